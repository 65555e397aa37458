"""The C-ABI library loads without a GPU, exports every symbol include/ts_ffn.h
declares, and rejects bad arguments before touching the device."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "ts_ffn.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2406_05955_gb300 import binding, build

    build.build()
    return binding.lib()


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(ts_[a-z_0-9]+)\s*\(", text)))


def test_header_symbols_exported(lib):
    from paper_2406_05955_gb300 import binding

    names = _declared()
    assert len(names) >= 20
    raw = ctypes.CDLL(binding.LIB_PATH)
    for n in names:
        assert hasattr(raw, n), f"{n} declared in ts_ffn.h but not exported"
    assert set(names) == set(binding.SIGNATURES), "binding signatures and header disagree"


def test_debug_library_exports_the_same_symbols(lib):
    from paper_2406_05955_gb300 import build

    assert os.path.exists(build.DEBUG_LIB), "build() also makes the range-checked debug library"
    raw = ctypes.CDLL(build.DEBUG_LIB)
    for n in _declared():
        assert hasattr(raw, n), f"{n} not exported by the debug library"


def test_scratch_checks_reject_null_handles(lib):
    from paper_2406_05955_gb300.binding import TS_ERR_INVALID_ARG

    assert lib.ts_ffn_check_scratch(None, None) == TS_ERR_INVALID_ARG
    assert lib.ts_moe_check_scratch(None, None) == TS_ERR_INVALID_ARG
    assert lib.ts_predictor_check_scratch(None, None) == TS_ERR_INVALID_ARG
    assert lib.ts_ffn_poke_guard(None, 0) == TS_ERR_INVALID_ARG


def test_status_strings_and_version(lib):
    from paper_2406_05955_gb300 import binding

    names = [binding.status_str(s) for s in range(8)]
    assert names == ["TS_OK", "TS_ERR_INVALID_ARG", "TS_ERR_CUDA", "TS_ERR_OOM", "TS_ERR_BAD_INDEX",
                     "TS_ERR_TIMEOUT", "TS_ERR_UNSUPPORTED", "TS_ERR_SCRATCH"]
    assert binding.status_str(99) == "TS_ERR_UNKNOWN"
    assert lib.ts_version() >= 100


def test_argument_validation_without_device(lib):
    from paper_2406_05955_gb300.binding import TS_BF16, TS_ERR_INVALID_ARG, TS_F32

    h = ctypes.c_void_p()
    good = 0x10000
    assert lib.ts_ffn_create(None, 64, 32, TS_BF16, good, good, good, 1) == TS_ERR_INVALID_ARG
    assert lib.ts_ffn_create(ctypes.byref(h), 0, 32, TS_BF16, good, good, good, 1) == TS_ERR_INVALID_ARG
    assert lib.ts_ffn_create(ctypes.byref(h), 64, 0, TS_BF16, good, good, good, 1) == TS_ERR_INVALID_ARG
    assert lib.ts_ffn_create(ctypes.byref(h), 64, 32, 7, good, good, good, 1) == TS_ERR_INVALID_ARG
    assert lib.ts_ffn_create(ctypes.byref(h), 64, 32, TS_BF16, None, good, good, 1) == TS_ERR_INVALID_ARG
    assert lib.ts_ffn_create(ctypes.byref(h), 64, 32, TS_BF16, good + 2, good, good, 1) == TS_ERR_INVALID_ARG
    assert lib.ts_ffn_create(ctypes.byref(h), 12, 32, TS_BF16, good, good, good, 1) == TS_ERR_INVALID_ARG
    assert lib.ts_ffn_create(ctypes.byref(h), 6, 32, TS_F32, good, good, good, 1) == TS_ERR_INVALID_ARG
    assert lib.ts_ffn_create(ctypes.byref(h), 64, 32, TS_BF16, good, good, good, 0) == TS_ERR_INVALID_ARG
    assert lib.ts_ffn_create(ctypes.byref(h), 64, 32, TS_BF16, good, good, good, 65) == TS_ERR_INVALID_ARG
    assert h.value is None
    assert lib.ts_ffn_forward(None, good, 1, good, None, None, 0) == TS_ERR_INVALID_ARG
    assert lib.ts_ffn_gate_up(None, good, 1, None, None, 0) == TS_ERR_INVALID_ARG
    assert lib.ts_ffn_down(None, 1, good, None) == TS_ERR_INVALID_ARG
    assert lib.ts_stack_forward(None, 1, good, 1, None, None, None) == TS_ERR_INVALID_ARG
    assert lib.ts_ffn_get_active(None, None, 0, None, None, None, None) == TS_ERR_INVALID_ARG
    assert lib.ts_ffn_get_error(None, None) == TS_ERR_INVALID_ARG
    assert lib.ts_moe_create(None, 64, 8, 2, TS_BF16, good, good, 1) == TS_ERR_INVALID_ARG
    assert lib.ts_moe_create(ctypes.byref(h), 64, 8, 5, TS_BF16, good, good, 1) == TS_ERR_INVALID_ARG
    assert lib.ts_moe_create(ctypes.byref(h), 64, 17, 2, TS_BF16, good, good, 1) == TS_ERR_INVALID_ARG
    assert lib.ts_moe_create(ctypes.byref(h), 64, 8, 2, TS_BF16, good, good, 9) == TS_ERR_INVALID_ARG
    assert lib.ts_moe_forward(None, good, 1, good, None) == TS_ERR_INVALID_ARG
    assert lib.ts_moe_stack_forward(None, 1, good, 1, None) == TS_ERR_INVALID_ARG
    assert lib.ts_moe_get_routing(None, None, None, None) == TS_ERR_INVALID_ARG
    assert lib.ts_moe_get_active(None, None, 0, 0, None, None, None, None) == TS_ERR_INVALID_ARG
    assert lib.ts_moe_get_error(None, None) == TS_ERR_INVALID_ARG
    assert lib.ts_graph_launch(None, None) == TS_ERR_INVALID_ARG
    assert lib.ts_graph_capture_stack(None, None, 0, None, 0, None, None) == TS_ERR_INVALID_ARG
    assert lib.ts_graph_capture_stack_fused(None, None, 0, None, 0, None, None) == TS_ERR_INVALID_ARG
    lib.ts_ffn_destroy(None)
    lib.ts_moe_destroy(None)
    lib.ts_graph_destroy(None)


def test_binding_refuses_cpu_tensors():
    """The product path has no CPU fallback: CPU tensors are an error."""
    import torch

    import paper_2406_05955_gb300 as ts

    w = torch.zeros(8, 64, dtype=torch.bfloat16)
    with pytest.raises(TypeError):
        ts.Ffn(w, w, w)


def test_debug_environment_selects_the_debug_library(lib):
    """TS_FFN_DEBUG=1 makes the binding load libtsffn_debug.so (checked in a child process)."""
    import subprocess
    import sys

    code = ("import sys; sys.path.insert(0, %r); from paper_2406_05955_gb300 import binding; "
            "binding.lib(); print(binding.LIB_PATH)") % ROOT
    env = dict(os.environ, TS_FFN_DEBUG="1")
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    assert r.stdout.strip().endswith(os.path.join("debug", "libtsffn_debug.so"))
