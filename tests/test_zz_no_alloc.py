"""ts_ffn_forward_noalloc (no handle, static device scratch) through the C ABI.

It must give what ts_ffn_forward gives on the same inputs, on two calls in a
row (the second reuses the scratch the first left behind), in detected and
predictor-list mode, and at the size limits; sizes above the limits are
refused without launching anything. The file sorts last so that the entry
point also runs after every other GPU test in the same process.
"""
import numpy as np
import pytest
import torch

from paper_2406_05955_gb300 import workload as wl

from _parity import check_y, rel_l2

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ts():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    import paper_2406_05955_gb300 as ts

    ts.lib()
    return ts


def _layer(d, m, act, seed, dtype=torch.bfloat16):
    L = wl.ffn_layer(d, m, activation=act, dtype=dtype, seed=seed, device=torch.device("cuda"))
    return L.w_gate, L.w_up, L.w_down


@pytest.mark.parametrize("d,m,B,act,dtype", [
    (4096, 14336, 1, 0.10, torch.bfloat16),   # one Mistral-7B-shaped layer, one token
    (1024, 3584, 5, 0.20, torch.bfloat16),    # ragged batch
    (512, 1408, 12, 0.25, torch.float32),     # two passes of the token loop
    (1024, 16384, 64, 0.10, torch.bfloat16),  # both size limits
])
def test_noalloc_matches_handle_forward(ts, d, m, B, act, dtype):
    from paper_2406_05955_gb300 import binding

    wg, wu, wd = _layer(d, m, act, seed=900 + B, dtype=dtype)
    ffn = ts.Ffn(wg, wu, wd, max_batch=B)
    dt = "bf16" if dtype == torch.bfloat16 else "f32"
    for call in range(2):
        x = wl.tokens(B, d, dtype=dtype, seed=910 + 7 * call + B).cuda()
        y_ref = ffn.forward(x).double().cpu().numpy()
        y = torch.full((B, d), float("nan"), dtype=torch.float32, device="cuda")
        binding.ffn_forward_noalloc(wg, wu, wd, x, y)
        y = y.double().cpu().numpy()
        assert np.isfinite(y).all(), f"call {call}: output not fully written"
        check_y(y, y_ref, dt, f"call {call}")
        assert rel_l2(y, y_ref) <= 1e-5, f"call {call}"
    assert ffn.get_error() == 0


def test_noalloc_predictor_list(ts):
    from paper_2406_05955_gb300 import binding

    d, m, B = 4096, 14336, 3
    L = wl.ffn_layer(d, m, activation=0.10, dtype=torch.bfloat16, seed=950, device=torch.device("cuda"))
    lst = wl.predictor_list(L.offsets.cpu(), 1434, seed=951).cuda()
    ffn = ts.Ffn(L.w_gate, L.w_up, L.w_down, max_batch=B)
    for call in range(2):
        x = wl.tokens(B, d, seed=952 + call).cuda()
        y_ref = ffn.forward(x, active_idx=lst).double().cpu().numpy()
        y = torch.empty(B, d, dtype=torch.float32, device="cuda")
        binding.ffn_forward_noalloc(L.w_gate, L.w_up, L.w_down, x, y, active_idx=lst)
        check_y(y.double().cpu().numpy(), y_ref, "bf16", f"call {call}")


def test_noalloc_refuses_sizes_above_limits(ts):
    from paper_2406_05955_gb300 import binding

    lib = binding.lib()
    dev = torch.device("cuda")
    d = 512
    m = 16385
    w = torch.zeros(m, d, dtype=torch.bfloat16, device=dev)
    x = torch.zeros(65, d, dtype=torch.bfloat16, device=dev)
    y = torch.zeros(65, d, dtype=torch.float32, device=dev)
    s = torch.cuda.current_stream().cuda_stream
    args = (binding.TS_BF16, w.data_ptr(), w.data_ptr(), w.data_ptr(), x.data_ptr())
    assert lib.ts_ffn_forward_noalloc(d, m, *args, 1, y.data_ptr(), s, None, 0) == binding.TS_ERR_UNSUPPORTED
    assert lib.ts_ffn_forward_noalloc(d, 1024, *args, 65, y.data_ptr(), s, None, 0) == binding.TS_ERR_UNSUPPORTED
    assert lib.ts_ffn_forward_noalloc(d, 1024, *args, -1, y.data_ptr(), s, None, 0) == binding.TS_ERR_INVALID_ARG
    assert lib.ts_ffn_forward_noalloc(d, 1024, *args, 0, y.data_ptr(), s, None, 0) == binding.TS_OK
    torch.cuda.synchronize()
    assert not y.any(), "a refused call wrote its output"
