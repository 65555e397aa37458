"""The debug build (-DTS_DEBUG: every gathered row index is range-checked
into the status word before the gather) must compute bit for bit what the
release build computes and record no error, on the kernel families of the
decode path. The debug library runs in a child process (TS_FFN_DEBUG=1), the
release library here, on the same seeded inputs."""
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

from paper_2406_05955_gb300 import workload as wl

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

# (d, m, batch, activation, list length or 0): batch-1/2 rows kernel, a
# predictor list, the 8-token tensor-core pass, the wide tcgen05 path
CASES = [(4096, 14336, 1, 0.10, 0), (4096, 14336, 2, 0.10, 1434), (512, 2048, 8, 0.25, 0),
         (1024, 2048, 32, 0.10, 0)]

CHILD = r"""
import sys, numpy as np, torch
sys.path.insert(0, {root!r})
import paper_2406_05955_gb300 as ts
from paper_2406_05955_gb300 import binding, workload as wl
assert binding.LIB_PATH.endswith("libtsffn_debug.so"), binding.LIB_PATH
out = {{}}
for i, (d, m, B, act, nl) in enumerate({cases!r}):
    L = wl.ffn_layer(d, m, activation=act, dtype=torch.bfloat16, seed=9200 + i)
    f = ts.Ffn(L.w_gate.cuda(), L.w_up.cuda(), L.w_down.cuda(), max_batch=B)
    idx = wl.predictor_list(L.offsets, nl, seed=9300 + i).cuda() if nl else None
    y = f.forward(wl.tokens(B, d, seed=9400 + i).cuda(), active_idx=idx)
    assert f.get_error() == 0, f"case {{i}}: status {{f.get_error()}}"
    out[f"y{{i}}"] = y.cpu().numpy()
np.savez({path!r}, **out)
"""


def test_debug_build_matches_release(tmp_path):
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    import paper_2406_05955_gb300 as ts
    from paper_2406_05955_gb300 import build as b

    b.build()
    assert os.path.exists(b.DEBUG_LIB), "the debug library was not built"
    path = str(tmp_path / "debug_out.npz")
    env = dict(os.environ, TS_FFN_DEBUG="1")
    r = subprocess.run([sys.executable, "-c", CHILD.format(root=ROOT, cases=CASES, path=path)], env=env,
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    got = np.load(path)
    for i, (d, m, B, act, nl) in enumerate(CASES):
        L = wl.ffn_layer(d, m, activation=act, dtype=torch.bfloat16, seed=9200 + i)
        f = ts.Ffn(L.w_gate.cuda(), L.w_up.cuda(), L.w_down.cuda(), max_batch=B)
        idx = wl.predictor_list(L.offsets, nl, seed=9300 + i).cuda() if nl else None
        y = f.forward(wl.tokens(B, d, seed=9400 + i).cuda(), active_idx=idx).cpu().numpy()
        assert f.get_error() == 0
        assert np.array_equal(got[f"y{i}"], y), f"case {i}: debug and release outputs differ"
