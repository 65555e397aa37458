"""One-GPU emulation of the neuron-range split of the FFN across devices.

The FFN of Eq. 1 is a sum over neurons, so it splits by neuron range: device
p would own rows [m p / P, m (p+1) / P) of W_gate, W_up and W_down, compute a
partial y over its rows, and one all-reduce (a sum of batch x d fp32 values)
would complete the layer. Every box here has one GPU, so the split is
emulated: P handles on the row ranges of one layer, each run on the same
activations, their outputs summed on the host. The sum must equal the
single-handle forward and the fp64 oracle within the bf16 tolerance, and the
handles' active sets, shifted by their range offset, must partition the full
handle's sets.
"""
import numpy as np
import pytest
import torch

import oracle
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


@pytest.mark.parametrize("P,B,d,m", [(2, 1, 4096, 14336), (2, 4, 4096, 14336), (4, 2, 1024, 3001),
                                     (3, 16, 1024, 2048)])
def test_neuron_range_split_sums_to_the_full_forward(ts, P, B, d, m):
    dev = torch.device("cuda")
    L = wl.ffn_layer(d, m, activation=0.10, dtype=torch.bfloat16, seed=97 + P + B, device=dev)
    x = wl.tokens(B, d, dtype=torch.bfloat16, seed=98 + B, device=dev)
    full = ts.Ffn(L.w_gate, L.w_up, L.w_down, max_batch=B)
    y_full = full.forward(x).double().cpu().numpy()
    g_full, b_full = full.get_active(-1)

    y_sum = np.zeros((B, d), np.float64)
    g_parts, b_parts = [], []
    bounds = [m * p // P for p in range(P + 1)]
    for p in range(P):
        r0, r1 = bounds[p], bounds[p + 1]
        shard = ts.Ffn(L.w_gate[r0:r1].contiguous(), L.w_up[r0:r1].contiguous(), L.w_down[r0:r1].contiguous(),
                       max_batch=B)
        y_sum += shard.forward(x).double().cpu().numpy()  # the all-reduce, on the host
        g, b = shard.get_active(-1)
        g_parts.append(np.asarray(g, np.int64) + r0)
        b_parts.append(np.asarray(b, np.int64) + r0)
        assert shard.get_error() == 0
        shard.close()

    # the shards' active sets partition the full handle's (same fp32 dot products per row)
    np.testing.assert_array_equal(np.concatenate(g_parts), np.asarray(g_full, np.int64))
    np.testing.assert_array_equal(np.concatenate(b_parts), np.asarray(b_full, np.int64))
    # the summed partials equal the full forward up to fp32 summation order
    assert rel_l2(y_sum, y_full) <= 1e-5
    ref = oracle.ffn(x.cpu(), L.w_gate.cpu(), L.w_up.cpu(), L.w_down.cpu())
    check_y(y_sum, ref["y"], "bf16", f"{P} shards")
    full.close()
