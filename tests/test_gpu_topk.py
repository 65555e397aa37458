"""Top-k magnitude mask (Eq. 3 and Eq. 4) on the GPU, through the C ABI
(ts_ffn_forward_topk), against the fp64 oracle (oracle.ffn_topk).

Kept sets: per token the GPU's kept active neurons equal the oracle's kept
neurons with Combined > 0, except (a) neurons the dReLU masks themselves
excuse (pre-activation within NEAR_ZERO of 0, as for the plain FFN) and (b)
near-ties at the cut: neurons whose Combined is within CUT_REL of the keep-th
largest oracle value (the GPU ranks fp32 c values, the oracle fp64 ones); the
numbers of kept neurons must agree within the excused ones. y: the bf16 /
fp32 tolerances of the plain FFN.
"""
import numpy as np
import pytest
import torch

from paper_2406_05955_gb300 import workload as wl

import oracle
from _parity import NEAR_ZERO, check_y, rel_l2

pytestmark = pytest.mark.gpu
CUT_REL = 1e-5


@pytest.fixture(scope="module")
def ts():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    import paper_2406_05955_gb300 as ts

    ts.lib()
    return ts


def _check_kept(gpu_both, ref, t, keep):
    c = ref["c"][t]
    g, u = ref["g"][t], ref["u"][t]
    want = np.nonzero(ref["sel"][t] & (c > 0))[0]
    got = np.asarray(gpu_both, np.int64)
    assert np.all(np.diff(got) > 0), "kept list not strictly ascending"
    srt = np.sort(c)[::-1]
    cut = srt[keep - 1] if 0 < keep <= len(srt) else 0.0
    near_cut = np.abs(c - cut) <= CUT_REL * max(srt[0], 1e-30)
    near_zero = (np.abs(g) < NEAR_ZERO) | (np.abs(u) < NEAR_ZERO)
    diff = np.setxor1d(got, want)
    bad = diff[~(near_cut[diff] | near_zero[diff])] if diff.size else diff
    assert bad.size == 0, f"token {t}: kept set differs at {bad[:10]}"
    return int(diff.size)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("B", [1, 2, 3, 8, 11])  # 1-2: row kernel without its down partial; 3+: 4-8 token passes
@pytest.mark.parametrize("keep_frac", [0.0, 0.0003, 0.03, 0.10, 1.0])
def test_topk_matches_oracle(ts, dtype, B, keep_frac):
    d, m = 1024, 3584
    L = wl.ffn_layer(d, m, activation=0.25, dtype=dtype, seed=71 + B)
    x = wl.tokens(B, d, dtype=dtype, seed=72 + B)
    keep = int(round(keep_frac * m))
    dev = torch.device("cuda")
    ffn = ts.Ffn(L.w_gate.to(dev), L.w_up.to(dev), L.w_down.to(dev), max_batch=B)
    y = ffn.forward_topk(x.to(dev), keep).double().cpu().numpy()
    ref = oracle.ffn_topk(x, L.w_gate, L.w_up, L.w_down, keep)
    check_y(y, ref["y"], "bf16" if dtype == torch.bfloat16 else "f32")
    for t in range(B):
        _check_kept(ffn.get_active(t)[1], ref, t, keep)
    assert ffn.get_error() == 0


@pytest.mark.parametrize("B", [1, 2])
def test_topk_full_size_layer(ts, B):
    d, m = 4096, 14336
    L = wl.ffn_layer(d, m, activation=0.10, dtype=torch.bfloat16, seed=81)
    x = wl.tokens(B, d, dtype=torch.bfloat16, seed=82)
    keep = 717  # 5% of the neurons, half of the ~10% dReLU keeps
    dev = torch.device("cuda")
    ffn = ts.Ffn(L.w_gate.to(dev), L.w_up.to(dev), L.w_down.to(dev), max_batch=B)
    y = ffn.forward_topk(x.to(dev), keep).double().cpu().numpy()
    ref = oracle.ffn_topk(x, L.w_gate, L.w_up, L.w_down, keep)
    check_y(y, ref["y"], "bf16")
    for t in range(B):
        _check_kept(ffn.get_active(t)[1], ref, t, keep)
        assert len(ffn.get_active(t)[1]) <= keep


def test_topk_keep_all_equals_forward_and_is_deterministic(ts):
    d, m, B = 1024, 3584, 5
    L = wl.ffn_layer(d, m, activation=0.10, dtype=torch.bfloat16, seed=91)
    x = wl.tokens(B, d, dtype=torch.bfloat16, seed=92).cuda()
    ffn = ts.Ffn(L.w_gate.cuda(), L.w_up.cuda(), L.w_down.cuda(), max_batch=B)
    y_plain = ffn.forward(x).double().cpu().numpy()
    y_all = ffn.forward_topk(x, m)
    y_again = ffn.forward_topk(x, m)
    assert torch.equal(y_all, y_again)
    assert rel_l2(y_all.double().cpu().numpy(), y_plain) <= 1e-5
    y_none = ffn.forward_topk(x, 0)
    assert not torch.any(y_none)


def test_topk_rejects_bad_arguments(ts):
    from paper_2406_05955_gb300 import binding

    d, m = 256, 100
    L = wl.ffn_layer(d, m, activation=0.10, dtype=torch.bfloat16, seed=93)
    ffn = ts.Ffn(L.w_gate.cuda(), L.w_up.cuda(), L.w_down.cuda(), max_batch=2)
    x = wl.tokens(2, d, dtype=torch.bfloat16, seed=94).cuda()
    for keep in (-1, m + 1):
        with pytest.raises(binding.TsError):
            ffn.forward_topk(x, keep)
