"""Pins for the oracle's top-k magnitude mask (Eq. 3 and Eq. 4), against things
other than the oracle: a hand-worked layer with a tie, the two limits (keep all
= the plain dReLU FFN, keep none = 0), an independent numpy restatement on
random layers (library matmuls and a stable sort), and mistakes planted in a
CPU restatement (smallest instead of largest, ties to the higher index,
ranking by |gate| instead of |Combined|, one neuron too many), which the
hand-worked case rejects.
"""
import numpy as np
import pytest
import torch

from paper_2406_05955_gb300 import workload as wl

import oracle


def _f32(a):
    return np.ascontiguousarray(np.asarray(a, np.float32))


# x = e_0, so g_j = W_gate[j][0] and u_j = W_up[j][0]:
#   g = (2, -1, 1, 1), u = (1, 3, 5, 5)  ->  Combined = (2, 0, 5, 5)
# keep 1 -> {2} (the tie 2/3 goes to the lower index), keep 2 -> {2, 3},
# keep 3 -> {0, 2, 3}, keep 4 -> all (neuron 1 adds 0).
D, M = 4, 4
X = _f32([[1, 0, 0, 0]])
WG = _f32([[2, 0, 0, 0], [-1, 0, 0, 0], [1, 0, 0, 0], [1, 0, 0, 0]])
WU = _f32([[1, 0, 0, 0], [3, 0, 0, 0], [5, 0, 0, 0], [5, 0, 0, 0]])
WD = _f32([[1, 0, 0, 0], [0, 1, 0, 0], [0, 0, 1, 0], [0, 0, 0, 1]])
EXPECT = {0: [], 1: [2], 2: [2, 3], 3: [0, 2, 3], 4: [0, 1, 2, 3]}
C = np.array([2.0, 0.0, 5.0, 5.0])


@pytest.mark.parametrize("keep", sorted(EXPECT))
def test_topk_handworked(keep):
    r = oracle.ffn_topk(X, WG, WU, WD, keep)
    assert list(np.nonzero(r["sel"][0])[0]) == EXPECT[keep]
    y = np.zeros(D)
    for j in EXPECT[keep]:
        y += C[j] * WD[j].astype(np.float64)
    assert np.array_equal(r["y"][0], y)


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_topk_limits(dtype):
    L = wl.ffn_layer(128, 96, activation=0.25, dtype=dtype, seed=41)
    x = wl.tokens(3, 128, dtype=dtype, seed=42)
    full = oracle.ffn(x, L.w_gate, L.w_up, L.w_down)
    r = oracle.ffn_topk(x, L.w_gate, L.w_up, L.w_down, 96)
    assert r["sel"].all()
    assert np.array_equal(r["y"], full["y"])  # keep all: the plain FFN, same summation order
    z = oracle.ffn_topk(x, L.w_gate, L.w_up, L.w_down, 0)
    assert not z["sel"].any() and not z["y"].any()
    with pytest.raises(ValueError):
        oracle.ffn_topk(x, L.w_gate, L.w_up, L.w_down, 97)


def _numpy_topk(x, wg, wu, wd, keep):
    """Independent restatement: float64 matmuls, Combined, a stable sort."""
    g, u = x @ wg.T, x @ wu.T
    c = np.maximum(g, 0) * np.maximum(u, 0)
    sel = np.zeros_like(c, np.uint8)
    for b in range(c.shape[0]):
        order = np.argsort(-np.abs(c[b]), kind="stable")  # equal keys keep index order
        sel[b, order[:keep]] = 1
    return (c * sel) @ wd, sel, c


@pytest.mark.parametrize("keep", [0, 3, 17, 50])
def test_topk_random_against_numpy(keep):
    L = wl.ffn_layer(64, 50, activation=0.50, dtype=torch.float32, seed=43)
    x = wl.tokens(3, 64, dtype=torch.float32, seed=44)
    r = oracle.ffn_topk(x, L.w_gate, L.w_up, L.w_down, keep)
    xv, wg, wu, wd = (t.double().numpy() for t in (x, L.w_gate, L.w_up, L.w_down))
    y, sel, c = _numpy_topk(xv, wg, wu, wd, keep)
    # the draw has no near-tie at the cut among non-zero values
    for b in range(3):
        srt = np.sort(c[b])[::-1]
        if 0 < keep < 50 and srt[keep - 1] > 0:
            assert srt[keep - 1] - srt[keep] > 1e-9
    assert np.array_equal(r["sel"], sel)
    assert np.allclose(r["y"], y, rtol=1e-12, atol=1e-12)


def _planted(keep, mistake):
    g, u = WG[:, 0].astype(np.float64), WU[:, 0].astype(np.float64)
    c = np.maximum(g, 0) * np.maximum(u, 0)
    key = np.abs(g) if mistake == "rank_by_gate" else np.abs(c)
    idx = np.arange(M)
    if mistake == "smallest":
        order = np.lexsort((idx, key))
    elif mistake == "ties_to_higher":
        order = np.lexsort((-idx, -key))
    else:
        order = np.lexsort((idx, -key))
    k = keep + 1 if mistake == "one_too_many" else keep
    return sorted(order[:k].tolist())


@pytest.mark.parametrize("mistake", [None, "smallest", "ties_to_higher", "rank_by_gate", "one_too_many"])
def test_topk_pins_reject_planted_mistakes(mistake):
    agree = all(_planted(k, mistake) == EXPECT[k] for k in (1, 2, 3))
    assert agree == (mistake is None)
