"""Activation predictor (the reading of Sec. 7's per-layer predictor: a
two-layer ReLU MLP whose K best-scored neurons form the list) on the GPU,
through the C ABI (ts_predict, ts_stack_forward_predicted), against the fp64
oracle (oracle.predict).

Scores: fp32 accumulation over identical inputs, relative L2 <= TIGHT_REL of
the oracle's fp64 scores. Lists: exactly K strictly ascending ids in range;
the set equals the oracle's except near-ties at the cut -- neurons whose
oracle key is within CUT_REL * max|key| of the K-th largest oracle key (the
GPU ranks fp32 scores, the oracle fp64 ones). In stack mode the GPU also
normalises h itself, so the cut window is STACK_CUT_REL. The FFN that the
list drives is then checked with the predictor-mode tolerances over the GPU's
own list.
"""
import numpy as np
import pytest
import torch

from paper_2406_05955_gb300 import workload as wl

import oracle
from _parity import TIGHT_REL, check_sets, check_y, rel_l2

pytestmark = pytest.mark.gpu
CUT_REL = 1e-5
STACK_CUT_REL = 1e-4


@pytest.fixture(scope="module")
def ts():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    import paper_2406_05955_gb300 as ts

    ts.lib()
    return ts


def _check_list(got, ref_scores, K, cut_rel=CUT_REL):
    """Compare a GPU list with the oracle's top-K of max-over-tokens keys; return excused ids."""
    got = np.asarray(got, np.int64)
    m = ref_scores.shape[1]
    assert got.size == K, f"list has {got.size} ids, want {K}"
    if K == 0:
        return 0
    assert np.all(np.diff(got) > 0), "list not strictly ascending"
    assert got[0] >= 0 and got[-1] < m, "list id out of range"
    key = ref_scores.max(axis=0)
    order = np.lexsort((np.arange(m), -key))
    want = np.sort(order[:K])
    cut = key[order[K - 1]]
    near = np.abs(key - cut) <= cut_rel * max(float(np.max(np.abs(key))), 1e-30)
    diff = np.setxor1d(got, want)
    bad = diff[~near[diff]] if diff.size else diff
    assert bad.size == 0, f"list differs at {bad[:10]} (not near the cut {cut:.6g})"
    return int(diff.size)


def _inputs(d, r, m, B, dtype, seed, act=0.10):
    L = wl.ffn_layer(d, m, activation=act, dtype=dtype, seed=seed)
    P = wl.predictor_weights(d, r, m, L.offsets, dtype=dtype, seed=seed + 1)
    x = wl.tokens(B, d, dtype=dtype, seed=seed + 2)
    return L, P, x


@pytest.mark.parametrize("dtype,r", [(torch.bfloat16, 256), (torch.bfloat16, 512), (torch.bfloat16, 2048),
                                     (torch.float32, 128), (torch.float32, 512)])
@pytest.mark.parametrize("B", [1, 3, 8])
@pytest.mark.parametrize("K_frac", [0.0, 0.0003, 0.10, 0.5, 1.0])
def test_predict_matches_oracle(ts, dtype, r, B, K_frac):
    d, m = 1024, 3584
    L, P, x = _inputs(d, r, m, B, dtype, seed=1000 + r + B)
    K = int(round(K_frac * m))
    dev = torch.device("cuda")
    pred = ts.Predictor(P.w1.to(dev), P.w2.to(dev), max_batch=B)
    scores = torch.full((B, m), float("nan"), dtype=torch.float32, device=dev)
    lst = pred.predict(x.to(dev), K, scores=scores).cpu().numpy()
    ref = oracle.predict(x, P.w1, P.w2, K)
    if K > 0:
        err = rel_l2(scores.double().cpu().numpy(), ref["scores"])
        assert err <= TIGHT_REL, f"scores rel L2 {err:.3e}"
    _check_list(lst, ref["scores"], K)


# 16384 fills the single-CTA register select exactly (16 keys per thread);
# 16385 and 20000 take the radix select over keys in shared memory
@pytest.mark.parametrize("m,K", [(1, 1), (5, 3), (1000, 999), (4097, 410), (33, 32), (16384, 1638),
                                 (16385, 1639), (20000, 3000)])
def test_predict_ragged_sizes(ts, m, K):
    d, r, B = 256, 256, 2
    L, P, x = _inputs(d, r, m, B, torch.bfloat16, seed=1100 + m)
    dev = torch.device("cuda")
    pred = ts.Predictor(P.w1.to(dev), P.w2.to(dev), max_batch=B)
    lst = pred.predict(x.to(dev), K).cpu().numpy()
    _check_list(lst, oracle.predict(x, P.w1, P.w2, K)["scores"], K)


def test_predict_ties_go_to_the_lower_id(ts):
    """Duplicated W2 rows give exactly equal fp32 scores: the lower ids win."""
    d, r, m, B = 256, 256, 512, 1
    L, P, x = _inputs(d, r, m, B, torch.bfloat16, seed=1200)
    w2 = P.w2.clone()
    w2[256:] = w2[:256]  # neuron j + 256 ties with neuron j
    dev = torch.device("cuda")
    pred = ts.Predictor(P.w1.to(dev), w2.to(dev), max_batch=B)
    for K in (1, 7, 100, 255, 256, 257, 511):
        lst = pred.predict(x.to(dev), K).cpu().numpy()
        ref = oracle.predict(x, P.w1, w2, K)
        _check_list(lst, ref["scores"], K)
        # each tie pair (j, j+256) keeps j before j+256
        s = set(lst.tolist())
        assert all((j - 256) in s for j in s if j >= 256), f"K={K}: a higher twin kept without its lower one"


@pytest.mark.parametrize("m", [3584, 14336, 20000])
def test_predict_all_scores_equal(ts, m):
    """W2 = 0 makes every score exactly 0: all keys tie (one histogram bin holds
    them all), so the list is the K lowest ids."""
    d, r, B = 256, 256, 1
    L, P, x = _inputs(d, r, m, B, torch.bfloat16, seed=1250 + m)
    w2 = torch.zeros_like(P.w2)
    dev = torch.device("cuda")
    pred = ts.Predictor(P.w1.to(dev), w2.to(dev), max_batch=B)
    for K in (1, m // 10, m - 1, m):
        lst = pred.predict(x.to(dev), K).cpu().numpy()
        assert np.array_equal(lst, np.arange(K)), f"m={m} K={K}"


def test_predict_full_size_mistral(ts):
    """d=4096, m=14336, r=512, K=1434 (10%): the benchmark's predictor layer."""
    cfg = wl.WORKLOADS["mistral7b-ffn-stack-bf16-b1-prednet"]
    d, m, r, K = cfg["d"], cfg["m"], cfg["rank"], cfg["k"]
    L, P, x = _inputs(d, r, m, 1, torch.bfloat16, seed=1300)
    dev = torch.device("cuda")
    pred = ts.Predictor(P.w1.to(dev), P.w2.to(dev), max_batch=1)
    scores = torch.empty(1, m, dtype=torch.float32, device=dev)
    lst = pred.predict(x.to(dev), K, scores=scores)
    ref = oracle.predict(x, P.w1, P.w2, K)
    assert rel_l2(scores.double().cpu().numpy(), ref["scores"]) <= TIGHT_REL
    _check_list(lst.cpu().numpy(), ref["scores"], K)
    # the list drives the FFN's predictor mode
    ffn = ts.Ffn(L.w_gate.to(dev), L.w_up.to(dev), L.w_down.to(dev), max_batch=1)
    y = ffn.forward(x.to(dev), active_idx=lst).double().cpu().numpy()
    rows = lst.cpu().numpy()
    ref_y = oracle.ffn(x, L.w_gate, L.w_up, L.w_down, rows=rows)
    check_y(y, ref_y["y"], "bf16")
    check_sets(*ffn.get_active(0), ref_y, 0, rows=rows)


def test_predict_is_deterministic(ts):
    d, r, m, B = 1024, 512, 3584, 4
    L, P, x = _inputs(d, r, m, B, torch.bfloat16, seed=1400)
    dev = torch.device("cuda")
    pred = ts.Predictor(P.w1.to(dev), P.w2.to(dev), max_batch=B)
    s1 = torch.empty(B, m, dtype=torch.float32, device=dev)
    s2 = torch.empty_like(s1)
    a = pred.predict(x.to(dev), 358, scores=s1).clone()
    b = pred.predict(x.to(dev), 358, scores=s2).clone()
    assert torch.equal(a, b) and torch.equal(s1, s2)


@pytest.mark.parametrize("B", [1, 4])
def test_stack_predicted_teacher_forced(ts, B):
    d, m, r, n_layers = 1024, 3584, 256, 3
    K = m // 10
    dev = torch.device("cuda")
    layers = [wl.ffn_layer(d, m, activation=0.10, dtype=torch.bfloat16, seed=wl.layer_seed(1500, l))
              for l in range(n_layers)]
    preds = [wl.predictor_weights(d, r, m, L.offsets, dtype=torch.bfloat16, seed=wl.layer_seed(1550, l))
             for l, L in enumerate(layers)]
    ffns = [ts.Ffn(L.w_gate.to(dev), L.w_up.to(dev), L.w_down.to(dev), max_batch=B) for L in layers]
    gp = [ts.Predictor(P.w1.to(dev), P.w2.to(dev), max_batch=B) for P in preds]
    h = wl.residual(B, d, seed=1501).numpy()
    for l in range(n_layers):
        x = oracle.rmsnorm(h, oracle.BF16)
        hg = torch.from_numpy(h.copy()).to(dev)
        buf = torch.empty(K, dtype=torch.int32, device=dev)
        ts.stack_forward_predicted([ffns[l]], [gp[l]], hg, [K], [buf])
        rows = buf.cpu().numpy()
        _check_list(rows, oracle.predict(x, preds[l].w1, preds[l].w2, K)["scores"], K, STACK_CUT_REL)
        ref = oracle.ffn(x, layers[l].w_gate, layers[l].w_up, layers[l].w_down, rows=rows)
        y_gpu = hg.double().cpu().numpy() - h.astype(np.float64)
        check_y(y_gpu, ref["y"], "bf16", f"layer {l}")
        for t in range(B):
            check_sets(*ffns[l].get_active(t), ref, t, rows=rows)
        assert ffns[l].get_error() == 0
        h = (h.astype(np.float64) + ref["y"]).astype(np.float32)


def test_stack_predicted_graph_equals_direct_and_k_zero(ts):
    d, m, r, n_layers, B = 1024, 3584, 512, 3, 2
    Ks = [358, 0, 1000]
    dev = torch.device("cuda")
    layers = [wl.ffn_layer(d, m, activation=0.10, dtype=torch.bfloat16, seed=wl.layer_seed(1600, l))
              for l in range(n_layers)]
    ffns = [ts.Ffn(L.w_gate.to(dev), L.w_up.to(dev), L.w_down.to(dev), max_batch=B) for L in layers]
    gp = []
    for l, L in enumerate(layers):
        P = wl.predictor_weights(d, r, m, L.offsets, dtype=torch.bfloat16, seed=wl.layer_seed(1650, l))
        gp.append(ts.Predictor(P.w1.to(dev), P.w2.to(dev), max_batch=B))
    h0 = wl.residual(B, d, seed=1601).to(dev)
    bufs_d = [torch.empty(max(k, 1), dtype=torch.int32, device=dev) for k in Ks]
    bufs_g = [torch.empty(max(k, 1), dtype=torch.int32, device=dev) for k in Ks]
    hd = h0.clone()
    ts.stack_forward_predicted(ffns, gp, hd, Ks, bufs_d)
    hg = h0.clone()
    g = ts.Graph.stack_predicted(ffns, gp, hg, Ks, bufs_g)
    g.launch()
    torch.cuda.synchronize()
    assert torch.equal(hd, hg)
    for k, a, b in zip(Ks, bufs_d, bufs_g):
        assert torch.equal(a[:k], b[:k])
    # K = 0 on one layer: that layer adds nothing
    h1 = h0.clone()
    ts.stack_forward_predicted(ffns[1:2], gp[1:2], h1, [0], [bufs_d[1]])
    assert torch.equal(h1, h0)


def test_predict_rejects_bad_arguments(ts):
    from paper_2406_05955_gb300 import binding

    d, r, m = 256, 256, 100
    L, P, x = _inputs(d, r, m, 2, torch.bfloat16, seed=1700)
    dev = torch.device("cuda")
    pred = ts.Predictor(P.w1.to(dev), P.w2.to(dev), max_batch=2)
    for K in (-1, m + 1):
        with pytest.raises(binding.TsError):
            pred.predict(x.to(dev), K)
    x3 = wl.tokens(3, d, dtype=torch.bfloat16, seed=1701).to(dev)
    with pytest.raises(binding.TsError):
        pred.predict(x3, 10)  # batch above max_batch
    # hidden widths without a kernel, too large a batch
    bad_r = torch.zeros(300, d, dtype=torch.bfloat16, device=dev)
    with pytest.raises(binding.TsError) as e:
        ts.Predictor(bad_r, torch.zeros(m, 300, dtype=torch.bfloat16, device=dev))
    assert e.value.status == binding.TS_ERR_UNSUPPORTED
    with pytest.raises(binding.TsError) as e:
        ts.Predictor(P.w1.to(dev), P.w2.to(dev), max_batch=9)
    assert e.value.status == binding.TS_ERR_UNSUPPORTED
    # a predictor whose m does not match the layer
    ffn = ts.Ffn(L.w_gate.to(dev), L.w_up.to(dev), L.w_down.to(dev), max_batch=2)
    other = wl.predictor_weights(d, r, m + 8, torch.zeros(m + 8), dtype=torch.bfloat16, seed=1702)
    wrong = ts.Predictor(other.w1.to(dev), other.w2.to(dev), max_batch=2)
    h = wl.residual(2, d, seed=1703).to(dev)
    with pytest.raises(binding.TsError):
        ts.stack_forward_predicted([ffn], [wrong], h, [10], [torch.empty(10, dtype=torch.int32, device=dev)])
