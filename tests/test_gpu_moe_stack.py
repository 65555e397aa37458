"""GPU parity of the MoE layer (Sec. 4) and the multi-layer stacks against the oracle.

MoE: routing (top-k with the lower index winning ties; a different pick is
excused only where the oracle's k-th and (k+1)-th logits are within NEAR_ZERO,
and y is then compared under the GPU's pick), routing weights, per-expert active
sets and y. Stacks: teacher-forced per layer (the GPU gets the oracle's
residual), graph replay against direct launches, and the full 32-layer
Mistral-shaped stack in the launch configuration the benchmark times.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2406_05955_gb300 import workload as wl

from _parity import NEAR_ZERO, check_sets, check_y, rel_l2

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ts():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    import paper_2406_05955_gb300 as ts

    ts.lib()
    return ts


def _moe_inputs(d, m, E, seed, act=0.20, dtype=torch.bfloat16):
    experts = [wl.ffn_layer(d, m, activation=act, dtype=dtype, seed=wl.layer_seed(seed, 0, e))
               for e in range(E)]
    wr = wl.router(E, d, dtype=dtype, seed=seed + 99)
    return experts, wr


def _check_routing(sel_gpu, w_gpu, ref, top_k):
    """Return the selection to compare y under, after checking it against the oracle."""
    sel = ref["sel"].copy()
    w = ref["w"].copy()
    for t in range(sel.shape[0]):
        if list(sel_gpu[t]) != list(ref["sel"][t]):
            lg = np.sort(ref["logits"][t])[::-1]
            assert lg[top_k - 1] - lg[top_k] < NEAR_ZERO, f"token {t}: routing differs without a near tie"
            sel[t] = sel_gpu[t]
            z = np.exp(ref["logits"][t, sel[t]] - ref["logits"][t, sel[t][0]])
            w[t] = z / z.sum()
        assert np.allclose(w_gpu[t], w[t], rtol=1e-5, atol=1e-6), f"token {t}: routing weights"
    return sel, w


@pytest.mark.parametrize("B", [1, 2, 5, 8])
@pytest.mark.parametrize("top_k", [1, 2])
def test_moe_layer_small(ts, B, top_k):
    d, m, E = 512, 1024, 8
    experts, wr = _moe_inputs(d, m, E, seed=100 + B)
    x = wl.tokens(B, d, dtype=torch.bfloat16, seed=B)
    dev = torch.device("cuda")
    ex = [ts.Ffn(L.w_gate.to(dev), L.w_up.to(dev), L.w_down.to(dev), max_batch=B) for L in experts]
    moe = ts.Moe(wr.to(dev), ex, top_k=top_k, max_batch=B)
    y = moe.forward(x.to(dev)).double().cpu().numpy()
    sel_g, w_g = moe.get_routing(B)
    triples = [(L.w_gate, L.w_up, L.w_down) for L in experts]
    ref0 = oracle.router(x, wr, top_k)
    sel, w = _check_routing(sel_g, w_g, ref0, top_k)
    ref = oracle.moe(x, wr, triples, top_k=top_k, sel=sel, w=w)
    check_y(y, ref["y"], "bf16")
    for e, per_tok in ref["expert_out"].items():
        for t, r in per_tok.items():
            one = {k: r[k][None] for k in ("g", "u", "gate_mask", "both_mask")}
            check_sets(*moe.get_active(e, t), one, 0)
    assert moe.get_error() == 0


@pytest.mark.parametrize("B", [1, 8])
def test_moe_layer_mixtral_size(ts, B):
    d, m, E = 4096, 14336, 8
    experts, wr = _moe_inputs(d, m, E, seed=300)
    x = wl.tokens(B, d, dtype=torch.bfloat16, seed=301)
    dev = torch.device("cuda")
    ex = [ts.Ffn(L.w_gate.to(dev), L.w_up.to(dev), L.w_down.to(dev), max_batch=B) for L in experts]
    moe = ts.Moe(wr.to(dev), ex, top_k=2, max_batch=B)
    y = moe.forward(x.to(dev)).double().cpu().numpy()
    sel_g, w_g = moe.get_routing(B)
    sel, w = _check_routing(sel_g, w_g, oracle.router(x, wr, 2), 2)
    ref = oracle.moe(x, wr, [(L.w_gate, L.w_up, L.w_down) for L in experts], top_k=2, sel=sel, w=w)
    check_y(y, ref["y"], "bf16")
    for e, per_tok in ref["expert_out"].items():
        t, r = next(iter(per_tok.items()))
        one = {k: r[k][None] for k in ("g", "u", "gate_mask", "both_mask")}
        check_sets(*moe.get_active(e, t), one, 0)
        frac = r["both_mask"].mean()
        assert 0.15 < frac < 0.25  # ~20% per expert


def test_moe_identical_experts_equal_single_ffn(ts):
    d, m, B = 1024, 2048, 4
    L = wl.ffn_layer(d, m, activation=0.20, dtype=torch.bfloat16, seed=7)
    dev = torch.device("cuda")
    wg, wu, wd = L.w_gate.to(dev), L.w_up.to(dev), L.w_down.to(dev)
    ex = [ts.Ffn(wg, wu, wd, max_batch=B) for _ in range(8)]
    moe = ts.Moe(wl.router(8, d, seed=8).to(dev), ex, top_k=2, max_batch=B)
    x = wl.tokens(B, d, seed=9).to(dev)
    y_moe = moe.forward(x).double().cpu().numpy()
    y_one = ex[0].forward(x).double().cpu().numpy()
    assert rel_l2(y_moe, y_one) <= 1e-5


@pytest.mark.parametrize("B", [1, 3, 16])
@pytest.mark.parametrize("predictor", [False, True])
def test_stack_teacher_forced(ts, B, predictor):
    d, m, n_layers = 1024, 3584, 4
    layers = [wl.ffn_layer(d, m, activation=0.10, dtype=torch.bfloat16, seed=wl.layer_seed(500, l))
              for l in range(n_layers)]
    lists = [wl.predictor_list(L.offsets, m // 10, seed=l) for l, L in enumerate(layers)] if predictor else None
    dev = torch.device("cuda")
    ffns = [ts.Ffn(L.w_gate.to(dev), L.w_up.to(dev), L.w_down.to(dev), max_batch=B) for L in layers]
    h0 = wl.residual(B, d, seed=501).numpy()
    h = h0
    for l, L in enumerate(layers):
        rows = None if lists is None else lists[l].numpy()
        x = oracle.rmsnorm(h, oracle.BF16)
        ref = oracle.ffn(x, L.w_gate, L.w_up, L.w_down, rows=rows)
        hg = torch.from_numpy(h.copy()).to(dev)
        idx = None if lists is None else [lists[l].to(dev)]
        ts.stack_forward([ffns[l]], hg, active_idx=idx)
        y_gpu = hg.double().cpu().numpy() - h.astype(np.float64)
        check_y(y_gpu, ref["y"], "bf16", f"layer {l}")
        for t in range(B):
            check_sets(*ffns[l].get_active(t), ref, t, rows=rows)
        h = (h.astype(np.float64) + ref["y"]).astype(np.float32)


@pytest.mark.parametrize("B", [2, 16])
def test_stack_graph_equals_direct(ts, B):
    d, m, n_layers = 1024, 3584, 3
    layers = [wl.ffn_layer(d, m, activation=0.10, dtype=torch.bfloat16, seed=wl.layer_seed(600, l))
              for l in range(n_layers)]
    dev = torch.device("cuda")
    ffns = [ts.Ffn(L.w_gate.to(dev), L.w_up.to(dev), L.w_down.to(dev), max_batch=B) for L in layers]
    h0 = wl.residual(B, d, seed=601).to(dev)
    h_direct = h0.clone()
    ts.stack_forward(ffns, h_direct)
    h_graph = h0.clone()
    g = ts.Graph.stack(ffns, h_graph)
    g.launch()
    torch.cuda.synchronize()
    assert torch.equal(h_direct, h_graph)
    h_graph.copy_(h0)
    g.launch()
    g.launch()
    ts.stack_forward(ffns, h_direct)
    torch.cuda.synchronize()
    assert torch.equal(h_direct, h_graph)


@pytest.mark.parametrize("B", [1, 8])
def test_moe_stack_teacher_forced(ts, B):
    d, m, E, n_layers = 1024, 2048, 8, 2
    dev = torch.device("cuda")
    moes, refs = [], []
    for l in range(n_layers):
        experts, wr = _moe_inputs(d, m, E, seed=wl.layer_seed(700, l))
        ex = [ts.Ffn(L.w_gate.to(dev), L.w_up.to(dev), L.w_down.to(dev), max_batch=B) for L in experts]
        moes.append(ts.Moe(wr.to(dev), ex, top_k=2, max_batch=B))
        refs.append((experts, wr))
    h = wl.residual(B, d, seed=701).numpy()
    for l in range(n_layers):
        experts, wr = refs[l]
        x = oracle.rmsnorm(h, oracle.BF16)
        hg = torch.from_numpy(h.copy()).to(dev)
        ts.moe_stack_forward([moes[l]], hg)
        sel, w = _check_routing(*moes[l].get_routing(B), oracle.router(x, wr, 2), 2)
        ref = oracle.moe(x, wr, [(L.w_gate, L.w_up, L.w_down) for L in experts], top_k=2, sel=sel, w=w)
        y_gpu = hg.double().cpu().numpy() - h.astype(np.float64)
        check_y(y_gpu, ref["y"], "bf16", f"layer {l}")
        h = (h.astype(np.float64) + ref["y"]).astype(np.float32)


def test_mistral_stack_32_layers_graph(ts):
    """The benchmark's workload and launch configuration: 32 layers in one graph, batch 1.

    The graph must give the same bits as direct launches; sampled layers are
    compared with the oracle teacher-forced (the GPU gets the oracle's residual
    at that layer), which is the parity gate for stacks. The free-running
    divergence over 32 layers is reported, not gated: each layer re-rounds the
    normalised activations to bf16, so a GPU/oracle difference within the
    per-layer tolerance can flip a rounding decision and a dReLU mask bit, and
    those flips propagate through every later layer; its size follows the
    input, not the kernels.
    """
    cfg = wl.WORKLOADS["mistral7b-ffn-stack-bf16-b1-act10"]
    d, m, n_layers = cfg["d"], cfg["m"], cfg["layers"]
    dev = torch.device("cuda")
    layers = [wl.ffn_layer(d, m, activation=cfg["activation"], dtype=torch.bfloat16,
                           seed=wl.layer_seed(cfg["seed"], l), device=dev) for l in range(n_layers)]
    ffns = [ts.Ffn(L.w_gate, L.w_up, L.w_down, max_batch=1) for L in layers]
    h0 = wl.residual(1, d, seed=cfg["seed"] - 1, device=dev)
    hg = h0.clone()
    g = ts.Graph.stack(ffns, hg)
    g.launch()
    hd = h0.clone()
    ts.stack_forward(ffns, hd)
    torch.cuda.synchronize()
    assert torch.equal(hg, hd), "graph replay and direct launches differ"
    assert all(f.get_error() == 0 for f in ffns)

    host = [(L.w_gate.cpu(), L.w_up.cpu(), L.w_down.cpu()) for L in layers]
    st = oracle.stack(h0.cpu().numpy(), host, record=True)
    for l in (0, 1, 15, 31):
        rec = st["layers"][l]
        ref = oracle.ffn(rec["x"], *host[l])
        hl = torch.from_numpy(rec["h_in"].copy()).to(dev)
        ts.stack_forward([ffns[l]], hl)
        y_gpu = hl.double().cpu().numpy() - rec["h_in"].astype(np.float64)
        check_y(y_gpu, ref["y"], "bf16", f"layer {l}")
        check_sets(*ffns[l].get_active(0), ref, 0)

    dy_gpu = hg.double().cpu().numpy() - h0.double().cpu().numpy()
    dy_ref = st["h"].astype(np.float64) - h0.double().cpu().numpy()
    err = rel_l2(dy_gpu, dy_ref)
    print(f"free-running 32-layer divergence of h_32 - h_0: rel L2 {err:.3e} (reported, not gated)")
    assert np.isfinite(err)
