"""GPU parity of the INT4 weight path (4-bit codes + binary16 group scales, the
storage of the paper's INT4 models, Tables 7-9) against the fp64 oracle, which
decodes the same rows exactly. Activations are bf16; batches run in passes of
up to two tokens on the tensor-core gate+up kernel."""
import numpy as np
import pytest
import torch

import oracle
from paper_2406_05955_gb300 import workload as wl

from _parity import check_sets, check_y, rel_l2

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ts():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    import paper_2406_05955_gb300 as ts

    ts.lib()
    return ts


def _ffn(ts, L, max_batch):
    dev = torch.device("cuda")
    return ts.Ffn(L.w_gate.to(dev), L.w_up.to(dev), L.w_down.to(dev), max_batch=max_batch)


@pytest.mark.parametrize("d,m,B,act", [
    (4096, 14336, 1, 0.10),   # a Mistral-shaped layer, one token
    (4096, 14336, 2, 0.10),   # two tokens in one pass
    (256, 1001, 3, 0.25),     # ragged chunks, a pass of 2 then 1
    (512, 2048, 5, 1.0),      # all active, three passes
])
def test_int4_layer(ts, d, m, B, act):
    L = wl.ffn_layer_int4(d, m, activation=act, seed=8800 + m + B)
    x = wl.tokens(B, d, seed=8801)
    f = _ffn(ts, L, B)
    y = f.forward(x.cuda()).double().cpu().numpy()
    ref = oracle.ffn(x, L.w_gate, L.w_up, L.w_down)
    check_y(y, ref["y"], "bf16")
    for t in range(B):
        check_sets(*f.get_active(t), ref, t)
    assert f.get_error() == 0


@pytest.mark.parametrize("list_len", [0, 700, 14336])
def test_int4_predictor_lists(ts, list_len):
    d, m = 4096, 14336
    L = wl.ffn_layer_int4(d, m, activation=0.10, seed=8810)
    rows = wl.predictor_list(L.offsets, list_len, seed=8811).numpy()
    x = wl.tokens(1, d, seed=8812)
    f = _ffn(ts, L, 1)
    idx = torch.as_tensor(rows).cuda()  # borrowed by the handle until get_active
    y = f.forward(x.cuda(), active_idx=idx).double().cpu().numpy()
    ref = oracle.ffn(x, L.w_gate, L.w_up, L.w_down, rows=rows)
    check_y(y, ref["y"], "bf16")
    check_sets(*f.get_active(0), ref, 0, rows=rows)


def test_int4_stack_teacher_forced_and_graph(ts):
    d, m, n_layers = 1024, 3584, 3
    layers = [wl.ffn_layer_int4(d, m, activation=0.10, seed=wl.layer_seed(8820, l)) for l in range(n_layers)]
    ffns = [_ffn(ts, L, 1) for L in layers]
    h = wl.residual(1, d, seed=8821).numpy()
    for l, L in enumerate(layers):
        x = oracle.rmsnorm(h, oracle.BF16)
        ref = oracle.ffn(x, L.w_gate, L.w_up, L.w_down)
        hg = torch.from_numpy(h.copy()).cuda()
        ts.stack_forward([ffns[l]], hg)
        check_y(hg.double().cpu().numpy() - h.astype(np.float64), ref["y"], "bf16", f"layer {l}")
        check_sets(*ffns[l].get_active(0), ref, 0)
        h = (h.astype(np.float64) + ref["y"]).astype(np.float32)
    h0 = wl.residual(1, d, seed=8822).cuda()
    hd, hgr = h0.clone(), h0.clone()
    ts.stack_forward(ffns, hd)
    g = ts.Graph.stack(ffns, hgr)
    g.launch()
    torch.cuda.synchronize()
    assert torch.equal(hd, hgr)


@pytest.mark.parametrize("B", [1, 2])
def test_int4_moe(ts, B):
    d, m, E = 512, 1024, 8
    experts = [wl.ffn_layer_int4(d, m, activation=0.20, seed=wl.layer_seed(8830, 0, e)) for e in range(E)]
    wr = wl.router(E, d, seed=8831)
    x = wl.tokens(B, d, seed=8832)
    dev = torch.device("cuda")
    ex = [_ffn(ts, L, B) for L in experts]
    moe = ts.Moe(wr.to(dev), ex, top_k=2, max_batch=B)
    y = moe.forward(x.to(dev)).double().cpu().numpy()
    sel, w = moe.get_routing(B)
    ref0 = oracle.router(x, wr, 2)
    assert np.array_equal(sel, ref0["sel"])
    ref = oracle.moe(x, wr, [(L.w_gate, L.w_up, L.w_down) for L in experts], top_k=2, sel=sel, w=w)
    check_y(y, ref["y"], "bf16")


def test_int4_deterministic(ts):
    L = wl.ffn_layer_int4(4096, 14336, activation=0.10, seed=8840)
    f = _ffn(ts, L, 2)
    x = wl.tokens(2, 4096, seed=8841).cuda()
    first = f.forward(x).clone()
    for _ in range(3):
        assert torch.equal(f.forward(x), first)
    assert rel_l2(first.double().cpu().numpy(), first.double().cpu().numpy()) == 0.0
