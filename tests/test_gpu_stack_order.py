"""A stack's layers overlap on the GPU (each reduction lets the next layer's
first kernel be scheduled before its own dependency wait, and that kernel
starts its weight copies early): the whole-stack call and its graph must
give bit for bit what the same layers give called one at a time, for the
batch-1/2 bf16 stacks, predictor lists, the predicted stack's kernels, and
INT4 stacks whose batch runs in several passes of two tokens on one handle."""
import pytest
import torch

from paper_2406_05955_gb300 import workload as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ts():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    import paper_2406_05955_gb300 as ts

    ts.lib()
    return ts


def _layers(ts, d, m, n, B, int4, seed):
    out = []
    for l in range(n):
        if int4:
            L = wl.ffn_layer_int4(d, m, activation=0.10, seed=wl.layer_seed(seed, l))
        else:
            L = wl.ffn_layer(d, m, activation=0.10, dtype=torch.bfloat16, seed=wl.layer_seed(seed, l))
        out.append((L, ts.Ffn(L.w_gate.cuda(), L.w_up.cuda(), L.w_down.cuda(), max_batch=B)))
    return out


@pytest.mark.parametrize("B,int4,lists", [(1, False, False), (2, False, False), (1, False, True),
                                          (1, True, False), (5, True, False)])
def test_stack_equals_layer_by_layer(ts, B, int4, lists):
    d, m, n = 1024, 3584, 4
    layers = _layers(ts, d, m, n, B, int4, seed=9500 + B + 10 * int4)
    ffns = [f for _, f in layers]
    idx = [wl.predictor_list(L.offsets, 400, seed=9600 + l).cuda() for l, (L, _) in enumerate(layers)] \
        if lists else None
    h0 = wl.residual(B, d, seed=9501).cuda()
    h_one = h0.clone()
    for l in range(n):
        ts.stack_forward([ffns[l]], h_one, active_idx=None if idx is None else [idx[l]])
    h_all = h0.clone()
    ts.stack_forward(ffns, h_all, active_idx=idx)
    h_graph = h0.clone()
    g = ts.Graph.stack(ffns, h_graph, active_idx=idx)
    g.launch()
    torch.cuda.synchronize()
    assert torch.equal(h_all, h_one), "whole stack differs from the layers called one at a time"
    assert torch.equal(h_graph, h_one), "the stack's graph differs from the layers called one at a time"
    for f in ffns:
        assert f.get_error() == 0


def test_predicted_stack_equals_layer_by_layer(ts):
    d, m, n, r, K = 1024, 3584, 3, 256, 358
    layers = _layers(ts, d, m, n, 1, False, seed=9700)
    ffns = [f for _, f in layers]
    preds = []
    for l, (L, _) in enumerate(layers):
        P = wl.predictor_weights(d, r, m, L.offsets, seed=9710 + l)
        preds.append(ts.Predictor(P.w1.cuda(), P.w2.cuda(), max_batch=1))
    h0 = wl.residual(1, d, seed=9701).cuda()
    bufs = [torch.empty(K, dtype=torch.int32, device="cuda") for _ in range(n)]
    h_one = h0.clone()
    for l in range(n):
        ts.stack_forward_predicted([ffns[l]], [preds[l]], h_one, [K], [bufs[l]])
    lists_one = [b.clone() for b in bufs]
    h_all = h0.clone()
    ts.stack_forward_predicted(ffns, preds, h_all, [K] * n, bufs)
    torch.cuda.synchronize()
    assert torch.equal(h_all, h_one)
    for l in range(n):
        assert torch.equal(bufs[l], lists_one[l]), f"layer {l}: predicted lists differ"
