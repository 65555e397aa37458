"""The fused layer stack (one persistent cooperative launch per decode step).

Its per-layer work is the unfused stack's code and its reduction adds the
partial down projections in the unfused reduction's order, so a fused replay
must give the unfused graph's bits exactly. Single-layer fused graphs are
compared with the fp64 oracle teacher-forced (the stack's parity gate), the
multi-layer graphs with the unfused graph bit for bit, in detected and
predictor-list mode, at batch 1 and 2.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2406_05955_gb300 import workload as wl

from _parity import check_y

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ts():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    import paper_2406_05955_gb300 as ts

    ts.lib()
    return ts


def _layers(d, m, n, seed, dev, act=0.10):
    return [wl.ffn_layer(d, m, activation=act, dtype=torch.bfloat16, seed=wl.layer_seed(seed, l), device=dev)
            for l in range(n)]


@pytest.mark.parametrize("B,d,m,n_layers,lists", [(1, 4096, 14336, 32, False), (2, 4096, 14336, 4, False),
                                                  (1, 1024, 3001, 5, False), (1, 4096, 14336, 8, True),
                                                  (2, 512, 1408, 3, True)])
def test_fused_stack_equals_unfused_bitwise(ts, B, d, m, n_layers, lists):
    dev = torch.device("cuda")
    layers = _layers(d, m, n_layers, 4242 + d + B, dev)
    ffns = [ts.Ffn(L.w_gate, L.w_up, L.w_down, max_batch=B) for L in layers]
    idx = None
    if lists:
        idx = [wl.predictor_list(L.offsets, m // 10, seed=l + 5).to(dev) for l, L in enumerate(layers)]
    h0 = wl.residual(B, d, seed=77 + B, device=dev)
    h_unf, h_fus = h0.clone(), h0.clone()
    g_unf = ts.Graph.stack(ffns, h_unf, active_idx=idx)
    g_fus = ts.Graph.stack_fused(ffns, h_fus, active_idx=idx)
    for rep in range(3):
        h_unf.copy_(h0)
        h_fus.copy_(h0)
        g_unf.launch()
        torch.cuda.synchronize()
        sets_unf = [f.get_active(-1) for f in ffns]
        g_fus.launch()
        torch.cuda.synchronize()
        assert torch.equal(h_unf, h_fus), f"replay {rep}: fused and unfused stacks differ"
        for l, f in enumerate(ffns):
            g, b = f.get_active(-1)
            np.testing.assert_array_equal(g, sets_unf[l][0])
            np.testing.assert_array_equal(b, sets_unf[l][1])
    assert all(f.get_error() == 0 for f in ffns)
    g_unf.close()
    g_fus.close()


@pytest.mark.parametrize("B", [1, 2])
def test_fused_single_layer_matches_oracle(ts, B):
    """Teacher-forced: every sampled layer as a one-layer fused graph on the
    oracle's residual, its output against the oracle's FFN of rmsnorm(h)."""
    d, m = 4096, 14336
    dev = torch.device("cuda")
    for l in (0, 7):
        L = wl.ffn_layer(d, m, activation=0.10, dtype=torch.bfloat16, seed=wl.layer_seed(900, l), device=dev)
        f = ts.Ffn(L.w_gate, L.w_up, L.w_down, max_batch=B)
        h_in = wl.residual(B, d, seed=901 + l, device=dev)
        h = h_in.clone()
        g = ts.Graph.stack_fused([f], h)
        g.launch()
        torch.cuda.synchronize()
        x = oracle.rmsnorm(h_in.cpu().numpy(), oracle.BF16)
        ref = oracle.ffn(x, L.w_gate.cpu(), L.w_up.cpu(), L.w_down.cpu())
        y_gpu = h.double().cpu().numpy() - h_in.double().cpu().numpy()
        check_y(y_gpu, ref["y"], "bf16", f"layer {l}")
        gs, bs = f.get_active(-1)
        want_b = np.nonzero(ref["both_mask"].any(axis=0))[0]
        near = (np.abs(ref["g"]).min(axis=0) < 1e-4) | (np.abs(ref["u"]).min(axis=0) < 1e-4)
        diff = np.setxor1d(bs, want_b)
        assert near[diff].all(), f"layer {l}: union both set differs at {diff[~near[diff]][:10]}"
        assert f.get_error() == 0
        g.close()


def test_fused_stack_replays_are_deterministic_and_time_out_free(ts):
    d, m, n_layers = 2048, 8192, 6
    dev = torch.device("cuda")
    layers = _layers(d, m, n_layers, 31, dev)
    ffns = [ts.Ffn(L.w_gate, L.w_up, L.w_down, max_batch=1) for L in layers]
    h0 = wl.residual(1, d, seed=3, device=dev)
    h = h0.clone()
    g = ts.Graph.stack_fused(ffns, h)
    outs = []
    for _ in range(4):
        h.copy_(h0)
        g.launch()
        torch.cuda.synchronize()
        outs.append(h.clone())
    assert all(torch.equal(outs[0], o) for o in outs[1:])
    assert all(f.get_error() == 0 for f in ffns)
    g.close()


def test_fused_stack_unsupported_cases(ts):
    dev = torch.device("cuda")
    L = wl.ffn_layer(512, 1408, activation=0.10, dtype=torch.float32, seed=1, device=dev)
    f32 = ts.Ffn(L.w_gate, L.w_up, L.w_down, max_batch=4)
    h = torch.zeros(1, 512, device=dev)
    with pytest.raises(ts.TsError) as e:
        ts.Graph.stack_fused([f32], h)
    assert e.value.status == 6  # TS_ERR_UNSUPPORTED: fp32 rows
    Lb = wl.ffn_layer(512, 1408, activation=0.10, dtype=torch.bfloat16, seed=1, device=dev)
    fb = ts.Ffn(Lb.w_gate, Lb.w_up, Lb.w_down, max_batch=4)
    h4 = torch.zeros(4, 512, device=dev)
    with pytest.raises(ts.TsError) as e:
        ts.Graph.stack_fused([fb], h4)
    assert e.value.status == 6  # batch 4 takes the unfused passes
    f32.close()
    fb.close()
