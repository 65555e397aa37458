"""GPU parity of the single sparse dReLU FFN (C ABI) against the fp64 oracle.

Covers: the fp32 d=512/m=1408 workload token by token; ragged shapes (partial
row chunks, partial column slices, batches split into passes); the
Mistral-shaped layer at full size; the activation sweep; predictor lists
(Sec. 7) including empty, full, exact and bad lists; the two-step entry points;
determinism; and argument errors.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2406_05955_gb300 import workload as wl

from _parity import check_sets, check_y, union_mask

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ts():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    import paper_2406_05955_gb300 as ts

    ts.lib()
    return ts


def _dt(dtype):
    return "f32" if dtype == torch.float32 else "bf16"


def _run(ts, L, x, rows=None, max_batch=None):
    dev = torch.device("cuda")
    ffn = ts.Ffn(L.w_gate.to(dev), L.w_up.to(dev), L.w_down.to(dev), max_batch=max_batch or x.shape[0])
    idx = None if rows is None else torch.as_tensor(rows, dtype=torch.int32).to(dev)
    y = ffn.forward(x.to(dev), active_idx=idx)
    torch.cuda.synchronize()
    return ffn, y.double().cpu().numpy()


def test_fp32_d512_m1408_sixteen_tokens(ts):
    cfg = wl.WORKLOADS["drelu-ffn-fp32-d512-m1408"]
    L = wl.ffn_layer(cfg["d"], cfg["m"], mu=cfg["mu"], dtype=torch.float32, seed=cfg["seed"])
    xs = wl.tokens(cfg["n_tokens"], cfg["d"], dtype=torch.float32, seed=cfg["seed"] + 1)
    dev = torch.device("cuda")
    ffn = ts.Ffn(L.w_gate.to(dev), L.w_up.to(dev), L.w_down.to(dev), max_batch=1)
    ref = oracle.ffn(xs, L.w_gate, L.w_up, L.w_down)
    flips = 0
    for t in range(cfg["n_tokens"]):
        y = ffn.forward(xs[t:t + 1].to(dev)).double().cpu().numpy()
        check_y(y[0], ref["y"][t], "f32", f"token {t}")
        g, b = ffn.get_active(0)
        one = {k: ref[k][t:t + 1] for k in ("g", "u", "gate_mask", "both_mask")}
        flips += check_sets(g, b, one, 0)
    assert flips <= 2
    frac = ref["both_mask"].mean()
    assert 0.05 < frac < 0.15  # ~10% both-active (mu = -0.7)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("d,m,B", [(8, 1, 1), (64, 7, 2), (136, 33, 3), (264, 1001, 5), (520, 777, 8),
                                   (1032, 515, 13), (256, 64, 1)])
def test_ragged_shapes(ts, dtype, d, m, B):
    L = wl.ffn_layer(d, m, activation=0.25, dtype=dtype, seed=d + m)
    x = wl.tokens(B, d, dtype=dtype, seed=B)
    ffn, y = _run(ts, L, x)
    ref = oracle.ffn(x, L.w_gate, L.w_up, L.w_down)
    check_y(y, ref["y"], _dt(dtype))
    for t in range(B):
        check_sets(*ffn.get_active(t), ref, t)
    g, b = ffn.get_active(-1)
    assert np.setxor1d(b, union_mask(ref, "both_mask")).size <= 2


@pytest.mark.parametrize("B", [1, 4, 16])
def test_mistral_layer_full_size(ts, B):
    L = wl.ffn_layer(4096, 14336, activation=0.10, dtype=torch.bfloat16, seed=11)
    x = wl.tokens(B, 4096, dtype=torch.bfloat16, seed=12)
    ffn, y = _run(ts, L, x)
    ref = oracle.ffn(x, L.w_gate, L.w_up, L.w_down)
    check_y(y, ref["y"], "bf16")
    flips = sum(check_sets(*ffn.get_active(t), ref, t) for t in range(B))
    assert flips <= 4 * B
    assert 0.08 < ref["both_mask"].mean() < 0.12 and 0.25 < ref["gate_mask"].mean() < 0.31


@pytest.mark.parametrize("act", [0.05, 0.25, 0.50, 1.0])
@pytest.mark.parametrize("B", [1, 4, 16, 64])
def test_activation_sweep(ts, act, B):
    d, m = 1024, 3584
    L = wl.ffn_layer(d, m, activation=act, dtype=torch.bfloat16, seed=int(act * 100) + B)
    x = wl.tokens(B, d, dtype=torch.bfloat16, seed=B + 7)
    ffn, y = _run(ts, L, x)
    ref = oracle.ffn(x, L.w_gate, L.w_up, L.w_down)
    check_y(y, ref["y"], "bf16")
    for t in (0, B - 1):
        check_sets(*ffn.get_active(t), ref, t)
    g, b = ffn.get_active(-1)
    assert np.setxor1d(b, union_mask(ref, "both_mask")).size <= 2 * B
    if act >= 1.0:
        assert len(b) == m


@pytest.mark.parametrize("B", [1, 3, 8, 16])
def test_predictor_lists(ts, B):
    d, m = 4096, 14336
    L = wl.ffn_layer(d, m, activation=0.10, dtype=torch.bfloat16, seed=21)
    x = wl.tokens(B, d, dtype=torch.bfloat16, seed=22)
    lst = wl.predictor_list(L.offsets, 1434, seed=23).numpy()
    ffn, y = _run(ts, L, x, rows=lst)
    ref = oracle.ffn(x, L.w_gate, L.w_up, L.w_down, rows=lst)
    check_y(y, ref["y"], "bf16")
    for t in range(B):
        check_sets(*ffn.get_active(t), ref, t, rows=lst)
    assert ffn.get_error() == 0


def test_predictor_edge_lists(ts):
    d, m = 512, 1000
    L = wl.ffn_layer(d, m, activation=0.10, dtype=torch.bfloat16, seed=31)
    x = wl.tokens(2, d, dtype=torch.bfloat16, seed=32)
    full = oracle.ffn(x, L.w_gate, L.w_up, L.w_down)
    # empty list: nothing is computed, y = 0
    ffn, y = _run(ts, L, x, rows=np.zeros(0, np.int32))
    assert not np.any(y)
    # the whole neuron range: identical to detected mode
    ffn, y = _run(ts, L, x, rows=np.arange(m, dtype=np.int32))
    check_y(y, full["y"], "bf16")
    # exactly the union of both-active neurons: identical result
    act = union_mask(full, "both_mask").astype(np.int32)
    ffn, y = _run(ts, L, x, rows=act)
    check_y(y, full["y"], "bf16")
    # one listed neuron, ragged chunk
    one = np.asarray([m - 1], np.int32)
    ffn, y = _run(ts, L, x, rows=one)
    check_y(y, oracle.ffn(x, L.w_gate, L.w_up, L.w_down, rows=one)["y"], "bf16")


@pytest.mark.parametrize("rows", [[5, 3, 9], [1, 1, 2], [0, 999, 1000], [-4, 2]])
def test_bad_predictor_list_sets_status(ts, rows):
    d, m = 256, 1000
    L = wl.ffn_layer(d, m, activation=0.10, dtype=torch.bfloat16, seed=33)
    x = wl.tokens(1, d, dtype=torch.bfloat16, seed=34)
    ffn, y = _run(ts, L, x, rows=np.asarray(rows, np.int32))
    assert ffn.get_error() == ts.binding.TS_ERR_BAD_INDEX
    assert ffn.get_error() == 0  # cleared by the read
    assert np.isfinite(y).all()


def test_two_step_entry_points_and_determinism(ts):
    d, m, B = 4096, 14336, 2
    L = wl.ffn_layer(d, m, activation=0.10, dtype=torch.bfloat16, seed=41)
    x = wl.tokens(B, d, dtype=torch.bfloat16, seed=42).cuda()
    dev = torch.device("cuda")
    ffn = ts.Ffn(L.w_gate.to(dev), L.w_up.to(dev), L.w_down.to(dev), max_batch=B)
    y1 = ffn.forward(x).clone()
    y2 = ffn.forward(x).clone()
    ffn.gate_up(x)
    y3 = ffn.down(B)
    torch.cuda.synchronize()
    assert torch.equal(y1, y2) and torch.equal(y1, y3)


def test_argument_errors(ts):
    dev = torch.device("cuda")
    d, m = 64, 32
    L = wl.ffn_layer(d, m, dtype=torch.bfloat16, seed=1)
    wg, wu, wd = (w.to(dev) for w in (L.w_gate, L.w_up, L.w_down))
    ffn = ts.Ffn(wg, wu, wd, max_batch=2)
    x = wl.tokens(3, d, dtype=torch.bfloat16).to(dev)
    with pytest.raises(ts.TsError) as e:
        ffn.forward(x)  # batch 3 > max_batch 2
    assert e.value.status == ts.binding.TS_ERR_INVALID_ARG
    with pytest.raises(ts.TsError):
        ffn.forward(x[:1], active_idx=torch.arange(m + 1, dtype=torch.int32, device=dev))
    # a weight pointer off the 16-byte grid
    flat = torch.zeros(m * d + 1, dtype=torch.bfloat16, device=dev)
    with pytest.raises(ts.TsError):
        ts.Ffn(flat[1:].view(m, d), wu, wd)
    # d * 2 bytes not a multiple of 16
    L2 = wl.ffn_layer(12, 8, dtype=torch.bfloat16, seed=2)
    with pytest.raises(ts.TsError):
        ts.Ffn(L2.w_gate.to(dev), L2.w_up.to(dev), L2.w_down.to(dev))
    # batch 0 is a no-op
    y = torch.full((0, d), 7.0, device=dev)
    ffn.forward(x[:0], y=y)
