"""Pins for the fp64 CPU oracle, against things other than the oracle itself.

Each test ties the oracle to something the paper or mathematics fixes:
hand-worked examples of Eq. 1/Eq. 2, exact integer brute force, the
sparse == dense identity, the all-active special case (a plain ReGLU FFN,
computed by a library matmul), linearity in W_down, permutation and batch
invariants, the predictor restriction (Sec. 7), the top-k router (Sec. 4), and
the stack glue's closed forms. ``test_pins_reject_planted_mistakes`` shows the
pins fail for plausible mistakes planted in a CPU restatement of the formula.
"""
import json
import os
import random

import numpy as np
import pytest
import torch

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "drelu_handworked.json")


def _golden_cases():
    with open(GOLDEN) as f:
        return json.load(f)["cases"]


def _store(a, dtype):
    """Exact small values as oracle storage (float32 or bf16 bits)."""
    t = torch.tensor(np.asarray(a, np.float64), dtype=torch.float32)
    if dtype == "bf16":
        t32 = t.clone()
        t = t.to(torch.bfloat16)
        assert torch.equal(t.float(), t32), "fixture values must be exact in bf16"
    return t


def _mask_lists(mask):
    return [list(np.nonzero(row)[0]) for row in mask]


# ---------------------------------------------------------------------------
# 1. Hand-worked examples (Eq. 1 + Eq. 2), fp32 and bf16 storage
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_handworked_examples(oracle_mod, dtype):
    for case in _golden_cases():
        x, wg, wu, wd = (_store(case[k], dtype) for k in ("x", "w_gate", "w_up", "w_down"))
        r = oracle_mod.ffn(x, wg, wu, wd)
        assert np.array_equal(r["g"], np.asarray(case["g"], np.float64)), case["name"]
        assert np.array_equal(r["u"], np.asarray(case["u"], np.float64)), case["name"]
        assert _mask_lists(r["gate_mask"]) == case["gate_active"], case["name"]
        assert _mask_lists(r["both_mask"]) == case["both_active"], case["name"]
        assert np.array_equal(r["y"], np.asarray(case["y"], np.float64)), case["name"]
        for p in case.get("predictor", []):
            rp = oracle_mod.ffn(x, wg, wu, wd, rows=np.asarray(p["rows"], np.int32))
            assert np.array_equal(rp["y"], np.asarray(p["y"], np.float64)), p["why"]
            assert _mask_lists(rp["gate_mask"]) == p["gate_active"], p["why"]
            assert _mask_lists(rp["both_mask"]) == p["both_active"], p["why"]


# ---------------------------------------------------------------------------
# 2. Brute force with small integers: every sum exact, every sign pattern hit
# ---------------------------------------------------------------------------
def _exact_ffn(x, wg, wu, wd, rows=None):
    """Pure-Python integer evaluation of Eq. 1 with Eq. 2 (exact)."""
    B, d = len(x), len(x[0])
    m = len(wg)
    take = set(range(m)) if rows is None else set(rows)
    ys, gates, boths = [], [], []
    for b in range(B):
        g = [sum(wg[j][i] * x[b][i] for i in range(d)) for j in range(m)]
        u = [sum(wu[j][i] * x[b][i] for i in range(d)) for j in range(m)]
        c = [max(0, g[j]) * max(0, u[j]) if j in take else 0 for j in range(m)]
        ys.append([sum(c[j] * wd[j][i] for j in range(m)) for i in range(d)])
        gates.append([j for j in range(m) if j in take and g[j] > 0])
        boths.append([j for j in range(m) if j in take and g[j] > 0 and u[j] > 0])
    return ys, gates, boths


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_brute_force_small_integers(oracle_mod, dtype):
    rng = random.Random(7)
    patterns = set()
    for trial in range(60):
        d = rng.randint(1, 8)
        m = rng.randint(1, 16)
        B = rng.randint(1, 3)
        ri = lambda: rng.randint(-3, 3)  # noqa: E731
        x = [[ri() for _ in range(d)] for _ in range(B)]
        wg = [[ri() for _ in range(d)] for _ in range(m)]
        wu = [[ri() for _ in range(d)] for _ in range(m)]
        wd = [[ri() for _ in range(d)] for _ in range(m)]
        rows = None
        if trial % 3 == 2:
            rows = sorted(rng.sample(range(m), rng.randint(0, m)))
        ys, gates, boths = _exact_ffn(x, wg, wu, wd, rows)
        r = oracle_mod.ffn(_store(x, dtype), _store(wg, dtype), _store(wu, dtype), _store(wd, dtype),
                           rows=None if rows is None else np.asarray(rows, np.int32))
        assert np.array_equal(r["y"], np.asarray(ys, np.float64))
        assert _mask_lists(r["gate_mask"]) == gates
        assert _mask_lists(r["both_mask"]) == boths
        for b in range(B):
            for j in range(m):
                g = sum(wg[j][i] * x[b][i] for i in range(d))
                u = sum(wu[j][i] * x[b][i] for i in range(d))
                patterns.add((int(np.sign(g)), int(np.sign(u))))
    assert patterns == {(a, b) for a in (-1, 0, 1) for b in (-1, 0, 1)}


# ---------------------------------------------------------------------------
# 3. Sparse == dense: skipping inactive neurons is exact (adding +0 is exact)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_sparse_sum_equals_dense_definition_bit_exact(oracle_mod, dtype):
    from paper_2406_05955_gb300 import workload as wl

    L = wl.ffn_layer(64, 300, activation=0.10, dtype=dtype, seed=3)
    x = wl.tokens(3, 64, dtype=dtype, seed=4)
    r = oracle_mod.ffn(x, L.w_gate, L.w_up, L.w_down)
    wd = oracle_mod.values(L.w_down)
    for b in range(3):
        act = np.nonzero(r["both_mask"][b])[0]
        assert 0 < act.size < 300
        y = np.zeros(64)
        for j in act:  # ascending j, only both-active neurons
            y = y + (r["g"][b, j] * r["u"][b, j]) * wd[j]
        assert np.array_equal(y, r["y"][b])
        # the oracle restricted to the active set gives the same bits
        rs = oracle_mod.ffn(x[b:b + 1], L.w_gate, L.w_up, L.w_down, rows=act.astype(np.int32))
        assert np.array_equal(rs["y"][0], r["y"][b])


# ---------------------------------------------------------------------------
# 4. All-active special case == ReGLU FFN by a library matmul
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_all_active_reduces_to_reglu(oracle_mod, dtype):
    from paper_2406_05955_gb300 import workload as wl

    L = wl.ffn_layer(96, 200, activation=1.0, dtype=dtype, seed=5)
    x = wl.tokens(4, 96, dtype=dtype, seed=6)
    r = oracle_mod.ffn(x, L.w_gate, L.w_up, L.w_down)
    assert r["both_mask"].all() and r["gate_mask"].all()
    X = oracle_mod.values(x)
    Wg, Wu, Wd = (oracle_mod.values(w) for w in (L.w_gate, L.w_up, L.w_down))
    ref = (np.maximum(X @ Wg.T, 0.0) * (X @ Wu.T)) @ Wd
    err = np.linalg.norm(r["y"] - ref) / np.linalg.norm(ref)
    assert err <= 1e-12


# ---------------------------------------------------------------------------
# 5. Linearity in W_down (masks do not depend on it)
# ---------------------------------------------------------------------------
def test_linearity_in_w_down(oracle_mod):
    rng = np.random.default_rng(11)
    d, m, B = 48, 120, 2
    x = rng.standard_normal((B, d)).astype(np.float32)
    wg = (rng.standard_normal((m, d)) / 7).astype(np.float32)
    wu = (rng.standard_normal((m, d)) / 7).astype(np.float32)
    # dyadic values with few bits, so alpha*A + beta*B is exact in fp32
    A = (rng.integers(-64, 65, (m, d)) / 64.0).astype(np.float32)
    Bm = (rng.integers(-64, 65, (m, d)) / 64.0).astype(np.float32)
    alpha, beta = 2.0, -0.5
    C = (alpha * A.astype(np.float64) + beta * Bm.astype(np.float64)).astype(np.float32)
    assert np.array_equal(C.astype(np.float64), alpha * A.astype(np.float64) + beta * Bm.astype(np.float64))
    ra, rb, rc = (oracle_mod.ffn(x, wg, wu, W) for W in (A, Bm, C))
    assert np.array_equal(ra["both_mask"], rc["both_mask"])
    lhs = rc["y"]
    rhs = alpha * ra["y"] + beta * rb["y"]
    assert np.linalg.norm(lhs - rhs) / np.linalg.norm(rhs) <= 1e-12


# ---------------------------------------------------------------------------
# 6./7. Neuron permutation and batch invariants
# ---------------------------------------------------------------------------
def test_joint_neuron_permutation_invariance(oracle_mod):
    from paper_2406_05955_gb300 import workload as wl

    L = wl.ffn_layer(64, 256, activation=0.25, dtype=torch.float32, seed=8)
    x = wl.tokens(2, 64, dtype=torch.float32, seed=9)
    perm = torch.randperm(256, generator=torch.Generator().manual_seed(1))
    r0 = oracle_mod.ffn(x, L.w_gate, L.w_up, L.w_down)
    r1 = oracle_mod.ffn(x, L.w_gate[perm], L.w_up[perm], L.w_down[perm])
    assert np.array_equal(r1["both_mask"], r0["both_mask"][:, perm.numpy()])
    assert np.array_equal(r1["g"], r0["g"][:, perm.numpy()])
    assert np.linalg.norm(r1["y"] - r0["y"]) / np.linalg.norm(r0["y"]) <= 1e-12


def test_batch_rows_equal_single_token_runs(oracle_mod):
    from paper_2406_05955_gb300 import workload as wl

    L = wl.ffn_layer(64, 200, activation=0.10, dtype=torch.bfloat16, seed=10)
    x = wl.tokens(5, 64, dtype=torch.bfloat16, seed=11)
    rb = oracle_mod.ffn(x, L.w_gate, L.w_up, L.w_down)
    for b in range(5):
        r1 = oracle_mod.ffn(x[b:b + 1], L.w_gate, L.w_up, L.w_down)
        for k in ("y", "g", "u", "gate_mask", "both_mask"):
            assert np.array_equal(r1[k][0], rb[k][b])


# ---------------------------------------------------------------------------
# 8. Predictor lists (Sec. 7)
# ---------------------------------------------------------------------------
def test_predictor_list_restriction(oracle_mod):
    from paper_2406_05955_gb300 import workload as wl

    L = wl.ffn_layer(64, 300, activation=0.10, dtype=torch.bfloat16, seed=12)
    x = wl.tokens(1, 64, dtype=torch.bfloat16, seed=13)
    full = oracle_mod.ffn(x, L.w_gate, L.w_up, L.w_down)
    all_rows = np.arange(300, dtype=np.int32)
    r_all = oracle_mod.ffn(x, L.w_gate, L.w_up, L.w_down, rows=all_rows)
    assert np.array_equal(r_all["y"], full["y"])
    act = np.nonzero(full["both_mask"][0])[0].astype(np.int32)
    r_act = oracle_mod.ffn(x, L.w_gate, L.w_up, L.w_down, rows=act)
    assert np.array_equal(r_act["y"], full["y"])
    # a list that misses half the active neurons: exactly the restricted sum
    lst = wl.predictor_list(L.offsets, 60, seed=3).numpy()
    r_l = oracle_mod.ffn(x, L.w_gate, L.w_up, L.w_down, rows=lst)
    wd = oracle_mod.values(L.w_down)
    y = np.zeros(64)
    for j in sorted(set(lst.tolist()) & set(act.tolist())):
        y = y + (full["g"][0, j] * full["u"][0, j]) * wd[j]
    assert np.array_equal(r_l["y"][0], y)
    outside = np.setdiff1d(np.arange(300), lst)
    assert not r_l["gate_mask"][0, outside].any() and not r_l["both_mask"][0, outside].any()
    empty = oracle_mod.ffn(x, L.w_gate, L.w_up, L.w_down, rows=np.zeros(0, np.int32))
    assert not empty["y"].any()


@pytest.mark.parametrize("rows", [[3, 2], [1, 1], [-1, 4], [5, 300]])
def test_predictor_list_rejects_bad_lists(oracle_mod, rows):
    from paper_2406_05955_gb300 import workload as wl

    L = wl.ffn_layer(16, 300, dtype=torch.float32, seed=1)
    with pytest.raises(ValueError):
        oracle_mod.ffn(wl.tokens(1, 16, dtype=torch.float32), L.w_gate, L.w_up, L.w_down,
                       rows=np.asarray(rows, np.int32))


# ---------------------------------------------------------------------------
# 9./10. MoE (Sec. 4): identical experts, top-k by brute force, softmax closed form
# ---------------------------------------------------------------------------
def test_moe_identical_experts_equal_single_ffn(oracle_mod):
    from paper_2406_05955_gb300 import workload as wl

    L = wl.ffn_layer(64, 128, activation=0.20, dtype=torch.bfloat16, seed=14)
    x = wl.tokens(4, 64, dtype=torch.bfloat16, seed=15)
    wr = wl.router(8, 64, dtype=torch.bfloat16, seed=16)
    experts = [(L.w_gate, L.w_up, L.w_down)] * 8
    r = oracle_mod.moe(x, wr, experts, top_k=2)
    single = oracle_mod.ffn(x, L.w_gate, L.w_up, L.w_down)
    assert np.allclose(r["w"].sum(axis=1), 1.0, rtol=0, atol=1e-15)
    assert np.linalg.norm(r["y"] - single["y"]) / np.linalg.norm(single["y"]) <= 1e-12


def test_router_topk_brute_force_and_softmax(oracle_mod):
    from paper_2406_05955_gb300 import workload as wl

    x = wl.tokens(16, 64, dtype=torch.bfloat16, seed=17)
    wr = wl.router(8, 64, dtype=torch.bfloat16, seed=18)
    for k in (1, 2, 3):
        r = oracle_mod.router(x, wr, top_k=k)
        ref_logits = oracle_mod.values(x) @ oracle_mod.values(wr).T
        assert np.max(np.abs(r["logits"] - ref_logits)) <= 1e-12
        for t in range(16):
            order = sorted(range(8), key=lambda e: (-r["logits"][t, e], e))
            assert list(r["sel"][t]) == order[:k]
            z = np.exp(r["logits"][t, order[:k]] - r["logits"][t, order[0]])
            assert np.allclose(r["w"][t], z / z.sum(), rtol=1e-14, atol=0)
        if k == 2:
            l0, l1 = r["logits"][:, r["sel"][:, 0]].diagonal(), r["logits"][:, r["sel"][:, 1]].diagonal()
            assert np.allclose(r["w"][:, 0], 1.0 / (1.0 + np.exp(l1 - l0)), rtol=1e-14, atol=0)


def test_router_tie_goes_to_lower_index(oracle_mod):
    x = np.ones((1, 4), np.float32)
    wr = np.array([[0, 0, 0, 0], [1, 0, 0, 0], [0, 0, 1, 1], [1, 1, 0, 0], [2, 0, 0, 0]], np.float32)
    r = oracle_mod.router(x, wr, top_k=3)
    # logits (0, 1, 2, 2, 2): the three tied experts are taken in index order
    assert list(r["sel"][0]) == [2, 3, 4]
    assert np.allclose(r["w"][0], [1 / 3, 1 / 3, 1 / 3], rtol=1e-15)


# ---------------------------------------------------------------------------
# 11. Stack glue: closed forms and bf16 rounding vs torch's rounding routine
# ---------------------------------------------------------------------------
def test_rmsnorm_closed_form_and_bias_channel(oracle_mod):
    c = 3.0
    h = np.full((1, 8), c, np.float32)
    x = oracle_mod.rmsnorm(h, oracle_mod.F32, eps=1e-5)
    expect = np.float32(c / np.sqrt(c * c + 1e-5))
    assert np.all(x[0, :7] == expect) and x[0, 7] == 1.0
    # eps = 1 - mean(h^2) makes rms exactly 1: x = h, then bf16 rounding only
    vals = np.array([1 + 2 ** -8, 1 + 3 * 2 ** -8, -(1 + 2 ** -8), 0.5, 0.25, -0.75, 0.125, 0.0], np.float32)
    h = vals[None, :]
    eps = 1.0 - float(np.mean(vals[:].astype(np.float64) ** 2))
    assert eps > 0
    xb = oracle_mod.rmsnorm(h, oracle_mod.BF16, eps=eps)
    got = oracle_mod.bf16_bits_to_f64(xb[0])
    # ties go to even: 1+2^-8 -> 1, 1+3*2^-8 -> 1+2^-6; last entry is the bias channel
    assert list(got) == [1.0, 1 + 2 ** -6, -1.0, 0.5, 0.25, -0.75, 0.125, 1.0]


def test_rmsnorm_bf16_rounding_matches_torch(oracle_mod):
    rng = np.random.default_rng(19)
    h = (rng.standard_normal((6, 1024)) * rng.uniform(0.1, 30, (6, 1))).astype(np.float32)
    x32 = oracle_mod.rmsnorm(h, oracle_mod.F32)
    xb = oracle_mod.rmsnorm(h, oracle_mod.BF16)
    ref = torch.from_numpy(x32).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(xb, ref)
    rms = np.sqrt(np.mean(h.astype(np.float64) ** 2, axis=1, keepdims=True) + 1e-5)
    expect = (h / rms).astype(np.float32)
    expect[:, -1] = 1.0
    assert np.array_equal(x32, expect)


def test_stack_two_layers_by_hand(oracle_mod):
    from paper_2406_05955_gb300 import workload as wl

    layers = [wl.ffn_layer(32, 64, activation=0.25, dtype=torch.bfloat16, seed=20 + i) for i in range(2)]
    h0 = wl.residual(2, 32, seed=22).numpy()
    st = oracle_mod.stack(h0, [(L.w_gate, L.w_up, L.w_down) for L in layers])
    h = h0
    for L in layers:
        x = oracle_mod.rmsnorm(h, oracle_mod.BF16)
        y = oracle_mod.ffn(x, L.w_gate, L.w_up, L.w_down)["y"]
        h = (h.astype(np.float64) + y).astype(np.float32)
    assert np.array_equal(st["h"], h)


# ---------------------------------------------------------------------------
# 12. The pins catch plausible mistakes (planted in a CPU restatement)
# ---------------------------------------------------------------------------
def _formula(x, wg, wu, wd, mistake=None):
    """Eq. 1 + Eq. 2 in numpy, with an optional planted mistake; returns (y, gate, both)."""
    d = x.shape[1]
    m = wg.shape[0]
    g = x @ wg.T
    u = x @ wu.T
    if mistake == "sign":
        g = -g
    if mistake == "transposed_down":  # flat buffer read as [d][m]
        wd = wd.reshape(-1).reshape(d, m).T
    if mistake == "no_up_relu":
        c = np.maximum(g, 0) * u
    elif mistake == "relu_of_product":
        c = np.maximum(g * u, 0)
    else:
        c = np.maximum(g, 0) * np.maximum(u, 0)
    if mistake == "dropped_first_term":
        c = c.copy()
        c[:, 0] = 0
    gate = (g >= 0) if mistake == "ge_zero_mask" else (g > 0)
    both = gate & (u > 0)
    return c @ wd, gate, both


@pytest.mark.parametrize("mistake", ["sign", "no_up_relu", "relu_of_product", "ge_zero_mask",
                                     "transposed_down", "dropped_first_term"])
def test_pins_reject_planted_mistakes(mistake):
    def differs(x, wg, wu, wd, y_ref, gate_ref, both_ref):
        y, gate, both = _formula(x, wg, wu, wd, mistake)
        return (not np.array_equal(y, np.asarray(y_ref, np.float64))
                or _mask_lists(gate) != gate_ref or _mask_lists(both) != both_ref)

    caught = []
    for case in _golden_cases():
        x, wg, wu, wd = (np.asarray(case[k], np.float64) for k in ("x", "w_gate", "w_up", "w_down"))
        y, gate, both = _formula(x, wg, wu, wd)
        assert np.array_equal(y, np.asarray(case["y"], np.float64))
        caught.append(differs(x, wg, wu, wd, case["y"], case["gate_active"], case["both_active"]))
    rng = np.random.default_rng(3)
    for _ in range(50):
        d, m = 4, 6
        x = rng.integers(-3, 4, (2, d))
        wg, wu, wd = (rng.integers(-3, 4, (m, d)) for _ in range(3))
        ys, gates, boths = _exact_ffn(x.tolist(), wg.tolist(), wu.tolist(), wd.tolist())
        caught.append(differs(*(a.astype(np.float64) for a in (x, wg, wu, wd)), ys, gates, boths))
    assert any(caught), f"no pin catches the planted mistake {mistake!r}"
