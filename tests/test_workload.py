"""The seeded generator reproduces the activation rates its recipe states.

Closed form for a token x with bias channel x[d-1] = 1: the pre-activations of
neuron j are g = z_g + b_j, u = z_u + b_j with z ~ N(0, s^2), s^2 = sum_{i<d-1}
x_i^2 / d, and b_j ~ N(mu, sigma_b^2) shared by gate and up. Hence
P(g > 0) = Phi(mu / sqrt(s^2 + sigma_b^2)) and P(g > 0, u > 0) = E_b[Phi(b/s)^2].
Neurons are independent, so measured fractions are binomial around these.
"""
import math

import numpy as np
import pytest
import torch
from scipy.integrate import quad
from scipy.stats import norm

from paper_2406_05955_gb300 import workload as wl


def _closed_form(mu, sigma_b, s):
    p_gate = norm.cdf(mu / math.hypot(s, sigma_b))
    p_both = quad(lambda b: norm.pdf(b, mu, sigma_b) * norm.cdf(b / s) ** 2,
                  mu - 12 * sigma_b, mu + 12 * sigma_b)[0]
    return p_gate, p_both


@pytest.mark.parametrize("activation", [0.05, 0.10, 0.20, 0.25, 0.50])
def test_activation_fractions_match_closed_form(activation):
    d, m = 1024, 16384
    L = wl.ffn_layer(d, m, activation=activation, dtype=torch.float32, seed=31)
    x = wl.tokens(4, d, dtype=torch.float32, seed=32).double()
    g = x @ L.w_gate.double().T
    u = x @ L.w_up.double().T
    mu = wl.MU_FOR_ACTIVATION[activation]
    for t in range(4):
        s = math.sqrt(float((x[t, : d - 1] ** 2).sum()) / d)
        p_gate, p_both = _closed_form(mu, wl.SIGMA_B, s)
        f_gate = float((g[t] > 0).double().mean())
        f_both = float(((g[t] > 0) & (u[t] > 0)).double().mean())
        assert abs(f_gate - p_gate) <= 4 * math.sqrt(p_gate * (1 - p_gate) / m)
        assert abs(f_both - p_both) <= 4 * math.sqrt(p_both * (1 - p_both) / m)
    # the table's mu is the solution for unit s
    assert abs(_closed_form(mu, wl.SIGMA_B, 1.0)[1] - activation) < 5e-4


def test_all_active_offsets():
    L = wl.ffn_layer(64, 512, activation=1.0, dtype=torch.bfloat16, seed=1)
    x = wl.tokens(8, 64, dtype=torch.bfloat16, seed=2).float()
    assert (x @ L.w_gate.float().T > 0).all() and (x @ L.w_up.float().T > 0).all()


def test_bias_channel_and_shared_offsets():
    L = wl.ffn_layer(32, 100, activation=0.10, dtype=torch.bfloat16, seed=3)
    assert torch.equal(L.w_gate[:, -1], L.w_up[:, -1])
    assert torch.equal(L.w_gate[:, -1], L.offsets.to(torch.bfloat16))
    x = wl.tokens(3, 32, seed=4)
    assert (x[:, -1] == 1).all()


def test_seed_determinism():
    a = wl.ffn_layer(16, 40, seed=5)
    b = wl.ffn_layer(16, 40, seed=5)
    c = wl.ffn_layer(16, 40, seed=6)
    assert torch.equal(a.w_gate, b.w_gate) and torch.equal(a.w_down, b.w_down)
    assert not torch.equal(a.w_gate, c.w_gate)
    assert torch.equal(wl.tokens(2, 16, seed=1), wl.tokens(2, 16, seed=1))


def test_predictor_list_shape_and_skew():
    L = wl.ffn_layer(64, 14336, activation=0.10, dtype=torch.float32, seed=7)
    lst = wl.predictor_list(L.offsets, 1434, seed=8)
    a = lst.numpy()
    assert lst.dtype == torch.int32 and a.size == 1434
    assert np.all(np.diff(a) > 0) and a[0] >= 0 and a[-1] < 14336
    # Zipf over hotness: listed neurons are hotter than average
    assert float(L.offsets[lst.long()].mean()) > float(L.offsets.mean()) + 0.2
    assert wl.predictor_list(L.offsets, 0).numel() == 0
    assert torch.equal(wl.predictor_list(L.offsets, 14336), torch.arange(14336, dtype=torch.int32))


def test_workload_table_shapes():
    w = wl.WORKLOADS
    assert w["mistral7b-ffn-stack-bf16-b1-act10"]["d"] == 4096
    assert w["mistral7b-ffn-stack-bf16-b1-act10"]["m"] == 14336
    assert w["mixtral47b-moe-stack-bf16-top2"]["experts"] == 8
    assert w["drelu-ffn-fp32-d512-m1408"]["m"] == 1408
