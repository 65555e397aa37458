"""Pins for the oracle's activation predictor (the reading of Sec. 7's
predictor: a two-layer ReLU MLP whose K best-rated neurons form the list),
against things other than the oracle: a hand-worked case with a tie and a
clipped hidden unit, the batch rule (a neuron's key is its largest score over
the tokens), the limits K = 0 and K = m, an independent numpy restatement on
random weights (library matmuls and a stable sort), and mistakes planted in a
CPU restatement (no ReLU, min over tokens, ties to the higher index, the
smallest scores), which the pins reject.
"""
import numpy as np
import pytest
import torch

from paper_2406_05955_gb300 import workload as wl

import oracle


def _f32(a):
    return np.ascontiguousarray(np.asarray(a, np.float32))


# x = (1, 2, 1): h = (max(0, 1), max(0, -2)) = (1, 0);
# s = W2 h = (3, 1, -1, 3)  ->  K=1: {0} (tie with 3 goes to 0), K=2: {0, 3},
# K=3: {0, 1, 3}, K=4: all
X = _f32([[1, 2, 1]])
W1 = _f32([[1, 0, 0], [0, -1, 0]])
W2 = _f32([[3, 5], [1, 0], [-1, 0], [3, 7]])
EXPECT = {0: [], 1: [0], 2: [0, 3], 3: [0, 1, 3], 4: [0, 1, 2, 3]}


@pytest.mark.parametrize("K", sorted(EXPECT))
def test_predict_handworked(K):
    r = oracle.predict(X, W1, W2, K)
    assert r["list"].tolist() == EXPECT[K]
    assert np.array_equal(r["scores"][0], [3.0, 1.0, -1.0, 3.0])


def test_predict_batch_takes_the_largest_score():
    # token 2: x = (-1, 0, 1) -> h = (0, 0) -> s = 0 everywhere; token 3: x = (0, -1, 0) -> h = (0, 1)
    x = _f32([[1, 2, 1], [-1, 0, 1], [0, -1, 0]])
    r = oracle.predict(x, W1, W2, 2)
    # keys: max over tokens of (3, 1, -1, 3), (0, 0, 0, 0), (5, 0, 0, 7) = (5, 1, 0, 7)
    assert r["list"].tolist() == [0, 3]
    r = oracle.predict(x, W1, W2, 3)
    assert r["list"].tolist() == [0, 1, 3]


def _numpy_predict(x, w1, w2, K):
    h = np.maximum(x @ w1.T, 0)
    s = h @ w2.T
    key = s.max(axis=0)
    order = np.argsort(-key, kind="stable")
    return np.sort(order[:K]), s


@pytest.mark.parametrize("K", [0, 7, 40, 96])
@pytest.mark.parametrize("B", [1, 4])
def test_predict_random_against_numpy(K, B):
    d, r, m = 64, 16, 96
    L = wl.ffn_layer(d, m, activation=0.10, dtype=torch.float32, seed=51)
    P = wl.predictor_weights(d, r, m, L.offsets, dtype=torch.float32, seed=52)
    x = wl.tokens(B, d, dtype=torch.float32, seed=53)
    got = oracle.predict(x, P.w1, P.w2, K)
    lst, s = _numpy_predict(*(t.double().numpy() for t in (x, P.w1, P.w2)), K)
    key = np.sort(s.max(axis=0))[::-1]
    if 0 < K < m:
        assert key[K - 1] - key[K] > 1e-9  # no near-tie at the cut in this draw
    assert got["list"].tolist() == lst.tolist()
    assert np.allclose(got["scores"], s, rtol=1e-12, atol=1e-12)


def test_predict_bf16_and_limits():
    d, r, m = 128, 32, 200
    L = wl.ffn_layer(d, m, activation=0.10, dtype=torch.bfloat16, seed=54)
    P = wl.predictor_weights(d, r, m, L.offsets, dtype=torch.bfloat16, seed=55)
    x = wl.tokens(2, d, dtype=torch.bfloat16, seed=56)
    assert oracle.predict(x, P.w1, P.w2, m)["list"].tolist() == list(range(m))
    assert oracle.predict(x, P.w1, P.w2, 0)["list"].size == 0
    with pytest.raises(ValueError):
        oracle.predict(x, P.w1, P.w2, m + 1)


def _planted(x, K, mistake):
    h = x @ W1.T.astype(np.float64)
    if mistake != "no_relu":
        h = np.maximum(h, 0)
    s = h @ W2.T.astype(np.float64)
    key = s.min(axis=0) if mistake == "min_over_tokens" else s.max(axis=0)
    idx = np.arange(len(key))
    if mistake == "smallest":
        order = np.lexsort((idx, key))
    elif mistake == "ties_to_higher":
        order = np.lexsort((-idx, -key))
    else:
        order = np.lexsort((idx, -key))
    return sorted(order[:K].tolist())


@pytest.mark.parametrize("mistake", [None, "no_relu", "min_over_tokens", "ties_to_higher", "smallest"])
def test_predict_pins_reject_planted_mistakes(mistake):
    x1 = X.astype(np.float64)
    x3 = _f32([[1, 2, 1], [-1, 0, 1], [0, -1, 0]]).astype(np.float64)
    agree = all(_planted(x1, k, mistake) == EXPECT[k] for k in (1, 2, 3)) and \
        _planted(x3, 2, mistake) == [0, 3] and _planted(x3, 3, mistake) == [0, 1, 3]
    assert agree == (mistake is None)
