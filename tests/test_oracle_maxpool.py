"""Pins of the oracle's max-pooling option (Sec. 3.3: the SRH heads' window
scores are pooled across the token dimension, then the heads' vectors are
combined; with max pooling the order matters, so each head is pooled before
the head sum)."""
import math

import numpy as np
import pytest
import torch

import oracle
from oracle import compresskv_oracle as O
from oracle.brute import brute_unit


@pytest.mark.parametrize("P", [1, 3, 5, 7, 9])
def test_pool_max_matches_torch_max_pool1d(P):
    """Stride-1 max pooling with r = (P-1)/2 on each side is torch's
    max_pool1d with padding r (its padding never wins)."""
    rng = np.random.default_rng(P)
    for n in (1, 2, 5, 40):
        raw = rng.random(n) * rng.choice([1e-6, 1.0, 30.0])
        want = torch.nn.functional.max_pool1d(torch.tensor(raw)[None, None], P, stride=1,
                                              padding=(P - 1) // 2)[0, 0].numpy()
        if n < (P - 1) // 2 + 1:  # torch wants the padding within half the kernel
            want = np.array([raw[max(0, j - (P - 1) // 2): j + (P - 1) // 2 + 1].max()
                             for j in range(n)])
        assert np.array_equal(oracle.pool_max(raw, P), want)


def test_golden_heads_pooled_before_the_sum():
    """Two heads' window scores, P = 3, worked by hand:
    head 1 [1, 3, 2, 0, 5] -> max pool [3, 3, 3, 5, 5];
    head 2 [0, 1, 0, 4, 0] -> max pool [1, 1, 4, 4, 4];
    sum [4, 4, 7, 9, 9].  Pooling the head sum [1, 4, 2, 4, 5] instead would
    give [4, 4, 4, 5, 5]."""
    h1 = np.array([[1.0, 3.0, 2.0, 0.0, 5.0]])
    h2 = np.array([[0.0, 1.0, 0.0, 4.0, 0.0]])
    got = O.pool_heads([h1, h2], 5, 3, "max")
    assert got.tolist() == [4.0, 4.0, 7.0, 9.0, 9.0]
    # average pooling is linear: the order does not matter
    avg = O.pool_heads([h1, h2], 5, 3, "avg")
    assert np.allclose(avg, (np.array([1, 4, 2, 4, 5]) + np.array([4, 2, 4, 5, 0]) +
                             np.array([0, 1, 4, 2, 4])) / 3.0)


@pytest.mark.parametrize("seed", range(10))
def test_max_pooling_matches_brute_force(seed):
    rng = np.random.default_rng(100 + seed)
    L = int(rng.integers(1, 50))
    W = int(rng.integers(1, 7))
    P = int(rng.choice([1, 3, 5, 7]))
    d = int(rng.choice([2, 4, 8]))
    nh = int(rng.integers(1, 4))
    budget = int(rng.integers(W, max(W + 1, L + 4)))
    q = rng.standard_normal((nh, W, d)) * 0.8
    k = rng.standard_normal((L, d))
    scale = 1.0 / math.sqrt(d)
    res = oracle.compress_unit(q, k, W, P, budget, scale, pool_kind="max")
    raw_b, pooled_b, idx_b = brute_unit(q.tolist(), k.tolist(), W, P, budget, scale,
                                        pool_kind="max")
    np.testing.assert_allclose(res.raw, raw_b, rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(res.pooled, pooled_b, rtol=1e-12, atol=1e-15)
    assert res.indices.tolist() == idx_b


def test_max_pool_invariants():
    """P = 1 makes both kinds the raw score; otherwise every head's maximum
    over a window is at least that window's zero-padded mean, so the max
    pooled score is at least the average pooled score."""
    rng = np.random.default_rng(7)
    q = rng.standard_normal((3, 4, 8))
    k = rng.standard_normal((60, 8))
    s = 1 / math.sqrt(8)
    a1 = oracle.compress_unit(q, k, 4, 1, 30, s, pool_kind="avg")
    m1 = oracle.compress_unit(q, k, 4, 1, 30, s, pool_kind="max")
    np.testing.assert_allclose(m1.pooled, a1.pooled, rtol=1e-12, atol=0)
    np.testing.assert_allclose(m1.pooled, m1.raw, rtol=1e-12, atol=0)
    a7 = oracle.compress_unit(q, k, 4, 7, 30, s, pool_kind="avg")
    m7 = oracle.compress_unit(q, k, 4, 7, 30, s, pool_kind="max")
    assert np.all(m7.pooled >= a7.pooled - 1e-15)
    assert np.all(m7.pooled <= 3.0 * 4 + 1e-12)  # each head's window sum is at most W


def test_layer_scope_sums_each_heads_max_pool():
    """Per-layer selection with max pooling: the layer score is the sum over
    every SRH head of the layer of that head's max-pooled window score."""
    rng = np.random.default_rng(11)
    B, Hq, Hkv, W, d, L = 1, 4, 2, 3, 8, 30
    q = rng.standard_normal((B, Hq, W, d))
    k = rng.standard_normal((L, Hkv, d))
    v = rng.standard_normal((L, Hkv, d))
    mask = np.array([True, True, False, True])
    res = oracle.compress_layer(q, k, v, [0, L], mask, [12], W, 5, selection="layer",
                                pool_kind="max")
    s = oracle.default_scale(d)
    want = np.zeros(L - W)
    for h in np.flatnonzero(mask):
        A = oracle.window_attention(q[0, h], k[:, h // 2], s)
        want += oracle.pool_max(A[:, :L - W].sum(axis=0), 5)
    np.testing.assert_allclose(res.shared[0].pooled, want, rtol=1e-12, atol=0)


def _mutant_pool_the_sum(attn, n, P, kind):
    return O.pool_max(O.raw_scores(attn, n), P) if kind == "max" else O.pool_avg(
        O.raw_scores(attn, n), P)


def _mutant_window_one_short(raw, P):
    raw = np.asarray(raw, np.float64)
    r = (P - 1) // 2
    return np.array([raw[max(0, j - r): j + r].max() if raw[max(0, j - r): j + r].size else 0.0
                     for j in range(len(raw))])


@pytest.mark.parametrize("name,target,mutant", [
    ("max-pool the head sum", "pool_heads", _mutant_pool_the_sum),
    ("pooling window one short", "pool_max", _mutant_window_one_short),
])
def test_planted_max_pool_mistakes_are_caught(monkeypatch, name, target, mutant):
    monkeypatch.setattr(O, target, mutant)
    failures = 0
    for fn in (test_golden_heads_pooled_before_the_sum,
               lambda: test_pool_max_matches_torch_max_pool1d(3),
               lambda: test_max_pooling_matches_brute_force(1)):
        try:
            fn()
        except AssertionError:
            failures += 1
    assert failures > 0, f"planted mistake '{name}' went unnoticed"
