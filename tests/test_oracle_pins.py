"""Pins of the float64 oracle against things other than itself.

* a hand-worked example (tests/golden), derived from Sec. 3.3 / Sec. 4;
* a pure-Python brute force on tiny prompts (explicit loops, math.fsum);
* closed forms (all keys equal => uniform causal attention);
* invariants (rows sum to one, total mass W*|S|, index-set properties);
* the all-heads special case == SnapKV-style group scoring recomputed with
  torch's float64 softmax / avg_pool1d / stable sort;
* planted mistakes in the oracle (on the CPU) that these pins must catch.
"""
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest
import torch

import oracle
from oracle import compresskv_oracle as O
from oracle.brute import brute_unit

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _num(x):
    if isinstance(x, str):
        sign = -1.0 if x.startswith("-") else 1.0
        body = x.lstrip("-")
        mult = 1.0
        if body[0].isdigit():
            i = 0
            while body[i].isdigit():
                i += 1
            mult, body = float(body[:i]), body[i:]
        return sign * mult * {"ln2": math.log(2.0), "ln3": math.log(3.0)}[body]
    return float(x)


def _frac(s):
    return float(Fraction(s))


def _load_golden():
    with open(os.path.join(GOLDEN, "hand_worked_window2.json")) as f:
        return json.load(f)


def _golden_inputs(g, both_srh=False, head1_like_head0=False):
    keys = np.array(g["keys"], dtype=np.float64)
    q0 = np.array([[_num(v) for v in row] for row in g["q_head0"]])
    q1 = q0.copy() if head1_like_head0 else np.array([[_num(v) for v in row] for row in g["q_head1"]])
    L, d = keys.shape
    q_win = np.stack([q0, q1])[None]                       # [1, 2, W, d]
    k = keys[:, None, :]                                   # [L, 1, d]
    v = np.arange(L * d, dtype=np.float64).reshape(L, 1, d)
    mask = np.array([True, both_srh])
    return q_win, k, v, np.array([0, L]), mask


# ---------------------------------------------------------------------------
# hand-worked example
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("budget", [2, 3, 4, 5])
def test_golden_hand_worked_pool3(budget):
    g = _load_golden()
    q_win, k, v, cu, mask = _golden_inputs(g)
    res = oracle.compress_layer(q_win, k, v, cu, mask, [budget], g["window"], 3, scale=g["scale"])
    u = res.units[(0, 0)]
    np.testing.assert_allclose(u.raw, [_frac(x) for x in g["expected_raw"]], rtol=1e-14)
    np.testing.assert_allclose(u.pooled, [_frac(x) for x in g["expected_pooled_P3"]], rtol=1e-14)
    assert u.indices.tolist() == g["expected_indices_P3"][str(budget)]
    assert res.k_out[:, 0].tolist() == k[u.indices, 0].tolist()
    assert res.v_out[:, 0].tolist() == v[u.indices, 0].tolist()


def test_golden_hand_worked_pool1():
    g = _load_golden()
    q_win, k, v, cu, mask = _golden_inputs(g)
    res = oracle.compress_layer(q_win, k, v, cu, mask, [3], g["window"], 1, scale=g["scale"])
    u = res.units[(0, 0)]
    np.testing.assert_allclose(u.pooled, [_frac(x) for x in g["expected_raw"]], rtol=1e-14)
    assert u.indices.tolist() == g["expected_indices_P1"]["3"]


def test_golden_heads_are_summed():
    g = _load_golden()
    q_win, k, v, cu, mask = _golden_inputs(g, both_srh=True, head1_like_head0=True)
    res = oracle.compress_layer(q_win, k, v, cu, mask, [3], g["window"], 3, scale=g["scale"])
    u = res.units[(0, 0)]
    np.testing.assert_allclose(u.raw, [2 * _frac(x) for x in g["expected_raw"]], rtol=1e-14)
    np.testing.assert_allclose(u.pooled, [2 * _frac(x) for x in g["expected_pooled_P3"]], rtol=1e-14)
    assert u.indices.tolist() == g["expected_indices_P3"]["3"]


# ---------------------------------------------------------------------------
# brute force on tiny prompts
# ---------------------------------------------------------------------------
def _rand_case(rng, L, W, d, n_heads, scale_keys=1.0):
    q = rng.standard_normal((n_heads, W, d)) * 0.7
    k = rng.standard_normal((L, d)) * scale_keys
    return q, k


@pytest.mark.parametrize("seed", range(12))
def test_oracle_matches_brute_force(seed):
    rng = np.random.default_rng(seed)
    L = int(rng.integers(1, 65))
    W = int(rng.integers(1, 9))
    P = int(rng.choice([1, 3, 5, 7]))
    d = int(rng.choice([2, 4, 8]))
    nh = int(rng.integers(1, 4))
    budget = int(rng.integers(W, L + 6))
    q, k = _rand_case(rng, L, W, d, nh)
    scale = 1.0 / math.sqrt(d)
    res = oracle.compress_unit(q, k, W, P, budget, scale)
    raw_b, pooled_b, idx_b = brute_unit(q.tolist(), k.tolist(), W, P, budget, scale)
    np.testing.assert_allclose(res.raw, raw_b, rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(res.pooled, pooled_b, rtol=1e-12, atol=1e-15)
    assert res.indices.tolist() == idx_b


def test_brute_force_with_exact_ties():
    # Integer keys on a grid produce exact ties; both sides must break them
    # toward the lower position.
    rng = np.random.default_rng(7)
    L, W, d = 40, 4, 2
    k = rng.integers(0, 2, size=(L, d)).astype(np.float64)
    q = np.ones((2, W, d))
    for P in (1, 3):
        for budget in (W, W + 5, W + 17):
            res = oracle.compress_unit(q, k, W, P, budget, 0.5)
            _, _, idx_b = brute_unit(q.tolist(), k.tolist(), W, P, budget, 0.5)
            assert res.indices.tolist() == idx_b


# ---------------------------------------------------------------------------
# closed forms
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("P", [1, 3, 7])
def test_uniform_keys_closed_form(P):
    L, W, d, nh = 50, 6, 8, 3
    rng = np.random.default_rng(3)
    q = rng.standard_normal((nh, W, d))
    k = np.tile(rng.standard_normal(d), (L, 1))
    n = L - W
    res = oracle.compress_unit(q, k, W, P, budget=W + 10, scale=0.3, keep_attn=True)
    expect = nh * sum(1.0 / (n + w + 1) for w in range(W))
    np.testing.assert_allclose(res.raw, expect, rtol=1e-13)
    r = (P - 1) // 2
    counts = np.array([min(j, r) + min(n - 1 - j, r) + 1 for j in range(n)])
    np.testing.assert_allclose(res.pooled, expect * counts / P, rtol=1e-13)
    # interior positions tie exactly, so the lowest interior positions win
    assert res.indices[:10].tolist() == list(range(r, r + 10))
    assert res.indices[10:].tolist() == list(range(n, L))


# ---------------------------------------------------------------------------
# invariants
# ---------------------------------------------------------------------------
def test_softmax_rows_and_total_mass():
    rng = np.random.default_rng(11)
    L, W, d, nh = 300, 16, 32, 2
    q, k = _rand_case(rng, L, W, d, nh, scale_keys=2.0)
    res = oracle.compress_unit(q, k, W, 5, budget=64, scale=1 / math.sqrt(d), keep_attn=True)
    n = L - W
    window_mass = 0.0
    for A in res.attn:
        for w in range(W):
            p = L - W + w
            assert abs(A[w, : p + 1].sum() - 1.0) < 1e-12
            assert np.all(A[w, p + 1:] == 0.0)
        window_mass += A[:, n:].sum()
    assert abs(res.raw.sum() + window_mass - W * nh) < 1e-10


def test_selection_invariants():
    rng = np.random.default_rng(5)
    L, W, d = 500, 8, 16
    q, k = _rand_case(rng, L, W, d, 2, scale_keys=3.0)
    for budget in (W, W + 1, 100, L - 1, L, L + 40):
        res = oracle.compress_unit(q, k, W, 7, budget, 0.25)
        kept = min(budget, L)
        idx = res.indices
        assert len(idx) == kept
        assert np.all(np.diff(idx) > 0)
        assert idx[-W:].tolist() == list(range(L - W, L))
        n = L - W
        sel = set(idx[: kept - W].tolist())
        if 0 < res.k < n:
            tau = res.tau
            assert all(res.pooled[j] >= tau for j in sel)
            assert all(res.pooled[j] <= tau for j in range(n) if j not in sel)


def test_budget_edge_cases():
    rng = np.random.default_rng(9)
    q, k = _rand_case(rng, 20, 4, 4, 1)
    with pytest.raises(oracle.OracleError):
        oracle.compress_unit(q, k, 4, 3, budget=3, scale=0.5)
    assert oracle.compress_unit(q, k, 4, 3, budget=4, scale=0.5).indices.tolist() == [16, 17, 18, 19]
    assert oracle.compress_unit(q, k, 4, 3, budget=20, scale=0.5).indices.tolist() == list(range(20))
    assert oracle.compress_unit(q, k, 4, 3, budget=99, scale=0.5).indices.tolist() == list(range(20))
    # prompt no longer than the window: nothing scored, all kept
    q3, k3 = _rand_case(rng, 3, 4, 4, 1)
    r = oracle.compress_unit(q3, k3, 4, 3, budget=4, scale=0.5)
    assert r.indices.tolist() == [0, 1, 2] and r.raw.size == 0


def test_empty_srh_group_is_error():
    rng = np.random.default_rng(1)
    q_win = rng.standard_normal((1, 4, 2, 4))
    k = rng.standard_normal((10, 2, 4))
    mask = np.array([True, False, False, False])     # group 1 has no SRH head
    with pytest.raises(oracle.OracleError):
        oracle.compress_layer(q_win, k, k, [0, 10], mask, [4], 2, 3)


# ---------------------------------------------------------------------------
# all-heads mask == SnapKV-style group scoring via torch float64 routines
# ---------------------------------------------------------------------------
def _snapkv_group_torch(q_win, k, cu, W, P, budget, scale):
    """Independent route: torch softmax with a causal -inf mask, sum over
    heads and window, avg_pool1d(count_include_pad=True), stable sort."""
    out = {}
    B, Hq = q_win.shape[:2]
    Hkv = k.shape[1]
    G = Hq // Hkv
    for s in range(B):
        ks = torch.from_numpy(k[cu[s]:cu[s + 1]])
        L = ks.shape[0]
        n = L - W
        for g in range(Hkv):
            q = torch.from_numpy(q_win[s, g * G:(g + 1) * G])        # [G, W, d]
            logits = torch.einsum("hwd,ld->hwl", q, ks[:, g]) * scale
            pos = torch.arange(L)
            qpos = torch.arange(L - W, L)
            logits = logits.masked_fill(pos[None, None, :] > qpos[None, :, None], float("-inf"))
            attn = torch.softmax(logits, dim=-1)
            raw = attn[:, :, :n].sum(dim=(0, 1))
            pooled = torch.nn.functional.avg_pool1d(raw[None, None], P, 1, P // 2,
                                                    count_include_pad=True)[0, 0]
            kk = min(budget, L) - W
            order = torch.sort(-pooled, stable=True).indices[:kk]
            idx = torch.cat([torch.sort(order).values, torch.arange(n, L)])
            out[(s, g)] = (raw.numpy(), pooled.numpy(), idx.numpy())
    return out


def test_all_heads_equals_snapkv_torch():
    rng = np.random.default_rng(21)
    B, Hq, Hkv, W, d = 2, 8, 2, 8, 16
    lens = [300, 177]
    cu = np.concatenate([[0], np.cumsum(lens)])
    q_win = rng.standard_normal((B, Hq, W, d))
    k = rng.standard_normal((int(cu[-1]), Hkv, d)) * 1.5
    mask = np.ones(Hq, dtype=bool)
    res = oracle.compress_layer(q_win, k, k, cu, mask, [64, 40], W, 7, scale=0.25)
    ref = _snapkv_group_torch(q_win, k, cu, W, 7, 64, 0.25)
    ref2 = _snapkv_group_torch(q_win, k, cu, W, 7, 40, 0.25)
    for (s, g), u in res.units.items():
        raw_t, pooled_t, idx_t = (ref if s == 0 else ref2)[(s, g)]
        np.testing.assert_allclose(u.raw, raw_t, rtol=1e-12)
        np.testing.assert_allclose(u.pooled, pooled_t, rtol=1e-12)
        assert u.indices.tolist() == idx_t.tolist()


# ---------------------------------------------------------------------------
# planted mistakes: each must be caught by a pin above
# ---------------------------------------------------------------------------
def _mutant_no_causal(q_rows, k_unit, scale):
    q = np.asarray(q_rows, np.float64)
    k = np.asarray(k_unit, np.float64)
    z = (q @ k.T) * scale
    e = np.exp(z - z.max(axis=1, keepdims=True))
    return e / e.sum(axis=1, keepdims=True)


def _mutant_pool_exclude_pad(raw, P):
    n = len(raw)
    r = (P - 1) // 2
    return np.array([raw[max(0, j - r): j + r + 1].mean() for j in range(n)])


def _mutant_ties_high_index(pooled, k):
    order = sorted(range(len(pooled)), key=lambda j: (-float(pooled[j]), -j))
    return np.array(sorted(order[:k]), dtype=np.int64)


@pytest.mark.parametrize("name,target,mutant", [
    ("no causal mask", "window_attention", _mutant_no_causal),
    ("pool excludes padding", "pool_avg", _mutant_pool_exclude_pad),
    ("ties to higher index", "select_top", _mutant_ties_high_index),
])
def test_planted_mistakes_are_caught(monkeypatch, name, target, mutant):
    monkeypatch.setattr(O, target, mutant)
    failures = 0
    for fn in (lambda: test_golden_hand_worked_pool3(3),
               lambda: test_uniform_keys_closed_form(3),
               lambda: test_oracle_matches_brute_force(0),
               lambda: test_brute_force_with_exact_ties()):
        try:
            fn()
        except AssertionError:
            failures += 1
    assert failures > 0, f"planted mistake '{name}' went unnoticed"
