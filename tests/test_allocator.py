"""Error-aware layer budgets (CompressKV Sec. 3.4, Eq. 4; m = 32 and
M = 3 * B_per_layer from Sec. 4): the oracle pinned by a hand-worked example,
exact rational arithmetic and the allocation's invariants, then the
library's host implementation against the oracle, bit for bit."""
import json
import os
from fractions import Fraction

import numpy as np
import pytest

from oracle import allocator as A

HERE = os.path.dirname(__file__)


def _exact(errors, total, m, M, with_shares=False):
    """The same allocation in exact rational arithmetic (no floats at all):
    water filling with Fractions, then largest remainder, ties to the lower
    layer."""
    L = len(errors)
    e = [Fraction(x) for x in errors]
    s = sum(e)
    w = [x / s for x in e] if s else [Fraction(1, L)] * L
    rest, room = total - L * m, M - m
    share = [Fraction(0)] * L
    free = [True] * L
    left = Fraction(rest)
    while True:
        wf = sum(w[l] for l in range(L) if free[l])
        nf = sum(free)
        give = [(left * w[l] / wf if wf else left / nf) if free[l] else None for l in range(L)]
        over = [free[l] and give[l] > room for l in range(L)]
        if not any(over):
            for l in range(L):
                if free[l]:
                    share[l] = give[l]
            break
        for l in range(L):
            if over[l]:
                share[l], free[l] = Fraction(room), False
                left -= room
    base = [int(x) for x in share]  # shares are >= 0: int() is floor
    missing = rest - sum(base)
    order = sorted((l for l in range(L) if base[l] < room), key=lambda l: (-(share[l] - base[l]), l))
    for l in order[:missing]:
        base[l] += 1
    out = [m + b for b in base]
    return (out, share) if with_shares else out


def test_hand_worked_example():
    g = json.load(open(os.path.join(HERE, "golden", "allocator_hand_worked.json")))
    got = A.allocate_layer_budgets(g["layer_errors"], g["total_budget"], g["min_budget"],
                                   g["max_budget"])
    assert got == g["budgets"]


@pytest.mark.parametrize("seed", range(40))
def test_matches_exact_rational_allocation(seed):
    rng = np.random.default_rng(seed)
    L = int(rng.integers(1, 40))
    errors = [int(x) for x in rng.integers(0, 50, size=L)]  # small integers: exact in binary
    per = int(rng.integers(40, 400))
    total = L * per
    m = int(rng.integers(0, 40))
    M = max(m, int(rng.integers(per, 4 * per)))
    got = A.allocate_layer_budgets(errors, total, m, M)
    want, share = _exact(errors, total, m, M, with_shares=True)
    # The oracle computes its shares in IEEE double (the reading fixed for
    # the library); it equals the exact allocation except where exact
    # fractional parts tie, which double rounding may order either way.
    diff = [l for l in range(L) if got[l] != want[l]]
    assert sum(got) == total and len(diff) % 2 == 0
    fracs = {share[l] - int(share[l]) for l in diff}
    assert len(fracs) <= 1, (diff, fracs)


def test_equal_errors_split_evenly_lower_layers_first():
    assert A.allocate_layer_budgets([3.0] * 4, 402, 32, 200) == [101, 101, 100, 100]
    assert A.allocate_layer_budgets([0.0] * 3, 300, 32, 200) == [100, 100, 100]


def test_paper_defaults_and_bounds():
    rng = np.random.default_rng(7)
    err = rng.dirichlet([1.0] * 80)
    per = 328
    b = A.allocate_layer_budgets(err, 80 * per)  # m = 32, M = 3 * 328
    assert sum(b) == 80 * per
    assert min(b) >= 32 and max(b) <= 3 * per
    # the layer with the largest error is capped or at least as large as any other
    assert b[int(np.argmax(err))] == max(b)


@pytest.mark.parametrize("seed", range(20))
def test_invariants(seed):
    rng = np.random.default_rng(100 + seed)
    L = int(rng.integers(2, 100))
    err = rng.dirichlet([float(rng.uniform(0.2, 3.0))] * L) * float(rng.uniform(0.1, 1e4))
    per = int(rng.integers(32, 2048))
    total = L * per
    m, M = 32, 3 * per
    b = A.allocate_layer_budgets(err, total, m, M)
    assert sum(b) == total
    assert all(m <= x <= M for x in b)
    # monotone in the error: a larger error never gets a smaller budget
    order = np.argsort(err, kind="stable")
    bs = np.asarray(b)[order]
    assert np.all(np.diff(bs) >= -1)  # rounding may swap neighbours by one unit
    strict = [(i, j) for i in range(L) for j in range(L) if err[i] > err[j] * 1.01]
    assert all(b[i] >= b[j] for i, j in strict)
    # uncapped layers are proportional to the errors (within rounding)
    free = [l for l in range(L) if b[l] < M]
    if len(free) >= 2:
        rest = total - L * m - sum(M - m for l in range(L) if b[l] == M)
        wsum = sum(err[l] for l in free)
        for l in free:
            assert abs((b[l] - m) - rest * err[l] / wsum) <= 1.0 + 1e-6


def test_infeasible_requests():
    with pytest.raises(ValueError):
        A.allocate_layer_budgets([1, 1], 50, 32, 100)   # 2 * 32 > 50
    with pytest.raises(ValueError):
        A.allocate_layer_budgets([1, 1], 500, 32, 100)  # 500 > 2 * 100
    with pytest.raises(ValueError):
        A.allocate_layer_budgets([1, float("nan")], 100, 32, 100)


def test_planted_mistake_without_cap_is_caught():
    """A copy of the water filling that forgets the cap breaks the bound."""
    def no_cap(weights, amount, room):
        s = sum(weights)
        return [amount * w / s for w in weights]
    err = [1.0, 1.0, 1.0, 20.0]
    share = no_cap(A.normalise_errors(err), 400 - 4 * 32, 150 - 32)
    b = [32 + x for x in A.round_to_total(share, 400 - 4 * 32, 10 ** 9)]
    assert max(b) > 150
    assert max(A.allocate_layer_budgets(err, 400, 32, 150)) == 150


# --------------------------------------------------------------------------
# the library's host implementation (no GPU needed)
# --------------------------------------------------------------------------
def _lib():
    ckv = pytest.importorskip("paper_2606_24467_gb300")
    try:
        ckv.load()
    except Exception as exc:  # pragma: no cover - missing toolchain
        pytest.skip(f"library not built: {exc}")
    return ckv


@pytest.mark.parametrize("seed", range(60))
def test_library_matches_oracle_bit_for_bit(seed):
    ckv = _lib()
    rng = np.random.default_rng(1000 + seed)
    L = int(rng.integers(1, 128))
    err = rng.dirichlet([float(rng.uniform(0.1, 3.0))] * L) * float(rng.uniform(1e-3, 1e3))
    if seed % 7 == 0:
        err[rng.integers(0, L)] = 0.0
    per = int(rng.integers(16, 4096))
    total = L * per + int(rng.integers(0, L))
    m = int(rng.integers(0, per + 1))
    M = 0 if seed % 3 == 0 else max(int(np.ceil(total / L)), int(rng.integers(per, 4 * per)))
    want = A.allocate_layer_budgets(err, total, m, M if M > 0 else None)
    got = ckv.allocate_layer_budgets(err, total, m, M)
    assert got.tolist() == want


def test_library_error_codes():
    ckv = _lib()
    from paper_2606_24467_gb300 import compresskv as B
    with pytest.raises(ckv.CompressKVError) as e:
        ckv.allocate_layer_budgets([1.0, 1.0], 50, 32, 100)
    assert e.value.code == B.CKV_ERR_BUDGET
    with pytest.raises(ckv.CompressKVError) as e:
        ckv.allocate_layer_budgets([1.0, -1.0], 100, 32, 100)
    assert e.value.code == B.CKV_ERR_INVALID_ARG
