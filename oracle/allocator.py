"""Error-aware layer budget allocation (CompressKV Sec. 3.4, Eq. 4; the
bounds m = 32 and M = 3 * B_per_layer of Sec. 4) -- the oracle.

TEST INFRASTRUCTURE ONLY: imported by tests/ (and nothing on the product
path).  Plain Python floats (IEEE double), every sum taken in layer order.

Steps, in the paper's order:
  1. normalise the per-layer error scores:  e~_l = e_l / sum_k e_k  (Eq. 4;
     all-zero errors count as equal errors);
  2. give every layer the minimum m;
  3. distribute the remaining R = B_total - L*m in proportion to e~, no layer
     above M: a layer whose share would pass M - m gets exactly M - m and the
     rest is shared again over the others (water filling);
  4. round to integers so that the budgets add up to B_total exactly: every
     layer keeps floor(share), the missing units go to the largest fractional
     parts, ties to the lower layer index (reading R10).
Infeasible requests (L*m > B_total, B_total > L*M, m > M) raise ValueError.
"""
from __future__ import annotations

import math


def normalise_errors(errors):
    """Eq. 4 normalisation e~_l = e_l / sum_k e_k (uniform if every e_l = 0)."""
    errs = [float(e) for e in errors]
    for e in errs:
        if not (e >= 0.0) or math.isinf(e):
            raise ValueError("layer errors must be finite and >= 0")
    total = 0.0
    for e in errs:
        total += e
    if total == 0.0:
        return [1.0 / len(errs)] * len(errs)
    return [e / total for e in errs]


def water_fill(weights, amount, room):
    """Real shares x_l >= 0 with sum x_l = amount, x_l <= room, proportional
    to `weights` among the layers below `room`."""
    n = len(weights)
    share = [0.0] * n
    free = [True] * n
    left = float(amount)
    for _ in range(n):
        w_free = 0.0
        n_free = 0
        for l in range(n):
            if free[l]:
                w_free += weights[l]
                n_free += 1
        if n_free == 0:
            break
        give = [0.0] * n
        for l in range(n):
            if free[l]:
                give[l] = left * weights[l] / w_free if w_free > 0.0 else left / n_free
        over = [free[l] and give[l] > room for l in range(n)]
        if not any(over):
            for l in range(n):
                if free[l]:
                    share[l] = give[l]
            break
        for l in range(n):
            if over[l]:
                share[l] = float(room)
                left -= float(room)
                free[l] = False
    return share


def round_to_total(share, amount, room):
    """Integers b_l with sum b_l = amount: floor(share_l), then +1 to the
    largest fractional parts (ties to the lower index); if floors overshoot,
    -1 from the smallest fractional parts (ties to the higher index)."""
    n = len(share)
    base = [min(int(math.floor(x)), room) for x in share]
    frac = [share[l] - base[l] for l in range(n)]
    missing = amount - sum(base)
    if missing > 0:
        order = sorted((l for l in range(n) if base[l] < room), key=lambda l: (-frac[l], l))
        for l in order[:missing]:
            base[l] += 1
    elif missing < 0:
        order = sorted((l for l in range(n) if base[l] > 0), key=lambda l: (frac[l], -l))
        for l in order[:-missing]:
            base[l] -= 1
    return base


def allocate_layer_budgets(errors, total_budget: int, min_budget: int = 32,
                           max_budget: int | None = None):
    """Per-layer budgets (list of int) for `total_budget` KV pairs over the
    layers, following Sec. 3.4.  `max_budget` defaults to 3 * B_total / L
    (rounded down), the paper's M."""
    L = len(errors)
    if L < 1:
        raise ValueError("no layers")
    total_budget = int(total_budget)
    m = int(min_budget)
    M = int(max_budget) if max_budget is not None else (3 * total_budget) // L
    if m < 0 or M < m or L * m > total_budget or total_budget > L * M:
        raise ValueError("infeasible budget bounds")
    weights = normalise_errors(errors)
    rest = total_budget - L * m
    share = water_fill(weights, rest, M - m)
    extra = round_to_total(share, rest, M - m)
    return [m + x for x in extra]
