"""Pure-Python brute force of the CompressKV selection for tiny prompts.

TEST INFRASTRUCTURE ONLY (same rule as ``compresskv_oracle``).  It restates
Sec. 3.3 (window scoring, pooling, top-N retention) with explicit loops,
``math.exp`` and ``math.fsum`` over Python floats, and a full sort for the
top-k, so that the numpy oracle can be checked against an implementation
that shares none of its code.  Meant for prompts of at most a few dozen
tokens.
"""
from __future__ import annotations

import math


def brute_unit(q_heads, k_unit, window, pool_width, budget, scale, pool_kind="avg"):
    """q_heads: list over SRH heads of W lists of d floats; k_unit: L lists of
    d floats.  pool_kind "avg" pools the heads' sum; "max" takes, per head,
    the largest window-summed attention within the pooling window and sums
    those over the heads.  Returns (raw, pooled, indices) as Python lists."""
    L = len(k_unit)
    W = window
    if budget < W:
        raise ValueError("budget smaller than window")
    if L <= W:
        return [], [], list(range(L))
    n = L - W
    raw = [0.0] * n
    terms = [[] for _ in range(n)]
    head_terms = [[[] for _ in range(n)] for _ in q_heads]
    for hi, head in enumerate(q_heads):
        for w in range(W):
            p = L - W + w
            logits = []
            for j in range(p + 1):
                logits.append(scale * math.fsum(a * b for a, b in zip(head[w], k_unit[j])))
            top = max(logits)
            exps = [math.exp(x - top) for x in logits]
            z = math.fsum(exps)
            for j in range(n):
                terms[j].append(exps[j] / z)
                head_terms[hi][j].append(exps[j] / z)
    for j in range(n):
        raw[j] = math.fsum(terms[j])
    r = (pool_width - 1) // 2
    pooled = []
    if pool_kind == "max":
        head_raw = [[math.fsum(ht[j]) for j in range(n)] for ht in head_terms]
        for j in range(n):
            best = []
            for hr in head_raw:
                m = None
                for t in range(-r, r + 1):
                    if 0 <= j + t < n and (m is None or hr[j + t] > m):
                        m = hr[j + t]
                best.append(m)
            pooled.append(math.fsum(best))
    else:
        for j in range(n):
            acc = []
            for t in range(-r, r + 1):
                if 0 <= j + t < n:
                    acc.append(raw[j + t])
            pooled.append(math.fsum(acc) / pool_width)
    k = min(budget, L) - W
    ranked = sorted(range(n), key=lambda j: (-pooled[j], j))
    chosen = sorted(ranked[:k])
    return raw, pooled, chosen + list(range(n, L))


def brute_layer_shared(q_heads_per_group, k_per_group, window, pool_width, budget, scale):
    """Layer-shared selection (Sec. 3.3 read literally) by brute force: every
    group's SRH heads are scored against that group's keys, the pooled
    vectors of all groups are added (math.fsum, group order) and one top-k
    with ties to the lower position is kept for the whole layer.
    q_heads_per_group: per group, a list over its SRH heads (possibly empty)
    of W lists of d floats; k_per_group: per group, L lists of d floats.
    Returns (pooled_sum, indices)."""
    L = len(k_per_group[0])
    W = window
    if budget < W:
        raise ValueError("budget smaller than window")
    if L <= W:
        return [], list(range(L))
    n = L - W
    pooled_per_group = []
    for heads, keys in zip(q_heads_per_group, k_per_group):
        if heads:
            _, pooled, _ = brute_unit(heads, keys, window, pool_width, budget, scale)
            pooled_per_group.append(pooled)
    total = [math.fsum(pg[j] for pg in pooled_per_group) for j in range(n)]
    k = min(budget, L) - W
    ranked = sorted(range(n), key=lambda j: (-total[j], j))
    return total, sorted(ranked[:k]) + list(range(n, L))
