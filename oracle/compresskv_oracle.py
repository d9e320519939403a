"""CompressKV prefill-end compression oracle (float64, CPU).

TEST INFRASTRUCTURE ONLY.  This module is the slow, plain restatement of the
method that the CUDA path is checked against.  Only ``tests/``,
``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline / reference leg may
import it; the library (``paper_2606_24467_gb300``) never does, and this module
imports nothing from the library.

What it computes (CompressKV, Sec. 3.3 "Token Selection Driven by Semantic
Retrieval Heads", with the SnapKV-style local setting of Sec. 4
"Implementation Details": an observation window of the last ``W`` prompt
queries and 1-D pooling of width ``P`` across the token dimension):

for every sequence ``s`` and GQA KV group ``g`` (a *unit*):

1. ``S`` = the query heads of group ``g`` marked in the SRH mask (Sec. 3.3;
   heads are grouped contiguously, head ``h`` belongs to group ``h // G``).
2. For each ``h`` in ``S`` and window query ``w`` (prompt position
   ``p = L - W + w``): causal softmax attention over keys ``j <= p``,
   ``a[h, w, j] = exp(z_j - max z) / sum_j' exp(z_j' - max z)``,
   ``z_j = scale * <q[h, w], k[j]>``.
3. raw score of prefix token ``j < n = L - W``: the attention summed over the
   window queries and the SRH heads (Sec. 3.3: "summing over the observation
   window"; heads are combined by a sum, whose ranking equals the paper's
   average because ``|S|`` is fixed within a unit).
4. pooled score: average pooling of width ``P`` (stride 1, ``r = (P-1)/2``
   zeros of padding on each side, divisor ``P``) over the prefix scores; or,
   as an option, max pooling of each SRH head's window-summed attention
   over ``[j - r, j + r]`` before the heads are summed (``pool_heads``).
5. keep the ``k = min(B, L) - W`` prefix tokens with the largest pooled score
   (Sec. 3.3 "top N"; ties go to the lower position), plus the ``W`` window
   tokens, in ascending position order.
6. gather the retained K and V rows (Sec. 3.3: retained pairs are kept, the
   rest evicted).

Every step is written with plain numpy on float64 copies of the inputs; the
only library primitives are a dot product, ``exp`` and a sort.

Two selection scopes:

* per group (the default): steps 3-6 run per unit with the group's own SRH
  heads; a group with no SRH head is an error;
* per layer (Sec. 3.3 read literally: all heads of a layer share one set of
  retained indices chosen by the layer's SRH heads, whose pooled window
  scores are averaged): per sequence, every SRH head's attention (against
  its own group's keys) is summed over the window and pooled, the pooled
  vectors are summed over all SRH heads of the layer (the average times the
  fixed head count), the top ``k`` are kept and every KV group retains the
  same positions; groups without an SRH head are allowed.

Readings where the paper is silent (each also listed in the design notes): the softmax of window query ``w`` spans all causal keys
including earlier window keys, only prefix columns are scored; the budget
``B`` counts the window tokens; ``B < W`` is an error and ``B >= L`` keeps
everything; retained tokens are listed in ascending position.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np


class OracleError(ValueError):
    """Raised for inputs the method does not define (see module docstring)."""


# ---------------------------------------------------------------------------
# Step 1: SRH heads of a group (Sec. 3.3; GQA grouping)
# ---------------------------------------------------------------------------
def srh_heads(srh_mask, group: int, group_size: int) -> list[int]:
    """Query heads of KV group ``group`` that the SRH mask selects.

    Heads ``[group*G, (group+1)*G)`` share KV head ``group`` (contiguous GQA
    grouping).  Sec. 3.3 scores tokens with the selected heads only.
    """
    lo = group * group_size
    return [h for h in range(lo, lo + group_size) if bool(srh_mask[h])]


# ---------------------------------------------------------------------------
# Step 2: observation-window causal softmax (Sec. 3.3 / Sec. 4 window)
# ---------------------------------------------------------------------------
def window_attention(q_rows: np.ndarray, k_unit: np.ndarray, scale: float) -> np.ndarray:
    """Causal softmax attention of the last ``W`` queries of one head.

    q_rows: ``[W, d]`` window queries (row ``w`` sits at position ``L-W+w``).
    k_unit: ``[L, d]`` keys of the unit.
    Returns ``A`` of shape ``[W, L]``: ``A[w, j]`` is the attention weight of
    window query ``w`` on key ``j`` (zero for ``j > L-W+w``).
    """
    q = np.asarray(q_rows, dtype=np.float64)
    k = np.asarray(k_unit, dtype=np.float64)
    W = q.shape[0]
    L = k.shape[0]
    Z = (q @ k.T) * scale                      # [W, L] logits
    A = np.zeros((W, L), dtype=np.float64)
    for w in range(W):
        p = L - W + w                          # causal: keys 0..p only
        z = Z[w, : p + 1]
        e = np.exp(z - z.max())
        A[w, : p + 1] = e / e.sum()
    return A


# ---------------------------------------------------------------------------
# Step 3: raw prefix score (sum over window queries and SRH heads)
# ---------------------------------------------------------------------------
def raw_scores(attn_per_head: list[np.ndarray], n: int) -> np.ndarray:
    """Sum of the window attention over window queries and SRH heads, for the
    ``n`` prefix tokens (Sec. 3.3: the attention matrices of the selected heads
    are summed over the observation window)."""
    total = np.zeros(n, dtype=np.float64)
    for A in attn_per_head:
        total += A[:, :n].sum(axis=0)
    return total


# ---------------------------------------------------------------------------
# Step 4: 1-D average pooling over tokens (Sec. 3.3 / Sec. 4 kernel size)
# ---------------------------------------------------------------------------
def pool_avg(raw: np.ndarray, pool_width: int) -> np.ndarray:
    """Average pooling, stride 1, ``r = (P-1)//2`` zero padding per side,
    divisor ``P``; output has the input's length."""
    if pool_width < 1 or pool_width % 2 == 0:
        raise OracleError("pool width must be odd and >= 1")
    n = raw.shape[0]
    r = (pool_width - 1) // 2
    padded = np.concatenate([np.zeros(r), np.asarray(raw, np.float64), np.zeros(r)])
    out = np.zeros(n, dtype=np.float64)
    for j in range(n):
        out[j] = padded[j : j + pool_width].sum() / pool_width
    return out


def pool_max(raw: np.ndarray, pool_width: int) -> np.ndarray:
    """Max pooling, stride 1, over ``[j - r, j + r]`` clipped to the prefix
    (padding that never wins: scores are non-negative, so -inf and zero
    padding agree); output has the input's length."""
    if pool_width < 1 or pool_width % 2 == 0:
        raise OracleError("pool width must be odd and >= 1")
    raw = np.asarray(raw, np.float64)
    n = raw.shape[0]
    r = (pool_width - 1) // 2
    out = np.zeros(n, dtype=np.float64)
    for j in range(n):
        out[j] = raw[max(0, j - r): min(n, j + r + 1)].max()
    return out


def pool_heads(attn_per_head: list[np.ndarray], n: int, pool_width: int, pool_kind: str) -> np.ndarray:
    """Pooled score of a set of SRH heads (Sec. 3.3: pooling across the token
    dimension, then the heads' vectors combined by a sum).  Average pooling
    is linear, so it is applied to the head sum; max pooling is applied to
    each head's window-summed attention before the sum."""
    if pool_kind == "avg":
        return pool_avg(raw_scores(attn_per_head, n), pool_width)
    if pool_kind != "max":
        raise OracleError("pool kind must be 'avg' or 'max'")
    total = np.zeros(n, dtype=np.float64)
    for A in attn_per_head:
        total += pool_max(raw_scores([A], n), pool_width)
    return total


# ---------------------------------------------------------------------------
# Step 5: top-k prefix selection (Sec. 3.3 "top N")
# ---------------------------------------------------------------------------
def select_top(pooled: np.ndarray, k: int) -> np.ndarray:
    """Positions of the ``k`` largest pooled scores, ties to the lower
    position, returned in ascending position order."""
    n = pooled.shape[0]
    if k < 0 or k > n:
        raise OracleError("k out of range")
    order = sorted(range(n), key=lambda j: (-float(pooled[j]), j))
    return np.array(sorted(order[:k]), dtype=np.int64)


def kth_value(pooled: np.ndarray, k: int) -> float:
    """The k-th largest pooled score (``tau``); NaN when ``k == 0``."""
    if k <= 0:
        return float("nan")
    return float(np.sort(np.asarray(pooled, np.float64))[::-1][k - 1])


# ---------------------------------------------------------------------------
# Budget rule (reading of Sec. 3.4 / Sec. 4: budgets count the window tokens)
# ---------------------------------------------------------------------------
def kept_count(budget: int, length: int, window: int) -> int:
    """Number of tokens a sequence of ``length`` keeps under ``budget``."""
    if budget < window:
        raise OracleError("budget smaller than the observation window")
    return min(budget, length)


# ---------------------------------------------------------------------------
# One unit = (sequence, KV group)
# ---------------------------------------------------------------------------
@dataclass
class UnitResult:
    heads: list
    raw: np.ndarray          # [n]
    pooled: np.ndarray       # [n]
    k: int                   # selected prefix tokens
    tau: float               # k-th largest pooled score (NaN if k == 0)
    indices: np.ndarray      # [min(B, L)] ascending positions within the sequence
    attn: list = field(default_factory=list)  # per SRH head [W, L]


def compress_unit(q_heads: np.ndarray, k_unit: np.ndarray, window: int, pool_width: int,
                  budget: int, scale: float, keep_attn: bool = False,
                  pool_kind: str = "avg") -> UnitResult:
    """Steps 2-5 for one unit.

    q_heads: ``[|S|, W, d]`` window queries of the unit's SRH heads.
    k_unit:  ``[L, d]``.
    """
    L = k_unit.shape[0]
    W = window
    kept = kept_count(budget, L, W)
    if L <= W:
        # The whole prompt is inside the window: nothing to score, all kept.
        return UnitResult([], np.zeros(0), np.zeros(0), 0, float("nan"),
                          np.arange(L, dtype=np.int64))
    n = L - W
    if q_heads.shape[0] == 0:
        raise OracleError("KV group without any SRH head")
    attn = [window_attention(q_heads[i], k_unit, scale) for i in range(q_heads.shape[0])]
    raw = raw_scores(attn, n)
    pooled = pool_avg(raw, pool_width) if pool_kind == "avg" else pool_heads(attn, n, pool_width,
                                                                            pool_kind)
    k = kept - W
    sel = select_top(pooled, k)
    idx = np.concatenate([sel, np.arange(n, L, dtype=np.int64)])
    return UnitResult([], raw, pooled, k, kth_value(pooled, k), idx, attn if keep_attn else [])


# ---------------------------------------------------------------------------
# Softmax denominators of the window queries (the log-sum-exp a prefill
# attention kernel returns; the library's given-LSE entry point takes it)
# ---------------------------------------------------------------------------
def window_lse(q_win, k, cu_seqlens, window: int, scale: float | None = None) -> np.ndarray:
    """``[B, H_q, W]`` natural-log ``log sum_{j <= p} exp(z_j)`` of every
    window query (``p = L_s - W + w``, ``z_j = scale * <q, k_j>``, keys of
    the head's KV group); 0 where the sequence has no such position."""
    q_win = np.asarray(q_win, np.float64)
    k = np.asarray(k, np.float64)
    cu = [int(x) for x in cu_seqlens]
    B, H_q, W, d = q_win.shape
    G = H_q // k.shape[1]
    if scale is None:
        scale = default_scale(d)
    out = np.zeros((B, H_q, W), dtype=np.float64)
    for s in range(B):
        L = cu[s + 1] - cu[s]
        for h in range(H_q):
            ku = k[cu[s]:cu[s + 1], h // G]
            for w in range(W):
                p = L - W + w
                if p < 0:
                    continue
                z = scale * (ku[:p + 1] @ q_win[s, h, w])
                m = z.max()
                out[s, h, w] = m + math.log(np.exp(z - m).sum())
    return out


# ---------------------------------------------------------------------------
# One layer over a packed (cu_seqlens) batch, in the library's output layout
# ---------------------------------------------------------------------------
@dataclass
class SharedSelection:
    """Per-layer (shared) selection of one sequence."""
    pooled: np.ndarray       # [n] pooled scores summed over the layer's SRH heads
    k: int
    tau: float
    indices: np.ndarray      # [min(B, L)] ascending positions, the same for every group


@dataclass
class LayerResult:
    units: dict              # (s, g) -> UnitResult
    raw: np.ndarray          # [H_kv, sum_s n_s] float64
    pooled: np.ndarray       # [H_kv, sum_s n_s]
    indices: np.ndarray      # [H_kv, sum_s kept_s] int64
    cu_out: np.ndarray       # [B+1]
    cu_prefix: np.ndarray    # [B+1] offsets of the prefix scores
    k_out: np.ndarray        # [sum_s kept_s, H_kv, d]  (input dtype)
    v_out: np.ndarray
    shared: dict = field(default_factory=dict)  # s -> SharedSelection (layer scope)


def default_scale(head_dim: int) -> float:
    return 1.0 / math.sqrt(head_dim)


def compress_layer(q_win, k, v, cu_seqlens, srh_mask, budgets, window: int,
                   pool_width: int, scale: float | None = None,
                   keep_attn: bool = False, selection: str = "group",
                   pool_kind: str = "avg") -> LayerResult:
    """Oracle of one layer's compression.

    q_win: ``[B, H_q, W, d]`` window queries (position ``L_s - W + w``).
    k, v:  ``[T, H_kv, d]`` packed keys/values, sequence ``s`` at rows
           ``cu_seqlens[s] : cu_seqlens[s+1]``.
    srh_mask: ``[H_q]`` booleans; budgets: ``[B]`` ints (per sequence).
    selection: ``"group"`` or ``"layer"`` (see the module docstring).
    pool_kind: ``"avg"`` or ``"max"`` (``pool_heads``).
    """
    if selection not in ("group", "layer"):
        raise OracleError("selection must be 'group' or 'layer'")
    q_win = np.asarray(q_win)
    k = np.asarray(k)
    v = np.asarray(v)
    cu = [int(x) for x in cu_seqlens]
    B = len(cu) - 1
    H_q = q_win.shape[1]
    H_kv = k.shape[1]
    if H_q % H_kv != 0:
        raise OracleError("query heads must be a multiple of KV heads")
    G = H_q // H_kv
    if scale is None:
        scale = default_scale(k.shape[2])
    lengths = [cu[s + 1] - cu[s] for s in range(B)]
    n_s = [max(Ls - window, 0) for Ls in lengths]
    kept_s = [kept_count(int(budgets[s]), lengths[s], window) for s in range(B)]
    cu_prefix = np.concatenate([[0], np.cumsum(n_s)]).astype(np.int64)
    cu_out = np.concatenate([[0], np.cumsum(kept_s)]).astype(np.int64)
    raw = np.zeros((H_kv, int(cu_prefix[-1])), dtype=np.float64)
    pooled = np.zeros_like(raw)
    indices = np.zeros((H_kv, int(cu_out[-1])), dtype=np.int64)
    k_out = np.zeros((int(cu_out[-1]), H_kv, k.shape[2]), dtype=k.dtype)
    v_out = np.zeros((int(cu_out[-1]), H_kv, v.shape[2]), dtype=v.dtype)
    q64 = q_win.astype(np.float64)
    k64 = k.astype(np.float64)
    units = {}
    shared = {}
    if selection == "layer":
        if not any(srh_heads(srh_mask, g, G) for g in range(H_kv)) and any(
                Ls > window for Ls in lengths):
            raise OracleError("the layer has no SRH head")
        for s in range(B):
            Ls, n, kept = lengths[s], n_s[s], kept_s[s]
            layer_pooled = np.zeros(n, dtype=np.float64)
            for g in range(H_kv):
                heads = srh_heads(srh_mask, g, G)
                ku = k64[cu[s]:cu[s + 1], g]
                if heads and Ls > window:
                    # Sec. 3.3: each head's window-summed attention is pooled,
                    # then the heads' vectors are combined
                    attn = [window_attention(q64[s, h], ku, scale) for h in heads]
                    for A in attn:
                        layer_pooled += pool_heads([A], n, pool_width, pool_kind)
                    g_raw = raw_scores(attn, n)
                    g_pooled = pool_heads(attn, n, pool_width, pool_kind)
                else:
                    attn, g_raw, g_pooled = [], np.zeros(n), np.zeros(n)
                units[(s, g)] = UnitResult(heads, g_raw, g_pooled, 0, float("nan"),
                                           np.zeros(0, dtype=np.int64),
                                           attn if keep_attn else [])
                raw[g, cu_prefix[s]:cu_prefix[s + 1]] = g_raw
                pooled[g, cu_prefix[s]:cu_prefix[s + 1]] = g_pooled
            if Ls <= window:
                idx = np.arange(Ls, dtype=np.int64)
                kk, tau = 0, float("nan")
            else:
                kk = kept - window
                sel = select_top(layer_pooled, kk)
                idx = np.concatenate([sel, np.arange(n, Ls, dtype=np.int64)])
                tau = kth_value(layer_pooled, kk)
            shared[s] = SharedSelection(layer_pooled, kk, tau, idx)
            for g in range(H_kv):
                units[(s, g)].k, units[(s, g)].tau, units[(s, g)].indices = kk, tau, idx
                indices[g, cu_out[s]:cu_out[s + 1]] = idx
                rows = cu[s] + idx
                k_out[cu_out[s]:cu_out[s + 1], g] = k[rows, g]
                v_out[cu_out[s]:cu_out[s + 1], g] = v[rows, g]
        return LayerResult(units, raw, pooled, indices, cu_out, cu_prefix, k_out, v_out, shared)
    for s in range(B):
        for g in range(H_kv):
            heads = srh_heads(srh_mask, g, G)
            if not heads and lengths[s] > window:
                raise OracleError(f"KV group {g} has no SRH head")
            qh = q64[s, heads] if heads else np.zeros((0, window, k.shape[2]))
            ku = k64[cu[s]:cu[s + 1], g]
            res = compress_unit(qh, ku, window, pool_width, int(budgets[s]), scale, keep_attn,
                                pool_kind)
            res.heads = heads
            units[(s, g)] = res
            raw[g, cu_prefix[s]:cu_prefix[s + 1]] = res.raw
            pooled[g, cu_prefix[s]:cu_prefix[s + 1]] = res.pooled
            indices[g, cu_out[s]:cu_out[s + 1]] = res.indices
            rows = cu[s] + res.indices
            k_out[cu_out[s]:cu_out[s + 1], g] = k[rows, g]
            v_out[cu_out[s]:cu_out[s + 1], g] = v[rows, g]
    return LayerResult(units, raw, pooled, indices, cu_out, cu_prefix, k_out, v_out)


# ---------------------------------------------------------------------------
# Head-level budgets (Sec. 4.6: the token selection combined with a budget
# per head group from a head-level allocator), outputs packed group-major
# ---------------------------------------------------------------------------
@dataclass
class HeadBudgetResult:
    units: dict              # (s, g) -> UnitResult, each with its own budget
    cu_out: np.ndarray       # [H_kv, B+1] first output row of (s, g); end of group g
    indices: np.ndarray      # [rows] int64
    k_out: np.ndarray        # [rows, d]
    v_out: np.ndarray


def compress_layer_head_budgets(q_win, k, v, cu_seqlens, srh_mask, group_budgets, window: int,
                                pool_width: int, scale: float | None = None) -> HeadBudgetResult:
    """Per (sequence, group) selection with budget ``group_budgets[s][g]``;
    group g's compressed sequences follow each other, then group g+1's."""
    q_win = np.asarray(q_win)
    k = np.asarray(k)
    v = np.asarray(v)
    cu = [int(x) for x in cu_seqlens]
    B = len(cu) - 1
    H_q, H_kv = q_win.shape[1], k.shape[1]
    G = H_q // H_kv
    if scale is None:
        scale = default_scale(k.shape[2])
    gb = np.asarray(group_budgets).reshape(B, H_kv)
    q64, k64 = q_win.astype(np.float64), k.astype(np.float64)
    units, idx_parts, k_parts, v_parts = {}, [], [], []
    cu_out = np.zeros((H_kv, B + 1), dtype=np.int64)
    row = 0
    for g in range(H_kv):
        heads = srh_heads(srh_mask, g, G)
        for s in range(B):
            cu_out[g, s] = row
            L = cu[s + 1] - cu[s]
            if not heads and L > window:
                raise OracleError(f"KV group {g} has no SRH head")
            qh = q64[s, heads] if heads else np.zeros((0, window, k.shape[2]))
            res = compress_unit(qh, k64[cu[s]:cu[s + 1], g], window, pool_width, int(gb[s, g]),
                                scale)
            res.heads = heads
            units[(s, g)] = res
            idx_parts.append(res.indices)
            k_parts.append(k[cu[s] + res.indices, g])
            v_parts.append(v[cu[s] + res.indices, g])
            row += len(res.indices)
        cu_out[g, B] = row
    d = k.shape[2]
    cat = lambda parts, dt: (np.concatenate(parts) if parts else np.zeros((0, d), dt))
    return HeadBudgetResult(units, cu_out,
                            np.concatenate(idx_parts) if idx_parts else np.zeros(0, np.int64),
                            cat(k_parts, k.dtype), cat(v_parts, v.dtype))

