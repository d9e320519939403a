"""Seeded synthetic inputs shared by the tests, the bench and the oracle checks.

This module only draws inputs; it holds none of the method's arithmetic (no
attention, pooling or selection).  Recipe (stated once more in the design
notes):

* window queries ``q_win[B, H_q, W, d]`` and keys ``k[T, H_kv, d]`` are
  i.i.d. N(0, 1)/sqrt(128), values ``v`` are N(0, 1); drawn in float32 and
  cast to the workload dtype (the oracle reads the cast values);
* attention sinks: tokens 0-3 of every sequence get the key
  ``gamma * u_g`` where ``u_g`` is the unit mean direction of all ``G*W``
  window queries of the group and ``gamma`` makes their mean scaled logit +4;
* needles: positions drawn without replacement from ``[4, n - P)`` with
  spacing >= P; key ``gain * |k| * (0.8 c_g + 0.6 r)`` where ``c_g`` is the
  unit mean direction of the group's SRH window queries, ``r`` a random unit
  vector orthogonal to it and ``|k|`` the replaced key's norm (cosine 0.8);
* SRH masks: per layer and group, a seeded count in ``srh_per_group`` of
  heads chosen without replacement;
* budgets: per-layer shares drawn from a Dirichlet, a floor of ``W + 16``,
  largest-remainder rounding; see ``layer_budgets``.
"""
from __future__ import annotations

import math

import numpy as np
import torch

from .configs import Workload

_TORCH_DTYPES = {"fp16": torch.float16, "bf16": torch.bfloat16, "fp32": torch.float32}


def torch_dtype(name: str) -> torch.dtype:
    return _TORCH_DTYPES[name]


def _rng(cfg: Workload, *stream) -> np.random.Generator:
    return np.random.default_rng([cfg.seed, *stream])


def _torch_gen(cfg: Workload, layer: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(cfg.seed * 1_000_003 + layer * 7919 + 17)
    return g


# ---------------------------------------------------------------------------
# Host-side (small) draws
# ---------------------------------------------------------------------------
def sequence_lengths(cfg: Workload) -> list[int]:
    if cfg.length_range is None:
        return [cfg.seq_len] * cfg.batch
    lo, hi = cfg.length_range
    return [int(x) for x in _rng(cfg, 1).integers(lo, hi + 1, size=cfg.batch)]


def cu_seqlens(lengths) -> np.ndarray:
    return np.concatenate([[0], np.cumsum(lengths)]).astype(np.int32)


def srh_masks(cfg: Workload) -> np.ndarray:
    """bool ``[n_layers, H_q]``."""
    rng = _rng(cfg, 2)
    G = cfg.group_size
    out = np.zeros((cfg.n_layers, cfg.num_q_heads), dtype=bool)
    lo, hi = cfg.srh_per_group
    for l in range(cfg.n_layers):
        for g in range(cfg.num_kv_heads):
            c = int(rng.integers(lo, hi + 1))
            heads = rng.choice(G, size=min(c, G), replace=False)
            out[l, g * G + heads] = True
    return out


def _largest_remainder(real: np.ndarray, total: int) -> np.ndarray:
    base = np.floor(real).astype(np.int64)
    rest = total - int(base.sum())
    if rest > 0:
        frac = real - base
        order = sorted(range(len(real)), key=lambda i: (-frac[i], i))
        for i in order[:rest]:
            base[i] += 1
    return base


def _split(shares: np.ndarray, mean: float, floor: int) -> np.ndarray:
    n = len(shares)
    total = int(round(mean * n))
    extra = max(total - floor * n, 0)
    return floor + _largest_remainder(shares * extra, extra)


def _split_capped(weights: np.ndarray, mean: float, floor: int, cap: int) -> np.ndarray:
    """Floor per layer, the rest in proportion to ``weights``, no layer above
    ``cap`` (overflow goes to the layers still below it)."""
    n = len(weights)
    extra = float(max(int(round(mean * n)) - floor * n, 0))
    alloc = np.zeros(n)
    free = np.ones(n, dtype=bool)
    room = float(cap - floor)
    for _ in range(n):
        w = np.where(free, weights, 0.0)
        if extra <= 1e-9 or w.sum() <= 0:
            break
        give = extra * w / w.sum()
        over = free & (alloc + give > room)
        if not over.any():
            alloc += give
            extra = 0.0
            break
        extra -= float((room - alloc[over]).sum())
        alloc[over] = room
        free &= ~over
    total_extra = int(round(alloc.sum()))
    return floor + _largest_remainder(alloc, total_extra)


def layer_budgets(cfg: Workload, lengths) -> np.ndarray:
    """int32 ``[n_layers, batch]``; every budget is >= W and <= the length
    (a sequence shorter than W keeps itself whole, so W is used there)."""
    rng = _rng(cfg, 3)
    nl, W = cfg.n_layers, cfg.window
    floor = W + 16
    out = np.zeros((nl, len(lengths)), dtype=np.int64)
    if cfg.budget_rule == "fixed":
        out[:] = int(cfg.budget_mean)
    elif cfg.budget_rule == "dirichlet":
        shares = rng.dirichlet([cfg.budget_alpha] * nl)
        out[:] = _split(shares, cfg.budget_mean, floor)[:, None]
    elif cfg.budget_rule == "frac_dirichlet":
        shares = rng.dirichlet([cfg.budget_alpha] * nl)
        for s, Ls in enumerate(lengths):
            out[:, s] = _split(shares, max(round(cfg.budget_mean * Ls), floor), floor)
    elif cfg.budget_rule == "error_profile":
        err = rng.dirichlet([cfg.budget_alpha] * nl)
        floor = max(32, floor)
        cap = 3 * int(cfg.budget_mean)
        out[:] = _split_capped(err, cfg.budget_mean, floor, cap)[:, None]
    else:
        raise ValueError(cfg.budget_rule)
    for s, Ls in enumerate(lengths):
        out[:, s] = np.clip(out[:, s], W, max(Ls, W))
    return out.astype(np.int32)


def needle_positions(cfg: Workload, layer: int, seq: int, group: int, n_prefix: int,
                     count: int | None = None) -> list[int]:
    count = cfg.needles_per_group if count is None else count
    lo, hi = 4, n_prefix - cfg.pool_width
    if hi <= lo or count <= 0:
        return []
    rng = _rng(cfg, 4, layer, seq, group)
    cand = rng.permutation(np.arange(lo, hi))
    chosen: list[int] = []
    for c in cand:
        c = int(c)
        if all(abs(c - x) >= cfg.pool_width for x in chosen):
            chosen.append(c)
            if len(chosen) == count:
                break
    return sorted(chosen)


# ---------------------------------------------------------------------------
# One layer's tensors
# ---------------------------------------------------------------------------
def make_layer(cfg: Workload, layer: int, device="cpu", lengths=None, masks=None,
               budgets=None, needle_gain: float = 1.0, sinks: bool = True,
               streaming_heads: bool = False) -> dict:
    """Tensors of one layer.

    Returns a dict with ``q_win [B, H_q, W, d]``, ``k``/``v [T, H_kv, d]`` (in
    the workload dtype, on ``device``), ``cu_seqlens`` (int32 numpy),
    ``srh_mask`` (bool numpy ``[H_q]``), ``budgets`` (int32 numpy ``[B]``)
    and ``needles`` ({(s, g): positions}).

    ``streaming_heads=True`` turns the non-SRH heads of every group into
    streaming heads that attend the first tokens and the end of the prompt
    (the head type the paper's SRH selection is built to outvote).
    """
    lengths = sequence_lengths(cfg) if lengths is None else list(lengths)
    masks = srh_masks(cfg) if masks is None else masks
    budgets = layer_budgets(cfg, lengths) if budgets is None else budgets
    mask = np.asarray(masks[layer], dtype=bool)
    bud = np.asarray(budgets[layer], dtype=np.int32)
    B, Hq, Hkv, d, W = len(lengths), cfg.num_q_heads, cfg.num_kv_heads, cfg.head_dim, cfg.window
    G = Hq // Hkv
    cu = cu_seqlens(lengths)
    T = int(cu[-1])
    gen = _torch_gen(cfg, layer, device)
    f32 = dict(device=device, dtype=torch.float32)
    inv = 1.0 / math.sqrt(128.0)
    q = torch.randn((B, Hq, W, d), generator=gen, **f32) * inv
    k = torch.randn((T, Hkv, d), generator=gen, **f32) * inv
    v = torch.randn((T, Hkv, d), generator=gen, **f32)
    scale = 1.0 / math.sqrt(d)
    needles = {}
    for s in range(B):
        Ls = int(lengths[s])
        base = int(cu[s])
        n_prefix = Ls - W
        for g in range(Hkv):
            heads = list(range(g * G, (g + 1) * G))
            srh = [h for h in heads if mask[h]]
            others = [h for h in heads if not mask[h]]
            c = None
            if srh:
                qs = q[s, srh].reshape(-1, d).mean(0)
                c = qs / qs.norm().clamp_min(1e-12)
            pos = needle_positions(cfg, layer, s, g, max(n_prefix, 0)) if srh else []
            if pos and needle_gain > 0:
                gpos = torch.tensor([base + p for p in pos], device=device, dtype=torch.long)
                r = torch.randn((len(pos), d), generator=gen, **f32)
                r = r - (r @ c)[:, None] * c[None, :]
                r = r / r.norm(dim=1, keepdim=True).clamp_min(1e-12)
                norms = k[gpos, g].norm(dim=1, keepdim=True)
                k[gpos, g] = needle_gain * norms * (0.8 * c[None, :] + 0.6 * r)
            if streaming_heads and others and c is not None and Ls > 0:
                # Sink-and-recency heads: their queries point along u; the sinks and the
                # last ``recent`` prefix tokens carry keys along u, so these
                # heads put their mass on the start and the end of the prompt.
                # u is orthogonal to every SRH window query, so the SRH heads
                # do not see the sink/recency keys at all.
                basis, _ = torch.linalg.qr(q[s, srh].reshape(-1, d).T)
                u = torch.randn(d, generator=gen, **f32)
                u = u - basis @ (basis.T @ u)
                u = u / u.norm().clamp_min(1e-12)
                noise = torch.randn((len(others), W, d), generator=gen, **f32) * 0.1 * inv
                q[s, others] = u + noise
                ns = min(4, Ls)
                k[base:base + ns, g] = (8.0 / scale) * u
                recent = min(max(n_prefix, 0), 2 * (int(bud[s]) - W) + W)
                if recent > 0:
                    lo = base + n_prefix - recent
                    k[lo:base + n_prefix, g] = (5.3 / scale) * u + k[lo:base + n_prefix, g]
            elif sinks and Ls > 0:
                qg = q[s, heads].reshape(-1, d)
                mean_all = qg.mean(0)
                u = mean_all / mean_all.norm().clamp_min(1e-12)
                gamma = 4.0 / (scale * float((qg @ u).mean().clamp_min(1e-6)))
                ns = min(4, Ls)
                k[base:base + ns, g] = gamma * u
            needles[(s, g)] = pos
    dt = torch_dtype(cfg.dtype)
    return dict(q_win=q.to(dt), k=k.to(dt), v=v.to(dt), cu_seqlens=cu, srh_mask=mask,
                budgets=bud, needles=needles, lengths=list(lengths))
