"""Behaviour of the oracle on the synthetic workloads (Sec. 1 / Sec. 2 motivation).

Streaming heads attend the first and the last tokens of a prompt; when they
are summed with the other heads of a GQA group they push mid-prompt evidence
out of the cache.  Scoring with the SRH heads only keeps it.  The generator
plants needles aligned with the SRH queries; these tests check that the
oracle recovers them, and that all-heads scoring loses them once the other
heads are made streaming-like.
"""
import numpy as np

import oracle
import workloads as wl


def _recovery(cfg, gain, streaming, all_heads):
    bud = np.full((1, 1), cfg.window + 7 * cfg.needles_per_group + 16, np.int32)
    d = wl.make_layer(cfg, 0, budgets=bud, needle_gain=gain, streaming_heads=streaming)
    q = d["q_win"].float().numpy()
    k = d["k"].float().numpy()
    mask = np.ones(cfg.num_q_heads, bool) if all_heads else d["srh_mask"]
    res = oracle.compress_layer(q, k, k, d["cu_seqlens"], mask, d["budgets"],
                                cfg.window, cfg.pool_width)
    hits = []
    for g in range(cfg.num_kv_heads):
        kept = set(res.units[(0, g)].indices.tolist())
        hits.append(sum(p in kept for p in d["needles"][(0, g)]))
    return hits


CFG = wl.get("c1").scaled(seq_len=2048, srh_per_group=(1, 1))


def test_srh_scoring_recovers_needles():
    hits = _recovery(CFG, gain=100.0, streaming=False, all_heads=False)
    assert min(hits) >= 15, hits


def test_srh_scoring_beats_all_heads_under_streaming_heads():
    srh = _recovery(CFG, gain=100.0, streaming=True, all_heads=False)
    allh = _recovery(CFG, gain=100.0, streaming=True, all_heads=True)
    assert min(srh) >= 15, srh
    assert max(allh) <= 8, allh
    assert sum(srh) >= 2 * sum(allh) + 64
