"""Acceptance checks of a device result against the oracle.

TEST INFRASTRUCTURE ONLY (imported by tests/, __graft_entry__.smoke() and
bench.py's parity spot check).

Tolerances (per-token scores and index sets):
* raw and pooled scores: |gpu - oracle| <= 1e-3 * |oracle| + 1e-5;
* retained index sets: identical, except for prefix tokens whose oracle
  pooled score lies within 1e-3 relative of the k-th largest oracle pooled
  score (a near-tie that fp32 may order either way);
* the W window positions are always the last W entries;
* gathered K/V rows: bit-exact copies of the input rows at the device's own
  indices.
"""
from __future__ import annotations

import numpy as np

RTOL = 1e-3
ATOL = 1e-5


def check_scores(name, gpu, ref, rtol=RTOL, atol=ATOL):
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    assert gpu.shape == ref.shape, f"{name}: shape {gpu.shape} vs {ref.shape}"
    err = np.abs(gpu - ref)
    bad = ~(err <= rtol * np.abs(ref) + atol)  # NaN or inf anywhere fails
    if bad.any():
        i = np.unravel_index(np.argmax(np.where(bad, np.nan_to_num(err, nan=np.inf), -np.inf)),
                             err.shape)
        raise AssertionError(f"{name}: {int(bad.sum())} of {bad.size} outside tolerance; "
                             f"worst at {i}: gpu={gpu[i]!r} oracle={ref[i]!r}")


def check_unit_indices(gpu_idx, unit, L, window, rel=RTOL, where=""):
    """gpu_idx: the device's retained positions of one unit (1-D)."""
    gpu_idx = np.asarray(gpu_idx, np.int64)
    ref_idx = unit.indices
    assert gpu_idx.shape == ref_idx.shape, f"{where}: {gpu_idx.shape} kept vs {ref_idx.shape}"
    if gpu_idx.size:
        assert np.all(np.diff(gpu_idx) > 0), f"{where}: indices not strictly ascending"
        assert gpu_idx.min() >= 0 and gpu_idx.max() < L, f"{where}: index out of range"
    kept = gpu_idx.size
    if kept >= L:
        assert gpu_idx.tolist() == list(range(L)), f"{where}: keep-all expected"
        return 0
    n = L - window
    assert gpu_idx[-window:].tolist() == list(range(n, L)), f"{where}: window not kept"
    if unit.k == 0:
        return 0
    diff = set(gpu_idx[:-window].tolist()) ^ set(ref_idx[:-window].tolist())
    tau = unit.tau
    for j in diff:
        if abs(unit.pooled[j] - tau) > rel * tau:
            raise AssertionError(f"{where}: token {j} differs (oracle pooled {unit.pooled[j]!r}, "
                                 f"k-th {tau!r})")
    return len(diff)


def check_gather_bits(k_bits, v_bits, k_out_bits, v_out_bits, indices, cu_seqlens, cu_out):
    """All *_bits are integer views (int16) of the tensors, as numpy arrays."""
    H = k_bits.shape[1]
    for s in range(len(cu_out) - 1):
        o0, o1 = int(cu_out[s]), int(cu_out[s + 1])
        base = int(cu_seqlens[s])
        for g in range(H):
            rows = base + np.asarray(indices[g, o0:o1], np.int64)
            if not np.array_equal(k_out_bits[o0:o1, g], k_bits[rows, g]):
                raise AssertionError(f"K rows differ for sequence {s} group {g}")
            if not np.array_equal(v_out_bits[o0:o1, g], v_bits[rows, g]):
                raise AssertionError(f"V rows differ for sequence {s} group {g}")


def check_layer(res, gpu_raw, gpu_pooled, gpu_indices, cu_seqlens, window):
    """Scores and index sets of a whole layer; returns the number of
    tolerated near-tie differences."""
    check_scores("raw", gpu_raw, res.raw)
    check_scores("pooled", gpu_pooled, res.pooled)
    ties = 0
    H = res.raw.shape[0]
    for (s, g), unit in res.units.items():
        L = int(cu_seqlens[s + 1] - cu_seqlens[s])
        o0, o1 = int(res.cu_out[s]), int(res.cu_out[s + 1])
        ties += check_unit_indices(gpu_indices[g, o0:o1], unit, L, window,
                                   where=f"seq {s} group {g}")
    assert len(res.units) == H * (len(cu_seqlens) - 1)
    return ties
