"""Max pooling (CKV_POOL_MAX) on the device vs the float64 oracle, through
the C ABI (needs a GB300).  Each SRH head's window-summed attention is
max-pooled over [j - r, j + r] of the prefix and the heads' pooled vectors
are summed (Sec. 3.3: pooling across the token dimension before the heads
are combined).  Acceptance as for average pooling: raw and pooled scores
within 1e-3 relative + 1e-5 absolute (raw scores are the heads' sum, as with
average pooling), index sets identical except near-ties within 1e-3 of the
k-th pooled score, K/V rows bit-exact at the device's indices."""
import numpy as np
import pytest
import torch

import oracle
import paper_2606_24467_gb300 as ckv
import workloads as wl
from oracle import compare

pytestmark = pytest.mark.gpu

RTOL = 1e-4  # per-head raw scores of the persistent kernel (fp32 exponentials)
TABLE_RTOL = 2.0 ** -11 + 2e-5  # the separate kernels' fp16 exponent table (W not a multiple of 16)


def _bits(t):
    return t.detach().cpu().contiguous().view(torch.int16).numpy()


def _run(d, cfg, dev, selection="group", mask=None):
    mask = d["srh_mask"] if mask is None else mask
    q, k, v = d["q_win"].to(dev), d["k"].to(dev), d["v"].to(dev)
    prob = ckv.Problem(q, k, d["cu_seqlens"], cfg.window, cfg.pool_width, selection=selection,
                       pool="max")
    out = ckv.LayerOutputs(prob, d["budgets"], 128, k.dtype, dev)
    ws = ckv.workspace(prob, dev)
    cu_out = ckv.compress_layer(prob, q, k, v, mask, d["budgets"], out.indices, out.k_out,
                                out.v_out, ws, raw=out.raw, pooled=out.pooled)
    torch.cuda.synchronize()
    assert ckv.read_device_status(ws) == 0
    res = oracle.compress_layer(d["q_win"].float().numpy(), d["k"].float().numpy(),
                                d["v"].float().numpy(), d["cu_seqlens"], mask, d["budgets"],
                                cfg.window, cfg.pool_width, selection=selection, pool_kind="max")
    assert np.array_equal(cu_out, res.cu_out)
    return out, cu_out, res


def _check_group_scope(d, cfg, dev, mask=None):
    out, cu_out, res = _run(d, cfg, dev, mask=mask)
    idx = out.indices.cpu().numpy()
    raw, pooled = out.raw.cpu().numpy(), out.pooled.cpu().numpy()
    compare.check_layer(res, raw, pooled, idx, d["cu_seqlens"], cfg.window)
    rtol = RTOL if cfg.window % 16 == 0 else TABLE_RTOL
    compare.check_scores("raw", raw, res.raw, rtol=rtol, atol=1e-8)
    compare.check_scores("pooled (max)", pooled, res.pooled, rtol=rtol, atol=1e-8)
    compare.check_gather_bits(_bits(d["k"]), _bits(d["v"]), _bits(out.k_out), _bits(out.v_out),
                              idx, d["cu_seqlens"], cu_out)
    return res


def test_llama8b_4k_single_layer_max_pool(cuda_device):
    """The 1-layer L=4096 workload with max pooling, in full."""
    cfg = wl.get("c1")
    _check_group_scope(wl.make_layer(cfg, 0), cfg, cuda_device)


def test_llama8b_32k_layer_max_pool(cuda_device):
    """One full-size layer of the L=32K Llama-3.1-8B workload (1-2 SRH heads
    per group), max pooling."""
    cfg = wl.get("c2")
    _check_group_scope(wl.make_layer(cfg, 5), cfg, cuda_device)


@pytest.mark.parametrize("W,P,heads", [(32, 7, 3), (16, 5, 4), (8, 3, 2)])
def test_max_pool_head_counts_and_windows(cuda_device, W, P, heads):
    """Several SRH heads per group (the pooled sum has that many terms), a
    ragged batch with edge lengths; W = 8 takes the separate scoring kernels
    for the per-head rounds, the others the persistent kernel."""
    lens = [1500, 0, 5, W, W + 1, 129, 1023]
    cfg = wl.get("c1").scaled(seq_len=0, batch=len(lens), window=W, pool_width=P,
                              srh_per_group=(heads, heads), dtype="bf16")
    d = wl.make_layer(cfg, 0, lengths=lens, budgets=np.array([[W + 77] * len(lens)], np.int32))
    _check_group_scope(d, cfg, cuda_device)


def test_layer_scope_max_pool(cuda_device):
    """Per-layer (shared) selection with max pooling: one top-k per sequence
    over every SRH head's max-pooled score, groups without an SRH head
    allowed."""
    cfg = wl.get("c1").scaled(seq_len=2000, batch=2)
    d = wl.make_layer(cfg, 0)
    mask = np.zeros(cfg.num_q_heads, bool)
    mask[[0, 1, 9, 30]] = True  # groups 0, 2, 7; the others have none
    out, cu_out, res = _run(d, cfg, cuda_device, selection="layer", mask=mask)
    idx = out.indices.cpu().numpy()
    compare.check_scores("raw", out.raw.cpu().numpy(), res.raw, rtol=RTOL, atol=1e-8)
    compare.check_scores("pooled (max)", out.pooled.cpu().numpy(), res.pooled, rtol=RTOL,
                         atol=1e-8)
    cu = d["cu_seqlens"]
    for s, sh in res.shared.items():
        o0, o1 = int(cu_out[s]), int(cu_out[s + 1])
        rows = idx[:, o0:o1]
        assert np.all(rows == rows[0:1]), f"seq {s}: groups disagree"
        unit = oracle.compresskv_oracle.UnitResult([], np.zeros(0), sh.pooled, sh.k, sh.tau,
                                                   sh.indices)
        compare.check_unit_indices(rows[0], unit, int(cu[s + 1] - cu[s]), cfg.window,
                                   where=f"seq {s}")
    compare.check_gather_bits(_bits(d["k"]), _bits(d["v"]), _bits(out.k_out), _bits(out.v_out),
                              idx, cu, cu_out)


def test_max_pool_differs_from_average(cuda_device):
    """The option changes the selection: on the same layer, the max-pooled
    scores differ from the average-pooled ones (both checked against the
    oracle elsewhere)."""
    cfg = wl.get("c1")
    d = wl.make_layer(cfg, 0)
    res = _check_group_scope(d, cfg, cuda_device)
    avg = oracle.compress_layer(d["q_win"].float().numpy(), d["k"].float().numpy(),
                                d["v"].float().numpy(), d["cu_seqlens"], d["srh_mask"],
                                d["budgets"], cfg.window, cfg.pool_width)
    assert not np.allclose(res.pooled, avg.pooled)
