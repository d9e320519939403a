"""Per-layer (shared) selection on the device vs the oracle, through the C
ABI (needs a GB300).  Sec. 3.3 read literally: per sequence, the pooled
scores of every group's SRH heads are summed, one top-k is kept and every KV
group retains the same positions.  Acceptance as for per-group selection:
scores within 1e-3 relative + 1e-5 absolute, index sets identical except
near-ties within 1e-3 of the k-th summed score, K/V bit-exact."""
import numpy as np
import pytest
import torch

import oracle
import paper_2606_24467_gb300 as ckv
import workloads as wl
from oracle import compare

pytestmark = pytest.mark.gpu


def _bits(t):
    return t.detach().cpu().contiguous().view(torch.int16).numpy()


def run_both(d, window, pool_width, dev, mask=None):
    mask = d["srh_mask"] if mask is None else mask
    q, k, v = d["q_win"].to(dev), d["k"].to(dev), d["v"].to(dev)
    prob = ckv.Problem(q, k, d["cu_seqlens"], window, pool_width, selection="layer")
    out = ckv.LayerOutputs(prob, d["budgets"], 128, k.dtype, dev)
    ws = ckv.workspace(prob, dev)
    cu_out = ckv.compress_layer(prob, q, k, v, mask, d["budgets"], out.indices, out.k_out,
                                out.v_out, ws, raw=out.raw, pooled=out.pooled)
    torch.cuda.synchronize()
    assert ckv.read_device_status(ws) == 0
    res = oracle.compress_layer(d["q_win"].float().numpy(), d["k"].float().numpy(),
                                d["v"].float().numpy(), d["cu_seqlens"], mask, d["budgets"],
                                window, pool_width, selection="layer")
    return out, cu_out, res


def check_layer_scope(d, window, pool_width, dev, mask=None):
    out, cu_out, res = run_both(d, window, pool_width, dev, mask)
    assert np.array_equal(cu_out, res.cu_out)
    compare.check_scores("raw", out.raw.cpu().numpy(), res.raw)
    compare.check_scores("pooled", out.pooled.cpu().numpy(), res.pooled)
    idx = out.indices.cpu().numpy()
    cu = d["cu_seqlens"]
    H = idx.shape[0]
    for s, sh in res.shared.items():
        o0, o1 = int(cu_out[s]), int(cu_out[s + 1])
        rows = idx[:, o0:o1]
        assert np.all(rows == rows[0:1]), f"seq {s}: groups disagree"
        L = int(cu[s + 1] - cu[s])
        unit = oracle.compresskv_oracle.UnitResult([], np.zeros(0), sh.pooled, sh.k, sh.tau,
                                                   sh.indices)
        compare.check_unit_indices(rows[0], unit, L, window, where=f"seq {s}")
    compare.check_gather_bits(_bits(d["k"]), _bits(d["v"]), _bits(out.k_out), _bits(out.v_out),
                              idx, cu, cu_out)
    assert H == d["k"].shape[1]
    return out, res


def test_layer_scope_4k(cuda_device):
    cfg = wl.get("c1")
    d = wl.make_layer(cfg, 0)
    check_layer_scope(d, cfg.window, cfg.pool_width, cuda_device)


@pytest.mark.parametrize("dtype", ["fp16", "bf16"])
def test_layer_scope_ragged_with_srh_free_groups(cuda_device, dtype):
    lens = [1000, 0, 5, 33, 161, 257, 700]
    cfg = wl.get("c1").scaled(dtype=dtype, batch=len(lens), seq_len=0, srh_per_group=(1, 2))
    bud = np.array([[64, 40, 40, 33, 100, 250, 5000]], np.int32)
    d = wl.make_layer(cfg, 0, lengths=lens, budgets=bud)
    mask = d["srh_mask"].copy()
    G = cfg.num_q_heads // cfg.num_kv_heads
    mask[2 * G:4 * G] = False  # groups 2 and 3 have no SRH head
    out, res = check_layer_scope(d, cfg.window, cfg.pool_width, cuda_device, mask=mask)
    pooled = out.pooled.cpu().numpy()
    assert np.all(pooled[2:4] == 0.0)


def test_layer_scope_full_size_llama8b_32k(cuda_device):
    cfg = wl.get("c2")
    d = wl.make_layer(cfg, 9)
    check_layer_scope(d, cfg.window, cfg.pool_width, cuda_device)


def test_layer_scope_stage_entry_points(cuda_device):
    """compresskv_score + compresskv_select (per-layer) equal the fused call."""
    cfg = wl.get("c1").scaled(seq_len=3000, batch=2)
    d = wl.make_layer(cfg, 0)
    dev = cuda_device
    q, k, v = d["q_win"].to(dev), d["k"].to(dev), d["v"].to(dev)
    prob = ckv.Problem(q, k, d["cu_seqlens"], cfg.window, cfg.pool_width, selection="layer")
    ws = ckv.workspace(prob, dev)
    fused = ckv.LayerOutputs(prob, d["budgets"], 128, k.dtype, dev)
    ckv.compress_layer(prob, q, k, v, d["srh_mask"], d["budgets"], fused.indices, fused.k_out,
                       fused.v_out, ws)
    staged = ckv.LayerOutputs(prob, d["budgets"], 128, k.dtype, dev)
    ckv.score(prob, q, k, d["srh_mask"], staged.raw, ws)
    ckv.select(prob, staged.raw, d["budgets"], staged.indices, ws)
    torch.cuda.synchronize()
    a, b = fused.indices.cpu().numpy(), staged.indices.cpu().numpy()
    res = oracle.compress_layer(d["q_win"].float().numpy(), d["k"].float().numpy(),
                                d["v"].float().numpy(), d["cu_seqlens"], d["srh_mask"],
                                d["budgets"], cfg.window, cfg.pool_width, selection="layer")
    for s, sh in res.shared.items():
        o0, o1 = int(res.cu_out[s]), int(res.cu_out[s + 1])
        L = int(d["cu_seqlens"][s + 1] - d["cu_seqlens"][s])
        unit = oracle.compresskv_oracle.UnitResult([], np.zeros(0), sh.pooled, sh.k, sh.tau,
                                                   sh.indices)
        for arr in (a, b):
            compare.check_unit_indices(arr[0, o0:o1], unit, L, cfg.window)
