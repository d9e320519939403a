"""Head-level budgets on the device (a budget per (sequence, KV group),
outputs packed group-major) vs the oracle, through the C ABI (needs a
GB300).  Index sets identical except near-ties within 1e-3 of the unit's
k-th pooled score; K/V rows bit-exact."""
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


def run(d, window, pool_width, dev, gb):
    q, k, v = d["q_win"].to(dev), d["k"].to(dev), d["v"].to(dev)
    prob = ckv.Problem(q, k, d["cu_seqlens"], window, pool_width)
    cu_host, rows = ckv.head_budget_layout(prob, gb)
    idx = torch.empty(max(rows, 1), dtype=torch.int32, device=dev)
    k_out = torch.empty((max(rows, 1), 128), dtype=k.dtype, device=dev)
    v_out = torch.empty_like(k_out)
    ws = ckv.workspace(prob, dev)
    cu_out = ckv.compress_layer_head_budgets(prob, q, k, v, d["srh_mask"], gb, idx, k_out, v_out,
                                             ws)
    torch.cuda.synchronize()
    assert ckv.read_device_status(ws) == 0
    assert np.array_equal(cu_out, cu_host)
    res = oracle.compress_layer_head_budgets(d["q_win"].float().numpy(), d["k"].float().numpy(),
                                             d["v"].float().numpy(), d["cu_seqlens"],
                                             d["srh_mask"], gb, window, pool_width)
    assert np.array_equal(cu_out, res.cu_out)
    gi = idx.cpu().numpy()[:rows]
    kb, vb = _bits(d["k"]), _bits(d["v"])
    ko, vo = _bits(k_out)[:rows], _bits(v_out)[:rows]
    cu = d["cu_seqlens"]
    for (s, g), unit in res.units.items():
        p0, p1 = int(cu_out[g, s]), int(cu_out[g, s + 1])
        L = int(cu[s + 1] - cu[s])
        compare.check_unit_indices(gi[p0:p1], unit, L, window, where=f"seq {s} group {g}")
        src = int(cu[s]) + gi[p0:p1].astype(np.int64)
        assert np.array_equal(ko[p0:p1], kb[src, g]) and np.array_equal(vo[p0:p1], vb[src, g])
    return res


def test_head_budgets_4k(cuda_device):
    cfg = wl.get("c1")
    d = wl.make_layer(cfg, 0)
    rng = np.random.default_rng(3)
    gb = rng.integers(cfg.window, 600, size=(1, cfg.num_kv_heads)).astype(np.int32)
    run(d, cfg.window, cfg.pool_width, cuda_device, gb)


def test_head_budgets_ragged_batch(cuda_device):
    lens = [1000, 0, 5, 33, 161, 700]
    cfg = wl.get("c1").scaled(dtype="bf16", batch=len(lens), seq_len=0, srh_per_group=(1, 2))
    d = wl.make_layer(cfg, 0, lengths=lens, budgets=np.full((1, len(lens)), 64, np.int32))
    rng = np.random.default_rng(5)
    gb = rng.integers(cfg.window, 300, size=(len(lens), cfg.num_kv_heads)).astype(np.int32)
    gb[0, 3] = 5000  # keep all
    gb[2, :] = cfg.window
    run(d, cfg.window, cfg.pool_width, cuda_device, gb)


def test_head_budgets_full_size_llama8b_32k(cuda_device):
    cfg = wl.get("c2")
    d = wl.make_layer(cfg, 2)
    rng = np.random.default_rng(7)
    gb = rng.integers(64, 1024, size=(1, cfg.num_kv_heads)).astype(np.int32)
    run(d, cfg.window, cfg.pool_width, cuda_device, gb)
