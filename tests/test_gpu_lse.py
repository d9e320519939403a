"""Given-LSE scoring on the device (the window queries' log-sum-exp supplied,
as a prefill attention kernel has it) vs the oracle's definition, through the
C ABI (needs a GB300).  The scores are summed in fp32 straight from the
logits, so they are held to a tighter bound than the table path."""
import numpy as np
import pytest
import torch

import oracle
import paper_2606_24467_gb300 as ckv
import workloads as wl
from oracle import compare

pytestmark = pytest.mark.gpu

RTOL = 1e-4  # fp32 exponentials of fp32 logits with an fp32 LSE


def _bits(t):
    return t.detach().cpu().contiguous().view(torch.int16).numpy()


def run_lse(d, window, pool_width, dev, selection="group", mask=None):
    mask = d["srh_mask"] if mask is None else mask
    lse64 = oracle.window_lse(d["q_win"].float().numpy(), d["k"].float().numpy(),
                              d["cu_seqlens"], window)
    lse = torch.tensor(lse64, dtype=torch.float32, device=dev)
    q, k, v = d["q_win"].to(dev), d["k"].to(dev), d["v"].to(dev)
    prob = ckv.Problem(q, k, d["cu_seqlens"], window, pool_width, selection=selection)
    out = ckv.LayerOutputs(prob, d["budgets"], 128, k.dtype, dev)
    ws = ckv.workspace(prob, dev)
    cu_out = ckv.compress_layer_lse(prob, q, k, v, lse, mask, d["budgets"], out.indices,
                                    out.k_out, out.v_out, ws, raw=out.raw,
                                    pooled=out.pooled if selection == "group" else None)
    torch.cuda.synchronize()
    assert ckv.read_device_status(ws) == 0
    res = oracle.compress_layer(d["q_win"].float().numpy(), d["k"].float().numpy(),
                                d["v"].float().numpy(), d["cu_seqlens"], mask, d["budgets"],
                                window, pool_width, selection=selection)
    return out, cu_out, res


def test_lse_path_4k(cuda_device):
    cfg = wl.get("c1")
    d = wl.make_layer(cfg, 0)
    out, cu_out, res = run_lse(d, cfg.window, cfg.pool_width, cuda_device)
    assert np.array_equal(cu_out, res.cu_out)
    raw, pooled = out.raw.cpu().numpy(), out.pooled.cpu().numpy()
    compare.check_scores("raw", raw, res.raw, rtol=RTOL, atol=1e-8)
    compare.check_scores("pooled", pooled, res.pooled, rtol=RTOL, atol=1e-8)
    idx = out.indices.cpu().numpy()
    compare.check_layer(res, raw, pooled, idx, d["cu_seqlens"], cfg.window)
    compare.check_gather_bits(_bits(d["k"]), _bits(d["v"]), _bits(out.k_out), _bits(out.v_out),
                              idx, d["cu_seqlens"], cu_out)


@pytest.mark.parametrize("dtype", ["fp16", "bf16"])
def test_lse_path_ragged(cuda_device, dtype):
    lens = [1000, 0, 5, 33, 160, 161, 257, 700]
    cfg = wl.get("c1").scaled(dtype=dtype, batch=len(lens), seq_len=0, srh_per_group=(1, 3))
    bud = np.array([[64, 40, 40, 33, 100, 161, 250, 5000]], np.int32)
    d = wl.make_layer(cfg, 0, lengths=lens, budgets=bud)
    out, cu_out, res = run_lse(d, cfg.window, cfg.pool_width, cuda_device)
    raw, pooled = out.raw.cpu().numpy(), out.pooled.cpu().numpy()
    compare.check_scores("raw", raw, res.raw, rtol=RTOL, atol=1e-8)
    idx = out.indices.cpu().numpy()
    compare.check_layer(res, raw, pooled, idx, d["cu_seqlens"], cfg.window)
    compare.check_gather_bits(_bits(d["k"]), _bits(d["v"]), _bits(out.k_out), _bits(out.v_out),
                              idx, d["cu_seqlens"], cu_out)


def test_lse_path_layer_scope(cuda_device):
    cfg = wl.get("c1").scaled(seq_len=2500, batch=2)
    d = wl.make_layer(cfg, 0)
    mask = d["srh_mask"].copy()
    mask[:4] = False  # group 0 without SRH head
    out, cu_out, res = run_lse(d, cfg.window, cfg.pool_width, cuda_device, selection="layer",
                               mask=mask)
    raw = out.raw.cpu().numpy()
    compare.check_scores("raw", raw, res.raw, rtol=RTOL, atol=1e-8)
    assert np.all(raw[0] == 0.0)
    idx = out.indices.cpu().numpy()
    for s, sh in res.shared.items():
        o0, o1 = int(cu_out[s]), int(cu_out[s + 1])
        assert np.all(idx[:, o0:o1] == idx[0:1, o0:o1])
        L = int(d["cu_seqlens"][s + 1] - d["cu_seqlens"][s])
        unit = oracle.compresskv_oracle.UnitResult([], np.zeros(0), sh.pooled, sh.k, sh.tau,
                                                   sh.indices)
        compare.check_unit_indices(idx[0, o0:o1], unit, L, cfg.window)


@pytest.mark.parametrize("n_layers,batch", [(2, 1), (3, 2)])
def test_lse_path_multi_layer(cuda_device, n_layers, batch):
    """Several layers in one given-LSE call (compress_layers_lse): each
    layer's block of the outputs against the oracle on that layer."""
    dev = cuda_device
    cfg = wl.get("c2").scaled(seq_len=2000, n_layers=n_layers, batch=batch)
    lengths = wl.sequence_lengths(cfg)
    masks = wl.srh_masks(cfg)
    budgets = wl.layer_budgets(cfg, lengths)
    layers = [wl.make_layer(cfg, l, lengths=lengths, masks=masks, budgets=budgets)
              for l in range(n_layers)]
    T = layers[0]["k"].shape[0]
    lse = torch.cat([torch.tensor(oracle.window_lse(lay["q_win"].float().numpy(),
                                                    lay["k"].float().numpy(),
                                                    lay["cu_seqlens"], cfg.window),
                                  dtype=torch.float32) for lay in layers]).to(dev)
    k_all = torch.cat([lay["k"] for lay in layers]).to(dev)
    v_all = torch.cat([lay["v"] for lay in layers]).to(dev)
    q_all = torch.cat([lay["q_win"] for lay in layers]).to(dev)
    cu = np.concatenate([np.asarray(lay["cu_seqlens"][:-1], np.int64) + l * T
                         for l, lay in enumerate(layers)] + [[n_layers * T]]).astype(np.int32)
    b_all = np.concatenate([np.asarray(lay["budgets"]).reshape(-1) for lay in layers])
    m_all = np.stack([np.asarray(lay["srh_mask"]) for lay in layers])
    prob = ckv.Problem(q_all, k_all, cu, cfg.window, cfg.pool_width)
    out = ckv.LayerOutputs(prob, b_all, 128, k_all.dtype, dev)
    ws = ckv.workspace(prob, dev)
    cu_out = ckv.compress_layers_lse(prob, n_layers, q_all, k_all, v_all, lse, m_all, b_all,
                                     out.indices, out.k_out, out.v_out, ws, raw=out.raw,
                                     pooled=out.pooled)
    torch.cuda.synchronize()
    assert ckv.read_device_status(ws) == 0
    n = np.maximum(np.diff(cu) - cfg.window, 0)
    cu_prefix = np.concatenate([[0], np.cumsum(n)])
    raw, pooled = out.raw.cpu().numpy(), out.pooled.cpu().numpy()
    idx = out.indices.cpu().numpy()
    k_bits, v_bits = _bits(out.k_out), _bits(out.v_out)
    for l, lay in enumerate(layers):
        s0, s1 = l * batch, (l + 1) * batch
        p0, p1 = cu_prefix[s0], cu_prefix[s1]
        o0, o1 = cu_out[s0], cu_out[s1]
        res = oracle.compress_layer(lay["q_win"].float().numpy(), lay["k"].float().numpy(),
                                    lay["v"].float().numpy(), lay["cu_seqlens"],
                                    lay["srh_mask"], lay["budgets"], cfg.window,
                                    cfg.pool_width)
        assert np.array_equal(cu_out[s0:s1 + 1] - o0, res.cu_out)
        compare.check_scores("raw", raw[:, p0:p1], res.raw, rtol=RTOL, atol=1e-8)
        compare.check_layer(res, raw[:, p0:p1], pooled[:, p0:p1], idx[:, o0:o1],
                            lay["cu_seqlens"], cfg.window)
        compare.check_gather_bits(_bits(lay["k"]), _bits(lay["v"]), k_bits[o0:o1],
                                  v_bits[o0:o1], idx[:, o0:o1], lay["cu_seqlens"],
                                  cu_out[s0:s1 + 1] - o0)


def test_lse_in_host_memory_refused(cuda_device):
    # every other argument is a valid device buffer; the library checks the
    # LSE pointer with cudaPointerGetAttributes and refuses host memory before
    # anything is enqueued (the binding's own check is bypassed here)
    from ctypes import POINTER, c_int32, c_void_p

    from paper_2606_24467_gb300 import compresskv as B
    cfg = wl.get("c1").scaled(seq_len=600)
    d = wl.make_layer(cfg, 0)
    dev = cuda_device
    q, k, v = d["q_win"].to(dev), d["k"].to(dev), d["v"].to(dev)
    prob = ckv.Problem(q, k, d["cu_seqlens"], cfg.window, cfg.pool_width)
    out = ckv.LayerOutputs(prob, d["budgets"], 128, k.dtype, dev)
    ws = ckv.workspace(prob, dev)
    lse = torch.zeros((prob.batch, q.shape[1], cfg.window), dtype=torch.float32)  # host
    m = np.ascontiguousarray(np.asarray(d["srh_mask"], np.uint8))
    b, bp = B._i32(d["budgets"])
    cu_out = np.zeros(prob.batch + 1, np.int32)
    rc = ckv.load().compresskv_compress_layer_lse(
        prob.ref, B._ptr(q), B._ptr(k), B._ptr(v), c_void_p(lse.data_ptr()), lse.stride(0),
        lse.stride(1), c_void_p(m.ctypes.data), bp, B._ptr(out.indices),
        cu_out.ctypes.data_as(POINTER(c_int32)), B._ptr(out.k_out), B._ptr(out.v_out), None,
        None, B._ptr(ws), ws.numel(), B._stream(None))
    assert rc == B.CKV_ERR_INVALID_ARG
