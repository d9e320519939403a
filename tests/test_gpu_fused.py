"""The persistent per-group kernel of compresskv_compress_layers against the
float64 oracle, through the C ABI (needs a GB300).

Besides parity with the oracle (tolerances as in test_gpu_parity.py), the
kernel's scores depend only on the unit itself: its softmax statistics
restart on a fixed grid of 16-tile chunks of every unit and each tile of that
grid always goes to the same epilogue warpgroup, so a layer compressed alone
and the same layer inside a larger call give identical bits.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2606_24467_gb300 as ckv
import workloads as wl
from oracle import compare

pytestmark = pytest.mark.gpu

RTOL = 1e-4  # fp32 exponentials of fp32 logits, fp32 merged denominators


def _bits(t):
    return t.detach().cpu().contiguous().view(torch.int16).numpy()


def _layers(cfg):
    lengths = wl.sequence_lengths(cfg)
    masks = wl.srh_masks(cfg)
    budgets = wl.layer_budgets(cfg, lengths)
    return [wl.make_layer(cfg, l, lengths=lengths, masks=masks, budgets=budgets)
            for l in range(cfg.n_layers)]


def _pack(layers, dev, lengths_per_layer=None):
    """K/V/Q of several layers packed as one batch (block l = layer l)."""
    Ts = [lay["k"].shape[0] for lay in layers]
    k_all = torch.cat([lay["k"] for lay in layers]).to(dev)
    v_all = torch.cat([lay["v"] for lay in layers]).to(dev)
    q_all = torch.cat([lay["q_win"] for lay in layers]).to(dev)
    offs = np.concatenate([[0], np.cumsum(Ts)])
    cu = np.concatenate([np.asarray(lay["cu_seqlens"][:-1], np.int64) + offs[l]
                         for l, lay in enumerate(layers)] + [[offs[-1]]]).astype(np.int32)
    b_all = np.concatenate([np.asarray(lay["budgets"]).reshape(-1) for lay in layers])
    m_all = np.stack([np.asarray(lay["srh_mask"]) for lay in layers])
    return q_all, k_all, v_all, cu, b_all, m_all


def _run_call(layers, cfg, dev, scores=True):
    q_all, k_all, v_all, cu, b_all, m_all = _pack(layers, dev)
    prob = ckv.Problem(q_all, k_all, cu, cfg.window, cfg.pool_width)
    out = ckv.LayerOutputs(prob, b_all, 128, k_all.dtype, dev, scores=scores)
    ws = ckv.workspace(prob, dev)
    cu_out = ckv.compress_layers(prob, len(layers), q_all, k_all, v_all, m_all, b_all,
                                 out.indices, out.k_out, out.v_out, ws, raw=out.raw,
                                 pooled=out.pooled)
    torch.cuda.synchronize()
    assert ckv.read_device_status(ws) == 0
    return out, cu_out, cu


def _block(out, cu_out, cu, l, B, window):
    """Layer l's block of a packed call's outputs (host arrays)."""
    n = np.maximum(np.diff(cu) - window, 0)
    cu_prefix = np.concatenate([[0], np.cumsum(n)])
    s0, s1 = l * B, (l + 1) * B
    p0, p1 = cu_prefix[s0], cu_prefix[s1]
    o0, o1 = cu_out[s0], cu_out[s1]
    blk = {"indices": out.indices[:, o0:o1].cpu().numpy(),
           "k_out": _bits(out.k_out[o0:o1]), "v_out": _bits(out.v_out[o0:o1]),
           "cu_out": cu_out[s0:s1 + 1] - o0}
    if out.raw is not None:
        blk["raw"] = out.raw[:, p0:p1].cpu().numpy()
        blk["pooled"] = out.pooled[:, p0:p1].cpu().numpy()
    return blk


def _check_block(blk, lay, cfg):
    res = oracle.compress_layer(lay["q_win"].float().numpy(), lay["k"].float().numpy(),
                                lay["v"].float().numpy(), lay["cu_seqlens"], lay["srh_mask"],
                                lay["budgets"], cfg.window, cfg.pool_width)
    assert np.array_equal(blk["cu_out"], res.cu_out)
    if "raw" in blk:
        compare.check_layer(res, blk["raw"], blk["pooled"], blk["indices"], lay["cu_seqlens"],
                            cfg.window)
        compare.check_scores("raw", blk["raw"], res.raw, rtol=RTOL, atol=1e-8)
        compare.check_scores("pooled", blk["pooled"], res.pooled, rtol=RTOL, atol=1e-8)
    else:
        for (s, g), unit in res.units.items():
            L = int(lay["cu_seqlens"][s + 1] - lay["cu_seqlens"][s])
            o0, o1 = int(res.cu_out[s]), int(res.cu_out[s + 1])
            compare.check_unit_indices(blk["indices"][g, o0:o1], unit, L, cfg.window)
    compare.check_gather_bits(_bits(lay["k"]), _bits(lay["v"]), blk["k_out"], blk["v_out"],
                              blk["indices"], lay["cu_seqlens"], blk["cu_out"])


def test_layer_alone_equals_layer_in_a_larger_call(cuda_device):
    """Scores, indices and K/V of a layer are bit-identical whether it is
    compressed alone or as one block of a six-layer call (ragged batch)."""
    dev = cuda_device
    cfg = wl.get("c2").scaled(seq_len=0, n_layers=6, batch=3, length_range=(900, 5200))
    layers = _layers(cfg)
    big, cu_out, cu = _run_call(layers, cfg, dev)
    for l in (0, 3, 5):
        alone, cu_out1, cu1 = _run_call([layers[l]], cfg, dev)
        a = _block(alone, cu_out1, cu1, 0, cfg.batch, cfg.window)
        b = _block(big, cu_out, cu, l, cfg.batch, cfg.window)
        for key in ("raw", "pooled", "indices", "k_out", "v_out", "cu_out"):
            assert np.array_equal(a[key].view(np.uint8) if a[key].dtype != np.int32 else a[key],
                                  b[key].view(np.uint8) if b[key].dtype != np.int32 else b[key]), (l, key)
        _check_block(b, layers[l], cfg)


def test_many_short_layers_with_edge_lengths(cuda_device):
    """Forty layers of a batch of 5 prompts with lengths 0, 1, W, W+1 and
    tile edges in one call: more units than chunks, empty and window-only
    sequences, per-layer masks and budgets."""
    dev = cuda_device
    lens = [0, 33, 32, 129, 1023]
    cfg = wl.get("c2").scaled(seq_len=0, n_layers=40, batch=len(lens), srh_per_group=(1, 3))
    lengths = lens
    masks = wl.srh_masks(cfg)
    budgets = wl.layer_budgets(cfg, lengths)
    layers = [wl.make_layer(cfg, l, lengths=lengths, masks=masks, budgets=budgets)
              for l in range(cfg.n_layers)]
    out, cu_out, cu = _run_call(layers, cfg, dev)
    for l in (0, 17, 39):
        _check_block(_block(out, cu_out, cu, l, cfg.batch, cfg.window), layers[l], cfg)


def test_repeat_call_is_bit_identical(cuda_device):
    dev = cuda_device
    cfg = wl.get("c2").scaled(seq_len=9000, n_layers=3)
    layers = _layers(cfg)
    a, ca, _ = _run_call(layers, cfg, dev)
    b, cb, _ = _run_call(layers, cfg, dev)
    assert np.array_equal(ca, cb)
    assert torch.equal(a.raw.view(torch.int32), b.raw.view(torch.int32))
    assert torch.equal(a.pooled.view(torch.int32), b.pooled.view(torch.int32))
    assert torch.equal(a.indices, b.indices)
    assert torch.equal(a.k_out.view(torch.int16), b.k_out.view(torch.int16))


def test_full_32_layer_llama8b_32k_in_one_call(cuda_device):
    """The benchmark step itself: all 32 layers of the L=32K Llama-3.1-8B
    workload in one call (256 units of 16 chunks each, more units than CTAs,
    so pass-2 chunks wait for merges of units spread over many CTAs).  The
    first and last layers
    are checked against the oracle unit by unit."""
    dev = cuda_device
    cfg = wl.get("c2")
    layers = _layers(cfg)
    out, cu_out, cu = _run_call(layers, cfg, dev, scores=False)
    for l in (0, cfg.n_layers - 1):
        _check_block(_block(out, cu_out, cu, l, cfg.batch, cfg.window), layers[l], cfg)


def test_bounded_wait_runs_out_and_the_workspace_recovers(cuda_device):
    """The failure path of the persistent kernel: a wait that cannot complete
    (the test hook's counter, before anything is issued) runs out after 2 ms;
    the call returns, every CTA stops, the device status reads
    CKV_ERR_DEVICE_TIMEOUT and, after workspace_init, the same call on the
    same workspace is correct again."""
    dev = cuda_device
    cfg = wl.get("c2").scaled(seq_len=9000, n_layers=4)
    layers = _layers(cfg)
    q_all, k_all, v_all, cu, b_all, m_all = _pack(layers, dev)
    prob = ckv.Problem(q_all, k_all, cu, cfg.window, cfg.pool_width)
    out = ckv.LayerOutputs(prob, b_all, 128, k_all.dtype, dev, scores=True)
    ws = ckv.workspace(prob, dev)

    def call():
        return ckv.compress_layers(prob, len(layers), q_all, k_all, v_all, m_all, b_all,
                                   out.indices, out.k_out, out.v_out, ws, raw=out.raw,
                                   pooled=out.pooled)

    ckv.debug_stall_next_fused_call(2_000_000)
    call()
    torch.cuda.synchronize()
    assert ckv.read_device_status(ws) == ckv.compresskv.CKV_ERR_DEVICE_TIMEOUT
    ckv.compresskv._check(ckv.load().compresskv_workspace_init(ckv.compresskv._ptr(ws), ws.numel(),
                                                               None), "workspace_init")
    cu_out = call()
    torch.cuda.synchronize()
    assert ckv.read_device_status(ws) == 0
    for l in (0, 3):
        _check_block(_block(out, cu_out, cu, l, cfg.batch, cfg.window), layers[l], cfg)


def test_ragged_odd_chunks_repeated_calls(cuda_device):
    """A Qwen-shaped (7 query heads per group, 4 KV heads) ragged batch over
    several layers, lengths chosen so that many units end in chunks of one or
    an odd number of K tiles (the two UMMA warps then take unequal shares),
    compressed repeatedly on one workspace: every call leaves a clean device
    status and the same bits, and one layer matches the oracle."""
    dev = cuda_device
    lens = [2048 * 3 + 128, 2048 + 128 * 5, 128 * 3 + 40, 2048 * 2 + 1, 8000, 128 + 33]
    cfg = wl.get("c4").scaled(seq_len=0, n_layers=5, batch=len(lens))
    masks = wl.srh_masks(cfg)
    budgets = wl.layer_budgets(cfg, lens)
    layers = [wl.make_layer(cfg, l, lengths=lens, masks=masks, budgets=budgets)
              for l in range(cfg.n_layers)]
    q_all, k_all, v_all, cu, b_all, m_all = _pack(layers, dev)
    prob = ckv.Problem(q_all, k_all, cu, cfg.window, cfg.pool_width)
    out = ckv.LayerOutputs(prob, b_all, 128, k_all.dtype, dev, scores=False)
    ws = ckv.workspace(prob, dev)
    first = None
    for _ in range(12):
        cu_out = ckv.compress_layers(prob, len(layers), q_all, k_all, v_all, m_all, b_all,
                                     out.indices, out.k_out, out.v_out, ws)
        torch.cuda.synchronize()
        assert ckv.read_device_status(ws) == 0
        got = (out.indices.clone(), out.k_out.view(torch.int16).clone())
        if first is None:
            first = got
        else:
            assert torch.equal(first[0], got[0]) and torch.equal(first[1], got[1])
    _check_block(_block(out, cu_out, cu, 2, cfg.batch, cfg.window), layers[2], cfg)


def test_wide_groups_in_a_call_of_many_masks(cuda_device):
    """Six layers of a Llama-70B-shaped problem (8 query heads per group,
    W = 64) with three SRH heads in every group: 192 query rows per unit, the
    most the persistent kernel's shared memory takes with two Q buffers and a
    K stage per UMMA warp.  More masks than the separate path takes in one
    call, so the call must run in the persistent kernel."""
    dev = cuda_device
    lens = [3000, 2048 + 77]
    cfg = wl.get("c5").scaled(seq_len=0, n_layers=6, batch=len(lens), srh_per_group=(3, 3))
    masks = wl.srh_masks(cfg)
    assert int(np.asarray(masks).reshape(cfg.n_layers, cfg.num_kv_heads, -1).sum(-1).min()) == 3
    budgets = wl.layer_budgets(cfg, lens)
    layers = [wl.make_layer(cfg, l, lengths=lens, masks=masks, budgets=budgets)
              for l in range(cfg.n_layers)]
    out, cu_out, cu = _run_call(layers, cfg, dev)
    for l in (0, 5):
        _check_block(_block(out, cu_out, cu, l, cfg.batch, cfg.window), layers[l], cfg)


def test_groups_of_every_row_class_in_one_call(cuda_device):
    """Groups of 64, 128 and 192 query rows (one to three SRH heads at W = 64)
    in one call, whose largest group sets the kernel's shared-memory and TMEM
    layout for all of them.  Every layer matches the oracle, and a layer
    compressed alone gives the same bits as inside the call."""
    dev = cuda_device
    lens = [2500, 2048 + 300]
    cfg = wl.get("c5").scaled(seq_len=0, n_layers=3, batch=len(lens), srh_per_group=(1, 3))
    masks = wl.srh_masks(cfg)
    rows = np.asarray(masks).reshape(cfg.n_layers, cfg.num_kv_heads, -1).sum(-1) * cfg.window
    assert {64, 128, 192} <= set(rows.ravel().tolist())
    budgets = wl.layer_budgets(cfg, lens)
    layers = [wl.make_layer(cfg, l, lengths=lens, masks=masks, budgets=budgets)
              for l in range(cfg.n_layers)]
    big, cu_out, cu = _run_call(layers, cfg, dev)
    for l in range(cfg.n_layers):
        _check_block(_block(big, cu_out, cu, l, cfg.batch, cfg.window), layers[l], cfg)
    alone, cu_out1, cu1 = _run_call([layers[1]], cfg, dev)
    a = _block(alone, cu_out1, cu1, 0, cfg.batch, cfg.window)
    b = _block(big, cu_out, cu, 1, cfg.batch, cfg.window)
    for key in ("raw", "pooled", "indices", "k_out", "v_out", "cu_out"):
        assert np.array_equal(a[key], b[key]), key


def test_thirty_two_query_heads_per_group(cuda_device):
    """The most query heads per KV group the persistent kernel takes (64
    query / 2 KV heads), the smallest window (W = 16), one to four SRH heads
    per group, fp16, pooling width 9: every layer against the oracle."""
    dev = cuda_device
    lens = [1500, 2100]
    cfg = wl.get("c1").scaled(seq_len=0, n_layers=3, batch=len(lens), num_q_heads=64,
                              num_kv_heads=2, window=16, pool_width=9, srh_per_group=(1, 4),
                              budget_rule="dirichlet", budget_mean=120)
    masks = wl.srh_masks(cfg)
    budgets = wl.layer_budgets(cfg, lens)
    layers = [wl.make_layer(cfg, l, lengths=lens, masks=masks, budgets=budgets)
              for l in range(cfg.n_layers)]
    out, cu_out, cu = _run_call(layers, cfg, dev)
    for l in range(cfg.n_layers):
        _check_block(_block(out, cu_out, cu, l, cfg.batch, cfg.window), layers[l], cfg)


@pytest.mark.parametrize("window,pool_width,dtype", [(16, 1, "bf16"), (48, 3, "fp16"),
                                                     (80, 5, "bf16")])
def test_windows_and_pool_widths(cuda_device, window, pool_width, dtype):
    """Windows whose query rows end in a partial 32-column group (W = 48, 80)
    or fill one exactly (W = 16 x 2 heads), pooling widths 1, 3 and 5, fp16
    and bf16, with one or two SRH heads per group (up to 160 rows)."""
    dev = cuda_device
    lens = [2048 * 2 + 77, 700]
    cfg = wl.get("c2").scaled(seq_len=0, n_layers=2, batch=len(lens), window=window,
                              pool_width=pool_width, dtype=dtype, srh_per_group=(1, 2),
                              budget_mean=200)
    masks = wl.srh_masks(cfg)
    budgets = wl.layer_budgets(cfg, lens)
    layers = [wl.make_layer(cfg, l, lengths=lens, masks=masks, budgets=budgets)
              for l in range(cfg.n_layers)]
    out, cu_out, cu = _run_call(layers, cfg, dev)
    for l in range(cfg.n_layers):
        _check_block(_block(out, cu_out, cu, l, cfg.batch, cfg.window), layers[l], cfg)
