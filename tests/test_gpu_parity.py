"""CUDA path vs. the float64 oracle, through the C ABI (needs a GB300).

Tolerances (acceptance, see oracle/compare.py): raw and pooled scores within
1e-3 relative + 1e-5 absolute (and, as a guard on the device's arithmetic,
within 2^-11 relative: the fp16 exponent table's rounding); retained index
sets identical except for near-ties within 1e-3 of the k-th pooled score;
K/V rows bit-exact at the device's indices; device results deterministic.
"""
import math

import numpy as np
import pytest
import torch

import oracle
import paper_2606_24467_gb300 as ckv
import workloads as wl
from oracle import compare

pytestmark = pytest.mark.gpu

EXPO_RTOL = 2.0 ** -11 + 2e-5


def _bits(t):
    return t.detach().cpu().contiguous().view(torch.int16).numpy()


def run_gpu(d, window, pool_width, dev, mask=None, scale=0.0, budgets=None, k=None, v=None,
            q=None):
    q = d["q_win"].to(dev) if q is None else q
    k = d["k"].to(dev) if k is None else k
    v = d["v"].to(dev) if v is None else v
    mask = d["srh_mask"] if mask is None else mask
    budgets = d["budgets"] if budgets is None else budgets
    prob = ckv.Problem(q, k, d["cu_seqlens"], window, pool_width, scale=scale)
    out = ckv.LayerOutputs(prob, budgets, 128, k.dtype, dev)
    ws = ckv.workspace(prob, dev)
    cu_out = ckv.compress_layer(prob, q, k, v, mask, budgets, out.indices, out.k_out, out.v_out,
                                ws, raw=out.raw, pooled=out.pooled)
    torch.cuda.synchronize()
    assert ckv.read_device_status(ws) == 0
    return out, cu_out


def run_oracle(d, window, pool_width, mask=None, scale=None, budgets=None):
    mask = d["srh_mask"] if mask is None else mask
    budgets = d["budgets"] if budgets is None else budgets
    return oracle.compress_layer(d["q_win"].float().numpy(), d["k"].float().numpy(),
                                 d["v"].float().numpy(), d["cu_seqlens"], mask, budgets,
                                 window, pool_width, scale=scale)


def check(d, window, pool_width, dev, mask=None, budgets=None, scale=None, **kw):
    out, cu_out = run_gpu(d, window, pool_width, dev, mask=mask, budgets=budgets,
                          scale=scale or 0.0, **kw)
    res = run_oracle(d, window, pool_width, mask=mask, budgets=budgets, scale=scale)
    assert np.array_equal(cu_out, res.cu_out)
    idx = out.indices.cpu().numpy()
    raw_gpu, pooled_gpu = out.raw.cpu().numpy(), out.pooled.cpu().numpy()
    ties = compare.check_layer(res, raw_gpu, pooled_gpu, idx, d["cu_seqlens"], window)
    # Tighter than the acceptance tolerance: the device's only coarse rounding
    # is the fp16 exponent table (relative 2^-11 per term, all terms >= 0);
    # the rest is fp32 arithmetic.
    compare.check_scores("raw (fp16 table bound)", raw_gpu, res.raw, rtol=EXPO_RTOL, atol=1e-8)
    compare.check_scores("pooled (fp16 table bound)", pooled_gpu, res.pooled, rtol=EXPO_RTOL,
                         atol=1e-8)
    compare.check_gather_bits(_bits(d["k"]), _bits(d["v"]), _bits(out.k_out), _bits(out.v_out),
                              idx, d["cu_seqlens"], cu_out)
    return out, res, ties


# ---------------------------------------------------------------------------
def test_llama8b_4k_single_layer(cuda_device):
    """The 1-layer L=4096 fp16 workload, in full."""
    cfg = wl.get("c1")
    d = wl.make_layer(cfg, 0)
    check(d, cfg.window, cfg.pool_width, cuda_device)


@pytest.mark.parametrize("dtype", ["fp16", "bf16"])
def test_ragged_batch_edge_lengths(cuda_device, dtype):
    # lengths around the window and the 128-token tiles, plus an empty sequence
    lens = [1000, 0, 5, 32, 33, 160, 161, 255, 256, 257, 128 + 32, 1, 700]
    cfg = wl.get("c1").scaled(dtype=dtype, batch=len(lens), seq_len=0, srh_per_group=(1, 3))
    bud = np.array([[64, 40, 40, 40, 33, 100, 161, 200, 32, 250, 64, 40, 5000]], np.int32)
    d = wl.make_layer(cfg, 0, lengths=lens, budgets=bud)
    check(d, cfg.window, cfg.pool_width, cuda_device)


@pytest.mark.parametrize("W,P,heads", [(8, 5, 4), (16, 3, 3), (32, 1, 2), (64, 7, 3), (64, 9, 4),
                                       (5, 7, 3), (7, 1, 1), (128, 7, 2)])
def test_window_pool_and_srh_counts(cuda_device, W, P, heads):
    """Query-row counts |S|*W from 7 to 256 (MMA N padding), pooling widths."""
    cfg = wl.get("c1").scaled(seq_len=1500, window=W, pool_width=P, srh_per_group=(heads, heads),
                              dtype="bf16")
    bud = np.array([[W + 77]], np.int32)
    d = wl.make_layer(cfg, 0, budgets=bud)
    check(d, W, P, cuda_device)


def test_all_heads_mask_is_snapkv_group_scoring(cuda_device):
    cfg = wl.get("c1").scaled(seq_len=2500)
    d = wl.make_layer(cfg, 0)
    check(d, cfg.window, cfg.pool_width, cuda_device, mask=np.ones(32, bool))


def test_budget_extremes(cuda_device):
    lens = [900, 900, 900, 900, 900]
    cfg = wl.get("c1").scaled(batch=5, seq_len=900, dtype="bf16")
    bud = np.array([[32, 33, 899, 900, 4096]], np.int32)  # window only .. keep all
    d = wl.make_layer(cfg, 0, lengths=lens, budgets=bud)
    out, res, _ = check(d, cfg.window, cfg.pool_width, cuda_device)
    assert res.cu_out.tolist() == [0, 32, 65, 964, 1864, 2764]


def test_exact_ties_break_to_lower_position(cuda_device):
    """All keys equal: every interior pooled score ties exactly, so the lowest
    interior positions must be kept (closed form of the oracle pins)."""
    cfg = wl.get("c1").scaled(seq_len=600, dtype="bf16")
    d = wl.make_layer(cfg, 0, sinks=False, needle_gain=0.0)
    d["k"][:] = d["k"][0:1]
    out, res, ties = check(d, cfg.window, cfg.pool_width, cuda_device)
    assert ties == 0
    r = (cfg.pool_width - 1) // 2
    k = 128 - cfg.window
    idx = out.indices.cpu().numpy()
    for g in range(8):
        assert idx[g, :k].tolist() == list(range(r, r + k))


def test_selection_full_search_paths(cuda_device):
    """The fused call's selection lists the keys at or above a sampled lower
    bound and falls back to a search over all of a unit's keys when that list
    would exceed 4096 keys.  Equal keys at L = 10000 (about 10000 tied
    candidates) and a budget of 9000 at L = 12000 take the fallback; both must
    still equal the oracle (ties to the lowest interior positions)."""
    cfg = wl.get("c1").scaled(seq_len=10000, dtype="bf16")
    d = wl.make_layer(cfg, 0, sinks=False, needle_gain=0.0)
    d["k"][:] = d["k"][0:1]
    out, res, ties = check(d, cfg.window, cfg.pool_width, cuda_device)
    assert ties == 0
    r = (cfg.pool_width - 1) // 2
    k = 128 - cfg.window
    idx = out.indices.cpu().numpy()
    for g in range(8):
        assert idx[g, :k].tolist() == list(range(r, r + k))

    cfg = wl.get("c1").scaled(seq_len=12000, dtype="bf16", srh_per_group=(1, 2))
    d = wl.make_layer(cfg, 0, budgets=np.array([[9000]], np.int32))
    check(d, cfg.window, cfg.pool_width, cuda_device)


def test_selection_second_sampled_bound(cuda_device):
    """A unit whose few top keys sit where the selection samples: strong
    needles at eleven of the sample positions of the first slice (L = 10000,
    8 units: a cluster of 10 CTAs -- about 80 CTAs per launch --, 1024
    positions and 25 evenly spaced samples each) make the first sampled
    bound the 10th needle, so fewer than k = 96 keys reach it and a second,
    looser bound is taken.  The result must equal the oracle."""
    cfg = wl.get("c1").scaled(seq_len=10000, dtype="bf16")
    d = wl.make_layer(cfg, 0, sinks=False, needle_gain=0.0)
    G = cfg.num_q_heads // cfg.num_kv_heads
    C, slice_len, per_cta = 10, 1024, 25
    pos = [(t * slice_len) // per_cta for t in range(1, 12)]
    for g in range(cfg.num_kv_heads):
        qm = d["q_win"][0, g * G:(g + 1) * G].float().mean(dim=(0, 1))
        key = (qm / qm.norm() * 6.0).to(d["k"].dtype)
        for i, p in enumerate(pos):
            d["k"][p, g] = key * (1.0 + 0.01 * i)  # distinct needle strengths
    out, res, ties = check(d, cfg.window, cfg.pool_width, cuda_device)
    # the construction: on the oracle's pooled scores the first bound (the
    # r-th largest sample, r = ceil(mu + 3 sqrt(mu)) + 2) leaves fewer than k
    # keys at or above it
    n = 10000 - cfg.window
    k = 128 - cfg.window
    samples = []
    for c in range(C):
        lo_c = min(n, c * slice_len)
        ln = min(n, lo_c + slice_len) - lo_c
        ns = min(256 // C, ln)
        samples += [lo_c + (t * ln) // ns for t in range(ns)]
    mu = k * len(samples) / n
    r = min(len(samples), math.ceil(mu + 3 * math.sqrt(mu)) + 2)
    for g in range(cfg.num_kv_heads):
        pooled = res.pooled[g]
        bound = np.sort(pooled[samples])[::-1][r - 1]
        assert (pooled >= bound).sum() < k


def test_strided_inputs(cuda_device):
    """K and V as views of one packed KV tensor; Q as a slice of a larger window."""
    cfg = wl.get("c1").scaled(seq_len=777, dtype="bf16", srh_per_group=(2, 2))
    d = wl.make_layer(cfg, 0)
    T = d["k"].shape[0]
    kv = torch.empty((T, 2, 8, 128), dtype=torch.bfloat16, device=cuda_device)
    kv[:, 0] = d["k"].to(cuda_device)
    kv[:, 1] = d["v"].to(cuda_device)
    qbig = torch.zeros((1, 32, 48, 128), dtype=torch.bfloat16, device=cuda_device)
    qbig[:, :, 16:] = d["q_win"].to(cuda_device)
    check(d, cfg.window, cfg.pool_width, cuda_device, k=kv[:, 0], v=kv[:, 1],
          q=qbig[:, :, 16:])


def test_explicit_scale(cuda_device):
    cfg = wl.get("c1").scaled(seq_len=1200, dtype="bf16")
    d = wl.make_layer(cfg, 0)
    check(d, cfg.window, cfg.pool_width, cuda_device, scale=0.5)


def test_stage_entry_points_match_fused(cuda_device):
    cfg = wl.get("c1").scaled(seq_len=3000, dtype="bf16", batch=2, srh_per_group=(1, 2))
    d = wl.make_layer(cfg, 0, lengths=[3000, 1700],
                      budgets=np.array([[300, 150]], np.int32))
    dev = cuda_device
    q, k, v = d["q_win"].to(dev), d["k"].to(dev), d["v"].to(dev)
    fused, cu_fused = run_gpu(d, cfg.window, cfg.pool_width, dev)
    prob = ckv.Problem(q, k, d["cu_seqlens"], cfg.window, cfg.pool_width)
    out = ckv.LayerOutputs(prob, d["budgets"], 128, k.dtype, dev)
    ws = ckv.workspace(prob, dev)
    ckv.score(prob, q, k, d["srh_mask"], out.raw, ws)
    cu_out = ckv.select(prob, out.raw, d["budgets"], out.indices, ws, pooled=out.pooled)
    ckv.gather(prob, out.indices, cu_out, k, v, out.k_out, out.v_out, ws)
    torch.cuda.synchronize()
    assert np.array_equal(cu_out, cu_fused)
    for a, b in ((out.raw, fused.raw), (out.pooled, fused.pooled), (out.indices, fused.indices)):
        assert torch.equal(a, b)
    assert torch.equal(out.k_out.view(torch.int16), fused.k_out.view(torch.int16))
    assert torch.equal(out.v_out.view(torch.int16), fused.v_out.view(torch.int16))


def test_deterministic(cuda_device):
    cfg = wl.get("c1").scaled(seq_len=5000, dtype="bf16", srh_per_group=(1, 2))
    d = wl.make_layer(cfg, 0)
    a, _ = run_gpu(d, cfg.window, cfg.pool_width, cuda_device)
    b, _ = run_gpu(d, cfg.window, cfg.pool_width, cuda_device)
    assert torch.equal(a.raw.view(torch.int32), b.raw.view(torch.int32))
    assert torch.equal(a.indices, b.indices)


def test_gather_reports_bad_index(cuda_device):
    cfg = wl.get("c1").scaled(seq_len=300, dtype="bf16")
    d = wl.make_layer(cfg, 0)
    dev = cuda_device
    k, v = d["k"].to(dev), d["v"].to(dev)
    prob = ckv.Problem(d["q_win"].to(dev), k, d["cu_seqlens"], cfg.window, cfg.pool_width)
    ws = ckv.workspace(prob, dev)
    cu_out = np.array([0, 10], np.int32)
    idx = torch.arange(10, dtype=torch.int32, device=dev).repeat(8, 1).contiguous()
    idx[3, 4] = 300  # one past the end of the sequence
    k_out = torch.zeros((10, 8, 128), dtype=k.dtype, device=dev)
    v_out = torch.zeros_like(k_out)
    ckv.gather(prob, idx, cu_out, k, v, k_out, v_out, ws)
    assert ckv.read_device_status(ws) == ckv.compresskv.CKV_ERR_DEVICE_INDEX
    assert torch.equal(k_out[4, 3], torch.zeros_like(k_out[4, 3]))
    assert torch.equal(k_out[5, 3], k[5, 3])


def test_v_in_page_locked_host_memory(cuda_device):
    """V read in place from page-locked host memory (only the kept rows cross
    the host link) gives the same outputs as V on the device, through the
    fused call and the gather entry point; pageable host memory is refused
    before anything is enqueued."""
    cfg = wl.get("c1").scaled(seq_len=2500, dtype="bf16", batch=2, srh_per_group=(1, 2))
    d = wl.make_layer(cfg, 0, lengths=[2500, 1300], budgets=np.array([[260, 130]], np.int32))
    dev = cuda_device
    ref, cu_ref = run_gpu(d, cfg.window, cfg.pool_width, dev)
    v_host = d["v"].contiguous().pin_memory()
    out, cu_out = run_gpu(d, cfg.window, cfg.pool_width, dev, v=v_host)
    assert np.array_equal(cu_out, cu_ref)
    assert torch.equal(out.indices, ref.indices)
    assert torch.equal(out.k_out.view(torch.int16), ref.k_out.view(torch.int16))
    assert torch.equal(out.v_out.view(torch.int16), ref.v_out.view(torch.int16))
    q, k = d["q_win"].to(dev), d["k"].to(dev)
    prob = ckv.Problem(q, k, d["cu_seqlens"], cfg.window, cfg.pool_width)
    ws = ckv.workspace(prob, dev)
    k2, v2 = torch.zeros_like(out.k_out), torch.zeros_like(out.v_out)
    ckv.gather(prob, out.indices, cu_out, k, v_host, k2, v2, ws)
    torch.cuda.synchronize()
    assert ckv.read_device_status(ws) == 0
    assert torch.equal(v2.view(torch.int16), ref.v_out.view(torch.int16))
    pageable = d["v"].contiguous()
    assert not pageable.is_pinned()
    o3 = ckv.LayerOutputs(prob, d["budgets"], 128, k.dtype, dev)
    with pytest.raises(ckv.CompressKVError) as e:
        ckv.compress_layer(prob, q, k, pageable, d["srh_mask"], d["budgets"], o3.indices,
                           o3.k_out, o3.v_out, ws)
    assert e.value.code == ckv.compresskv.CKV_ERR_INVALID_ARG
    with pytest.raises(ckv.CompressKVError):
        ckv.gather(prob, out.indices, cu_out, k, pageable, k2, v2, ws)
    torch.cuda.synchronize()
    assert ckv.read_device_status(ws) == 0


# ---------------------------------------------------------------------------
# full-size layers of the benchmark workloads (every unit of a sampled layer)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("name,layer", [("c2", 5), ("c3", 17), ("c4", 3), ("c5", 40)])
def test_full_size_layer(cuda_device, name, layer):
    cfg = wl.get(name)
    d = wl.make_layer(cfg, layer)
    check(d, cfg.window, cfg.pool_width, cuda_device)


@pytest.mark.parametrize("n_layers,batch", [(2, 1), (3, 2), (4, 1)])
def test_multi_layer_call(cuda_device, n_layers, batch):
    """Several layers in one call (compress_layers): the layers' K/V and
    window queries packed as one batch, one SRH mask per layer.  Every
    layer's block of the outputs equals the oracle on that layer alone."""
    dev = cuda_device
    cfg = wl.get("c2").scaled(seq_len=3000, n_layers=n_layers, batch=batch)
    lengths = wl.sequence_lengths(cfg)
    masks = wl.srh_masks(cfg)
    budgets = wl.layer_budgets(cfg, lengths)
    layers = [wl.make_layer(cfg, l, lengths=lengths, masks=masks, budgets=budgets)
              for l in range(n_layers)]
    T = layers[0]["k"].shape[0]
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
    cu_out = ckv.compress_layers(prob, n_layers, q_all, k_all, v_all, m_all, b_all, out.indices,
                                 out.k_out, out.v_out, ws, raw=out.raw, pooled=out.pooled)
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
        res = run_oracle(lay, cfg.window, cfg.pool_width)
        assert np.array_equal(cu_out[s0:s1 + 1] - o0, res.cu_out)
        compare.check_layer(res, raw[:, p0:p1], pooled[:, p0:p1], idx[:, o0:o1],
                            lay["cu_seqlens"], cfg.window)
        compare.check_scores("raw (fp16 table bound)", raw[:, p0:p1], res.raw, rtol=EXPO_RTOL,
                             atol=1e-8)
        compare.check_gather_bits(_bits(lay["k"]), _bits(lay["v"]), k_bits[o0:o1], v_bits[o0:o1],
                                  idx[:, o0:o1], lay["cu_seqlens"], cu_out[s0:s1 + 1] - o0)


def test_multi_layer_call_rejects_bad_mask_counts(cuda_device):
    cfg = wl.get("c1").scaled(seq_len=500, batch=2)
    d = wl.make_layer(cfg, 0, lengths=[500, 400])
    dev = cuda_device
    q, k, v = d["q_win"].to(dev), d["k"].to(dev), d["v"].to(dev)
    prob = ckv.Problem(q, k, d["cu_seqlens"], cfg.window, cfg.pool_width)
    out = ckv.LayerOutputs(prob, d["budgets"], 128, k.dtype, dev)
    ws = ckv.workspace(prob, dev)
    masks = np.stack([d["srh_mask"]] * 3)
    for n_masks, code in ((3, ckv.compresskv.CKV_ERR_INVALID_ARG),   # does not divide the batch
                          (0, ckv.compresskv.CKV_ERR_INVALID_ARG)):
        with pytest.raises(ckv.CompressKVError) as e:
            ckv.compress_layers(prob, n_masks, q, k, v, masks[:max(n_masks, 1)], d["budgets"],
                                out.indices, out.k_out, out.v_out, ws)
        assert e.value.code == code
    torch.cuda.synchronize()
    assert ckv.read_device_status(ws) == 0


def test_graph_captured_multilayer_step_matches(cuda_device):
    """Several layers back to back in one CUDA graph: consecutive kernels
    overlap (programmatic dependent launch) and share one workspace; every
    layer must still equal its own eager result and the oracle."""
    dev = cuda_device
    cfg = wl.get("c2").scaled(seq_len=6000, n_layers=4)
    lengths = wl.sequence_lengths(cfg)
    masks = wl.srh_masks(cfg)
    budgets = wl.layer_budgets(cfg, lengths)
    layers = [wl.make_layer(cfg, l, lengths=lengths, masks=masks, budgets=budgets)
              for l in range(cfg.n_layers)]
    dl = [{k: lay[k].to(dev) for k in ("q_win", "k", "v")} for lay in layers]
    probs = [ckv.Problem(d["q_win"], d["k"], lay["cu_seqlens"], cfg.window, cfg.pool_width)
             for d, lay in zip(dl, layers)]
    ws = ckv.workspace(probs[0], dev)
    outs = [ckv.LayerOutputs(probs[l], budgets[l], 128, torch.bfloat16, dev)
            for l in range(cfg.n_layers)]

    def step():
        for l, (d, lay) in enumerate(zip(dl, layers)):
            o = outs[l]
            ckv.compress_layer(probs[l], d["q_win"], d["k"], d["v"], lay["srh_mask"],
                               lay["budgets"], o.indices, o.k_out, o.v_out, ws, raw=o.raw,
                               pooled=o.pooled)

    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        step()
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    eager = [(o.raw.clone(), o.indices.clone(), o.k_out.clone()) for o in outs]
    for o in outs:
        o.raw.zero_()
        o.indices.zero_()
        o.k_out.zero_()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, capture_error_mode="thread_local"):
        step()
    for _ in range(3):
        graph.replay()
    torch.cuda.synchronize()
    assert ckv.read_device_status(ws) == 0
    for l, o in enumerate(outs):
        raw_e, idx_e, k_e = eager[l]
        assert torch.equal(o.raw, raw_e), l
        assert torch.equal(o.indices, idx_e), l
        assert torch.equal(o.k_out.view(torch.int16), k_e.view(torch.int16)), l
        res = run_oracle(layers[l], cfg.window, cfg.pool_width)
        compare.check_layer(res, o.raw.cpu().numpy(), o.pooled.cpu().numpy(),
                            o.indices.cpu().numpy(), layers[l]["cu_seqlens"], cfg.window)
