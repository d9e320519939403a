"""compresskv_compress_layer_noalloc: the variant for callers that cannot
allocate device memory (for example a plugin inside an inference engine that
owns all of HBM and offers no allocator).  It uses the library's built-in
static scratch instead of a caller workspace, so its results must equal the
regular entry point's, on consecutive calls that reuse the same scratch.

Kept in its own file, collected last.
"""
import numpy as np
import pytest
import torch

import paper_2606_24467_gb300 as ckv
import workloads as wl
from oracle import compare
from paper_2606_24467_gb300 import compresskv as B


def _layer():
    cfg = wl.get("c1").scaled(dtype="bf16", batch=2, seq_len=0, srh_per_group=(1, 2))
    d = wl.make_layer(cfg, 0, lengths=[3000, 1300], budgets=np.array([[256, 100]], np.int32))
    return cfg, d


@pytest.mark.gpu
def test_noalloc_matches_workspace_entry_point_twice(cuda_device):
    dev = cuda_device
    cfg, d = _layer()
    q, k, v = d["q_win"].to(dev), d["k"].to(dev), d["v"].to(dev)
    prob = ckv.Problem(q, k, d["cu_seqlens"], cfg.window, cfg.pool_width)
    assert ckv.workspace_size(prob) <= B.STATIC_SCRATCH_BYTES

    ref = ckv.LayerOutputs(prob, d["budgets"], 128, k.dtype, dev)
    ws = ckv.workspace(prob, dev)
    cu_ref = ckv.compress_layer(prob, q, k, v, d["srh_mask"], d["budgets"], ref.indices,
                                ref.k_out, ref.v_out, ws, raw=ref.raw, pooled=ref.pooled)
    torch.cuda.synchronize()
    assert ckv.read_device_status(ws) == 0

    for call in range(2):
        out = ckv.LayerOutputs(prob, d["budgets"], 128, k.dtype, dev)
        status = torch.full((1,), -123, dtype=torch.int32, device=dev)
        cu_out = ckv.compress_layer_noalloc(prob, q, k, v, d["srh_mask"], d["budgets"],
                                            out.indices, out.k_out, out.v_out, raw=out.raw,
                                            pooled=out.pooled, device_status=status)
        torch.cuda.synchronize()
        assert int(status.item()) == 0, call
        assert np.array_equal(cu_out, cu_ref)
        compare.check_scores("raw", out.raw.cpu().numpy(), ref.raw.cpu().numpy())
        compare.check_scores("pooled", out.pooled.cpu().numpy(), ref.pooled.cpu().numpy())
        assert torch.equal(out.indices, ref.indices), call
        assert torch.equal(out.k_out.view(torch.int16), ref.k_out.view(torch.int16)), call
        assert torch.equal(out.v_out.view(torch.int16), ref.v_out.view(torch.int16)), call


def test_noalloc_rejects_problems_beyond_the_static_scratch():
    # 2^21 prefix tokens x 8 groups x 2 score vectors x 4 B = 128 MiB of scratch
    L = 1 << 21
    q = torch.zeros((1, 32, 32, 128), dtype=torch.bfloat16)
    # an overlapping host view: only shapes and strides are read, never the data
    k = torch.zeros((L - 1) * 8 + 7 * 8 + 128, dtype=torch.bfloat16).as_strided(
        (L, 8, 128), (8, 8, 1))
    prob = ckv.Problem(q, k, [0, L], 32, 7)
    assert ckv.workspace_size(prob) > B.STATIC_SCRATCH_BYTES
    with pytest.raises(ckv.CompressKVError) as e:
        ckv.compress_layer_noalloc(prob, q, k, k, np.ones(32, np.uint8), [256],
                                   None, None, None, stream=0)
    assert e.value.code == B.CKV_ERR_STATIC_SCRATCH
