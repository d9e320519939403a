"""The C ABI library without a GPU: it builds, loads, exports every function
include/compresskv.h declares, and rejects bad arguments on the host before
anything is enqueued (these calls make no CUDA call)."""
import ctypes
import os
import re

import numpy as np
import pytest
import torch

import paper_2606_24467_gb300 as ckv
from paper_2606_24467_gb300 import compresskv as B

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include",
                      "compresskv.h")


def _declared():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"\b(compresskv_\w+)\s*\(", text)))


def test_header_and_binding_agree():
    assert _declared() == sorted(B.EXPORTED)


def test_library_loads_and_exports_every_symbol():
    lib = ckv.load()
    for name in _declared():
        assert hasattr(lib, name), name
    assert ckv.status_string(-3) == "budget smaller than the observation window"
    assert ckv.status_string(0) == "ok"


def _problem(L=(300, 40), Hq=8, Hkv=2, W=32, P=7, dtype=torch.bfloat16, **kw):
    cu = np.concatenate([[0], np.cumsum(L)]).astype(np.int32)
    q = torch.zeros((len(L), Hq, W, 128), dtype=dtype)
    k = torch.zeros((int(cu[-1]), Hkv, 128), dtype=dtype)
    return ckv.Problem(q, k, cu, W, P, **kw), q, k


def test_workspace_size_and_layout():
    prob, q, k = _problem()
    n = ckv.workspace_size(prob)
    assert n >= 2 * 2 * (268 + 8) * 4
    cu_prefix, cu_out = ckv.output_layout(prob, [100, 100])
    assert cu_prefix.tolist() == [0, 268, 276]
    assert cu_out.tolist() == [0, 100, 140]


def test_budget_below_window_is_rejected():
    prob, q, k = _problem()
    with pytest.raises(ckv.CompressKVError) as e:
        ckv.output_layout(prob, [31, 100])
    assert e.value.code == B.CKV_ERR_BUDGET


def _fake_dev_ptr(n=1 << 20):
    # An aligned address that is never dereferenced: every call below fails
    # validation on the host first.
    return 1 << 30


def test_invalid_shapes_rejected():
    lib = ckv.load()
    prob, q, k = _problem()
    s = prob.struct
    for field, value, code in (("head_dim", 64, B.CKV_ERR_UNSUPPORTED),
                               ("pool_width", 4, B.CKV_ERR_INVALID_ARG),
                               ("window", 0, B.CKV_ERR_INVALID_ARG),
                               ("num_q_heads", 7, B.CKV_ERR_INVALID_ARG),
                               ("dtype", 5, B.CKV_ERR_INVALID_ARG),
                               ("pool_kind", 2, B.CKV_ERR_INVALID_ARG),
                               ("kv_token_stride", 100, B.CKV_ERR_INVALID_ARG)):
        old = getattr(s, field)
        setattr(s, field, value)
        assert lib.compresskv_workspace_size(prob.ref) == 0
        rc = lib.compresskv_output_layout(prob.ref, None, None, None)
        assert rc == code, (field, rc)
        setattr(s, field, old)


def test_compress_layer_host_errors():
    lib = ckv.load()
    prob, q, k = _problem()
    vp = ctypes.c_void_p
    ws = vp(_fake_dev_ptr())
    n = ckv.workspace_size(prob)
    mask_ok = np.zeros(8, np.uint8)
    mask_ok[[1, 6]] = 1
    mask_empty = np.zeros(8, np.uint8)
    mask_empty[1] = 1  # group 1 (heads 4-7) has no SRH head
    bud, bp = B._i32([64, 64])
    cu_out = (ctypes.c_int32 * 3)()

    def call(mask, budgets_ptr=bp, workspace=ws, wsn=n, qptr=vp(1 << 30)):
        return lib.compresskv_compress_layer(
            prob.ref, qptr, vp(1 << 30), vp(1 << 30), vp(mask.ctypes.data), budgets_ptr,
            vp(1 << 30), cu_out, vp(1 << 30), vp(1 << 30), None, None, workspace, wsn, None)

    assert call(mask_empty) == B.CKV_ERR_EMPTY_SRH_GROUP
    assert call(mask_ok, workspace=vp(None)) == B.CKV_ERR_WORKSPACE
    assert call(mask_ok, wsn=n - 1) == B.CKV_ERR_WORKSPACE
    assert call(mask_ok, workspace=vp((1 << 30) + 16)) == B.CKV_ERR_WORKSPACE
    b2, bp2 = B._i32([64, 10])
    assert call(mask_ok, budgets_ptr=bp2) == B.CKV_ERR_BUDGET
    big = np.ones(8, np.uint8)          # 4 heads x W=32 = 128 rows: fine
    prob.struct.window = 80             # 4 x 80 = 320 rows > 256: unsupported
    b3, bp3 = B._i32([100, 100])
    # the workspace bound grows with the window (exponent rows of G*W)
    assert call(big, budgets_ptr=bp3, wsn=ckv.workspace_size(prob)) == B.CKV_ERR_UNSUPPORTED


def test_compress_layers_host_errors():
    """The multi-layer call checks its mask count against the packed batch
    and each mask's groups against its own block of sequences."""
    lib = ckv.load()
    prob, q, k = _problem()  # batch 2: two one-sequence blocks
    vp = ctypes.c_void_p
    ws = vp(_fake_dev_ptr())
    n = ckv.workspace_size(prob)
    mask_ok = np.zeros(8, np.uint8)
    mask_ok[[1, 6]] = 1
    mask_empty = np.zeros(8, np.uint8)
    mask_empty[1] = 1  # group 1 (heads 4-7) has no SRH head
    bud, bp = B._i32([64, 64])
    cu_out = (ctypes.c_int32 * 3)()

    def call(n_masks, masks, p=prob, budgets_ptr=bp, wsn=n):
        m = np.ascontiguousarray(np.stack(masks))
        return lib.compresskv_compress_layers(
            p.ref, n_masks, vp(1 << 30), vp(1 << 30), vp(1 << 30), vp(m.ctypes.data),
            budgets_ptr, vp(1 << 30), cu_out, vp(1 << 30), vp(1 << 30), None, None, ws, wsn,
            None)

    assert call(0, [mask_ok]) == B.CKV_ERR_INVALID_ARG
    assert call(3, [mask_ok] * 3) == B.CKV_ERR_INVALID_ARG   # 3 does not divide batch 2
    assert call(2, [mask_ok, mask_empty]) == B.CKV_ERR_EMPTY_SRH_GROUP  # second block
    assert call(2, [mask_empty, mask_ok]) == B.CKV_ERR_EMPTY_SRH_GROUP  # first block
    # one mask for both sequences is the single-layer call: the empty group fails too
    assert call(1, [mask_empty]) == B.CKV_ERR_EMPTY_SRH_GROUP
    # per-layer selection runs the separate kernels: at most 4 masks per call
    p5, _, _ = _problem(L=(100,) * 5, selection="layer")
    b5, bp5 = B._i32([64] * 5)
    cu_out = (ctypes.c_int32 * 6)()
    assert call(5, [mask_ok] * 5, p=p5, budgets_ptr=bp5,
                wsn=ckv.workspace_size(p5)) == B.CKV_ERR_UNSUPPORTED
    # per-group selection runs the persistent kernel: at most 256 masks
    p257, _, _ = _problem(L=(40,) * 257)
    b257, bp257 = B._i32([32] * 257)
    cu_out = (ctypes.c_int32 * 258)()
    assert call(257, [mask_ok] * 257, p=p257, budgets_ptr=bp257,
                wsn=ckv.workspace_size(p257)) == B.CKV_ERR_UNSUPPORTED


def test_compress_layers_lse_host_errors():
    lib = ckv.load()
    prob, q, k = _problem()
    vp = ctypes.c_void_p
    ws = vp(_fake_dev_ptr())
    n = ckv.workspace_size(prob)
    mask_ok = np.zeros(8, np.uint8)
    mask_ok[[1, 6]] = 1
    mask_empty = np.zeros(8, np.uint8)
    mask_empty[1] = 1
    bud, bp = B._i32([64, 64])
    cu_out = (ctypes.c_int32 * 3)()

    def call(n_masks, masks, lse=vp(1 << 30)):
        m = np.ascontiguousarray(np.stack(masks))
        return lib.compresskv_compress_layers_lse(
            prob.ref, n_masks, vp(1 << 30), vp(1 << 30), vp(1 << 30), lse, 8 * 32, 32,
            vp(m.ctypes.data), bp, vp(1 << 30), cu_out, vp(1 << 30), vp(1 << 30), None, None,
            ws, n, None)

    assert call(0, [mask_ok]) == B.CKV_ERR_INVALID_ARG
    assert call(3, [mask_ok] * 3) == B.CKV_ERR_INVALID_ARG
    assert call(2, [mask_ok, mask_ok], lse=vp(None)) == B.CKV_ERR_INVALID_ARG
    assert call(2, [mask_ok, mask_empty]) == B.CKV_ERR_EMPTY_SRH_GROUP


def test_compress_layers_binding_checks_mask_shape():
    prob, q, k = _problem()
    with pytest.raises(ckv.CompressKVError) as e:
        ckv.compress_layers(prob, 2, q, k, k, np.ones((3, 8), np.uint8), [64, 64], k, k, k,
                            torch.zeros(16, dtype=torch.uint8))
    assert e.value.code == B.CKV_ERR_INVALID_ARG


def test_selection_scope_validation():
    lib = ckv.load()
    prob, q, k = _problem()
    prob.struct.selection = 2
    assert lib.compresskv_workspace_size(prob.ref) == 0
    assert lib.compresskv_output_layout(prob.ref, None, None, None) == B.CKV_ERR_INVALID_ARG
    with pytest.raises(ckv.CompressKVError):
        _problem(selection="heads")
    # the per-layer scope keeps an extra row of summed scores in the workspace
    g, _, _ = _problem()
    lay, _, _ = _problem(selection="layer")
    assert ckv.workspace_size(lay) >= ckv.workspace_size(g) + (268 + 8) * 4


def test_layer_scope_host_errors():
    lib = ckv.load()
    prob, q, k = _problem(selection="layer")
    vp = ctypes.c_void_p
    n = ckv.workspace_size(prob)
    bud, bp = B._i32([64, 64])
    cu_out = (ctypes.c_int32 * 3)()
    no_srh = np.zeros(8, np.uint8)  # no SRH head anywhere in the layer
    rc = lib.compresskv_compress_layer(
        prob.ref, vp(1 << 30), vp(1 << 30), vp(1 << 30), vp(no_srh.ctypes.data), bp,
        vp(1 << 30), cu_out, vp(1 << 30), vp(1 << 30), None, None, vp(1 << 30), n, None)
    assert rc == B.CKV_ERR_EMPTY_SRH_GROUP
    # per-layer selection has no per-group pooled output in compresskv_select
    rc = lib.compresskv_select(prob.ref, vp(1 << 30), bp, vp(1 << 30), cu_out, vp(1 << 30),
                               vp(1 << 30), n, None)
    assert rc == B.CKV_ERR_INVALID_ARG


def test_head_budget_host_errors_and_layout():
    lib = ckv.load()
    prob, q, k = _problem()
    cu, rows = ckv.head_budget_layout(prob, [[100, 50], [300, 40]])
    assert cu.tolist() == [[0, 100, 140], [140, 190, 230]] and rows == 230
    vp = ctypes.c_void_p
    n = ckv.workspace_size(prob)
    mask = np.ones(8, np.uint8)
    cu_out = (ctypes.c_int32 * 6)()

    def call(gb, problem=prob):
        b, bp = B._i32(np.asarray(gb).reshape(-1))
        return lib.compresskv_compress_layer_head_budgets(
            problem.ref, vp(1 << 30), vp(1 << 30), vp(1 << 30), vp(mask.ctypes.data), bp,
            vp(1 << 30), cu_out, vp(1 << 30), vp(1 << 30), None, None, vp(1 << 30), n, None)

    assert call([[100, 31], [100, 100]]) == B.CKV_ERR_BUDGET
    lay, _, _ = _problem(selection="layer")
    assert call([[100, 100], [100, 100]], lay) == B.CKV_ERR_INVALID_ARG


def test_binding_checks_single_mask_length():
    prob, q, k = _problem()
    ws = torch.zeros(16, dtype=torch.uint8)
    for call in (lambda m: ckv.compress_layer(prob, q, k, k, m, [64, 64], k, k, k, ws),
                 lambda m: ckv.score(prob, q, k, m, k, ws),
                 lambda m: ckv.compress_layer_noalloc(prob, q, k, k, m, [64, 64], k, k, k),
                 lambda m: ckv.compress_layer_head_budgets(prob, q, k, k, m,
                                                           np.full((2, 2), 64), k, k, k, ws)):
        with pytest.raises(ckv.CompressKVError) as e:
            call(np.ones(7, np.uint8))  # num_q_heads is 8
        assert e.value.code == B.CKV_ERR_INVALID_ARG


def test_binding_checks_lse_tensor():
    prob, q, k = _problem()
    ws = torch.zeros(16, dtype=torch.uint8)
    mask = np.zeros(8, np.uint8)
    mask[[1, 6]] = 1
    good_shape = (2, 8, 32)
    bad = [torch.zeros(good_shape, dtype=torch.float32),            # host memory
           torch.zeros((2, 2, 32), dtype=torch.float32),            # [B, H_kv, W]
           torch.zeros(good_shape, dtype=torch.float64),            # dtype
           torch.zeros((2, 8, 64), dtype=torch.float32)[:, :, ::2]]  # strided rows
    for lse in bad:
        with pytest.raises(ckv.CompressKVError) as e:
            ckv.compress_layer_lse(prob, q, k, k, lse, mask, [64, 64], k, k, k, ws)
        assert e.value.code == B.CKV_ERR_INVALID_ARG
        with pytest.raises(ckv.CompressKVError) as e:
            ckv.compress_layers_lse(prob, 2, q, k, k, lse, np.stack([mask, mask]), [64, 64], k,
                                    k, k, ws)
        assert e.value.code == B.CKV_ERR_INVALID_ARG



def test_stall_hook_limits():
    """The failure-path test hook takes 0 (cancel) or 0.1 ms .. 2 s."""
    for bad in (-1, 99_999, 2_000_000_001):
        with pytest.raises(ckv.CompressKVError):
            ckv.debug_stall_next_fused_call(bad)
    ckv.debug_stall_next_fused_call(1_000_000)
    ckv.debug_stall_next_fused_call(0)  # cancelled: no later call stalls


def test_max_pooling_workspace_and_unsupported_calls():
    """CKV_POOL_MAX: the workspace grows by one raw-score row per group head
    slot (G rows per group); the calls that cannot pool per head refuse it
    on the host."""
    lib = ckv.load()
    prob, q, k = _problem()
    s = prob.struct
    avg = lib.compresskv_workspace_size(prob.ref)
    s.pool_kind = B.CKV_POOL_MAX
    mx = lib.compresskv_workspace_size(prob.ref)
    G = s.num_q_heads // s.num_kv_heads
    p_total = sum(max(int(prob._cu[i + 1] - prob._cu[i]) - s.window, 0) for i in range(s.batch))
    assert mx >= avg + G * s.num_kv_heads * p_total * 4
    assert mx <= avg + 256 + (G * s.num_kv_heads * p_total * 4 + 255) // 256 * 256 + 256
    vp = ctypes.c_void_p
    ws = vp(_fake_dev_ptr())
    bud, bp = B._i32([64, 64])
    cu_out = (ctypes.c_int32 * 3)()
    rc = lib.compresskv_select(prob.ref, vp(_fake_dev_ptr()), bp, vp(_fake_dev_ptr()), cu_out, None,
                               ws, mx, None)
    assert rc == B.CKV_ERR_UNSUPPORTED
    s.pool_kind = B.CKV_POOL_AVG
