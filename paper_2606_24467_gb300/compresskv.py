"""ctypes binding of libcompresskv (include/compresskv.h).

Argument marshalling only: every step of the compression path runs in the
library's CUDA kernels.  PyTorch supplies device memory and streams.  There
is no fallback: if the library is missing or fails to load, importing the
binding raises.
"""
from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, c_float, c_int32, c_int64, c_size_t, c_void_p

import numpy as np
import torch

from . import _build

CKV_OK = 0
CKV_ERR_INVALID_ARG = -1
CKV_ERR_UNSUPPORTED = -2
CKV_ERR_BUDGET = -3
CKV_ERR_EMPTY_SRH_GROUP = -4
CKV_ERR_WORKSPACE = -5
CKV_ERR_CUDA = -6
CKV_ERR_DEVICE_TIMEOUT = -7
CKV_ERR_DEVICE_INDEX = -8
CKV_ERR_STATIC_SCRATCH = -9
STATIC_SCRATCH_BYTES = 16 * 1024 * 1024
CKV_DTYPE_F16 = 0
CKV_DTYPE_BF16 = 1
CKV_POOL_AVG = 0
CKV_POOL_MAX = 1
CKV_SELECT_PER_GROUP = 0
CKV_SELECT_PER_LAYER = 1
KERNEL_KINDS = {1: "score", 2: "combine", 3: "select", 4: "gather", 5: "fused"}

EXPORTED = (
    "compresskv_workspace_size",
    "compresskv_workspace_init",
    "compresskv_output_layout",
    "compresskv_score",
    "compresskv_select",
    "compresskv_gather",
    "compresskv_compress_layer",
    "compresskv_compress_layers",
    "compresskv_compress_layer_noalloc",
    "compresskv_compress_layer_lse",
    "compresskv_compress_layers_lse",
    "compresskv_compress_layer_head_budgets",
    "compresskv_read_device_status",
    "compresskv_debug_stall_next_fused_call",
    "compresskv_allocate_layer_budgets",
    "compresskv_status_string",
)


class CkvTrace(ctypes.Structure):
    _fields_ = [("events", POINTER(c_void_p)), ("kinds", POINTER(c_int32)),
                ("capacity", c_int32), ("count", c_int32), ("launches", c_int64)]


class CkvProblem(ctypes.Structure):
    _fields_ = [("batch", c_int32), ("num_q_heads", c_int32), ("num_kv_heads", c_int32),
                ("head_dim", c_int32), ("window", c_int32), ("pool_width", c_int32),
                ("dtype", c_int32), ("pool_kind", c_int32), ("scale", c_float),
                ("selection", c_int32), ("cu_seqlens", POINTER(c_int32)),
                ("kv_token_stride", c_int64), ("kv_head_stride", c_int64),
                ("q_batch_stride", c_int64), ("q_head_stride", c_int64),
                ("q_win_stride", c_int64), ("trace", POINTER(CkvTrace))]


class CompressKVError(RuntimeError):
    def __init__(self, code: int, what: str):
        super().__init__(f"{what}: {status_string(code)} ({code})")
        self.code = code


_LIB = None


def library_path() -> str:
    return _build.LIB_PATH


def load(build_if_missing: bool = True) -> ctypes.CDLL:
    """Load libcompresskv (building it first if it is absent or stale)."""
    global _LIB
    if _LIB is not None:
        return _LIB
    path = library_path()
    if build_if_missing and _build.needs_build():
        _build.build()
    if not os.path.exists(path):
        raise RuntimeError(f"libcompresskv not built ({path}); run __graft_entry__.build()")
    lib = ctypes.CDLL(path)
    vp, pp = c_void_p, POINTER(CkvProblem)
    i32p = POINTER(c_int32)
    sig = {
        "compresskv_workspace_size": (c_size_t, [pp]),
        "compresskv_workspace_init": (c_int32, [vp, c_size_t, vp]),
        "compresskv_output_layout": (c_int32, [pp, i32p, i32p, i32p]),
        "compresskv_score": (c_int32, [pp, vp, vp, vp, vp, vp, c_size_t, vp]),
        "compresskv_select": (c_int32, [pp, vp, i32p, vp, i32p, vp, vp, c_size_t, vp]),
        "compresskv_gather": (c_int32, [pp, vp, i32p, vp, vp, vp, vp, vp, vp]),
        "compresskv_compress_layer": (c_int32, [pp, vp, vp, vp, vp, i32p, vp, i32p, vp, vp,
                                                 vp, vp, vp, c_size_t, vp]),
        "compresskv_compress_layers": (c_int32, [pp, c_int32, vp, vp, vp, vp, i32p, vp, i32p, vp,
                                                  vp, vp, vp, vp, c_size_t, vp]),
        "compresskv_compress_layer_noalloc": (c_int32, [pp, vp, vp, vp, vp, i32p, vp, i32p, vp,
                                                         vp, vp, vp, vp, vp]),
        "compresskv_compress_layer_lse": (c_int32, [pp, vp, vp, vp, vp, c_int64, c_int64, vp, i32p,
                                                     vp, i32p, vp, vp, vp, vp, vp, c_size_t, vp]),
        "compresskv_compress_layers_lse": (c_int32, [pp, c_int32, vp, vp, vp, vp, c_int64,
                                                      c_int64, vp, i32p, vp, i32p, vp, vp, vp,
                                                      vp, vp, c_size_t, vp]),
        "compresskv_compress_layer_head_budgets": (c_int32, [pp, vp, vp, vp, vp, i32p, vp, i32p,
                                                              vp, vp, vp, vp, vp, c_size_t, vp]),
        "compresskv_read_device_status": (c_int32, [vp, vp, i32p]),
        "compresskv_debug_stall_next_fused_call": (c_int32, [ctypes.c_longlong]),
        "compresskv_allocate_layer_budgets": (c_int32, [POINTER(ctypes.c_double), c_int32,
                                                        c_int64, c_int32, c_int32, i32p]),
        "compresskv_status_string": (ctypes.c_char_p, [c_int32]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _LIB = lib
    return lib


def status_string(code: int) -> str:
    return load().compresskv_status_string(int(code)).decode()


def _check(code: int, what: str):
    if code != CKV_OK:
        raise CompressKVError(code, what)


def _ptr(t) -> c_void_p:
    if t is None:
        return c_void_p(None)
    return c_void_p(t.data_ptr())


def _stream(stream) -> c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def _i32(arr) -> tuple:
    a = np.ascontiguousarray(np.asarray(arr, dtype=np.int32))
    return a, a.ctypes.data_as(POINTER(c_int32))


class Problem:
    """One layer's problem description (wraps ``ckv_problem``).

    ``q_win`` is ``[B, H_q, W, d]`` and ``k`` is ``[T, H_kv, d]`` (any
    strides with ``d`` contiguous); only shapes, strides and dtype are read.
    """

    def __init__(self, q_win: torch.Tensor, k: torch.Tensor, cu_seqlens, window: int,
                 pool_width: int, scale: float = 0.0, trace: "Trace | None" = None,
                 selection: str = "group", pool: str = "avg"):
        """``selection``: "group" (each KV group keeps its own SRH heads'
        choice) or "layer" (one choice per sequence shared by every group);
        ``pool``: "avg" or "max" (each SRH head max-pooled, then summed)."""
        if k.dtype not in (torch.float16, torch.bfloat16) or q_win.dtype != k.dtype:
            raise CompressKVError(CKV_ERR_INVALID_ARG, "Q and K must share an f16/bf16 dtype")
        self._cu, cu_ptr = _i32(cu_seqlens)
        self.trace = trace
        s = CkvProblem()
        s.batch = len(self._cu) - 1
        s.num_q_heads = q_win.shape[1]
        s.num_kv_heads = k.shape[1]
        s.head_dim = k.shape[2]
        s.window = int(window)
        s.pool_width = int(pool_width)
        s.dtype = CKV_DTYPE_BF16 if k.dtype == torch.bfloat16 else CKV_DTYPE_F16
        if pool not in ("avg", "max"):
            raise CompressKVError(CKV_ERR_INVALID_ARG, "pool must be 'avg' or 'max'")
        s.pool_kind = CKV_POOL_MAX if pool == "max" else CKV_POOL_AVG
        s.scale = float(scale)
        if selection not in ("group", "layer"):
            raise CompressKVError(CKV_ERR_INVALID_ARG, "selection must be 'group' or 'layer'")
        s.selection = CKV_SELECT_PER_LAYER if selection == "layer" else CKV_SELECT_PER_GROUP
        s.cu_seqlens = cu_ptr
        s.kv_token_stride = k.stride(0)
        s.kv_head_stride = k.stride(1)
        s.q_batch_stride = q_win.stride(0)
        s.q_head_stride = q_win.stride(1)
        s.q_win_stride = q_win.stride(2)
        s.trace = ctypes.pointer(trace.struct) if trace is not None else None
        self.struct = s
        self.batch = s.batch
        self.num_kv_heads = s.num_kv_heads

    @property
    def ref(self):
        return ctypes.byref(self.struct)


class Trace:
    """Launch trace: ``capacity`` launches bracketed by CUDA events."""

    def __init__(self, capacity: int):
        """``capacity`` = 0 only counts launches (no events are recorded)."""
        self.events = [torch.cuda.Event(enable_timing=True) for _ in range(2 * capacity)]
        for e in self.events:  # torch creates the CUDA event on its first record
            e.record()
        if capacity:
            torch.cuda.synchronize()
        self._ev = (c_void_p * max(1, 2 * capacity))(*[e.cuda_event for e in self.events])
        self._kinds = (c_int32 * max(1, capacity))()
        self.struct = CkvTrace(ctypes.cast(self._ev, POINTER(c_void_p)),
                               ctypes.cast(self._kinds, POINTER(c_int32)), capacity, 0, 0)

    def reset(self):
        self.struct.count = 0
        self.struct.launches = 0

    @property
    def launches(self) -> int:
        return int(self.struct.launches)

    def records(self):
        """[(kind name, elapsed ms)] for the recorded launches (call after a sync)."""
        out = []
        for i in range(self.struct.count):
            out.append((KERNEL_KINDS.get(self._kinds[i], "?"),
                        self.events[2 * i].elapsed_time(self.events[2 * i + 1])))
        return out


def workspace_size(problem: Problem) -> int:
    n = load().compresskv_workspace_size(problem.ref)
    if n == 0:
        raise CompressKVError(CKV_ERR_INVALID_ARG, "compresskv_workspace_size")
    return int(n)


def workspace(problem: Problem, device=None, stream=None) -> torch.Tensor:
    """A zero-status workspace tensor for ``problem`` (256-byte aligned)."""
    n = workspace_size(problem)
    ws = torch.empty(n, dtype=torch.uint8, device=device or "cuda")
    assert ws.data_ptr() % 256 == 0
    _check(load().compresskv_workspace_init(_ptr(ws), n, _stream(stream)), "workspace_init")
    return ws


def output_layout(problem: Problem, budgets):
    b, bp = _i32(budgets)
    cu_prefix = np.zeros(problem.batch + 1, np.int32)
    cu_out = np.zeros(problem.batch + 1, np.int32)
    _check(load().compresskv_output_layout(problem.ref, bp,
                                           cu_prefix.ctypes.data_as(POINTER(c_int32)),
                                           cu_out.ctypes.data_as(POINTER(c_int32))),
           "output_layout")
    return cu_prefix, cu_out


def _mask(srh_mask, problem: "Problem"):
    """One layer's SRH mask as host bytes; the library reads num_q_heads of them."""
    m = np.ascontiguousarray(np.asarray(srh_mask).astype(np.uint8).reshape(-1))
    if m.size != int(problem.struct.num_q_heads):
        raise CompressKVError(CKV_ERR_INVALID_ARG, "srh_mask must have num_q_heads entries")
    return m, c_void_p(m.ctypes.data)


def _check_lse(problem: "Problem", lse_win, k, rows: int):
    """lse_win must be a float32 device tensor on K's device, [rows, H_q, W]
    with contiguous window rows: the scoring kernel reads every (sequence,
    SRH head, window row) element through the given strides."""
    W = int(problem.struct.window)
    shape = (int(rows), int(problem.struct.num_q_heads), W)
    if (not isinstance(lse_win, torch.Tensor) or lse_win.dtype != torch.float32
            or not lse_win.is_cuda or lse_win.device != k.device or tuple(lse_win.shape) != shape
            or lse_win.stride(2) != 1 or (shape[1] > 1 and lse_win.stride(1) < W)
            or (shape[0] > 1 and lse_win.stride(0) < 1)):
        raise CompressKVError(CKV_ERR_INVALID_ARG,
                              f"lse_win must be a float32 CUDA tensor on K's device of shape "
                              f"{shape} with contiguous window rows")


def score(problem: Problem, q_win, k, srh_mask, raw, ws, stream=None):
    m, mp = _mask(srh_mask, problem)
    _check(load().compresskv_score(problem.ref, _ptr(q_win), _ptr(k), mp, _ptr(raw), _ptr(ws),
                                   ws.numel(), _stream(stream)), "compresskv_score")


def select(problem: Problem, raw, budgets, indices, ws, pooled=None, stream=None) -> np.ndarray:
    b, bp = _i32(budgets)
    cu_out = np.zeros(problem.batch + 1, np.int32)
    _check(load().compresskv_select(problem.ref, _ptr(raw), bp, _ptr(indices),
                                    cu_out.ctypes.data_as(POINTER(c_int32)), _ptr(pooled),
                                    _ptr(ws), ws.numel(), _stream(stream)), "compresskv_select")
    return cu_out


def gather(problem: Problem, indices, cu_out, k, v, k_out, v_out, ws=None, stream=None):
    c, cp = _i32(cu_out)
    _check(load().compresskv_gather(problem.ref, _ptr(indices), cp, _ptr(k), _ptr(v),
                                    _ptr(k_out), _ptr(v_out), _ptr(ws), _stream(stream)),
           "compresskv_gather")


def compress_layer(problem: Problem, q_win, k, v, srh_mask, budgets, indices, k_out, v_out, ws,
                   raw=None, pooled=None, stream=None) -> np.ndarray:
    m, mp = _mask(srh_mask, problem)
    b, bp = _i32(budgets)
    cu_out = np.zeros(problem.batch + 1, np.int32)
    _check(load().compresskv_compress_layer(
        problem.ref, _ptr(q_win), _ptr(k), _ptr(v), mp, bp, _ptr(indices),
        cu_out.ctypes.data_as(POINTER(c_int32)), _ptr(k_out), _ptr(v_out), _ptr(raw),
        _ptr(pooled), _ptr(ws), ws.numel(), _stream(stream)), "compresskv_compress_layer")
    return cu_out


def compress_layers(problem: Problem, n_masks: int, q_win, k, v, srh_masks, budgets, indices,
                    k_out, v_out, ws, raw=None, pooled=None, stream=None) -> np.ndarray:
    """Several layers in one call: ``problem``'s batch packs ``n_masks`` blocks
    of sequences (block l = layer l: K ``[n_layers*T, H_kv, d]``, Q window
    ``[n_layers*B, H_q, W, d]``, cu_seqlens repeated per layer with offset
    l*T) and block l selects with ``srh_masks[l]`` (``[n_masks, H_q]``);
    budgets ``[n_layers*B]``; outputs as for compress_layer on that batch."""
    m = np.ascontiguousarray(np.asarray(srh_masks).astype(np.uint8).reshape(-1))
    if n_masks >= 1 and m.size != int(n_masks) * int(problem.struct.num_q_heads):
        raise CompressKVError(CKV_ERR_INVALID_ARG, "srh_masks must be [n_masks, num_q_heads]")
    b, bp = _i32(budgets)
    cu_out = np.zeros(problem.batch + 1, np.int32)
    _check(load().compresskv_compress_layers(
        problem.ref, int(n_masks), _ptr(q_win), _ptr(k), _ptr(v), c_void_p(m.ctypes.data), bp,
        _ptr(indices), cu_out.ctypes.data_as(POINTER(c_int32)), _ptr(k_out), _ptr(v_out),
        _ptr(raw), _ptr(pooled), _ptr(ws), ws.numel(), _stream(stream)),
        "compresskv_compress_layers")
    return cu_out


def compress_layer_noalloc(problem: Problem, q_win, k, v, srh_mask, budgets, indices, k_out,
                           v_out, raw=None, pooled=None, device_status=None,
                           stream=None) -> np.ndarray:
    """compress_layer without a workspace: the library's static scratch is
    used (for callers that cannot allocate device memory)."""
    m, mp = _mask(srh_mask, problem)
    b, bp = _i32(budgets)
    cu_out = np.zeros(problem.batch + 1, np.int32)
    _check(load().compresskv_compress_layer_noalloc(
        problem.ref, _ptr(q_win), _ptr(k), _ptr(v), mp, bp, _ptr(indices),
        cu_out.ctypes.data_as(POINTER(c_int32)), _ptr(k_out), _ptr(v_out), _ptr(raw),
        _ptr(pooled), _ptr(device_status), _stream(stream)), "compresskv_compress_layer_noalloc")
    return cu_out


def allocate_layer_budgets(layer_errors, total_budget: int, min_budget: int = 32,
                           max_budget: int = 0) -> np.ndarray:
    """Per-layer budgets from offline layer errors (Sec. 3.4); host only.
    `max_budget` <= 0 selects 3 * total_budget / n_layers."""
    err = np.ascontiguousarray(np.asarray(layer_errors, dtype=np.float64))
    out = np.zeros(err.size, dtype=np.int32)
    _check(load().compresskv_allocate_layer_budgets(
        err.ctypes.data_as(POINTER(ctypes.c_double)), int(err.size), int(total_budget),
        int(min_budget), int(max_budget), out.ctypes.data_as(POINTER(c_int32))),
        "compresskv_allocate_layer_budgets")
    return out


def compress_layer_lse(problem: Problem, q_win, k, v, lse_win, srh_mask, budgets, indices, k_out,
                       v_out, ws, raw=None, pooled=None, stream=None) -> np.ndarray:
    """compress_layer with the window queries' log-sum-exp given:
    ``lse_win`` is a float32 ``[B, H_q, W]`` tensor (window rows contiguous)."""
    _check_lse(problem, lse_win, k, problem.batch)
    m, mp = _mask(srh_mask, problem)
    b, bp = _i32(budgets)
    cu_out = np.zeros(problem.batch + 1, np.int32)
    _check(load().compresskv_compress_layer_lse(
        problem.ref, _ptr(q_win), _ptr(k), _ptr(v), _ptr(lse_win), lse_win.stride(0),
        lse_win.stride(1), mp, bp, _ptr(indices), cu_out.ctypes.data_as(POINTER(c_int32)),
        _ptr(k_out), _ptr(v_out), _ptr(raw), _ptr(pooled), _ptr(ws), ws.numel(), _stream(stream)),
        "compresskv_compress_layer_lse")
    return cu_out


def compress_layers_lse(problem: Problem, n_masks: int, q_win, k, v, lse_win, srh_masks, budgets,
                        indices, k_out, v_out, ws, raw=None, pooled=None,
                        stream=None) -> np.ndarray:
    """compress_layers with the window queries' log-sum-exp given, packed like
    the batch: ``lse_win`` is float32 ``[n_layers*B, H_q, W]``."""
    _check_lse(problem, lse_win, k, problem.batch)
    m = np.ascontiguousarray(np.asarray(srh_masks).astype(np.uint8).reshape(-1))
    if n_masks >= 1 and m.size != int(n_masks) * int(problem.struct.num_q_heads):
        raise CompressKVError(CKV_ERR_INVALID_ARG, "srh_masks must be [n_masks, num_q_heads]")
    b, bp = _i32(budgets)
    cu_out = np.zeros(problem.batch + 1, np.int32)
    _check(load().compresskv_compress_layers_lse(
        problem.ref, int(n_masks), _ptr(q_win), _ptr(k), _ptr(v), _ptr(lse_win),
        lse_win.stride(0), lse_win.stride(1), c_void_p(m.ctypes.data), bp, _ptr(indices),
        cu_out.ctypes.data_as(POINTER(c_int32)), _ptr(k_out), _ptr(v_out), _ptr(raw),
        _ptr(pooled), _ptr(ws), ws.numel(), _stream(stream)), "compresskv_compress_layers_lse")
    return cu_out


def head_budget_layout(problem: Problem, group_budgets) -> tuple[np.ndarray, int]:
    """Host-side output layout of compress_layer_head_budgets: cu_out
    ``[H_kv, B+1]`` (group-major packing) and the total number of rows."""
    b = np.asarray(group_budgets, dtype=np.int64).reshape(problem.batch, problem.num_kv_heads)
    lens = np.diff(np.asarray(problem._cu, dtype=np.int64))
    kept = np.minimum(b, lens[:, None])
    cu = np.zeros((problem.num_kv_heads, problem.batch + 1), dtype=np.int32)
    row = 0
    for g in range(problem.num_kv_heads):
        for s in range(problem.batch):
            cu[g, s] = row
            row += int(kept[s, g])
        cu[g, problem.batch] = row
    return cu, row


def compress_layer_head_budgets(problem: Problem, q_win, k, v, srh_mask, group_budgets, indices,
                                k_out, v_out, ws, raw=None, pooled=None,
                                stream=None) -> np.ndarray:
    """compress_layer with a budget per (sequence, KV group): ``group_budgets``
    is ``[B, H_kv]``; outputs are packed group-major (see head_budget_layout);
    returns cu_out ``[H_kv, B+1]``."""
    m, mp = _mask(srh_mask, problem)
    b, bp = _i32(np.asarray(group_budgets).reshape(-1))
    cu_out = np.zeros((problem.num_kv_heads, problem.batch + 1), np.int32)
    _check(load().compresskv_compress_layer_head_budgets(
        problem.ref, _ptr(q_win), _ptr(k), _ptr(v), mp, bp, _ptr(indices),
        cu_out.ctypes.data_as(POINTER(c_int32)), _ptr(k_out), _ptr(v_out), _ptr(raw),
        _ptr(pooled), _ptr(ws), ws.numel(), _stream(stream)),
        "compresskv_compress_layer_head_budgets")
    return cu_out


def debug_stall_next_fused_call(wait_ns: int) -> None:
    """Test hook: the next persistent-kernel call stalls on purpose and stops
    with CKV_ERR_DEVICE_TIMEOUT after `wait_ns` (see the header)."""
    _check(load().compresskv_debug_stall_next_fused_call(ctypes.c_longlong(int(wait_ns))),
           "compresskv_debug_stall_next_fused_call")


def read_device_status(ws, stream=None) -> int:
    out = c_int32(0)
    _check(load().compresskv_read_device_status(_ptr(ws), _stream(stream), ctypes.byref(out)),
           "read_device_status")
    return int(out.value)


class LayerOutputs:
    """Device buffers for one compressed layer, sized from the budgets."""

    def __init__(self, problem: Problem, budgets, head_dim: int, dtype, device, scores=True):
        cu_prefix, cu_out = output_layout(problem, budgets)
        H = problem.num_kv_heads
        self.cu_prefix, self.cu_out = cu_prefix, cu_out
        self.indices = torch.empty((H, int(cu_out[-1])), dtype=torch.int32, device=device)
        self.k_out = torch.empty((int(cu_out[-1]), H, head_dim), dtype=dtype, device=device)
        self.v_out = torch.empty_like(self.k_out)
        self.raw = torch.empty((H, int(cu_prefix[-1])), dtype=torch.float32, device=device) if scores else None
        self.pooled = torch.empty_like(self.raw) if scores else None
