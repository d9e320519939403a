"""CompressKV prefill-end KV-cache compression on one GB300 (sm_103a).

The compression path (window scoring with the SRH heads, pooling, budgeted
top-k, K/V gather) runs in the CUDA kernels of ``libcompresskv``; this
package holds the kernels' sources (``csrc/``), their nvcc build and a thin
ctypes binding of the C ABI in ``include/compresskv.h``.
"""
from . import compresskv  # noqa: F401
from .compresskv import (  # noqa: F401
    CompressKVError,
    LayerOutputs,
    Problem,
    Trace,
    allocate_layer_budgets,
    compress_layer,
    compress_layer_head_budgets,
    compress_layer_lse,
    compress_layer_noalloc,
    compress_layers,
    compress_layers_lse,
    debug_stall_next_fused_call,
    gather,
    head_budget_layout,
    load,
    output_layout,
    read_device_status,
    score,
    select,
    status_string,
    workspace,
    workspace_size,
)
