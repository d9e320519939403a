"""CompressKV float64 CPU oracle: test infrastructure, never the product path.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline
and reference legs import this package.
"""
from .compresskv_oracle import (  # noqa: F401
    OracleError,
    compress_layer,
    compress_layer_head_budgets,
    compress_unit,
    default_scale,
    kept_count,
    kth_value,
    pool_avg,
    pool_heads,
    pool_max,
    raw_scores,
    select_top,
    srh_heads,
    window_attention,
    window_lse,
)
