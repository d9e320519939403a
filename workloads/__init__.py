"""Seeded synthetic workloads (inputs only) for tests and the bench."""
from .configs import ALIASES, WORKLOADS, Workload, get  # noqa: F401
from .generate import (  # noqa: F401
    cu_seqlens,
    layer_budgets,
    make_layer,
    needle_positions,
    sequence_lengths,
    srh_masks,
    torch_dtype,
)
