"""The five synthetic workloads the compression path is measured and checked on.

Shapes follow the long-context models the paper evaluates (Llama-3.1-8B,
Qwen2.5-7B-like GQA, Llama-3.1-70B): GQA head counts, head_dim 128, and the
paper's local setting of an observation window plus 1-D pooling (Sec. 4,
"Implementation Details"; these workloads use W = 32/64 and pooling width 7).
Every tensor is synthetic and seeded; see ``workloads.generate``.
"""
from __future__ import annotations

from dataclasses import dataclass, replace


@dataclass(frozen=True)
class Workload:
    name: str
    description: str
    n_layers: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    batch: int
    seq_len: int                  # fixed length (ignored when length_range is set)
    dtype: str                    # "fp16" | "bf16"
    window: int
    pool_width: int
    srh_per_group: tuple          # (lo, hi) inclusive SRH heads per group per layer
    needles_per_group: int
    budget_rule: str              # "fixed" | "dirichlet" | "frac_dirichlet" | "error_profile"
    budget_mean: float            # tokens (or fraction of L for "frac_dirichlet")
    budget_alpha: float = 2.0
    length_range: tuple | None = None   # (lo, hi) inclusive, ragged batch
    seed: int = 0

    @property
    def group_size(self) -> int:
        return self.num_q_heads // self.num_kv_heads

    def scaled(self, **overrides) -> "Workload":
        """A copy with some fields replaced (small test variants)."""
        return replace(self, **overrides)


WORKLOADS = {
    "llama8b_L4k_1layer": Workload(
        name="llama8b_L4k_1layer",
        description="1 layer, Llama-3.1-8B GQA (32 Q / 8 KV heads, d=128), batch 1, L=4096, "
                    "fp16, W=32, P=7, B=128, 1 SRH head per group, 16 needles per group",
        n_layers=1, num_q_heads=32, num_kv_heads=8, head_dim=128, batch=1, seq_len=4096,
        dtype="fp16", window=32, pool_width=7, srh_per_group=(1, 1), needles_per_group=16,
        budget_rule="fixed", budget_mean=128, seed=101),
    "llama8b_L32k_32layers": Workload(
        name="llama8b_L32k_32layers",
        description="32 layers, Llama-3.1-8B GQA, batch 1, L=32768, bf16, W=32, P=7, "
                    "per-layer budgets Dirichlet(2) with mean 256, 1-2 SRH heads per group",
        n_layers=32, num_q_heads=32, num_kv_heads=8, head_dim=128, batch=1, seq_len=32768,
        dtype="bf16", window=32, pool_width=7, srh_per_group=(1, 2), needles_per_group=16,
        budget_rule="dirichlet", budget_mean=256, seed=202),
    "llama8b_L128k_32layers": Workload(
        name="llama8b_L128k_32layers",
        description="32 layers, Llama-3.1-8B GQA, batch 1, L=131072, bf16, W=32, P=7, "
                    "per-layer budgets Dirichlet(2) with mean 917 (0.7% of L), 64 needles per group",
        n_layers=32, num_q_heads=32, num_kv_heads=8, head_dim=128, batch=1, seq_len=131072,
        dtype="bf16", window=32, pool_width=7, srh_per_group=(1, 2), needles_per_group=64,
        budget_rule="dirichlet", budget_mean=917, seed=303),
    "qwen7b_ragged8_28layers": Workload(
        name="qwen7b_ragged8_28layers",
        description="28 layers, Qwen2.5-7B GQA (28 Q / 4 KV heads), bf16, batch 8 ragged "
                    "lengths U[8K, 64K] (cu_seqlens), W=32, P=7, budgets 3% of each length, 2 SRH heads per group",
        n_layers=28, num_q_heads=28, num_kv_heads=4, head_dim=128, batch=8, seq_len=0,
        dtype="bf16", window=32, pool_width=7, srh_per_group=(2, 2), needles_per_group=16,
        budget_rule="frac_dirichlet", budget_mean=0.03, length_range=(8192, 65536), seed=404),
    "llama70b_L32k_b4_80layers": Workload(
        name="llama70b_L32k_b4_80layers",
        description="80 layers, Llama-3.1-70B GQA (64 Q / 8 KV heads), bf16, batch 4, L=32768, "
                    "W=64, P=7, budgets from a Dirichlet(1) eviction-error profile with mean 1% of L, "
                    "1-3 SRH heads per group",
        n_layers=80, num_q_heads=64, num_kv_heads=8, head_dim=128, batch=4, seq_len=32768,
        dtype="bf16", window=64, pool_width=7, srh_per_group=(1, 3), needles_per_group=16,
        budget_rule="error_profile", budget_mean=328, budget_alpha=1.0, seed=505),
}

# Short aliases in the order the workloads are listed above.
ALIASES = {
    "c1": "llama8b_L4k_1layer",
    "c2": "llama8b_L32k_32layers",
    "c3": "llama8b_L128k_32layers",
    "c4": "qwen7b_ragged8_28layers",
    "c5": "llama70b_L32k_b4_80layers",
}


def get(name: str) -> Workload:
    return WORKLOADS[ALIASES.get(name, name)]
