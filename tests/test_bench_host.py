"""Host logic of the benchmark: how many layers one compress_layers call
packs (the most, up to four, whose exponent tables with the actual SRH rows
fit one 128 MiB set; two when a single layer's table does not)."""
import numpy as np

import bench
import workloads as wl


def _lpc(name):
    cfg = wl.get(name)
    lengths = wl.sequence_lengths(cfg)
    masks = wl.srh_masks(cfg)
    layers = [{"srh_mask": masks[l]} for l in range(cfg.n_layers)]
    return bench.layers_per_call(cfg, layers, lengths)


def test_expo_stride_matches_the_library_rule():
    assert [bench.expo_stride(r) for r in (0, 1, 8, 9, 32, 33, 64, 96, 192, 256)] == \
        [8, 8, 8, 16, 32, 64, 64, 128, 256, 256]


def test_layers_per_call_of_the_workloads():
    assert _lpc("c2") == 4   # ~25 MB of table per layer
    assert _lpc("c3") == 1   # ~100 MB per layer: one layer per set
    assert _lpc("c4") == 2   # a layer's table exceeds the set: two passes
    assert _lpc("c5") == 2


def test_layers_per_call_bounds():
    cfg = wl.get("c2").scaled(seq_len=1000, n_layers=8)
    lengths = wl.sequence_lengths(cfg)
    one_head = np.zeros(cfg.num_q_heads, bool)
    one_head[::cfg.num_q_heads // cfg.num_kv_heads] = True
    layers = [{"srh_mask": one_head} for _ in range(cfg.n_layers)]
    assert bench.layers_per_call(cfg, layers, lengths) == bench.MAX_LAYERS_PER_CALL
