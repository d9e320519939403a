"""Host logic of the benchmark: how many layers one compress_layers call
packs (every layer of the step, up to the 256 SRH masks one per-group call
takes), and the step's algorithmic bytes."""
import numpy as np

import bench
import workloads as wl


def _lpc(name):
    cfg = wl.get(name)
    lengths = wl.sequence_lengths(cfg)
    masks = wl.srh_masks(cfg)
    layers = [{"srh_mask": masks[l]} for l in range(cfg.n_layers)]
    return bench.layers_per_call(cfg, layers, lengths)


def test_layers_per_call_of_the_workloads():
    assert _lpc("c1") == 1
    assert _lpc("c2") == 32
    assert _lpc("c3") == 32
    assert _lpc("c4") == 28
    assert _lpc("c5") == 80


def test_layers_per_call_bounds():
    cfg = wl.get("c2").scaled(seq_len=1000, n_layers=300)
    lengths = wl.sequence_lengths(cfg)
    layers = [{"srh_mask": np.ones(cfg.num_q_heads, bool)} for _ in range(cfg.n_layers)]
    assert bench.layers_per_call(cfg, layers, lengths) == bench.MAX_LAYERS_PER_CALL == 256


def test_algorithmic_bytes_of_the_bench_step():
    # K once for scoring, the SRH query rows, and 4 x 256 B per kept token and
    # group (K and V rows read and written)
    cfg = wl.get("c2").scaled(n_layers=2, seq_len=1000)
    lengths = wl.sequence_lengths(cfg)
    mask = np.zeros(cfg.num_q_heads, bool)
    mask[[0, 5, 9, 13, 17, 21, 25, 29]] = True
    layers = [{"srh_mask": mask, "budgets": np.array([200])},
              {"srh_mask": mask, "budgets": np.array([2000])}]
    total, score = bench.algorithmic_bytes(cfg, layers, lengths)
    k_bytes = 1000 * 8 * 128 * 2
    q_bytes = 8 * 32 * 128 * 2
    assert score == 2 * (k_bytes + q_bytes)
    assert total == score + 4 * (200 + 1000) * 8 * 128 * 2
