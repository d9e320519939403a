"""The seeded generator: determinism and the recipe's stated properties."""
import numpy as np
import torch

import workloads as wl


def test_layer_is_deterministic():
    cfg = wl.get("c1").scaled(seq_len=512, n_layers=2)
    a = wl.make_layer(cfg, 0)
    b = wl.make_layer(cfg, 0)
    for key in ("q_win", "k", "v"):
        assert torch.equal(a[key].view(torch.int16), b[key].view(torch.int16))
    assert a["needles"] == b["needles"]
    c = wl.make_layer(cfg, 1)
    assert not torch.equal(a["k"], c["k"])


def test_shapes_and_dtypes():
    cfg = wl.get("c4").scaled(length_range=(300, 900), n_layers=3)
    lens = wl.sequence_lengths(cfg)
    d = wl.make_layer(cfg, 2)
    assert d["q_win"].shape == (8, 28, 32, 128)
    assert d["k"].shape == (sum(lens), 4, 128) and d["k"].dtype == torch.bfloat16
    assert d["cu_seqlens"].tolist() == [0] + np.cumsum(lens).tolist()
    assert d["srh_mask"].reshape(4, 7).sum(1).tolist() == [2, 2, 2, 2]


def test_budgets_follow_the_recipe():
    c2 = wl.get("c2")
    b = wl.layer_budgets(c2, wl.sequence_lengths(c2))
    assert b.shape == (32, 1) and b.sum() == 32 * 256 and b.min() >= 48
    c5 = wl.get("c5")
    b5 = wl.layer_budgets(c5, wl.sequence_lengths(c5))
    assert b5.min() >= 80 and b5.max() <= 3 * 328 and abs(b5.mean() - 328) < 1
    c4 = wl.get("c4")
    lens = wl.sequence_lengths(c4)
    b4 = wl.layer_budgets(c4, lens)
    for s, L in enumerate(lens):
        assert abs(b4[:, s].mean() - round(0.03 * L)) < 1


def test_srh_counts():
    for name, (lo, hi) in (("c2", (1, 2)), ("c5", (1, 3))):
        cfg = wl.get(name)
        m = wl.srh_masks(cfg).reshape(cfg.n_layers, cfg.num_kv_heads, cfg.group_size).sum(-1)
        assert m.min() >= lo and m.max() <= hi


def test_needles_spaced_and_in_range():
    cfg = wl.get("c3").scaled(seq_len=20000)
    pos = wl.needle_positions(cfg, 0, 0, 3, 20000 - 32)
    assert len(pos) == 64
    assert min(pos) >= 4 and max(pos) < 20000 - 32 - 7
    assert min(np.diff(pos)) >= 7
