"""Head-level budgets in the oracle (Sec. 4.6: the token selection under a
budget per head group): uniform budgets reproduce the per-layer-budget
selection, and each unit's selection is its own top-k."""
import numpy as np
import pytest

import oracle
from oracle import brute


def _case(seed, lens=(41, 30, 3)):
    rng = np.random.default_rng(seed)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    q = rng.normal(size=(len(lens), 8, 4, 16)) / 3
    k = rng.normal(size=(int(cu[-1]), 2, 16)) / 3
    v = rng.normal(size=(int(cu[-1]), 2, 16))
    mask = np.zeros(8, bool)
    mask[[0, 2, 5]] = True
    return q, k, v, cu, mask


def test_uniform_budgets_equal_the_per_sequence_layout():
    q, k, v, cu, mask = _case(1)
    bud = [14, 9, 6]
    a = oracle.compress_layer(q, k, v, cu, mask, bud, 4, 3)
    b = oracle.compress_layer_head_budgets(q, k, v, cu, mask, np.repeat([bud], 2, 0).T, 4, 3)
    for g in range(2):
        for s in range(3):
            o0, o1 = int(a.cu_out[s]), int(a.cu_out[s + 1])
            p0, p1 = int(b.cu_out[g, s]), int(b.cu_out[g, s + 1])
            assert a.indices[g, o0:o1].tolist() == b.indices[p0:p1].tolist()
            np.testing.assert_array_equal(a.k_out[o0:o1, g], b.k_out[p0:p1])


@pytest.mark.parametrize("seed", range(4))
def test_each_unit_matches_brute_force_with_its_own_budget(seed):
    q, k, v, cu, mask = _case(10 + seed)
    rng = np.random.default_rng(seed)
    gb = rng.integers(4, 40, size=(3, 2))
    res = oracle.compress_layer_head_budgets(q, k, v, cu, mask, gb, 4, 3)
    assert res.cu_out[-1, -1] == len(res.indices)
    for (s, g), unit in res.units.items():
        heads = [h for h in range(4 * g, 4 * g + 4) if mask[h]]
        rows = slice(int(cu[s]), int(cu[s + 1]))
        _, _, idx = brute.brute_unit([q[s, h].tolist() for h in heads], k[rows, g].tolist(), 4, 3,
                                     int(gb[s, g]), oracle.default_scale(16))
        p0, p1 = int(res.cu_out[g, s]), int(res.cu_out[g, s + 1])
        assert res.indices[p0:p1].tolist() == idx
