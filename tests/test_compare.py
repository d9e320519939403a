"""The acceptance helpers themselves: a score check must reject non-finite
device values (NaN compares false against any tolerance)."""
import numpy as np
import pytest

from oracle import compare


def test_scores_within_tolerance_pass():
    ref = np.array([1.0, 2e-3, 0.0])
    compare.check_scores("x", ref * (1 + 5e-4), ref)


@pytest.mark.parametrize("bad", [np.nan, np.inf, -np.inf])
def test_non_finite_scores_fail(bad):
    ref = np.array([1.0, 2e-3, 0.5])
    gpu = ref.copy()
    gpu[1] = bad
    with pytest.raises(AssertionError, match="outside tolerance"):
        compare.check_scores("x", gpu, ref)


def test_relative_error_above_tolerance_fails():
    ref = np.array([1.0, 0.25])
    with pytest.raises(AssertionError):
        compare.check_scores("x", ref * (1 + 2e-3), ref)
