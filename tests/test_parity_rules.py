"""The parity bars of tests/parity.py, on the CPU: each accepts what the
arithmetic allows and rejects a plain mistake."""

import numpy as np
import pytest

from oracle import conduit_oracle as O
from tests import parity as PT


def test_quota_band_accepts_quotas_of_perturbed_coefficients():
    """Coefficients within rtol of the fp64 ones (as binary32 ones are) give
    quotas inside the band: differences only next to a near-tie."""
    rng = np.random.default_rng(31)
    for trial in range(400):
        K = int(rng.integers(1, 9))
        n = rng.integers(1, 60, size=K)
        k = int(rng.integers(0, n.sum() + 1))
        c = rng.uniform(0.0, 2.0, size=K)
        if trial % 5 == 0:
            c[:] = 1.0 + (trial % 3) * 0.25           # equal weights: remainder ties
        pert = c * (1.0 + rng.uniform(-1e-6, 1e-6, size=K))
        PT.assert_quotas_in_band(O.image_quotas(pert, n, k), c, n, k, 1e-6)


def test_quota_band_rejects_a_unit_moved_away_from_a_tie():
    c, n, k = np.array([1.0, 2.0, 3.0]), [100, 100, 100], 61   # ideals 10.17, 20.33, 30.5
    assert O.image_quotas(c, n, k).tolist() == [10, 20, 31]
    PT.assert_quotas_in_band([10, 20, 31], c, n, k, 1e-5)
    with pytest.raises(AssertionError):
        PT.assert_quotas_in_band([11, 20, 30], c, n, k, 1e-5)   # the leftover unit went elsewhere
    with pytest.raises(AssertionError):
        PT.assert_quotas_in_band([10, 20, 30], c, n, k, 1e-5)   # a unit lost


def test_quota_band_allows_either_side_of_an_exact_tie():
    c, n, k = np.array([1.0, 1.0]), [10, 10], 5                 # ideals 2.5 and 2.5
    assert O.image_quotas(c, n, k).tolist() == [3, 2]           # ties to the lower image
    PT.assert_quotas_in_band([2, 3], c, n, k, 1e-6)


def test_selection_band_rejects_a_swap_outside_the_band():
    s = np.array([5.0, 4.0, 3.0, 2.0, 1.0])
    PT.assert_selection_ok([0, 1], None, s, [0, 1], 2, 1e-3)
    with pytest.raises(AssertionError):
        PT.assert_selection_ok([0, 2], None, s, [0, 1], 2, 1e-3)
    tie = np.array([5.0, 4.0, 4.0 * (1 + 1e-4), 1.0])
    PT.assert_selection_ok([0, 1], None, tie, [0, 2], 2, 1e-3)  # inside the band at the k-th value
