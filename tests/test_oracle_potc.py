"""Pins of the oracle's power-of-d-choices sweep (App. A.8, "Optimal
Candidate Set Size"): m balls into n bins, each ball to the least loaded of
d random bins.  The random bins come from SplitMix64's published output
sequence; placement is checked by hand, d = 1 against a brute-force count,
and the sweep against the shape App. A.8 reports (a sharp drop in maximum
load deviation from d = 1 to d = 2, little after)."""

import numpy as np
import pytest

from oracle import oracle as O


def test_choices_are_splitmix64_outputs_scaled():
    """Choice c is floor(x * n / 2^64) for x the (c+1)-th output of
    SplitMix64(seed) (the sequence itself is pinned to its published
    vector elsewhere)."""
    for seed in (0, 1234567, 2**63 + 5):
        xs = O.splitmix64_stream(seed, 200)
        for n in (1, 3, 8, 17, 32, 1000):
            assert [O.potc_choice(seed, c, n) for c in range(200)] == [(x * n) >> 64 for x in xs]


def test_placement_by_hand():
    """n = 3, d = 2: (0,1) -> 0 (tie: first); (0,1) -> 1; (1,0) -> 1 (tie:
    first); (2,2) -> 2; (0,2) -> 0 (tie: first)."""
    load = O.potc_place_all([[0, 1], [0, 1], [1, 0], [2, 2], [0, 2]], 3)
    assert load.tolist() == [2, 2, 1]
    # d = 3: (0,1,2) -> 0; (0,1,2) -> 1 (the first empty); (0,1,2) -> 2;
    # (2,1,0) with all loads 1 -> 2 (tie: first choice)
    load = O.potc_place_all([[0, 1, 2], [0, 1, 2], [0, 1, 2], [2, 1, 0]], 3)
    assert load.tolist() == [1, 1, 2]


def test_one_choice_is_a_plain_count_and_loads_sum_to_m():
    n, m, seed = 16, 4000, 77
    got = O.potc_max_loads(n, m, 1, 3, seed)
    for s in range(3):
        bins = [O.potc_choice(seed, s * m + t, n) for t in range(m)]
        assert got[s] == np.bincount(bins, minlength=n).max()
    rng = np.random.default_rng(3)
    ch = rng.integers(0, 7, (500, 3))
    load = O.potc_place_all(ch, 7)
    assert load.sum() == 500 and load.max() - load.min() <= 2      # three choices keep it tight


def test_more_bins_than_balls_and_one_bin():
    assert O.potc_max_loads(1, 123, 2, 2, 5).tolist() == [123, 123]
    assert all(x >= 1 for x in O.potc_max_loads(64, 10, 2, 5, 5))


def test_sweep_shape_of_app_a8():
    """n = 8..32 with m/n = 1,000: the mean maximum-load deviation falls by
    more than 10x from d = 1 to d = 2, and by less than one ball from d = 2
    to d = 3 (the near-exponential two-choice gain and its quick
    tapering)."""
    for n in (8, 16, 24, 32):
        m = 1000 * n
        dev = {d: O.potc_max_loads(n, m, d, 40, 100 + n).mean() - m / n for d in (1, 2, 3)}
        assert dev[1] > 10 * dev[2]
        assert dev[2] - dev[3] < 1.0
        assert dev[2] <= 3.0


def test_bad_arguments():
    with pytest.raises(ValueError):
        O.potc_max_loads(0, 10, 2, 1, 1)
    with pytest.raises(ValueError):
        O.potc_max_loads(4, 10, 65, 1, 1)
