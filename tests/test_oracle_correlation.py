"""Pins of the Appendix B correlation statistics (oracle side).

Appendix B defines R_Kendall = 2 / (N (N - 1)) sum_{i<j} sgn(x_i - x_j) sgn(y_i - y_j) (tau-a); the
tie-corrected tau-b is an extra figure.  The two agree without ties and differ with them.
"""
import itertools

import numpy as np
import pytest

import sr_inputs as si
from oracle.correlation import kendall_tau_a, kendall_tau_b, partial_final, pearson
from oracle.transformer import Transformer

scipy_stats = pytest.importorskip("scipy.stats")


def test_pearson_and_kendall_against_scipy():
    rng = np.random.default_rng(5)
    for n in (3, 10, 57):
        x = rng.standard_normal(n)
        y = 0.6 * x + rng.standard_normal(n)
        assert pearson(x, y) == pytest.approx(scipy_stats.pearsonr(x, y)[0], abs=1e-12)
        # no ties: tau-a and tau-b coincide, and scipy's (tau-b) gives both
        assert kendall_tau_a(x, y) == pytest.approx(scipy_stats.kendalltau(x, y)[0], abs=1e-12)
        assert kendall_tau_b(x, y) == pytest.approx(scipy_stats.kendalltau(x, y)[0], abs=1e-12)
        if n >= 10:
            xi, yi = np.round(x), np.round(y)       # heavy ties: the tau-b correction matters
            assert kendall_tau_b(xi, yi) == pytest.approx(scipy_stats.kendalltau(xi, yi)[0], abs=1e-12)
            assert abs(kendall_tau_a(xi, yi)) < abs(kendall_tau_b(xi, yi))


def test_kendall_tau_a_with_ties_by_hand():
    """x = (1, 1, 2, 3), y = (1, 2, 2, 3): of the 6 pairs, (0,1) ties in x and (1,2) ties in y, the other 4 are
    concordant.  Appendix B's statistic: 2 / (4 * 3) * 4 = 2/3; tau-b: 4 / sqrt(5 * 5) = 4/5."""
    x, y = [1, 1, 2, 3], [1, 2, 2, 3]
    assert kendall_tau_a(x, y) == pytest.approx(2.0 / 3.0, abs=1e-15)
    assert kendall_tau_b(x, y) == pytest.approx(0.8, abs=1e-15)
    # all of x tied: every pair contributes 0
    assert kendall_tau_a([5, 5, 5], [1, 2, 3]) == 0.0
    # two discordant pairs and one pair tied in y: 2 / (3 * 2) * (-1 - 1 + 0)
    assert kendall_tau_a([1, 2, 3], [2, 1, 1]) == pytest.approx(-2.0 / 3.0)


def test_closed_forms():
    x = np.arange(8.0)
    assert pearson(x, 3 * x + 1) == pytest.approx(1.0) and pearson(x, -x) == pytest.approx(-1.0)
    for tau in (kendall_tau_a, kendall_tau_b):
        assert tau(x, x ** 3) == 1.0 and tau(x, -x) == -1.0
        # one swapped neighbour pair among n: (C - D) / (n(n-1)/2) with D = 1
        y = x.copy()
        y[[3, 4]] = y[[4, 3]]
        assert tau(x, y) == pytest.approx((28 - 1 - 1) / 28)
        # brute force over all permutations of 5: the mean of tau over permutations is 0
        taus = [tau(np.arange(5), np.array(p)) for p in itertools.permutations(range(5))]
        assert np.mean(taus) == pytest.approx(0.0, abs=1e-12)


def test_library_statistics_match_the_oracle():
    """The tool's vectorised statistics (paper_2410_20290_gb300.correlation) equal the oracle's loops."""
    from paper_2410_20290_gb300 import correlation as tool
    rng = np.random.default_rng(9)
    for n in (2, 7, 40):
        x, y = np.round(rng.standard_normal(n), 1), np.round(rng.standard_normal(n), 1)
        ka, kb = tool.kendall(x, y)
        assert ka == pytest.approx(kendall_tau_a(x, y), abs=1e-12)
        assert kb == pytest.approx(kendall_tau_b(x, y), abs=1e-12)
        assert tool.pearson(x, y) == pytest.approx(pearson(x, y), abs=1e-12)


def test_partial_at_full_length_is_the_final_reward():
    w = si.WORKLOADS["tiny"]
    gen = Transformer(w.gen, si.random_weights(w.gen, 0, 0))
    rm = Transformer(w.rm, si.random_weights(w.rm, 0, 1))
    partial, final, stats = partial_final(gen, rm, w.prompt(0), w.N, (4, w.max_new), w.max_new, w.temperature,
                                          w.eos_bias, w.eos_id, 0)
    np.testing.assert_array_equal(partial[w.max_new], final)
    assert stats[w.max_new][0] == pytest.approx(1.0) and stats[w.max_new][1] == pytest.approx(1.0)
    assert -1.0 <= stats[4][1] <= 1.0 and -1.0 <= stats[4][2] <= 1.0
