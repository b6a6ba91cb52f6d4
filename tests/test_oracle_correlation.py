"""Pins of the Appendix B correlation statistics (oracle side)."""
import itertools

import numpy as np
import pytest

import sr_inputs as si
from oracle.correlation import kendall_tau_b, partial_final, pearson
from oracle.transformer import Transformer

scipy_stats = pytest.importorskip("scipy.stats")


def test_pearson_and_kendall_against_scipy():
    rng = np.random.default_rng(5)
    for n in (3, 10, 57):
        x = rng.standard_normal(n)
        y = 0.6 * x + rng.standard_normal(n)
        assert pearson(x, y) == pytest.approx(scipy_stats.pearsonr(x, y)[0], abs=1e-12)
        assert kendall_tau_b(x, y) == pytest.approx(scipy_stats.kendalltau(x, y)[0], abs=1e-12)
        if n >= 10:
            xi, yi = np.round(x), np.round(y)       # heavy ties: the tau-b correction matters
            assert kendall_tau_b(xi, yi) == pytest.approx(scipy_stats.kendalltau(xi, yi)[0], abs=1e-12)


def test_closed_forms():
    x = np.arange(8.0)
    assert pearson(x, 3 * x + 1) == pytest.approx(1.0) and pearson(x, -x) == pytest.approx(-1.0)
    assert kendall_tau_b(x, x ** 3) == 1.0 and kendall_tau_b(x, -x) == -1.0
    # one swapped neighbour pair among n: (C - D) / (n(n-1)/2) with D = 1
    y = x.copy()
    y[[3, 4]] = y[[4, 3]]
    assert kendall_tau_b(x, y) == pytest.approx((28 - 1 - 1) / 28)
    # brute force over all permutations of 5: the mean of tau over permutations is 0
    taus = [kendall_tau_b(np.arange(5), np.array(p)) for p in itertools.permutations(range(5))]
    assert np.mean(taus) == pytest.approx(0.0, abs=1e-12)


def test_partial_at_full_length_is_the_final_reward():
    w = si.WORKLOADS["tiny"]
    gen = Transformer(w.gen, si.random_weights(w.gen, 0, 0))
    rm = Transformer(w.rm, si.random_weights(w.rm, 0, 1))
    partial, final, stats = partial_final(gen, rm, w.prompt(0), w.N, (4, w.max_new), w.max_new, w.temperature,
                                          w.eos_bias, w.eos_id, 0)
    np.testing.assert_array_equal(partial[w.max_new], final)
    assert stats[w.max_new][0] == pytest.approx(1.0) and stats[w.max_new][1] == pytest.approx(1.0)
    assert -1.0 <= stats[4][1] <= 1.0
