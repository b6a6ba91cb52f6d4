"""Pins of the oracle's cut-off threshold and accepted set (Section 4.2)."""
import json
import os

import numpy as np
import pytest

from oracle.select import accepted_mask, cut_index, float_keys, key_to_float, r_cut, select_round

HERE = os.path.dirname(__file__)


def test_paper_two_response_example():
    """Section 4.1: partial rewards 2.92 (Y1) and -1.88 (Y2); the cut keeps Y1 and stops Y2."""
    ex = json.load(open(os.path.join(HERE, "golden", "paper_example.json")))
    r = np.array(ex["partial_rewards"], np.float32)
    rc = r_cut(r, ex["alpha"])
    assert rc == np.float32(ex["expected_r_cut"])
    assert accepted_mask(r, rc).tolist() == ex["expected_accepted"]
    # Y1's final reward is also the larger one, so the returned response is Y1
    assert int(np.argmax(ex["final_rewards"])) == ex["expected_best"]


def test_brute_force_order_statistic():
    rng = np.random.default_rng(3)
    for trial in range(300):
        b = int(rng.integers(1, 70))
        alpha = float(rng.uniform(0, 1))
        if trial % 3 == 0:
            r = rng.integers(-3, 4, b).astype(np.float32)       # many ties
        else:
            r = rng.standard_normal(b).astype(np.float32)
        k = min(int(np.floor(float(np.float32(alpha)) * b)), b - 1)
        want = sorted(r.tolist())[k]
        rc, mask, kk = select_round(r, alpha)
        assert kk == k and rc == want
        assert mask.tolist() == [x >= want for x in r.tolist()]


def test_size_rule_without_ties():
    """Distinct rewards: exactly b - floor(alpha b) survive (the top 1 - alpha proportion)."""
    rng = np.random.default_rng(4)
    for b in (1, 2, 3, 7, 64, 100, 1024):
        r = rng.permutation(b).astype(np.float32) - 17.5
        for alpha in (0.0, 0.1, 0.3, 0.5, 0.7, 0.9, 0.999):
            _, mask, k = select_round(r, alpha)
            assert mask.sum() == b - k
            assert k == min(int(np.floor(float(np.float32(alpha)) * b)), b - 1)


def test_alpha_ends_and_ties():
    r = np.array([0.5, -2.0, 3.0, 3.0, 1.0], np.float32)
    assert select_round(r, 0.0)[1].all()                           # alpha = 0: Best-of-N keeps all
    assert select_round(r, 1.0)[1].tolist() == [False, False, True, True, False]   # only the maximum (tied)
    assert select_round(np.full(9, 1.25, np.float32), 0.7)[1].all()  # all tied: all accepted


def test_float_key_order():
    rng = np.random.default_rng(5)
    x = np.concatenate([rng.standard_normal(5000) * 10 ** rng.uniform(-30, 30, 5000),
                        [0.0, -0.0, np.inf, -np.inf, 1e-45, -1e-45]]).astype(np.float32)
    k = float_keys(x)
    order_k = np.argsort(k, kind="stable")
    assert np.all(np.diff(x[order_k].astype(np.float64)) >= 0)
    assert float_keys([-0.0])[0] == float_keys([0.0])[0]
    assert float_keys([np.nan])[0] == float_keys([-np.inf])[0]
    for v in (0.0, 1.5, -2.25, 3.4e38, -1e-40):
        assert key_to_float(int(float_keys([v])[0])) == np.float32(v)


def test_cut_index_exact_product():
    # 0.7f * 1024 = 716.79998 -> 716 ; 0.5f * 7 = 3.5 -> 3 ; clamp at b - 1
    assert cut_index(0.7, 1024) == 716
    assert cut_index(0.5, 7) == 3
    assert cut_index(1.0, 5) == 4
    assert cut_index(0.0, 5) == 0
