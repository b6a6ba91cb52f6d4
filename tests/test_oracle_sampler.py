"""Pins of the oracle's sampler: Philox known answers, the series logarithm, Gumbel-max."""
import math

import numpy as np
import pytest

from oracle.flog import flog
from oracle.philox import philox4x32_10
from oracle.sampler import gumbel_noise, perturbed_logits, sample_token

# Known-answer vectors published with Random123 (Salmon et al., SC'11) for philox4x32_10.
KAT = [
    ((0, 0, 0, 0), (0, 0), (0x6627E8D5, 0xE169C58D, 0xBC57AC4C, 0x9B00DBD8)),
    ((0xFFFFFFFF,) * 4, (0xFFFFFFFF,) * 2, (0x408F276D, 0x41C83B0E, 0xA20BC7C6, 0x6D5451FD)),
    ((0x243F6A88, 0x85A308D3, 0x13198A2E, 0x03707344), (0xA4093822, 0x299F31D0),
     (0xD16CFE09, 0x94FDCCEB, 0x5001E420, 0x24126EA1)),
]


@pytest.mark.parametrize("ctr,key,want", KAT)
def test_philox_known_answers(ctr, key, want):
    got = philox4x32_10(*ctr, *key)
    assert tuple(int(x) for x in got) == want


def test_flog_error_bound():
    rng = np.random.default_rng(1)
    # the sampler's two ranges: u in [2^-24, 1) and -ln u in (0, 17)
    x = np.concatenate([rng.uniform(2.0 ** -24, 1.0, 200000), rng.uniform(1e-7, 17.0, 200000),
                        np.float32(2.0) ** -np.arange(1, 25, dtype=np.float32)]).astype(np.float32)
    ref = np.log(x.astype(np.float64))
    got = flog(x).astype(np.float64)
    ulp = np.spacing(np.abs(ref).astype(np.float32)).astype(np.float64)
    assert np.max(np.abs(got - ref) / ulp) <= 4.0
    assert flog(np.float32([1.0]))[0] == 0.0
    assert abs(float(flog(np.float32([math.e]))[0]) - 1.0) < 2e-7


def test_uniform_in_open_interval_and_keyed():
    g1 = gumbel_noise(123, 5, 7, 4096)
    g2 = gumbel_noise(123, 5, 7, 4096)
    g3 = gumbel_noise(123, 6, 7, 4096)
    assert np.array_equal(g1, g2)
    assert not np.array_equal(g1, g3)
    assert np.all(np.isfinite(g1))
    # a standard Gumbel has mean Euler-Mascheroni and variance pi^2/6
    g = np.concatenate([gumbel_noise(9, i, 0, 4096) for i in range(16)]).astype(np.float64)
    assert abs(g.mean() - 0.5772156649) < 0.02
    assert abs(g.var() - math.pi ** 2 / 6) < 0.05


def _chi2_ok(counts, probs, n):
    exp = probs * n
    stat = float(np.sum((counts - exp) ** 2 / exp))
    df = len(probs) - 1
    # Wilson-Hilferty upper 1e-4 quantile of chi-square(df)
    z = 3.719
    crit = df * (1 - 2 / (9 * df) + z * math.sqrt(2 / (9 * df))) ** 3
    return stat, crit


@pytest.mark.parametrize("T,bias", [(1.0, 0.0), (0.5, 1.0), (2.0, -1.5)])
def test_gumbel_max_matches_softmax(T, bias):
    """Gumbel-max theorem: argmax(z/T + g) is distributed as softmax((logit + bias e_eos) / T)."""
    logits = np.array([0.3, -1.2, 0.9, 0.0, 1.4, -0.4], np.float32)
    eos = 2
    n = 30000
    counts = np.zeros(len(logits))
    for i in range(n):
        counts[sample_token(logits, 77, i % 1000, i // 1000, T, bias, eos)] += 1
    adj = logits.astype(np.float64).copy()
    adj[eos] += bias
    p = np.exp(adj / T)
    p /= p.sum()
    stat, crit = _chi2_ok(counts, p, n)
    assert stat < crit, (stat, crit, counts / n, p)
    # the mistaken order "scale, then bias" must be rejected by the same test
    wrong = logits.astype(np.float64) / T
    wrong[eos] += bias
    q = np.exp(wrong)
    q /= q.sum()
    if bias != 0.0 and T != 1.0:
        stat_w, _ = _chi2_ok(counts, q, n)
        assert stat_w > crit


def test_ties_and_nan():
    inf = np.float32(np.inf)
    # equal +inf perturbed logits: the lowest id wins
    assert sample_token(np.array([0.0, inf, inf], np.float32), 1, 0, 0, 1.0, 0.0, 0) == 1
    # NaN counts as -inf and is never drawn
    for i in range(50):
        assert sample_token(np.array([np.nan, 0.0], np.float32), 3, i, 0, 1.0, 0.0, 5) == 1
    # temperature scales before the noise is added
    z = perturbed_logits(np.array([2.0, 4.0], np.float32), 3, 0, 0, 2.0, 0.0, 0)
    g = gumbel_noise(3, 0, 0, 2)
    assert np.array_equal(z, (np.array([1.0, 2.0], np.float32) + g).astype(np.float32))


def test_gumbel_noise_bound_for_skip_test():
    """The sampler kernel skips an id whose uniform satisfies 1 - u > exp(ap - best + margin), margin >= 1e-4: valid
    because the Gumbel noise as computed (two series logarithms) never exceeds -ln(1 - u) by 1e-5.  Checked over
    every one of the 2^23 uniforms the generator can produce."""
    w = np.arange(1 << 23, dtype=np.uint32)
    u = (w.astype(np.float32) + np.float32(0.5)) * np.float32(2.0 ** -23)
    g = -flog(-flog(u)).astype(np.float64)                      # the sampler's noise, as the kernel computes it
    one_minus_u = ((np.uint32(0x7FFFFF) - w).astype(np.float32) + np.float32(0.5)) * np.float32(2.0 ** -23)
    assert np.array_equal(one_minus_u.astype(np.float64), 1.0 - u.astype(np.float64))   # exact in float32
    bound = -np.log(one_minus_u.astype(np.float64))             # g(u) <= -ln(1 - u) since -ln u >= 1 - u
    assert np.max(g - bound) < 1e-5
    exact = -np.log(-np.log(u.astype(np.float64)))
    assert np.max(np.abs(g - exact)) < 1e-5 and np.max(np.abs(g)) < 17.0
