"""Pins of the self-likelihood reward (Section 5.3): s(Y) = ln p(Y | X) / len(Y) under the generator."""
import math

import numpy as np
import pytest

import sr_inputs as si
from oracle.logprob import token_logprob
from oracle.sr import DONE, best_of_n, run_workload
from oracle.transformer import Transformer


def test_uniform_logits_give_minus_log_v():
    for V in (2, 7, 512, 32000):
        l = np.full(V, 3.25, np.float32)
        for tok in (0, V // 2, V - 1):
            assert token_logprob(l, tok) == pytest.approx(-math.log(V), abs=1e-13)


def test_probabilities_from_the_plain_softmax():
    """Against the textbook softmax exp(l_v) / sum_u exp(l_u) (no shift), normalisation and shift invariance."""
    rng = np.random.default_rng(3)
    for V in (5, 64, 1000):
        l = (rng.standard_normal(V) * 2).astype(np.float32)
        e = np.exp(l.astype(np.float64))
        p = e / e.sum()
        lp = np.array([token_logprob(l, v) for v in range(V)])
        np.testing.assert_allclose(lp, np.log(p), rtol=0, atol=1e-12)
        assert np.exp(lp).sum() == pytest.approx(1.0, abs=1e-12)
        lp2 = np.array([token_logprob(l.astype(np.float64) + 40.0, v) for v in range(V)])
        np.testing.assert_allclose(lp2, lp, rtol=0, atol=1e-11)
    # NaN logits carry no probability (the sampler's rule)
    l = np.array([0.0, np.nan, 0.0], np.float32)
    assert token_logprob(l, 0) == pytest.approx(-math.log(2), abs=1e-14)
    assert token_logprob(l, 1) == float("-inf")


@pytest.fixture(scope="module")
def tiny():
    w = si.WORKLOADS["tiny"]
    gw, rw = si.random_weights(w.gen, 0, 0), si.random_weights(w.rm, 0, 1)
    gen, rm = Transformer(w.gen, gw), Transformer(w.rm, rw)
    prompt = w.prompt(0)
    bon = best_of_n(gen, rm, prompt, w.N, w.max_new, w.temperature, w.eos_bias, w.eos_id, 0, reward="logprob")
    return w, gw, rw, gen, rm, prompt, bon


def test_final_rewards_match_a_full_recompute(tiny):
    """The per-step accumulation equals ln p(Y | X) / len(Y) recomputed from one forward over prompt ++ Y:
    the token at response index t is scored by the logits of position P + t - 1."""
    w, gw, rw, gen, rm, prompt, bon = tiny
    P = len(prompt)
    for i, y in enumerate(bon[3][:4]):
        ids = np.array([list(prompt) + list(y)])
        logits = gen.logits(gen.forward(ids))[0]
        want = np.mean([token_logprob(logits[P + t - 1], y[t]) for t in range(len(y))])
        assert bon[4][i] == pytest.approx(want, rel=1e-5, abs=1e-6)


def test_alpha_zero_is_best_of_n_with_logprob_reward(tiny):
    w, gw, rw, gen, rm, prompt, bon = tiny
    res = run_workload(w, gw, rw, prompt, seed=0, alpha=0.0, reward="logprob")
    assert res.best_id == bon[0] and res.tokens == bon[1] and res.score == bon[2]
    assert res.rm_tokens == 0


def test_sr_with_logprob_reward_is_bounded_by_best_of_n(tiny):
    """Keyed noise: SR candidates follow their BoN trajectories, completed ones carry the BoN reward, so
    s(Y_SR) <= s(Y_BoN), with equality iff the BoN winner survived; rejections cut the lowest means."""
    w, gw, rw, gen, rm, prompt, bon = tiny
    for alpha in (0.25, 0.5, 0.9):
        res = run_workload(w, gw, rw, prompt, seed=0, alpha=alpha, reward="logprob")
        for i in range(w.N):
            assert res.all_tokens[i] == bon[3][i][:len(res.all_tokens[i])]
            if res.status[i] == DONE:
                assert res.final_reward[i] == bon[4][i]
        assert res.score <= bon[2]
        assert (res.score == bon[2]) == (res.status[bon[0]] == DONE)
        rd = res.rounds[0]
        assert np.all(rd.rewards[rd.accepted] >= rd.r_cut) and np.all(rd.rewards[~rd.accepted] < rd.r_cut)
