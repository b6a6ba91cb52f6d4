"""Pins of the oracle's Algorithm 1 against Best-of-N and brute force."""
import itertools

import numpy as np
import pytest

import sr_inputs as si
from oracle.sampler import perturbed_logits
from oracle.select import float_keys
from oracle.sr import DONE, REJECTED, SpeculativeRejection, best_of_n, run_workload, score_sequences
from oracle.transformer import Transformer


def _models(w: si.Workload, seed=0):
    gw = si.random_weights(w.gen, seed, 0)
    rw = si.random_weights(w.rm, seed, 1)
    return gw, rw, Transformer(w.gen, gw), Transformer(w.rm, rw)


@pytest.fixture(scope="module")
def tiny():
    w = si.WORKLOADS["tiny"]
    gw, rw, gen, rm = _models(w)
    prompt = w.prompt(0)
    bon = best_of_n(gen, rm, prompt, w.N, w.max_new, w.temperature, w.eos_bias, w.eos_id, 0)
    return w, gw, rw, gen, rm, prompt, bon


def test_alpha_zero_is_best_of_n(tiny):
    """Section 5.1: alpha = 0 with initial batch N is Best-of-N."""
    w, gw, rw, gen, rm, prompt, bon = tiny
    res = run_workload(w, gw, rw, prompt, seed=0, alpha=0.0)
    assert res.best_id == bon[0] and res.tokens == bon[1] and res.score == bon[2]
    # also in pool-sized waves under a memory trigger
    wp = w.replace(sched_kind=si.SCHED_POOL_FULL, pool_bytes=(1 + 3 * 5) * 16 * si.kv_bytes_per_token(w.gen))
    res = run_workload(wp, gw, rw, prompt, seed=0, alpha=0.0)
    assert res.best_id == bon[0] and res.tokens == bon[1] and res.score == bon[2]


def test_sr_trajectories_are_bon_trajectories(tiny):
    """Noise is keyed on (candidate, step): every SR candidate's tokens are a prefix of its BoN response,
    and completed candidates carry the same final reward, so s(Y_SR) <= s(Y_BoN)."""
    w, gw, rw, gen, rm, prompt, bon = tiny
    for alpha in (0.25, 0.5, 0.9):
        res = run_workload(w, gw, rw, prompt, seed=0, alpha=alpha)
        for i in range(w.N):
            assert res.all_tokens[i] == bon[3][i][:len(res.all_tokens[i])]
            if res.status[i] == DONE:
                assert res.all_tokens[i] == bon[3][i]
                assert res.final_reward[i] == bon[4][i]
        assert res.score <= bon[2]
        assert (res.score == bon[2]) == (res.status[bon[0]] == DONE)


def test_round_bookkeeping(tiny):
    w, gw, rw, gen, rm, prompt, bon = tiny
    res = run_workload(w, gw, rw, prompt, seed=0)
    assert len(res.rounds) == 1
    rd = res.rounds[0]
    assert rd.step == w.taus[0] and rd.batch == list(range(w.N))
    # partial rewards are the reward model on prompt ++ first tau_k tokens, tau_k = min(tau, l_k)
    trunc = [bon[3][i][:min(w.taus[0], len(bon[3][i]))] for i in range(w.N)]
    np.testing.assert_array_equal(rd.rewards, score_sequences(rm, prompt, trunc))
    assert rd.accepted.sum() == w.N - int(np.floor(np.float32(w.alpha) * w.N))
    for i, a in zip(rd.batch, rd.accepted):
        finished_early = len(bon[3][i]) <= w.taus[0]
        if finished_early:
            assert res.status[i] == DONE           # completed joins I whatever the cut says
        elif not a:
            assert res.status[i] == REJECTED and res.lengths[i] == w.taus[0]
        else:
            assert res.status[i] == DONE and res.lengths[i] == len(bon[3][i])
    done = [i for i in range(w.N) if res.status[i] == DONE]
    assert res.best_id == done[int(np.argmax(float_keys(res.final_reward[done])))]


def test_tiny_vocabulary_brute_force():
    """V = 4, max_new = 3: walk the whole 4^3 continuation tree with fixed noise, recomputing every
    node's logits from scratch; the sampled path must be the argmax path and the returned response the
    argmax of recomputed final rewards among completed candidates."""
    m = si.ModelDesc(n_layers=2, d_model=16, n_heads=2, n_kv_heads=1, head_dim=8, ffn_dim=24, vocab=4,
                     max_pos=16, dtype=si.DT_F32)
    rmd = m.replace(has_lm_head=0, has_scalar_head=1)
    gen = Transformer(m, si.random_weights(m, 21, 0, std=0.5))
    rm = Transformer(rmd, si.random_weights(rmd, 21, 1, std=0.5))
    prompt = [1, 3, 2]
    N, max_new, seed = 6, 3, 99
    z = {}
    for L in range(max_new):
        for prefix in itertools.product(range(4), repeat=L):
            logits = gen.logits(gen.forward([prompt + list(prefix)])[0, -1])
            for i in range(N):
                z[(i,) + prefix] = perturbed_logits(logits, seed, i, L, 1.0, 0.3, 0)
    paths = []
    for i in range(N):
        y = []
        while len(y) < max_new and (not y or y[-1] != 0):
            y.append(int(np.argmax(z[(i,) + tuple(y)])))
        paths.append(y)
    final = score_sequences(rm, prompt, paths)
    for alpha, taus in ((0.0, ()), (0.5, (1,)), (0.5, (2,))):
        sr = SpeculativeRejection(gen, rm, prompt, N, alpha, si.SCHED_FIXED, taus, max_new, 1.0, 0.3, 0, seed)
        res = sr.run()
        done = [i for i in range(N) if res.status[i] == DONE]
        for i in range(N):
            assert res.all_tokens[i] == paths[i][:len(res.all_tokens[i])]
        best = done[int(np.argmax(float_keys(final[done])))]
        assert res.best_id == best and res.tokens == paths[best]
        np.testing.assert_allclose(res.score, final[best], rtol=1e-5, atol=1e-6)
