"""Reward-model KV kept across rounds (sr_set_rm_cache) against the oracle, which rescores in full.

A partial reward s(X ++ Y^{<=tau}) (Eq. partial.reward.set) read with the cache runs only the positions added
since the candidate was last scored and attends to the cached ones; the oracle recomputes the whole sequence.
The two must agree within the reward tolerance, and Algorithm 1's decisions must come out the same.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import sr_inputs as si
from oracle.sr import SpeculativeRejection, score_sequences
from oracle.transformer import Transformer

pytestmark = pytest.mark.gpu
REWARD_REL = 1e-2


@pytest.fixture(scope="module")
def sr():
    from paper_2410_20290_gb300 import binding
    return binding


def reward_tol(r, R):
    R = np.asarray(R, np.float64)
    R = R[np.isfinite(R)]
    return REWARD_REL * max(abs(float(r)), float(np.sqrt(np.mean(R ** 2))) if R.size else 0.0)


def _ctx(sr, w, seed=0, cache_bytes=1 << 30, host=True):
    gw = si.random_weights(w.gen, seed, 0, perturb_norms=True)
    rw = si.random_weights(w.rm, seed, 1, perturb_norms=True)
    ctx = sr.sr_init(w.gen, si.pack_blob(w.gen, gw), w.rm, si.pack_blob(w.rm, rw), w.pool_bytes, 16, 0)
    sr.sr_set_rm_cache(ctx, cache_bytes)
    return ctx, gw, rw


@pytest.mark.parametrize("seed", [0, 1])
def test_tiny_several_rounds_with_cache_match_oracle(sr, seed):
    """Tiny fp32 workload with decision points at 8, 16, 32 and 48 tokens, free running: rounds, batch sizes,
    accepted counts, r_cut, the selected candidate, its tokens and score equal the oracle's (full rescoring);
    fewer reward-model positions are run than without the cache."""
    w = si.WORKLOADS["tiny"].replace(taus=(8, 16, 32, 48), alpha=0.3)
    ctx, gw, rw = _ctx(sr, w, seed)
    try:
        prompt = w.prompt(seed)
        toks, score, st = sr.sr_generate(ctx, prompt, w.N, w.alpha, w.sched_kind, w.taus, w.max_new,
                                          w.temperature, w.eos_bias, w.eos_id, seed)
        sr.sr_set_rm_cache(ctx, 0)
        toks0, score0, st0 = sr.sr_generate(ctx, prompt, w.N, w.alpha, w.sched_kind, w.taus, w.max_new,
                                            w.temperature, w.eos_bias, w.eos_id, seed)
    finally:
        sr.sr_destroy(ctx)
    ref = SpeculativeRejection(Transformer(w.gen, gw), Transformer(w.rm, rw), prompt, w.N, w.alpha,
                               w.sched_kind, w.taus, w.max_new, w.temperature, w.eos_bias, w.eos_id, seed).run()
    assert st["rounds"] == len(ref.rounds) >= 2
    for i, rd in enumerate(ref.rounds):
        assert st["b_per_round"][i] == len(rd.batch)
        assert st["accepted_per_round"][i] == int(rd.accepted.sum())
        assert abs(st["r_cut_per_round"][i] - rd.r_cut) <= reward_tol(rd.r_cut, rd.rewards)
    assert st["best_id"] == ref.best_id and list(toks) == ref.tokens
    assert abs(score - ref.score) <= reward_tol(ref.score, ref.final_reward)
    # the same run without the cache: same decisions, all positions run again
    assert st0["best_id"] == st["best_id"] and list(toks0) == list(toks)
    assert st["rm_tokens_cached"] > 0 and st0["rm_tokens_cached"] == 0
    assert st["rm_tokens"] + st["rm_tokens_cached"] == st0["rm_tokens"]


def _component_run(sr, w, ctx, gw, rw, prompt, seed, taus, alpha):
    """Rounds at `taus` through the component calls; every round's rewards (GPU, with the cache) against the
    oracle's full rescoring of the GPU's own sequences."""
    rm = Transformer(w.rm, rw)
    P, N = len(prompt), w.N
    max_pages = (P + w.max_new - 1) // 16 + 1
    n_pages = P // 16 + N * ((P + w.max_new - 2) // 16 + 1 - P // 16)
    b = sr.sr_batch_begin(ctx, prompt, N, w.max_new, w.temperature, w.eos_bias, w.eos_id, seed)
    try:
        g, worst = 1, 0.0
        for tau in list(taus) + [None]:
            while tau is None or g < tau:
                q = sr.sr_batch_query(ctx, b, N, w.max_new, max_pages, n_pages)
                if q["n_live"] == 0:
                    break
                sr.sr_decode_step(ctx, b, None)
                g += 1
            q = sr.sr_batch_query(ctx, b, N, w.max_new, max_pages, n_pages)
            batch = [i for i in range(N) if q["status"][i] in (0, 1)]
            if not batch:
                break
            rewards = sr.sr_score_partial(ctx, b, N)
            seqs = [q["tokens"][i][:q["lengths"][i]].tolist() for i in batch]
            want = score_sequences(rm, prompt, seqs)
            for a, r in zip(rewards, want):
                assert abs(a - r) <= reward_tol(r, want), (tau, a, r)
                worst = max(worst, abs(a - r) / max(reward_tol(r, want), 1e-30))
            if tau is None:
                break
            sr.sr_reject_compact(ctx, b, rewards, alpha)
    finally:
        sr.sr_batch_end(ctx, b)
    return worst


@pytest.mark.parametrize("cache_bytes", [1 << 30, None])
def test_tiny_component_rounds_with_cache(sr, cache_bytes):
    """Three rounds and a final scoring through the component calls.  cache_bytes None: a pool of 40 pages,
    too small to keep every candidate, so some candidates are stored and the rest rescored in full."""
    w = si.WORKLOADS["tiny"].replace(N=12)
    if cache_bytes is None:
        cache_bytes = 40 * 16 * si.kv_bytes_per_token(w.rm)
    ctx, gw, rw = _ctx(sr, w, 3, cache_bytes)
    try:
        _component_run(sr, w, ctx, gw, rw, w.prompt(2), 4, (10, 17, 33), 0.3)
    finally:
        sr.sr_destroy(ctx)


def test_bf16_reward_model_with_cache(sr):
    """16-bit path (GPT-2-small shape, 12 layers, LayerNorm, GELU, learned positions): rounds at 7 and 15 tokens
    and the final scoring with the cache, each against the oracle's full rescoring."""
    w = si.WORKLOADS["gpt2"].replace(N=12, max_new=28)
    ctx, gw, rw = _ctx(sr, w, 0)
    try:
        _component_run(sr, w, ctx, gw, rw, w.prompt(1), 9, (7, 15), 0.4)
    finally:
        sr.sr_destroy(ctx)


def test_gqa_head_dim_256_reward_model_with_cache(sr):
    """The 2B-shaped reward model (MHA, head_dim 256, GeGLU) at 2 layers with the Mistral-shaped generator:
    cached keys through the head-dim-256 prefill kernel (two 128-column value halves)."""
    base = si.WORKLOADS["mistral7b_rm2b"]
    w = si.shrink(base, 2, N=8, max_new=26, taus=(), prompt_len=21, sched_kind=si.SCHED_FIXED, pool_bytes=0)
    ctx, gw, rw = _ctx(sr, w, 1)
    try:
        _component_run(sr, w, ctx, gw, rw, w.prompt(0), 2, (9, 18), 0.5)
    finally:
        sr.sr_destroy(ctx)


def test_llama_width_reward_model_with_cache(sr):
    """8B widths (head_dim 128, 8 kv heads: the tensor-core prefill kernel reads the cached pages), 2 layers:
    rounds at 7 and 15 tokens and the final scoring with the cache, each against the oracle's full rescoring."""
    w = si.shrink(si.WORKLOADS["llama8b_n256"], 2, N=8, max_new=24, taus=(), prompt_len=40, pool_bytes=0)
    ctx, gw, rw = _ctx(sr, w, 2)
    try:
        _component_run(sr, w, ctx, gw, rw, w.prompt(3), 5, (7, 15), 0.5)
    finally:
        sr.sr_destroy(ctx)
