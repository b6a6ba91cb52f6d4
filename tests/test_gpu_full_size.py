"""Full-size GPU checks in the launch configuration the benchmark times.

The oracle cannot run 8B-shaped models end to end, so at the workloads' full sizes the checks are outputs the
oracle computes one by one from the GPU's own intermediate values -- sampled tokens from the GPU's logits
(bit-exact), r_cut and the accepted set from the GPU's partial rewards (bit-exact) -- and properties that hold at
any size: the memory trigger fires exactly when the free pages cannot cover the next step, the size rule of the
cut, and conservation of KV pages.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import sr_inputs as si
from oracle.pool import pool_pages
from oracle.sampler import sample_token
from oracle.select import select_round

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sr():
    from paper_2410_20290_gb300 import binding
    return binding


def _counts(sr, ctx, b):
    import ctypes
    nl, top, mp = ctypes.c_int(0), ctypes.c_int(0), ctypes.c_int(0)
    sr._check(sr.LIB.sr_batch_query(ctx, b, None, None, None, None, None, None, ctypes.addressof(nl),
                                    ctypes.addressof(top), ctypes.addressof(mp)))
    return nl.value, top.value


def _first_round(sr, w: si.Workload, prompt_index: int, sample_step: int = 3, n_sample: int = 12):
    prompt = w.prompt(prompt_index)
    P, N = len(prompt), w.N
    gb = si.device_weight_blob(w.gen, w.weight_seed, 0)
    rb = si.device_weight_blob(w.rm, w.weight_seed, 1)
    ctx = sr.sr_init(w.gen, gb, w.rm, rb, w.pool_bytes, 16, 0)
    del gb, rb
    torch.cuda.empty_cache()
    seed = 17
    n_pages = pool_pages(w.pool_bytes, si.kv_bytes_per_token(w.gen)) if w.pool_bytes else \
        P // 16 + N * ((P + w.max_new - 2) // 16 + 1 - P // 16)
    max_pages = (P + w.max_new - 1) // 16 + 1
    try:
        b = sr.sr_batch_begin(ctx, prompt, N, w.max_new, w.temperature, w.eos_bias, w.eos_id, seed)
        g = 1
        while True:
            n_live, free = _counts(sr, ctx, b)
            assert n_live > 0
            need = (P + g - 1) % 16 == 0
            if w.sched_kind == si.SCHED_POOL_FULL:
                if need and free < n_live:
                    break
            elif g == w.taus[0]:
                break
            if g == sample_step:
                q = sr.sr_batch_query(ctx, b, N, w.max_new, max_pages, n_pages)
                live = q["ids_live"]
                logits = np.zeros((len(live), w.gen.vocab), np.float32)
                sr.sr_decode_step(ctx, b, logits)
                assert np.all(np.isfinite(logits))
                q2 = sr.sr_batch_query(ctx, b, N, w.max_new, max_pages, n_pages)
                pick = np.linspace(0, len(live) - 1, n_sample).astype(int)
                for j in pick:
                    i = int(live[j])
                    assert q2["tokens"][i][g] == sample_token(logits[j], seed, i, g, w.temperature, w.eos_bias,
                                                              w.eos_id)
            else:
                sr.sr_decode_step(ctx, b, None)
            g += 1
        q = sr.sr_batch_query(ctx, b, N, w.max_new, max_pages, n_pages)
        round_batch = [i for i in range(N) if q["status"][i] in (0, 1)]
        rewards = sr.sr_score_partial(ctx, b, N)
        assert len(rewards) == len(round_batch) and np.all(np.isfinite(rewards))
        rc, acc, n_live_after = sr.sr_reject_compact(ctx, b, rewards, w.alpha)
        want_rc, want_mask, k = select_round(rewards, w.alpha)
        assert np.float32(rc) == np.float32(want_rc)
        assert acc.tolist() == [i for i, a in zip(round_batch, want_mask) if a]
        if len(np.unique(rewards)) == len(rewards):
            assert len(acc) == len(rewards) - k                      # the top (1 - alpha) proportion
        # page conservation: shared prompt pages + private pages of live candidates + free stack = the pool,
        # with no page held twice
        q = sr.sr_batch_query(ctx, b, N, w.max_new, max_pages, n_pages)
        n_sh = P // 16
        held = list(q["page_table"][q["ids_live"][0]][:n_sh]) if n_sh and q["n_live"] else []
        for i in q["ids_live"]:
            L = q["lengths"][i]
            last = P + L - 2
            held += list(q["page_table"][i][n_sh:last // 16 + 1])
        pages = held + q["free_stack"].tolist()
        assert len(pages) == len(set(pages)) == n_pages
        sr.sr_batch_end(ctx, b)
        return g, n_live_after
    finally:
        sr.sr_destroy(ctx)


def test_llama8b_n1024_first_round_full_size(sr):
    """Llama-3-8B-shaped generator and reward model, N = 1024, 60 GB pool, memory-triggered (the bench workload)."""
    w = si.WORKLOADS["llama8b_n1024"]
    g, n_live = _first_round(sr, w, 0)
    P = len(w.prompt(0))
    # without completions the closed form of the first trigger would be 11 + 16 * 26 = 427 for P = 262; pages
    # released by candidates that hit EOS can only delay it, by whole 16-token page periods
    assert P == 262 and g >= 427 and (g - 427) % 16 == 0
    assert 0 < n_live <= 1024 - int(np.floor(np.float32(w.alpha) * 1024))


def test_llama8b_n256_decision_point_full_size(sr):
    """Llama-3-8B shape, N = 256, one decision point at tau = 128, temperature 0.8, EOS bias +2."""
    w = si.WORKLOADS["llama8b_n256"]
    g, n_live = _first_round(sr, w, 0)
    assert g == 128 and 0 < n_live <= 128


def test_mistral_rm2b_first_round_full_size(sr):
    """Mistral-7B shape with the 2B reward model, N = 2048, 60 GB pool, memory-triggered, alpha = 0.5."""
    w = si.WORKLOADS["mistral7b_rm2b"]
    g, n_live = _first_round(sr, w, 0)
    # P = 512 fills 32 shared pages; 28578 free pages give 13 page periods for 2048 candidates: first trigger at
    # 1 + 16 * 13 = 209 without completions
    assert g >= 209 and (g - 209) % 16 == 0
    assert 0 < n_live <= 1024
