"""Oracle parity of the 8B-shaped path at the sizes the benchmark runs.

* Full depth: the Llama-3-8B-shaped workload as the benchmark runs it (32 layers, N = 1024, 60 GB pool,
  memory-triggered) through the component calls.  At sampled (candidate, step) positions the oracle follows the
  GPU's tokens through all 32 layers and gives the logits (max |delta| <= 5e-2) before and after the first
  rejection round -- the 1024-row phase runs the 256-row and CTA-pair GEMM kernels, the post-round phase the
  transposed split-K kernel -- and the first round's partial rewards through the 32-layer reward model
  (1e-2 x max(|r|, rms R)), Eq. partial.reward.set.
* Multi-chunk scoring: 2 layers at 8B widths, N = 1024 and a decision point at tau = 17, so the round's 17 408
  response rows are scored in two 16 384-row chunks; 64 sampled rewards on both sides of the chunk boundary
  against the oracle, and the same run with the self-likelihood reward of Section 5.3 against the oracle's
  log-probabilities.

The weights are drawn on the device (sr_inputs.device_weight_blob) and streamed to the oracle one layer at a
time, so the oracle's float64 weight copies stay at one layer.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import sr_inputs as si
from oracle.logprob import token_logprob
from oracle.sampler import perturbed_logits
from oracle.select import select_round
from oracle.transformer import Transformer, attention

pytestmark = pytest.mark.gpu
LOGIT_TOL = 5e-2
REWARD_REL = 1e-2


@pytest.fixture(scope="module")
def sr():
    from paper_2410_20290_gb300 import binding
    return binding


class StreamedModel:
    """The oracle's forward (oracle.transformer) of a model whose bf16 weights are a device blob in the sr.h
    layout, run one layer at a time: each layer's weights are widened to float32 (exact for bf16), copied to the
    host, used by the oracle's layer functions and dropped."""

    def __init__(self, m: si.ModelDesc, blob):
        self.m, self.blob = m, blob
        self.offs, off = {}, 0
        for name, shape in si.weight_layout(m):
            n = int(np.prod(shape))
            self.offs[name] = (off, shape)
            off += n
        assert off == blob.numel()

    def _part(self, names, rename=None):
        w = {}
        for n in names:
            off, shape = self.offs[n]
            w[rename(n) if rename else n] = self.blob[off:off + int(np.prod(shape))].float().cpu().numpy().reshape(shape)
        return Transformer(self.m.replace(n_layers=1, dtype=si.DT_F32), w)

    def hidden(self, *id_sets):
        """Each ids [B, T] at positions 0..T-1 -> final-normed hidden [B, T, d]; every layer is fetched once for
        all sets.  Returns ([hidden per set], the final-norm / head part)."""
        m = self.m
        sets = [np.asarray(ids) for ids in id_sets]
        poss = [np.broadcast_to(np.arange(ids.shape[1]), ids.shape) for ids in sets]
        emb = self._part(["tok_emb"] + (["pos_emb"] if m.pos == si.POS_LEARNED else []))
        xs = [emb.embed(ids, pos) for ids, pos in zip(sets, poss)]
        del emb
        for l in range(m.n_layers):
            names = [n for n, _ in si.weight_layout(m) if n.startswith(f"l{l}.")]
            t = self._part(names, rename=lambda k, l=l: "l0." + k[len(f"l{l}."):])
            for k_, pos in enumerate(poss):
                q, k, v = t.qkv(0, xs[k_], pos)
                x = t.attn_out(0, xs[k_], attention(q, k, v, pos, pos, m.window))
                xs[k_] = t.mlp(0, x)
            del t
        head = ["final_norm_w"] + (["final_norm_b"] if m.norm == si.NORM_LAYER else []) + \
            (["lm_head"] if m.has_lm_head else ["score_head"])
        fin = self._part(head)
        return [fin.final(x) for x in xs], fin


def _counts(sr, ctx, b):
    import ctypes
    nl, top, mp = ctypes.c_int(0), ctypes.c_int(0), ctypes.c_int(0)
    sr._check(sr.LIB.sr_batch_query(ctx, b, None, None, None, None, None, None, ctypes.addressof(nl),
                                    ctypes.addressof(top), ctypes.addressof(mp)))
    return nl.value, top.value


def _reward_tol(r, R):
    R = np.asarray(R, np.float64)
    return REWARD_REL * max(abs(float(r)), float(np.sqrt(np.mean(R ** 2))))


def _check_tokens(logits_want, toks_gpu, ids, steps, w, seed):
    """A sampled token must be the oracle's draw from its own logits wherever the oracle's top-2 perturbed gap
    exceeds twice the logit tolerance; closer calls may go either way within that tolerance."""
    for lw, t, i, g in zip(logits_want, toks_gpu, ids, steps):
        z = perturbed_logits(lw, seed, int(i), int(g), w.temperature, w.eos_bias, w.eos_id)
        top = np.sort(z)[-2:]
        if top[1] - top[0] > 2 * LOGIT_TOL:
            assert int(t) == int(np.argmax(z)), (i, g)


def test_llama8b_n1024_full_depth_logits_and_rewards(sr):
    """32 layers, N = 1024, 60 GB pool, prompt 6 of the workload (P = 73): logits at steps 1 and 2 (1024 live
    rows), partial rewards at the first memory-triggered round, and logits of the first step after it (about
    308 live rows), each for sampled candidates against the oracle's 32-layer forward on the GPU's tokens."""
    w = si.WORKLOADS["llama8b_n1024"]
    prompt = w.prompt(6)
    P, N, V, seed = len(prompt), w.N, w.gen.vocab, 23
    assert P == 73
    gb = si.device_weight_blob(w.gen, w.weight_seed, 0)
    rb = si.device_weight_blob(w.rm, w.weight_seed, 1)
    ctx = sr.sr_init(w.gen, gb, w.rm, rb, w.pool_bytes, 16, 0)
    max_pages = (P + w.max_new - 1) // 16 + 1
    n_pages = w.pool_bytes // (16 * si.kv_bytes_per_token(w.gen))
    early = {}       # step -> (ids, gpu logits rows, gpu tokens)
    try:
        b = sr.sr_batch_begin(ctx, prompt, N, w.max_new, w.temperature, w.eos_bias, w.eos_id, seed)
        g = 1
        while True:
            n_live, free = _counts(sr, ctx, b)
            if (P + g - 1) % 16 == 0 and free < n_live:
                break
            if g in (1, 2):
                q = sr.sr_batch_query(ctx, b, N, w.max_new, max_pages, n_pages)
                live = [int(i) for i in q["ids_live"]]
                assert len(live) == N - int(np.sum(q["status"] != 0))
                if g == 1:
                    early_ids = [live[0], live[len(live) // 2], live[-1]]
                rows = [live.index(i) for i in early_ids]        # still live at step 2 (no EOS at token 0 or 1)
                logits = np.zeros((len(live), V), np.float32)
                sr.sr_decode_step(ctx, b, logits)
                q2 = sr.sr_batch_query(ctx, b, N, w.max_new, max_pages, n_pages)
                early[g] = (logits[rows].copy(), [q2["tokens"][i][g] for i in early_ids], q2["tokens"].copy())
                del logits
            else:
                sr.sr_decode_step(ctx, b, None)
            g += 1
        g_round = g
        q = sr.sr_batch_query(ctx, b, N, w.max_new, max_pages, n_pages)
        batch = [i for i in range(N) if q["status"][i] in (0, 1)]
        rewards = sr.sr_score_partial(ctx, b, N)
        assert len(rewards) == len(batch) and np.all(np.isfinite(rewards))
        rc, acc, n_live_after = sr.sr_reject_compact(ctx, b, rewards, w.alpha)
        want_rc, want_mask, _ = select_round(rewards, w.alpha)
        assert np.float32(rc) == np.float32(want_rc)
        assert acc.tolist() == [i for i, a in zip(batch, want_mask) if a]
        q = sr.sr_batch_query(ctx, b, N, w.max_new, max_pages, n_pages)
        live = [int(i) for i in q["ids_live"]]
        assert len(live) == n_live_after and 0 < n_live_after <= 512      # the transposed split-K GEMM's range
        logits = np.zeros((len(live), V), np.float32)
        sr.sr_decode_step(ctx, b, logits)
        q2 = sr.sr_batch_query(ctx, b, N, w.max_new, max_pages, n_pages)
        late_ids = [live[0], live[-1]]
        late_rows = [0, len(live) - 1]
        late_logits = logits[late_rows].copy()
        late_toks = [q2["tokens"][i][g_round] for i in late_ids]
        late_seqs = np.array([list(prompt) + q["tokens"][i][:g_round].tolist() for i in late_ids])
        assert all(q["lengths"][i] == g_round for i in late_ids)
        late_rewards = [float(rewards[batch.index(i)]) for i in late_ids]
        del logits
        sr.sr_batch_end(ctx, b)
    finally:
        sr.sr_destroy(ctx)
    torch.cuda.empty_cache()

    gen = StreamedModel(w.gen, gb)
    # steps 1 and 2 from one forward over prompt ++ tokens 0..1; after the round, step g_round over
    # prompt ++ tokens 0..g_round-1 (the same sequences the reward model scored)
    lg1, tk1, toks = early[1]
    lg2, tk2, _ = early[2]
    seqs = np.array([list(prompt) + toks[i][:2].tolist() for i in early_ids])
    (hn_e, hn_l), fin = gen.hidden(seqs, late_seqs)
    want1 = fin.logits(hn_e[:, P])          # logits for token 1: the last input is token 0, at position P
    want2 = fin.logits(hn_e[:, P + 1])
    assert np.max(np.abs(lg1 - want1)) <= LOGIT_TOL
    assert np.max(np.abs(lg2 - want2)) <= LOGIT_TOL
    _check_tokens(want1, tk1, early_ids, [1] * 3, w, seed)
    _check_tokens(want2, tk2, early_ids, [2] * 3, w, seed)
    want = fin.logits(hn_l[:, -1])
    assert np.max(np.abs(late_logits - want)) <= LOGIT_TOL
    _check_tokens(want, late_toks, late_ids, [g_round] * 2, w, seed)
    del hn_e, hn_l, fin, gen
    rm = StreamedModel(w.rm, rb)
    (hn,), fin = rm.hidden(late_seqs)
    want_r = fin.score(hn[:, -1])
    for r_gpu, r_ref in zip(late_rewards, want_r):
        assert abs(r_gpu - r_ref) <= _reward_tol(r_ref, rewards), (r_gpu, r_ref)


@pytest.fixture(scope="module")
def chunked(sr):
    """2-layer 8B-width run, N = 1024, decision at tau = 17 (17 408 rows, two scoring chunks), with the reward
    model and with the self-likelihood reward (same seed, so the same tokens)."""
    base = si.WORKLOADS["llama8b_n256"]
    w = si.shrink(base, 2, N=1024, max_new=40, taus=(17,), prompt_len=73, pool_bytes=0)
    prompt = w.prompt(4)
    gb = si.device_weight_blob(w.gen, 5, 0)
    rb = si.device_weight_blob(w.rm, 5, 1)
    ctx = sr.sr_init(w.gen, gb, w.rm, rb, 0, 16, 0)
    P, N, seed = len(prompt), w.N, 31
    max_pages = (P + w.max_new - 1) // 16 + 1
    n_pages = P // 16 + N * ((P + w.max_new - 2) // 16 + 1 - P // 16)
    out = {"w": w, "prompt": prompt, "gb": gb, "rb": rb, "seed": seed}
    try:
        for kind in (sr.SR_REWARD_MODEL, sr.SR_REWARD_LOGPROB):
            sr.sr_set_reward(ctx, kind)
            b = sr.sr_batch_begin(ctx, prompt, N, w.max_new, w.temperature, w.eos_bias, w.eos_id, seed)
            for g in range(1, 17):
                sr.sr_decode_step(ctx, b, None)
            q = sr.sr_batch_query(ctx, b, N, w.max_new, max_pages, n_pages)
            rewards = sr.sr_score_partial(ctx, b, N)
            batch = [i for i in range(N) if q["status"][i] in (0, 1)]
            res = {"rewards": rewards, "batch": batch, "tokens": q["tokens"].copy(), "lengths": q["lengths"].copy()}
            if kind == sr.SR_REWARD_MODEL:
                rc, acc, _ = sr.sr_reject_compact(ctx, b, rewards, w.alpha)
                res["rc"], res["acc"] = rc, acc
            sr.sr_batch_end(ctx, b)
            out[kind] = res
    finally:
        sr.sr_destroy(ctx)
    return out


def _sample_ids(batch, lengths, tau):
    """64 candidates of full length tau: spread over the batch, and 8 on each side of the first chunk boundary
    (the chunk planner packs ids in order until 16 384 rows)."""
    full = [i for i in batch if lengths[i] == tau]
    rows, boundary = 0, None
    for j, i in enumerate(batch):
        if rows + lengths[i] > 16384:
            boundary = j
            break
        rows += lengths[i]
    assert boundary is not None, "the round must need two chunks"
    near = [i for i in batch[boundary - 8: boundary + 8] if lengths[i] == tau]
    spread = [full[k] for k in np.linspace(0, len(full) - 1, 64 - len(near)).astype(int)]
    return sorted(set(near + spread)), boundary


def test_multi_chunk_partial_rewards_match_oracle(sr, chunked):
    w, prompt = chunked["w"], chunked["prompt"]
    res = chunked[sr.SR_REWARD_MODEL]
    batch, lengths, rewards = res["batch"], res["lengths"], res["rewards"]
    assert len(batch) == w.N and sum(int(lengths[i]) for i in batch) > 16384
    ids, boundary = _sample_ids(batch, lengths, 17)
    assert len(ids) >= 60 and any(batch.index(i) < boundary for i in ids) and any(batch.index(i) >= boundary
                                                                                   for i in ids)
    seqs = np.array([list(prompt) + res["tokens"][i][:17].tolist() for i in ids])
    (hn,), fin = StreamedModel(w.rm, chunked["rb"]).hidden(seqs)
    want = fin.score(hn[:, -1])
    for i, r_ref in zip(ids, want):
        r_gpu = float(rewards[batch.index(i)])
        assert abs(r_gpu - r_ref) <= _reward_tol(r_ref, rewards), (i, r_gpu, r_ref)
    # the cut on the GPU's rewards is the oracle's order statistic, bit for bit
    want_rc, want_mask, _ = select_round(rewards, w.alpha)
    assert np.float32(res["rc"]) == np.float32(want_rc)
    assert res["acc"].tolist() == [i for i, a in zip(batch, want_mask) if a]
    # a sampled candidate clear of r_cut by more than the tolerance is on the oracle's side of it
    for i, r_ref in zip(ids, want):
        if abs(r_ref - want_rc) > _reward_tol(r_ref, rewards):
            assert (i in set(res["acc"].tolist())) == (r_ref >= want_rc)


def test_multi_chunk_self_likelihood_matches_oracle(sr, chunked):
    """Section 5.3 reward at 8B widths (fp16 path): mean ln p of the 17 generated tokens under the generator."""
    w, prompt = chunked["w"], chunked["prompt"]
    res = chunked[sr.SR_REWARD_LOGPROB]
    assert np.array_equal(res["tokens"], chunked[sr.SR_REWARD_MODEL]["tokens"])
    batch, lengths, rewards = res["batch"], res["lengths"], res["rewards"]
    ids, _ = _sample_ids(batch, lengths, 17)
    P = len(prompt)
    seqs = np.array([list(prompt) + res["tokens"][i][:17].tolist() for i in ids])
    (hn,), fin = StreamedModel(w.gen, chunked["gb"]).hidden(seqs)
    for j, i in enumerate(ids):
        lg = fin.logits(hn[j, P - 1:P + 16])        # logits for tokens 0..16
        want = np.mean([token_logprob(lg[t], int(res["tokens"][i][t])) for t in range(17)])
        r_gpu = float(rewards[batch.index(i)])
        assert abs(r_gpu - want) <= _reward_tol(want, rewards), (i, r_gpu, want)
