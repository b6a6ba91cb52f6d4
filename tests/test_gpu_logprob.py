"""GPU parity of the self-likelihood reward of Section 5.3 (s(Y) = ln p(Y | X) / len(Y) under the generator)."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import sr_inputs as si
from oracle.logprob import token_logprob
from oracle.pool import pool_pages
from oracle.sampler import sample_token
from oracle.sr import DONE, SpeculativeRejection
from oracle.transformer import Transformer

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sr():
    from paper_2410_20290_gb300 import binding
    return binding


@pytest.mark.parametrize("V,T,bias,eos", [(512, 1.0, 0.0, 0), (128256, 0.8, 2.0, 0), (37, 1.3, -1.0, 36)])
def test_sample_accumulates_token_logprob(sr, V, T, bias, eos):
    """Two sampling steps on the same rows: tokens bit-exact, and logprob_sum[id] equals the oracle's
    ln softmax(raw logits)[token] summed over both steps (fp32 log-sum-exp on the GPU)."""
    rng = np.random.default_rng(V)
    b = 6
    ids = rng.permutation(16)[:b].astype(np.int32)
    lp = torch.zeros(16, dtype=torch.float64, device="cuda")
    want = np.zeros(16)
    seed = 77
    for step in (0, 5):
        logits = (rng.standard_normal((b, V)) * 2.0).astype(np.float32)
        logits[1, :3] = np.nan
        steps = np.full(b, step, np.int32)
        out = torch.zeros(b, dtype=torch.int32, device="cuda")
        sr.sr_k_sample(torch.from_numpy(logits).cuda(), V, b, V, torch.from_numpy(ids).cuda(),
                       torch.from_numpy(steps).cuda(), seed, T, bias, eos, out, logprob_sum=lp)
        got = out.cpu().numpy()
        for r in range(b):
            tok = sample_token(logits[r], seed, int(ids[r]), step, T, bias, eos)
            assert got[r] == tok
            want[ids[r]] += token_logprob(logits[r], tok)
    np.testing.assert_allclose(lp.cpu().numpy(), want, rtol=0, atol=2e-5 * 2 * np.log(V))


def _oracle(w, gw, rw, prompt, seed, alpha):
    n_pages = pool_pages(w.pool_bytes, si.kv_bytes_per_token(w.gen)) if w.pool_bytes else 0
    o = SpeculativeRejection(Transformer(w.gen, gw), Transformer(w.rm, rw), prompt, w.N, alpha, w.sched_kind,
                             w.taus, w.max_new, w.temperature, w.eos_bias, w.eos_id, seed, n_pages,
                             reward="logprob")
    return o.run()


@pytest.mark.parametrize("seed,alpha", [(0, 0.5), (1, 0.5), (2, 0.0)])
def test_tiny_logprob_reward_free_running(sr, seed, alpha):
    """Tiny fp32 workload with the self-likelihood reward: same rounds, survivors, selected candidate, tokens
    and score as the oracle; no reward-model work."""
    w = si.WORKLOADS["tiny"]
    gw, rw = si.random_weights(w.gen, 0, 0), si.random_weights(w.rm, 0, 1)
    ctx = sr.sr_init(w.gen, si.pack_blob(w.gen, gw), w.rm, si.pack_blob(w.rm, rw), w.pool_bytes, 16, 0)
    try:
        sr.sr_set_reward(ctx, sr.SR_REWARD_LOGPROB)
        prompt = w.prompt(seed)
        toks, score, st = sr.sr_generate(ctx, prompt, w.N, alpha, w.sched_kind, w.taus, w.max_new,
                                          w.temperature, w.eos_bias, w.eos_id, seed)
        # back to the reward model: the same context scores with s again
        sr.sr_set_reward(ctx, sr.SR_REWARD_MODEL)
        _, _, st2 = sr.sr_generate(ctx, prompt, w.N, alpha, w.sched_kind, w.taus, w.max_new,
                                   w.temperature, w.eos_bias, w.eos_id, seed)
    finally:
        sr.sr_destroy(ctx)
    ref = _oracle(w, gw, rw, prompt, seed, alpha)
    assert st["best_id"] == ref.best_id
    assert list(toks) == ref.tokens
    assert abs(score - ref.score) <= 1e-4
    assert st["rounds"] == len(ref.rounds)
    for i, rd in enumerate(ref.rounds):
        assert st["b_per_round"][i] == len(rd.batch)
        assert st["accepted_per_round"][i] == int(rd.accepted.sum())
        assert abs(st["r_cut_per_round"][i] - rd.r_cut) <= 1e-4
    assert st["n_completed"] == sum(1 for s in ref.status if s == DONE)
    assert st["rm_tokens"] == 0 and st2["rm_tokens"] > 0
