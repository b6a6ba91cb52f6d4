"""LM head fused with sampling (the GEMM epilogue reduces each row's logits to one record per 64 vocabulary ids;
the logits are never stored) against sampling stored logits, and against the oracle's Gumbel-max.

The fused path picks 256 x 256 CTA-pair tiles from 512 rows and 128 x 256 tiles below; the unfused GEMM is pinned
to the same tiles (SR_GEMM_PAIR=1 / SR_GEMM_BN=256, read once per process, so each runs in a child process) so that
both see the same fp32 logits, and then the tokens must agree bit for bit: with k_sample on the stored logits and
with the oracle's sample_token (Section 3's sampling step) on them.
"""
import json
import os
import subprocess
import sys

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import sr_inputs as si

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import json, sys
sys.path.insert(0, {root!r})
import numpy as np, torch
import sr_inputs as si
from oracle import sampler as osamp
from paper_2410_20290_gb300 import binding as sr
cases = {cases!r}
bad = []
for (M, V, K, T, bias, eos, dt, seed) in cases:
    rng = np.random.default_rng(seed)
    tt = torch.bfloat16 if dt == si.DT_BF16 else torch.float16
    x = torch.from_numpy(rng.standard_normal((M, K)).astype(np.float32) / np.sqrt(K)).to(tt).cuda()
    W = torch.from_numpy(rng.standard_normal((V, K)).astype(np.float32) * 3.0).to(tt).cuda()
    ids = torch.from_numpy(rng.permutation(4096)[:M].astype(np.int32)).cuda()
    lens = torch.from_numpy(rng.integers(0, 3000, 4096).astype(np.int32)).cuda()
    sd = int(rng.integers(0, 2 ** 63))
    logits = torch.zeros(M, V, device="cuda")
    sr.sr_k_gemm(dt, x, W, logits, M, V, K, 0)
    steps = lens[ids.long()].contiguous()
    t_unf = torch.zeros(M, dtype=torch.int32, device="cuda")
    sr.sr_k_sample(logits, V, M, V, ids, steps, sd, T, bias, eos, t_unf)
    t_fus = torch.zeros(M, dtype=torch.int32, device="cuda")
    sr.sr_k_lm_head_sample(dt, x, W, M, V, K, ids, lens, sd, T, bias, eos, t_fus)
    torch.cuda.synchronize()
    L = logits.cpu().numpy()
    ih, sh = ids.cpu().numpy(), steps.cpu().numpy()
    rows = range(M) if M <= 64 else sorted(set(np.linspace(0, M - 1, 48).astype(int)))
    want = [osamp.sample_token(L[r], sd, int(ih[r]), int(sh[r]), T, bias, eos) for r in rows]
    fu, uf = t_fus.cpu().numpy(), t_unf.cpu().numpy()
    if not np.array_equal(fu, uf) or [int(fu[r]) for r in rows] != want:
        bad.append([M, V, K, int((fu != uf).sum())])
print("RESULT", json.dumps(bad))
"""


def _run(env, cases):
    r = subprocess.run([sys.executable, "-c", CHILD.format(root=ROOT, cases=cases)], cwd=ROOT,
                       env=dict(os.environ, **env), capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-3000:]
    line = [l for l in r.stdout.splitlines() if l.startswith("RESULT")][-1]
    return json.loads(line.split(" ", 1)[1])


F16, BF16 = si.DT_F16, si.DT_BF16


def test_fused_sampling_one_sm_tiles():
    """Below 512 rows: 128 x 256 tiles; ragged rows, vocabulary tails inside a tile, EOS bias, bf16 operands."""
    cases = [(1, 128256, 4096, 1.0, 1.0, 0, F16, 1), (5, 32000, 768, 0.7, 2.0, 7, F16, 2),
             (100, 128256, 4096, 1.0, 1.0, 0, F16, 3), (308, 128256, 4096, 1.0, 1.0, 0, F16, 4),
             (130, 1056, 256, 1.3, -1.0, 1055, F16, 5), (77, 32000, 512, 1.0, 0.0, -1, BF16, 6)]
    assert _run({"SR_GEMM_BN": "256"}, cases) == []


def test_fused_sampling_pair_tiles():
    """From 512 rows: CTA-pair 256 x 256 tiles; ragged pair rows (600, 1000) and the bench's 1024."""
    cases = [(512, 32000, 1024, 1.0, 1.0, 0, F16, 11), (600, 128256, 4096, 0.8, 2.0, 0, F16, 12),
             (1024, 128256, 4096, 1.0, 1.0, 0, F16, 13), (1000, 1056, 256, 1.0, 0.0, -1, BF16, 14)]
    assert _run({"SR_GEMM_PAIR": "1"}, cases) == []


GEN_CHILD = r"""
import json, sys
sys.path.insert(0, {root!r})
import numpy as np
import sr_inputs as si
from paper_2410_20290_gb300 import binding as sr
out = []
for name, reward in (("llama_small", sr.SR_REWARD_MODEL), ("llama_small", sr.SR_REWARD_LOGPROB)):
    w = si.shrink(si.WORKLOADS["llama8b_n256"], 2, N=24, max_new=40, taus=(12, 25), prompt_len=37, pool_bytes=0)
    gw, rw = si.random_weights(w.gen, 5, 0), si.random_weights(w.rm, 5, 1)
    ctx = sr.sr_init(w.gen, si.pack_blob(w.gen, gw), w.rm, si.pack_blob(w.rm, rw), w.pool_bytes, 16, 0)
    try:
        sr.sr_set_reward(ctx, reward)
        toks, score, st = sr.sr_generate(ctx, w.prompt(4), w.N, w.alpha, w.sched_kind, w.taus, w.max_new,
                                          w.temperature, w.eos_bias, w.eos_id, 9)
    finally:
        sr.sr_destroy(ctx)
    out.append([list(map(int, toks)), float(score), st["best_id"], st["b_per_round"], st["r_cut_per_round"]])
print("RESULT", json.dumps(out))
"""


def test_fused_sampling_generation_matches_unfused():
    """Whole generations (8B widths at 2 layers, 24 candidates, rounds at 12 and 25 tokens; reward model and the
    self-likelihood reward, whose log-sum-exp the fused records carry): the same tokens, rounds, cuts and
    choice with the fused sampler as with stored logits."""
    res = {}
    for flag in ("1", "0"):
        r = subprocess.run([sys.executable, "-c", GEN_CHILD.format(root=ROOT)], cwd=ROOT,
                           env=dict(os.environ, SR_FUSED_SAMPLE=flag), capture_output=True, text=True, timeout=900)
        assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-3000:]
        res[flag] = json.loads([l for l in r.stdout.splitlines() if l.startswith("RESULT")][-1].split(" ", 1)[1])
    for fu, uf in zip(res["1"], res["0"]):
        assert fu[0] == uf[0] and fu[2] == uf[2] and fu[3] == uf[3]
        assert np.allclose(fu[4], uf[4], rtol=1e-6, atol=1e-6) and abs(fu[1] - uf[1]) <= 1e-5 * max(1.0, abs(uf[1]))
