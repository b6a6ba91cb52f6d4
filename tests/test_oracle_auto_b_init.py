"""Pin of the automatic initial batch size (Algorithm 1, first step) against the oracle's own trigger."""
import pytest

import sr_inputs as si
from oracle.pool import auto_b_init, pool_pages
from oracle.sr import SpeculativeRejection
from oracle.transformer import Transformer


def _first_round_step(w, gen, rm, prompt, N, n_pages):
    o = SpeculativeRejection(gen, rm, prompt, N, 0.5, si.SCHED_POOL_FULL, (), w.max_new, w.temperature,
                             w.eos_bias, w.eos_id, 0, n_pages)
    try:
        res = o.run()
    except MemoryError:   # not even the prompt-tail pages fit: the batch fails before its first token
        return -1
    return res.rounds[0].step if res.rounds else None


@pytest.mark.parametrize("P,tau_min,n_pages", [(16, 8, 40), (21, 10, 45), (30, 17, 64), (5, 1, 12)])
def test_auto_b_init_is_the_largest_batch_reaching_tau_min(P, tau_min, n_pages):
    """With N = auto_b_init the first memory-triggered round comes at tau_min generated tokens or later; with
    N + 1 it comes earlier, or the batch cannot even take its prompt-tail pages (the oracle's trigger and pool,
    run step by step, decide).  EOS is disabled so every
    candidate keeps generating."""
    w = si.WORKLOADS["tiny"].replace(max_new=40, eos_id=-1)
    gen = Transformer(w.gen, si.random_weights(w.gen, 0, 0))
    rm = Transformer(w.rm, si.random_weights(w.rm, 0, 1))
    prompt = w.prompt(0)[:P] if len(w.prompt(0)) >= P else list(w.prompt(0)) * (P // len(w.prompt(0)) + 1)
    prompt = list(prompt)[:P]
    N = auto_b_init(n_pages, P, tau_min, n_max=64)
    assert 1 <= N < 64
    s = _first_round_step(w, gen, rm, prompt, N, n_pages)
    assert s is None or s >= tau_min
    s1 = _first_round_step(w, gen, rm, prompt, N + 1, n_pages)
    assert s1 is not None and s1 < tau_min


def test_auto_b_init_limits():
    assert auto_b_init(10, 16, 8, 64) == 9                      # 1 shared page, 1 private page each
    assert auto_b_init(10, 16, 8, 4) == 4                       # capped by n_max
    assert auto_b_init(0, 16, 8, 64) == 0                       # nothing fits
    # the 8B pool at P = 288: 28 610 pages, 18 shared, 27 private pages to reach 432 tokens
    assert pool_pages(60 * 10 ** 9, 128 * 1024) == 28610
    assert auto_b_init(28610, 288, 432, 4096) == (28610 - 18) // 27 == 1058


def test_library_auto_b_init_matches_the_oracle():
    """The C-ABI's host-side b_init equals the oracle's on a grid (integers: exact).  No GPU call."""
    from paper_2410_20290_gb300 import binding as sr
    for name in ("tiny", "gpt2", "llama8b_n1024"):
        w = si.WORKLOADS[name]
        kvt = si.kv_bytes_per_token(w.gen)
        for pool_bytes in (16 * kvt * 7, 16 * kvt * 100, 60 * 10 ** 9):
            for P in (1, 15, 16, 17, 288, 511):
                for tau in (1, 2, 16, 17, 432):
                    want = auto_b_init(pool_pages(pool_bytes, kvt), P, tau, 4096)
                    assert sr.sr_auto_b_init(w.gen, pool_bytes, P, tau, 4096) == want
