"""Pins of the oracle's page accounting and memory-triggered rounds."""
import numpy as np
import pytest

import sr_inputs as si
from oracle.pool import PagePool, private_pages_full
from oracle.sr import SpeculativeRejection
from oracle.transformer import Transformer


def test_lifo_order():
    p = PagePool(5)
    assert [p.pop() for _ in range(3)] == [4, 3, 2]
    p.push([7, 9])
    assert p.pop() == 9 and p.pop() == 7 and p.pop() == 1
    with pytest.raises(MemoryError):
        PagePool(0).pop()


def test_private_pages_full():
    # KV positions 0 .. P + max_new - 2
    assert private_pages_full(32, 1) == 0
    assert private_pages_full(32, 2) == 1
    assert private_pages_full(30, 1) == 1
    assert private_pages_full(30, 3) == 1       # positions 30, 31
    assert private_pages_full(30, 4) == 2       # position 32 opens a page


def _tiny(vocab=64):
    m = si.ModelDesc(n_layers=1, d_model=16, n_heads=2, n_kv_heads=2, head_dim=8, ffn_dim=32, vocab=vocab,
                     max_pos=256, dtype=si.DT_F32)
    return Transformer(m, si.random_weights(m, 1)), Transformer(m.replace(has_lm_head=0, has_scalar_head=1),
                                                               si.random_weights(m.replace(has_lm_head=0,
                                                                                           has_scalar_head=1), 1, 1))


@pytest.mark.parametrize("P,b,pages", [(32, 4, 2 + 4 * 3 + 1), (37, 3, 2 + 3 + 3 * 2 + 2), (16, 5, 1 + 5 * 4)])
def test_first_memory_trigger_closed_form(P, b, pages):
    """With no EOS, a page is needed at steps g with (P + g - 1) % 16 == 0; the first round runs at the
    first such step the free pages cannot cover: g* = (16 - P % 16) % 16 + 1 + 16 * floor(avail / b), where
    avail = pages - floor(P/16) - (b if P % 16 else 0)."""
    gen, rm = _tiny()
    prompt = list(np.arange(1, P + 1) % 60 + 1)
    sr = SpeculativeRejection(gen, rm, prompt, b, 0.5, si.SCHED_POOL_FULL, (), max_new=120, eos_bias=-1e30,
                              n_pool_pages=pages)
    res = sr.run()
    avail = pages - P // 16 - (b if P % 16 else 0)
    g_star = (16 - P % 16) % 16 + 1 + 16 * (avail // b)
    assert res.rounds[0].step == g_star
    assert len(res.rounds[0].batch) == b


def test_bon_waves_fit_the_pool():
    gen, rm = _tiny()
    P, N, max_new = 20, 7, 30
    per = private_pages_full(P, max_new)
    pages = P // 16 + 3 * per               # 3 candidates per wave -> waves of 3, 3, 1
    sr = SpeculativeRejection(gen, rm, list(range(1, P + 1)), N, 0.0, si.SCHED_POOL_FULL, (), max_new=max_new,
                              eos_bias=-1e30, n_pool_pages=pages)
    res = sr.run()
    assert all(L == max_new for L in res.lengths)
    assert sorted(res.free_stack) == sorted(set(range(pages)) - set(res.page_tables[0][:P // 16]))
