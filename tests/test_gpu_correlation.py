"""Appendix B partial-versus-final reward correlation through the component calls, against the oracle."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import sr_inputs as si
from oracle import correlation as oc
from oracle.transformer import Transformer

pytestmark = pytest.mark.gpu


def test_tiny_partial_final_correlation_matches_oracle():
    from paper_2410_20290_gb300 import binding as sr
    from paper_2410_20290_gb300.correlation import partial_final
    w = si.WORKLOADS["tiny"].replace(N=12)
    gw, rw = si.random_weights(w.gen, 0, 0), si.random_weights(w.rm, 0, 1)
    taus = (2, 8, 24, w.max_new + 5)
    ctx = sr.sr_init(w.gen, si.pack_blob(w.gen, gw), w.rm, si.pack_blob(w.rm, rw), 0, 16, 0)
    try:
        part, final, stats = partial_final(ctx, w.prompt(1), w.N, taus, w.max_new, w.temperature, w.eos_bias,
                                           w.eos_id, 1)
    finally:
        sr.sr_destroy(ctx)
    gen, rm = Transformer(w.gen, gw), Transformer(w.rm, rw)
    opart, ofinal, ostats = oc.partial_final(gen, rm, w.prompt(1), w.N, taus, w.max_new, w.temperature,
                                             w.eos_bias, w.eos_id, 1)
    tol = 1e-2 * max(float(np.sqrt(np.mean(ofinal.astype(np.float64) ** 2))), 1e-6)
    np.testing.assert_allclose(final, ofinal, rtol=0, atol=tol)
    for t in taus:
        np.testing.assert_allclose(part[t], opart[t], rtol=0, atol=tol)
        assert abs(stats[t][0] - ostats[t][0]) <= 1e-2
        # each pair whose order flips within the reward tolerance moves tau-a by 2 / (N (N - 1))
        assert abs(stats[t][1] - ostats[t][1]) <= 2.0 / (w.N * (w.N - 1) / 2) + 1e-9
        assert abs(stats[t][2] - ostats[t][2]) <= 3.0 / (w.N * (w.N - 1) / 2) + 1e-9
    assert stats[taus[-1]][0] == pytest.approx(1.0)
