"""Partial-versus-final reward correlation (Appendix B) through the library's component calls.

Runs one Best-of-N batch (no rejection) with `sr_batch_begin` / `sr_decode_step`, scores every
candidate with `sr_score_partial` when the batch has generated tau tokens for each tau in `taus`
(tau_k = min(tau, len(Y_k)), Eq. partial.reward.set) and once more when every candidate has completed
(the final rewards), and reports the Pearson correlation and Kendall's tau-b between the partial and
final rewards per tau.  With random-initialised weights the numbers describe only the synthetic models.

    python -m paper_2410_20290_gb300.correlation [workload] [tau ...]
"""
import json
import sys
from typing import Sequence


from . import binding as sr


def _n_live(ctx, batch) -> int:
    """Live candidates of the batch (sr_batch_query with only the count requested)."""
    import ctypes
    n = ctypes.c_int(0)
    sr._check(sr.LIB.sr_batch_query(ctx, batch, None, None, None, None, None, None, ctypes.addressof(n), None, None))
    return n.value


def partial_final(ctx, prompt, N: int, taus: Sequence[int], max_new: int, temperature: float, eos_bias: float,
                  eos_id: int, seed: int):
    """Partial rewards {tau: [N]} and final rewards [N] (ascending candidate id), and {tau: (pearson, tau_b)}."""
    from scipy import stats as st
    taus = sorted(set(int(t) for t in taus))
    b = sr.sr_batch_begin(ctx, prompt, N, max_new, temperature, eos_bias, eos_id, seed)
    partial = {}
    try:
        g = 1  # token 0 of every candidate is sampled by sr_batch_begin
        while True:
            if g in taus:
                partial[g] = sr.sr_score_partial(ctx, b, N)
            if _n_live(ctx, b) == 0:
                break
            sr.sr_decode_step(ctx, b)
            g += 1
        final = sr.sr_score_partial(ctx, b, N)
    finally:
        sr.sr_batch_end(ctx, b)
    for t in taus:  # decision points past the longest response score the complete responses
        partial.setdefault(t, final.copy())
    stats = {t: (float(st.pearsonr(partial[t], final)[0]), float(st.kendalltau(partial[t], final)[0])) for t in taus}
    return partial, final, stats


def main(argv):
    import sr_inputs as si
    name = argv[0] if argv else "tiny"
    w = si.WORKLOADS[name]
    taus = [int(t) for t in argv[1:]] or [max(1, w.max_new // 8), w.max_new // 4, w.max_new // 2]
    gw, rw = si.random_weights(w.gen, w.weight_seed, 0), si.random_weights(w.rm, w.weight_seed, 1)
    ctx = sr.sr_init(w.gen, si.pack_blob(w.gen, gw), w.rm, si.pack_blob(w.rm, rw), 0, 16, 0)
    try:
        _, _, stats = partial_final(ctx, w.prompt(0), w.N, taus, w.max_new, w.temperature, w.eos_bias, w.eos_id, 0)
    finally:
        sr.sr_destroy(ctx)
    print(json.dumps({"workload": name, "N": w.N,
                      "per_tau": {str(t): {"pearson": p, "kendall_tau_b": k} for t, (p, k) in stats.items()}}))


if __name__ == "__main__":
    main(sys.argv[1:])
