"""Partial-versus-final reward correlation (Appendix B) through the library's component calls.

Runs one Best-of-N batch (no rejection) with `sr_batch_begin` / `sr_decode_step`, scores every
candidate with `sr_score_partial` when the batch has generated tau tokens for each tau in `taus`
(tau_k = min(tau, len(Y_k)), Eq. partial.reward.set) and once more when every candidate has completed
(the final rewards), and reports per tau the Pearson correlation and Kendall's rank correlation of
Appendix B between the partial and final rewards, R_Kendall = 2 / (N (N - 1)) sum_{i<j} sgn(x_i - x_j)
sgn(y_i - y_j) (tau-a: tied pairs count 0), with the tie-corrected tau-b beside it.  With random-initialised weights the numbers describe only the synthetic models.

    python -m paper_2410_20290_gb300.correlation [workload] [tau ...]
"""
import json
import sys
from typing import Sequence


import numpy as np


def pearson(x, y) -> float:
    """Appendix B: sum (x_i - mean x)(y_i - mean y) / sqrt(sum (x_i - mean x)^2 sum (y_i - mean y)^2)."""
    x = np.asarray(x, np.float64)
    y = np.asarray(y, np.float64)
    dx, dy = x - x.mean(), y - y.mean()
    den = np.sqrt(np.sum(dx * dx) * np.sum(dy * dy))
    return float(np.sum(dx * dy) / den) if den > 0 else float("nan")


def kendall(x, y):
    """(tau-a, tau-b): tau-a = 2 / (n (n - 1)) sum_{i<j} sgn(x_i - x_j) sgn(y_i - y_j) (Appendix B);
    tau-b divides the same sum by sqrt((n0 - ties in x)(n0 - ties in y)), n0 = n (n - 1) / 2."""
    x = np.asarray(x, np.float64)
    y = np.asarray(y, np.float64)
    n = len(x)
    if n < 2:
        return float("nan"), float("nan")
    iu = np.triu_indices(n, 1)
    sx = np.sign(x[:, None] - x[None, :])[iu]
    sy = np.sign(y[:, None] - y[None, :])[iu]
    s = float(np.sum(sx * sy))
    n0 = n * (n - 1) / 2
    den_b = np.sqrt(float(np.count_nonzero(sx)) * float(np.count_nonzero(sy)))
    return s / n0, (s / den_b if den_b > 0 else float("nan"))


def _n_live(ctx, batch) -> int:
    """Live candidates of the batch (sr_batch_query with only the count requested)."""
    import ctypes

    from . import binding as sr
    n = ctypes.c_int(0)
    sr._check(sr.LIB.sr_batch_query(ctx, batch, None, None, None, None, None, None, ctypes.addressof(n), None, None))
    return n.value


def partial_final(ctx, prompt, N: int, taus: Sequence[int], max_new: int, temperature: float, eos_bias: float,
                  eos_id: int, seed: int):
    """Partial rewards {tau: [N]} and final rewards [N] (ascending candidate id), and
    {tau: (pearson, kendall tau-a, kendall tau-b)}."""
    from . import binding as sr
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
    stats = {t: (pearson(partial[t], final), *kendall(partial[t], final)) for t in taus}
    return partial, final, stats


def main(argv):
    import sr_inputs as si

    from . import binding as sr
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
                      "per_tau": {str(t): {"pearson": p, "kendall": ka, "kendall_tau_b": kb}
                                  for t, (p, ka, kb) in stats.items()}}))


if __name__ == "__main__":
    main(sys.argv[1:])
