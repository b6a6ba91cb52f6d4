"""Correlation between partial and final rewards (Appendix B), oracle side.

Appendix B measures how well the reward of a partial response Y^{<=tau} predicts the reward of the
complete response: for Best-of-N trajectories, the partial reward at each decision point tau
(tau_k = min(tau, len(Y_k)), Eq. partial.reward.set) against the final reward, summarised by the
Pearson correlation and Kendall's rank correlation.  Appendix B defines Kendall's statistic as
R_Kendall = 2 / (N (N - 1)) sum_{i<j} sgn(x_i - x_j) sgn(y_i - y_j), the plain tau-a (a tied pair
contributes 0 and the denominator counts every pair); that is what `kendall_tau_a` computes.  The
tie-corrected tau-b is kept as an extra figure.  Every statistic is written from its definition;
pinned against scipy, hand-computed vectors and brute force in tests/test_oracle_correlation.py.
Test infrastructure only.
"""
from typing import Sequence

import numpy as np

from .sr import best_of_n, score_sequences


def pearson(x, y) -> float:
    x = np.asarray(x, np.float64)
    y = np.asarray(y, np.float64)
    dx, dy = x - x.mean(), y - y.mean()
    den = np.sqrt(np.sum(dx * dx) * np.sum(dy * dy))
    return float(np.sum(dx * dy) / den) if den > 0 else float("nan")


def kendall_tau_a(x, y) -> float:
    """Appendix B: 2 / (n (n - 1)) sum_{i<j} sgn(x_i - x_j) sgn(y_i - y_j)."""
    x = np.asarray(x, np.float64)
    y = np.asarray(y, np.float64)
    n = len(x)
    if n < 2:
        return float("nan")
    total = 0
    for i in range(n):
        for j in range(i + 1, n):
            total += int(np.sign(x[i] - x[j])) * int(np.sign(y[i] - y[j]))
    return 2.0 * total / (n * (n - 1))


def kendall_tau_b(x, y) -> float:
    """(concordant - discordant) / sqrt((n0 - n1)(n0 - n2)) over all pairs; n1, n2 count pairs tied in x, y."""
    x = np.asarray(x, np.float64)
    y = np.asarray(y, np.float64)
    n = len(x)
    c = d = tx = ty = 0
    for i in range(n):
        for j in range(i + 1, n):
            sx, sy = np.sign(x[i] - x[j]), np.sign(y[i] - y[j])
            if sx == 0:
                tx += 1
            if sy == 0:
                ty += 1
            if sx * sy > 0:
                c += 1
            elif sx * sy < 0:
                d += 1
    n0 = n * (n - 1) // 2
    den = np.sqrt(float(n0 - tx) * float(n0 - ty))
    return float((c - d) / den) if den > 0 else float("nan")


def partial_final(gen, rm, prompt, N: int, taus: Sequence[int], max_new: int, temperature: float, eos_bias: float,
                  eos_id: int, seed: int):
    """Best-of-N responses; partial rewards at each tau, final rewards, and per-tau (Pearson, Kendall tau-a of
    Appendix B, Kendall tau-b)."""
    _, _, _, seqs, final = best_of_n(gen, rm, prompt, N, max_new, temperature, eos_bias, eos_id, seed)
    partial = {t: score_sequences(rm, prompt, [y[:min(t, len(y))] for y in seqs]) for t in taus}
    stats = {t: (pearson(partial[t], final), kendall_tau_a(partial[t], final), kendall_tau_b(partial[t], final))
             for t in taus}
    return partial, final, stats
