"""Cut-off threshold and accepted set of one rejection round (oracle side).

Section 4.2: the partial rewards R_partial = {s(Y_k^{<=tau_k}) : k = 1..b}
(Eq. partial.reward.set), the cut-off r_cut = q_alpha(R_partial), the alpha-th
lower quantile (Eq. cutoff.threshold), and the accepted set
I_accepted = {k : s(Y_k^{<=tau_k}) >= r_cut} (Eq. accepted.set).

Reading of the quantile (the paper gives no interpolation rule): the order
statistic  r_cut = sort_ascending(R)[k],  k = min(floor(alpha * b), b - 1),
0-based.  floor(alpha * b) is taken on the exact product of the float32 alpha
and the integer b (exact in float64).  So alpha = 0 keeps everyone (Best-of-N,
Section 5.1), and with distinct rewards exactly b - floor(alpha b) candidates
survive, the "top (1 - alpha) proportion".  Ties at r_cut are all accepted
(the ">=" of Eq. accepted.set).

Float order: rewards are compared through an order-preserving map to uint32
(-0.0 is folded onto +0.0; NaN orders as -inf), so the selection is exact.

Pinned in tests/test_oracle_select.py: brute force over sorted vectors, the
two-response example of Section 4.1 (partial rewards 2.92 and -1.88), the size
rule, ties and the alpha = 0 / alpha = 1 ends.
"""
import numpy as np


def float_keys(r) -> np.ndarray:
    r = np.asarray(r, dtype=np.float32).copy()
    r[np.isnan(r)] = -np.inf
    r[r == 0] = 0.0                      # fold -0.0 onto +0.0
    u = r.view(np.uint32)
    neg = (u >> np.uint32(31)) == 1
    return np.where(neg, ~u, u | np.uint32(0x80000000)).astype(np.uint32)


def key_to_float(k: int) -> float:
    k = np.uint32(k)
    u = np.uint32(k & np.uint32(0x7FFFFFFF)) if (k >> np.uint32(31)) else np.uint32(~k)
    return float(np.array([u], dtype=np.uint32).view(np.float32)[0])


def cut_index(alpha: float, b: int) -> int:
    k = int(np.floor(float(np.float32(alpha)) * b))
    return min(max(k, 0), b - 1)


def r_cut(rewards, alpha: float) -> float:
    """q_alpha(R): the k-th smallest reward, k = min(floor(alpha b), b - 1)."""
    keys = float_keys(rewards)
    k = cut_index(alpha, len(keys))
    return key_to_float(int(np.sort(keys)[k]))


def accepted_mask(rewards, threshold: float) -> np.ndarray:
    """[s_k >= r_cut] for each k, compared in the same exact key order."""
    keys = float_keys(rewards)
    return keys >= float_keys([threshold])[0]


def select_round(rewards, alpha: float, k_override: int = -1):
    """(r_cut, accepted mask, k) for one round; ``k_override`` forces the order-statistic index."""
    keys = float_keys(rewards)
    b = len(keys)
    k = cut_index(alpha, b) if k_override < 0 else min(k_override, b - 1)
    kc = int(np.sort(keys)[k])
    return key_to_float(kc), keys >= np.uint32(kc), k
