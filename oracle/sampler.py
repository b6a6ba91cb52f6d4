"""Gumbel-max sampling of the next token (oracle side).

Auto-regressive sampling draws y^{k+1} ~ p(. | X, y^{<=k}) (Section 3,
Eq. auto-regressive).  The oracle realises that draw with the Gumbel-max trick:
    y = argmax_v  z_v,   z_v = (logit_v + b * [v == eos]) * (1/T) + g_v,
    g_v = -ln(-ln u_v),  u_v uniform on (0, 1),
which samples exactly from softmax((logit + b e_eos) / T).  The EOS bias b is
added before temperature scaling.  Noise is keyed, not drawn from a stream, so
that a candidate's trajectory does not depend on which batch slot it occupies:
    key     = (seed mod 2^32, seed div 2^32)
    counter = (v div 4, orig_id, step, 0), word v mod 4 of Philox4x32-10
    u_v     = ((word >> 9) + 1/2) * 2^-23        (exact in float32, in (0, 1))
``step`` is the 0-based index of the generated token and ``orig_id`` the
candidate's index in 0..N-1.  Ties in z go to the lowest v; NaN logits count
as -inf.  An EOS id outside [0, V) means the vocabulary has no EOS.  All arithmetic is float32 with one rounding per operation, in the
order written here.

Pinned by tests/test_oracle_sampler.py (Gumbel-max frequencies vs the softmax,
chi-square; tie and NaN rules; Philox known-answer vectors).
"""
import numpy as np

from .flog import flog
from .philox import philox4x32_10

F = np.float32


def gumbel_noise(seed: int, orig_id: int, step: int, vocab: int) -> np.ndarray:
    v = np.arange(vocab, dtype=np.uint32)
    k0 = seed & 0xFFFFFFFF
    k1 = (seed >> 32) & 0xFFFFFFFF
    words = philox4x32_10(v >> np.uint32(2), np.uint32(orig_id), np.uint32(step), np.uint32(0), k0, k1)
    sel = (v & np.uint32(3)).astype(np.int64)
    x = np.choose(sel, words).astype(np.uint32)
    u = ((x >> np.uint32(9)).astype(np.float32) + F(0.5)) * F(2.0 ** -23)
    l1 = flog(u)            # ln u < 0
    l2 = flog(-l1)          # ln(-ln u)
    return (-l2).astype(np.float32)


def perturbed_logits(logits: np.ndarray, seed: int, orig_id: int, step: int, temperature: float,
                     eos_bias: float, eos_id: int) -> np.ndarray:
    logits = np.asarray(logits, dtype=np.float32)
    V = logits.shape[-1]
    inv_t = F(1) / F(temperature)
    adj = logits.copy()
    if 0 <= eos_id < V:
        adj[eos_id] = adj[eos_id] + F(eos_bias)
    adj = np.where(np.isnan(adj), F(-np.inf), adj).astype(np.float32)
    z = adj * inv_t
    return (z + gumbel_noise(seed, orig_id, step, V)).astype(np.float32)


def sample_token(logits: np.ndarray, seed: int, orig_id: int, step: int, temperature: float,
                 eos_bias: float, eos_id: int) -> int:
    z = perturbed_logits(logits, seed, orig_id, step, temperature, eos_bias, eos_id)
    return int(np.argmax(z))      # first maximum: ties go to the lowest id


def top2_gap(logits, seed, orig_id, step, temperature, eos_bias, eos_id) -> float:
    """Gap between the largest and second-largest perturbed logit (how close a draw was to flipping)."""
    z = perturbed_logits(logits, seed, orig_id, step, temperature, eos_bias, eos_id)
    a = np.partition(z, -2)[-2:]
    return float(a[1] - a[0])
