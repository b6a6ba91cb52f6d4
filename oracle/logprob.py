"""Self-likelihood reward of Section 5.3 (oracle side).

Section 5.3 scores a response with the generator itself instead of a reward model:
    s(Y) = (1 / len(Y)) ln p(Y | X) = (1 / len(Y)) sum_t ln p(y_t | X, y_<t),
the mean log-probability of its tokens under the model p.  Readings taken where the section is
silent (each also holds on the GPU):
  * p is the model's own distribution: softmax of the raw logits at temperature 1, without the EOS
    bias the sampler may add (both are sampling devices, not part of p).
  * ln p(v) = logit_v - ln sum_u exp(logit_u); NaN logits count as -inf (as in the sampler).
  * A partial response Y^{<=tau} is scored the same way over its tau tokens (Eq.
    partial.reward.set with this s); a completed response over all its tokens, EOS included.
Computed in float64 from the float32 logits.

Test infrastructure only: the product path never imports this package.
"""
import numpy as np


def token_logprob(logits, tok: int) -> float:
    """ln softmax(logits)[tok] with the log-sum-exp taken about the maximum, in float64."""
    l = np.asarray(logits, dtype=np.float64)
    l = np.where(np.isnan(l), -np.inf, l)
    m = np.max(l)
    if m == -np.inf:
        return float("-inf")
    lse = m + np.log(np.sum(np.exp(l - m)))
    return float(l[int(tok)] - lse)


def mean_logprob(logprob_sum: float, n_tokens: int) -> float:
    """s(Y) for a response of n_tokens tokens whose log-probabilities sum to logprob_sum."""
    return logprob_sum / n_tokens
