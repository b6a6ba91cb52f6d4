"""Algorithm 1 (Speculative Rejection) and plain Best-of-N, oracle side.

Algorithm 1 (Section 4.2): start b = b_init candidates; while b > 0, generate
until the decision token tau (tau_k = min(tau, l_k) for candidates that hit EOS
earlier), score every candidate of the batch with the reward model on prompt ++
partial response (Eq. partial.reward.set), take r_cut = q_alpha (Eq.
cutoff.threshold), keep I_accepted (Eq. accepted.set), add completed
sequences to I and shrink the batch; return argmax_{k in I} s(Y_k) (Eq.
output.SBoN).  Best-of-N (Section 3) is the same procedure with no rejection.

Readings taken where the paper is silent (each also holds on the GPU):
  * b_init is the caller's N.
  * Decision schedule: either fixed decision points (generated-token counts)
    or memory-triggered: before a decode step, when the free pages cannot give
    every live candidate the page it needs, a round runs at that step.
  * The batch of a round is every candidate that survived the previous round:
    the live ones (tau_k = tokens generated so far) and those that completed
    since (tau_k = l_k; partial reward = final reward).  Completed candidates
    join I whatever the cut says (they were not halted in the middle) and
    never continue; b <- |accepted and not completed|.
  * A candidate completes on EOS (kept as its last token) or at max_new
    tokens.  Its generator pages are released when it completes.
  * Memory-triggered rounds with too few pages freed by floor(alpha b)
    rejections raise the order-statistic index k to the smallest value whose
    rejections make room for the next step.
  * alpha = 0 with a memory trigger is Best-of-N run in pool-sized waves
    (every candidate is generated to the end; a wave holds as many candidates
    as the pool can take to max_new).
  * When b reaches 0, completed candidates not yet scored are scored; ties in
    the final argmax go to the lowest candidate id.
Token ``step`` g is the 0-based index of the generated token; token g is sampled
from the logits at position P + g - 1 (the prompt's last position for g = 0).

Pinned in tests/test_oracle_sr.py: alpha = 0 returns exactly what the plain
Best-of-N loop below returns; every candidate's tokens equal its Best-of-N
trajectory (noise is keyed on candidate id and step); tiny-vocabulary brute
force of the sampled path and of the final argmax.
"""
from __future__ import annotations

import dataclasses
from typing import Callable, List, Optional

import numpy as np

import sr_inputs as si
from .pool import PagePool, pool_pages, private_pages_full
from .logprob import mean_logprob, token_logprob
from .sampler import sample_token
from .select import cut_index, float_keys, select_round
from .transformer import Decoder, Transformer

LIVE, PENDING, DONE, REJECTED = 0, 1, 2, 3
PAGE = 16


@dataclasses.dataclass
class Round:
    step: int                 # generated tokens of the live candidates when the round ran
    batch: List[int]          # candidate ids in the round's batch, ascending
    rewards: np.ndarray       # partial rewards, aligned with batch
    k: int                    # order-statistic index used
    k_raised: bool
    r_cut: float
    accepted: np.ndarray      # bool mask aligned with batch


@dataclasses.dataclass
class Result:
    best_id: int
    tokens: List[int]
    score: float
    rounds: List[Round]
    status: List[int]
    lengths: List[int]
    final_reward: np.ndarray
    all_tokens: List[List[int]]
    page_tables: List[List[int]]
    free_stack: List[int]
    gen_tokens: int
    rm_tokens: int


def score_sequences(rm: Transformer, prompt, seqs: List[List[int]]) -> np.ndarray:
    """s(X ++ Y) for each response Y: final-normed hidden of the last position dotted with the score head."""
    out = np.zeros(len(seqs), np.float32)
    by_len = {}
    for i, y in enumerate(seqs):
        by_len.setdefault(len(y), []).append(i)
    for L, idx in by_len.items():
        ids = np.array([list(prompt) + list(seqs[i]) for i in idx])
        hn = rm.forward(ids)
        out[idx] = rm.score(hn[:, -1])
    return out


class SpeculativeRejection:
    def __init__(self, gen: Transformer, rm: Transformer, prompt, N: int, alpha: float, sched_kind: int,
                 taus=(), max_new: int = 64, temperature: float = 1.0, eos_bias: float = 0.0, eos_id: int = 0,
                 seed: int = 0, n_pool_pages: int = 0,
                 token_hook: Optional[Callable] = None, accept_hook: Optional[Callable] = None,
                 reward: str = "model"):
        if reward not in ("model", "logprob"):
            raise ValueError("reward must be 'model' or 'logprob'")
        self.reward = reward
        self.gen, self.rm = gen, rm
        self.prompt = [int(t) for t in prompt]
        self.N, self.alpha = N, float(np.float32(alpha))
        self.sched_kind, self.taus = sched_kind, tuple(taus)
        self.max_new, self.T, self.eos_bias, self.eos_id, self.seed = max_new, temperature, eos_bias, eos_id, seed
        P = len(self.prompt)
        if n_pool_pages <= 0:
            n_pool_pages = P // PAGE + N * private_pages_full(P, max_new)
        self.pool = PagePool(n_pool_pages)
        self.token_hook, self.accept_hook = token_hook, accept_hook

    # -- helpers ---------------------------------------------------------------
    def _release(self, i):
        """Return candidate i's private pages, ascending page index."""
        P = len(self.prompt)
        priv = self.page_table[i][P // PAGE:]
        self.pool.push(priv)
        self.page_table[i] = self.page_table[i][:P // PAGE]

    def _complete_if_done(self, i):
        y = self.tokens[i]
        if y[-1] == self.eos_id or len(y) == self.max_new:
            self.status[i] = PENDING
            self._release(i)

    def _sample(self, i, logits, g):
        tok = sample_token(logits, self.seed, i, g, self.T, self.eos_bias, self.eos_id)
        if self.token_hook is not None:
            tok = int(self.token_hook(i, g, tok, logits))
        self.tokens[i].append(tok)
        self.lp_sum[i] += token_logprob(logits, tok)
        self.gen_tokens += 1

    def _score(self, ids):
        if self.reward == "logprob":  # Section 5.3: mean log-probability under the generator itself
            return np.array([mean_logprob(self.lp_sum[i], len(self.tokens[i])) for i in ids], np.float32)
        r = score_sequences(self.rm, self.prompt, [self.tokens[i] for i in ids])
        self.rm_tokens += sum(len(self.tokens[i]) for i in ids)
        return r

    # -- one rejection round (Eqs. partial.reward.set, cutoff.threshold, accepted.set)
    def _round(self, g, wave, need_pages: bool):
        batch = [i for i in wave if self.status[i] in (LIVE, PENDING)]
        rewards = self._score(batch)
        b = len(batch)
        k0 = cut_index(self.alpha, b)
        k = k0
        if self.sched_kind == si.SCHED_POOL_FULL and need_pages:
            P = len(self.prompt)
            while True:
                _, mask, _ = select_round(rewards, self.alpha, k)
                live_acc = sum(1 for i, a in zip(batch, mask) if a and self.status[i] == LIVE)
                freed = sum(len(self.page_table[i]) - P // PAGE
                            for i, a in zip(batch, mask) if (not a) and self.status[i] == LIVE)
                if live_acc <= self.pool.n_free + freed or k == b - 1:
                    break
                k += 1
        rc, mask, k = select_round(rewards, self.alpha, k)
        if self.accept_hook is not None:
            mask = np.asarray(self.accept_hook(len(self.rounds), batch, rewards, mask), dtype=bool)
        for i, a, r in zip(batch, mask, rewards):
            if self.status[i] == PENDING:
                self.status[i] = DONE
                self.final_reward[i] = r
            elif not a:
                self.status[i] = REJECTED
                self._release(i)
        self.rounds.append(Round(g, batch, rewards, k, k != k0, rc, np.asarray(mask, dtype=bool)))
        self.snapshots.append(self._snapshot(g))

    def _snapshot(self, g):
        """Copy of the bookkeeping state (for comparisons; no effect on the run)."""
        return dict(step=g, status=list(self.status), lengths=[len(t) for t in self.tokens],
                    page_tables=[list(p) for p in self.page_table], free_stack=list(self.pool.stack))

    # -- Algorithm 1 ----------------------------------------------------------------
    def run(self) -> Result:
        P, N = len(self.prompt), self.N
        self.status = [LIVE] * N
        self.tokens: List[List[int]] = [[] for _ in range(N)]
        self.lp_sum = [0.0] * N
        self.final_reward = np.full(N, np.nan, np.float32)
        self.rounds: List[Round] = []
        self.snapshots: List[dict] = []
        self.gen_tokens = 0
        self.rm_tokens = P if self.reward == "model" else 0
        shared = [self.pool.pop() for _ in range(P // PAGE)]
        self.page_table = [list(shared) for _ in range(N)]
        dec = Decoder(self.gen, N, P + self.max_new)
        hn = dec.prefill(self.prompt, np.arange(N))
        logits0 = self.gen.logits(hn[-1])

        if self.sched_kind == si.SCHED_POOL_FULL and self.alpha == 0.0:
            per = private_pages_full(P, self.max_new)
            waves, start = [], 0
            while start < N:
                w = N - start if per == 0 else min(N - start, self.pool.n_free // per)
                if w <= 0:
                    raise MemoryError("KV pool cannot hold one candidate to max_new")
                waves.append(list(range(start, start + w)))
                start += w
        else:
            waves = [list(range(N))]

        for wave in waves:
            if P % PAGE:
                if self.pool.n_free < len(wave):
                    raise MemoryError("KV pool cannot hold the prompt tails")
                for i in wave:
                    self.page_table[i].append(self.pool.pop())
            for i in wave:
                self._sample(i, logits0, 0)
                self._complete_if_done(i)
            g = 1
            while True:
                live = [i for i in wave if self.status[i] == LIVE]
                if not live:
                    break
                need = (P + g - 1) % PAGE == 0
                if self.alpha > 0.0:
                    trig = (g in self.taus) if self.sched_kind == si.SCHED_FIXED else \
                           (need and self.pool.n_free < len(live))
                    if trig:
                        self._round(g, wave, need)
                        live = [i for i in wave if self.status[i] == LIVE]
                        if not live:
                            break
                if need:
                    if self.pool.n_free < len(live):
                        raise MemoryError("KV pool exhausted")
                    for i in live:
                        self.page_table[i].append(self.pool.pop())
                h = dec.step(live, [self.tokens[i][g - 1] for i in live], P + g - 1)
                logits = self.gen.logits(h)
                for j, i in enumerate(live):
                    self._sample(i, logits[j], g)
                    self._complete_if_done(i)
                g += 1
            pend = [i for i in wave if self.status[i] == PENDING]
            if pend:
                r = self._score(pend)
                for i, v in zip(pend, r):
                    self.status[i] = DONE
                    self.final_reward[i] = v

        done = [i for i in range(N) if self.status[i] == DONE]
        keys = float_keys(self.final_reward[done])
        best = done[int(np.argmax(keys))]          # first maximum = lowest id among ties
        return Result(best, list(self.tokens[best]), float(self.final_reward[best]), self.rounds,
                      list(self.status), [len(t) for t in self.tokens], self.final_reward.copy(),
                      [list(t) for t in self.tokens], [list(p) for p in self.page_table],
                      list(self.pool.stack), self.gen_tokens, self.rm_tokens)


def run_workload(w: si.Workload, gen_w: dict, rm_w: dict, prompt, seed: int = 0, alpha=None, **kw) -> Result:
    gen, rm = Transformer(w.gen, gen_w), Transformer(w.rm, rm_w)
    n_pages = pool_pages(w.pool_bytes, si.kv_bytes_per_token(w.gen)) if w.pool_bytes else 0
    sr = SpeculativeRejection(gen, rm, prompt, w.N, w.alpha if alpha is None else alpha, w.sched_kind, w.taus,
                              w.max_new, w.temperature, w.eos_bias, w.eos_id, seed, n_pages, **kw)
    return sr.run()


def best_of_n(gen: Transformer, rm: Transformer, prompt, N, max_new, temperature, eos_bias, eos_id, seed,
              reward: str = "model"):
    """Plain Best-of-N (Section 3): N independent responses, each decoded on its own, argmax of s
    (s = the reward model, or with reward="logprob" the mean log-probability of Section 5.3)."""
    P = len(prompt)
    seqs, rewards, lps = [], [], []
    for i in range(N):
        dec = Decoder(gen, 1, P + max_new)
        hn = dec.prefill(prompt, [0])
        logits = gen.logits(hn[-1])
        y, lp = [], 0.0
        for g in range(max_new):
            if g > 0:
                logits = gen.logits(dec.step([0], [y[-1]], P + g - 1)[0])
            y.append(sample_token(logits, seed, i, g, temperature, eos_bias, eos_id))
            lp += token_logprob(logits, y[-1])
            if y[-1] == eos_id:
                break
        seqs.append(y)
        lps.append(mean_logprob(lp, len(y)))
    rewards = score_sequences(rm, prompt, seqs) if reward == "model" else np.array(lps, np.float32)
    best = int(np.argmax(float_keys(rewards)))
    return best, seqs[best], float(rewards[best]), seqs, rewards
