"""CPU oracle for Speculative Rejection (arXiv 2410.20290) -- TEST INFRASTRUCTURE.

A plain, slow, deliberately unoptimised float32 NumPy implementation of what
the GPU path computes: the decoder-only transformer forward (full recompute and
a KV-cached decode), Gumbel-max sampling with Philox4x32-10 noise, the reward
model's scalar score, the cut-off threshold and accepted set of Section 4.2
(Eqs. partial.reward.set, cutoff.threshold, accepted.set), KV page accounting,
Algorithm 1 and plain Best-of-N.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline leg
may import this package.  It shares no code with the CUDA library and imports
nothing from it; both read the same seeded inputs from ``sr_inputs``.

Parity status per function (details in each module header):
  philox.philox4x32_10   pinned: Random123 known-answer vectors
  flog.flog              pinned: error bound against math.log
  sampler.*              pinned: Gumbel-max theorem (chi-square), tie/NaN rules
  select.*               pinned: brute-force sort, the paper's two-response
                         example (Section 4.1), the (1-alpha) size rule
  pool.PagePool          pinned: closed-form first-trigger step
  transformer.*          pinned: torch library routines (SDPA, norms, GELU),
                         KV-cache == recompute, RoPE relative-position property
  sr.*                   pinned: alpha=0 == Best-of-N, SR trajectories are
                         BoN trajectories, tiny-vocabulary brute force
  reward values          parity unpinned in absolute terms: no trained reward
                         model exists, so the paper fixes no value to match.
"""
