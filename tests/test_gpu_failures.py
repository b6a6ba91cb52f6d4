"""Failure paths on the GPU, made on the host or by a bounded wait that runs out -- never by a fault.

* SR_ERR_OOM: a KV pool too small for the prompt tails, and one too small for the next decode step even after
  the round's k is raised as far as it goes; the context stays usable.
* SR_ERR_TIMEOUT: the one-SM tensor-core GEMM's pipeline waits bounded to 1 ns (SR_GEMM_WAIT_NS, read once per
  process, so in a child process): the kernel gives up, drains the copies it issued, sets the error word and
  exits; the library reports the expired wait at its next read of the control words.
"""
import os
import subprocess
import sys

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import sr_inputs as si

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def sr():
    from paper_2410_20290_gb300 import binding
    return binding


def _ctx(sr, w, pages):
    gw, rw = si.random_weights(w.gen, 0, 0), si.random_weights(w.rm, 0, 1)
    kvt = si.kv_bytes_per_token(w.gen)
    return sr.sr_init(w.gen, si.pack_blob(w.gen, gw), w.rm, si.pack_blob(w.rm, rw), pages * 16 * kvt, 16, 0)


def _gen(sr, ctx, w, prompt, N, alpha, kind, taus):
    return sr.sr_generate(ctx, prompt, N, alpha, kind, taus, w.max_new, w.temperature, w.eos_bias, w.eos_id, 3)


def test_pool_too_small_for_prompt_tails(sr):
    """P = 21: one shared page and a 5-position tail page per candidate; 1 + 3 pages cannot admit 8."""
    w = si.WORKLOADS["tiny"].replace(prompt_len=21, max_new=40)
    ctx = _ctx(sr, w, 1 + 3)
    try:
        with pytest.raises(sr.SrError) as e:
            _gen(sr, ctx, w, w.prompt(0), 8, 0.5, si.SCHED_FIXED, (8,))
        assert e.value.status == sr.SR_ERR_OOM
        # the context stays usable: one candidate fits (its tail page and the two pages of positions 32..59)
        toks, score, st = _gen(sr, ctx, w, w.prompt(0), 1, 0.5, si.SCHED_FIXED, (8,))
        assert len(toks) >= 1 and np.isfinite(score)
    finally:
        sr.sr_destroy(ctx)


def test_pool_too_small_for_a_step(sr):
    """P = 16 (no tail): the first decode step opens a page for every candidate.  Fixed schedule, 4 free pages
    for 8 candidates: SR_ERR_OOM before the step.  Memory-triggered with no free page at all: the round raises k
    to b - 1, the rejected candidates hold no private page, so nothing is freed: SR_ERR_OOM."""
    w = si.WORKLOADS["tiny"].replace(prompt_len=16, max_new=40)
    ctx = _ctx(sr, w, 1 + 4)
    try:
        with pytest.raises(sr.SrError) as e:
            _gen(sr, ctx, w, w.prompt(1), 8, 0.5, si.SCHED_FIXED, (20,))
        assert e.value.status == sr.SR_ERR_OOM and "next decode step" in str(e.value)
    finally:
        sr.sr_destroy(ctx)
    ctx = _ctx(sr, w, 1)
    try:
        with pytest.raises(sr.SrError) as e:
            _gen(sr, ctx, w, w.prompt(1), 8, 0.5, si.SCHED_POOL_FULL, ())
        assert e.value.status == sr.SR_ERR_OOM
    finally:
        sr.sr_destroy(ctx)


CHILD = r"""
import sys
sys.path.insert(0, {root!r})
import sr_inputs as si
from paper_2410_20290_gb300 import binding as sr
w = si.WORKLOADS["gpt2"].replace(N=4, max_new=6, taus=(3,))
gw, rw = si.random_weights(w.gen, 0, 0), si.random_weights(w.rm, 0, 1)
ctx = sr.sr_init(w.gen, si.pack_blob(w.gen, gw), w.rm, si.pack_blob(w.rm, rw), 0, 16, 0)
try:
    sr.sr_generate(ctx, w.prompt(0), w.N, w.alpha, w.sched_kind, w.taus, w.max_new, w.temperature, w.eos_bias,
                   w.eos_id, 0)
    print("NO ERROR")
except sr.SrError as e:
    print("STATUS", e.status, str(e))
"""


def test_gemm_wait_expiry_reports_timeout():
    env = dict(os.environ, SR_GEMM_WAIT_NS="1", SR_GEMM_SKINNY="0", SR_GEMM_PAIR="0")
    r = subprocess.run([sys.executable, "-c", CHILD.format(root=ROOT)], cwd=ROOT, env=env, capture_output=True,
                       text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-2000:]
    from paper_2410_20290_gb300 import binding as b
    assert f"STATUS {b.SR_ERR_TIMEOUT}" in r.stdout and "wait expired" in r.stdout, r.stdout[-2000:]
