"""Time one libsr kernel on synthetic inputs through the C ABI (CUDA events, after warm-up).

  python -m paper_2410_20290_gb300.microbench gemm M N K [epilogue]
  python -m paper_2410_20290_gb300.microbench decode_attn b Hq Hkv dh len [shared_positions]
  python -m paper_2410_20290_gb300.microbench prefill_attn n_seq tau n_pre Hq Hkv dh
  python -m paper_2410_20290_gb300.microbench sample b V
  python -m paper_2410_20290_gb300.microbench decode_gemms M
  python -m paper_2410_20290_gb300.microbench lm_head_sample M V K

Prints one JSON line with the mean launch time and the achieved rate (TFLOP/s or GB/s) of the
algorithmic work.  Operands are sized by the shape given; choose shapes larger than the 129 MB L2
for DRAM-bound figures.  Used as the small-case command of the ncu captures under profiles/.
"""
from __future__ import annotations

import json
import sys

import numpy as np
import torch

from . import binding as sr

DT_F16 = 2


def _time(fn, iters=20, warm=3):
    for _ in range(warm):
        fn()
    torch.cuda.synchronize()
    st = torch.cuda.current_stream()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(st)
    for _ in range(iters):
        fn()
    b.record(st)
    torch.cuda.synchronize()
    return a.elapsed_time(b) / iters


def gemm(M, N, K, epi=0, iters=20):
    g = torch.Generator(device="cuda").manual_seed(0)
    A = torch.randn(M, K, device="cuda", generator=g).to(torch.float16)
    W = torch.randn(N, K, device="cuda", generator=g).to(torch.float16)
    C = torch.zeros(M, N // 2 if epi in (3, 4) else N, device="cuda",
                    dtype=torch.float32 if epi in (0, 1) else torch.float16)
    s = torch.cuda.current_stream().cuda_stream
    ms = _time(lambda: sr.sr_k_gemm(DT_F16, A, W, C, M, N, K, epi, s), iters)
    fl = 2.0 * M * N * K
    by = 2.0 * (M * K + N * K) + C.numel() * C.element_size()
    return dict(kernel="gemm", M=M, N=N, K=K, epi=epi, ms=ms, tflops=fl / ms / 1e9, gbs=by / ms / 1e6)


def decode_attn(b, Hq, Hkv, dh, L, shared=0, iters=20):
    """shared > 0: the first `shared` positions sit in pages common to every candidate (the prompt)."""
    pages = (L + 15) // 16
    sp = shared // 16
    pool = torch.randn(b * (pages - sp) + sp + 1, 2, Hkv, 16, dh, device="cuda").to(torch.float16)
    own = torch.randperm(b * (pages - sp), device="cuda").to(torch.int32).reshape(b, pages - sp) + sp
    pt = torch.cat([torch.arange(sp, device="cuda", dtype=torch.int32).expand(b, sp), own], 1).contiguous()
    ids = torch.arange(b, device="cuda", dtype=torch.int32)
    lens = torch.full((b,), L, device="cuda", dtype=torch.int32)
    q = torch.randn(b, Hq, dh, device="cuda").to(torch.float16)
    out = torch.zeros_like(q)
    s = torch.cuda.current_stream().cuda_stream
    ms = _time(lambda: sr.sr_k_decode_attention(DT_F16, q, pool, pt, pages, ids, lens, b, Hq, Hkv, dh, 0, out, s,
                                                shared_pos=shared), iters)
    by = (b * (L - shared) + shared) * Hkv * dh * 2 * 2 + 2 * q.numel() * 2    # shared positions counted once
    return dict(kernel="decode_attn", b=b, Hq=Hq, Hkv=Hkv, dh=dh, len=L, shared=shared, ms=ms, gbs=by / ms / 1e6)


def prefill_attn(n_seq, tau, n_pre, Hq, Hkv, dh, iters=10):
    rows = n_seq * tau
    q = torch.randn(rows, Hq, dh, device="cuda").to(torch.float16)
    k = torch.randn(rows, Hkv, dh, device="cuda").to(torch.float16)
    v = torch.randn(rows, Hkv, dh, device="cuda").to(torch.float16)
    kp = torch.randn(max(n_pre, 1), Hkv, dh, device="cuda").to(torch.float16)
    vp = torch.randn(max(n_pre, 1), Hkv, dh, device="cuda").to(torch.float16)
    off = torch.arange(0, rows + 1, tau, device="cuda", dtype=torch.int32)
    out = torch.zeros_like(q)
    s = torch.cuda.current_stream().cuda_stream
    ms = _time(lambda: sr.sr_k_prefill_attention(DT_F16, q, k, v, kp, vp, n_pre, off, n_seq, n_pre, Hq, Hkv, dh, 0, out, s),
               iters)
    fl = 4.0 * Hq * dh * n_seq * (tau * n_pre + tau * (tau + 1) / 2)
    return dict(kernel="prefill_attn", n_seq=n_seq, tau=tau, n_pre=n_pre, ms=ms, tflops=fl / ms / 1e9)


def sample(b, V, iters=20):
    logits = torch.randn(b, V, device="cuda")
    ids = torch.arange(b, device="cuda", dtype=torch.int32)
    steps = torch.zeros(b, device="cuda", dtype=torch.int32)
    out = torch.zeros(b, device="cuda", dtype=torch.int32)
    s = torch.cuda.current_stream().cuda_stream
    ms = _time(lambda: sr.sr_k_sample(logits, V, b, V, ids, steps, 7, 1.0, 1.0, 0, out, s), iters)
    return dict(kernel="sample", b=b, V=V, ms=ms, gbs=b * V * 4 / ms / 1e6)


def lm_head_sample(M, V, K, iters=10):
    """The LM head fused with sampling (sr_k_lm_head_sample) against the LM-head GEMM storing fp32 logits followed
    by the sampling pass over them (sr_k_gemm + sr_k_sample)."""
    g = torch.Generator(device="cuda").manual_seed(0)
    x = (torch.randn(M, K, device="cuda", generator=g) / K ** 0.5).to(torch.float16)
    W = torch.randn(V, K, device="cuda", generator=g).to(torch.float16)
    ids = torch.arange(M, device="cuda", dtype=torch.int32)
    lens = torch.full((max(M, 1),), 100, device="cuda", dtype=torch.int32)
    tok = torch.zeros(M, device="cuda", dtype=torch.int32)
    logits = torch.zeros(M, V, device="cuda")
    s = torch.cuda.current_stream().cuda_stream
    fused = _time(lambda: sr.sr_k_lm_head_sample(DT_F16, x, W, M, V, K, ids, lens, 7, 1.0, 1.0, 0, tok, s), iters)
    gemm = _time(lambda: sr.sr_k_gemm(DT_F16, x, W, logits, M, V, K, 0, s), iters)
    samp = _time(lambda: sr.sr_k_sample(logits, V, M, V, ids, lens, 7, 1.0, 1.0, 0, tok, s), iters)
    fl = 2.0 * M * V * K
    return dict(kernel="lm_head_sample", M=M, V=V, K=K, fused_ms=fused, gemm_ms=gemm, sample_ms=samp,
                unfused_ms=gemm + samp, fused_tflops=fl / fused / 1e9)


def decode_gemms(M, iters=5):
    """The five GEMMs of one decode step of the Llama-3-8B-shaped generator at M live rows (QKV, O + residual,
    gate/up + SwiGLU, down + residual, LM head), each launched `iters` times; per shape the mean time and the
    algorithmic bytes of one launch (operands read once, result written once; + the residual read)."""
    shapes = (("qkv", 6144, 4096, 0), ("o", 4096, 4096, 1), ("gate_up", 28672, 4096, 3), ("down", 4096, 14336, 1),
              ("lm_head", 128256, 4096, 0))
    out = []
    for name, N, K, epi in shapes:
        r = gemm(M, N, K, epi, iters)
        out_b = {0: 4 * M * N, 1: 8 * M * N, 3: M * N}[epi]
        r.update(name=name, alg_bytes=2 * (M * K + N * K) + out_b)
        out.append(r)
    return dict(kernel="decode_gemms", M=M, shapes=out)


def main(argv):
    kind, nums = argv[0], [int(x) for x in argv[1:]]
    fn = {"gemm": gemm, "decode_attn": decode_attn, "prefill_attn": prefill_attn, "sample": sample,
          "decode_gemms": decode_gemms, "lm_head_sample": lm_head_sample}[kind]
    print(json.dumps(fn(*nums)), flush=True)


if __name__ == "__main__":
    main(sys.argv[1:])
