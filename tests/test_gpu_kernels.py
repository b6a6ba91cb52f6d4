"""GPU parity of the individual kernels through the C ABI.

Integer results (sampled tokens, r_cut and accepted masks) must equal the oracle bit for bit on
identical inputs; GEMMs are compared with a plain PyTorch fp32 matmul of the same bf16 / fp32
operands; attention with the oracle's float64-accumulated attention on the same K/V values.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import sr_inputs as si
from oracle import sampler as osamp
from oracle import select as osel
from oracle import transformer as otr

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sr():
    from paper_2410_20290_gb300 import binding
    return binding


def dev(x, dtype=None):
    t = torch.from_numpy(np.ascontiguousarray(x)).cuda()
    return t if dtype is None else t.to(dtype)


# ------------------------------------------------------------------------------------------ sample
@pytest.mark.parametrize("V,T,bias,eos", [(512, 1.0, 0.0, 0), (32000, 0.8, 2.0, 0), (1000, 1.3, -1.0, 999),
                                          (128256, 1.0, 1.0, 0), (37, 0.5, 3.0, -1)])
def test_sample_bit_exact(sr, V, T, bias, eos):
    rng = np.random.default_rng(V)
    b = 9
    logits = (rng.standard_normal((b, V)) * 1.3).astype(np.float32)
    logits[0, :5] = np.nan
    ids = rng.integers(0, 4096, b).astype(np.int32)
    steps = rng.integers(0, 3000, b).astype(np.int32)
    seed = int(rng.integers(0, 2 ** 63))
    out = torch.zeros(b, dtype=torch.int32, device="cuda")
    sr.sr_k_sample(dev(logits), V, b, V, dev(ids), dev(steps), seed, T, bias, eos, out)
    got = out.cpu().numpy()
    want = [osamp.sample_token(logits[r], seed, int(ids[r]), int(steps[r]), T, bias, eos) for r in range(b)]
    assert got.tolist() == want
    # broadcast row (ld = 0), as used for token 0 of every candidate
    sr.sr_k_sample(dev(logits[1]), 0, b, V, dev(ids), dev(steps), seed, T, bias, eos, out)
    want = [osamp.sample_token(logits[1], seed, int(ids[r]), int(steps[r]), T, bias, eos) for r in range(b)]
    assert out.cpu().numpy().tolist() == want


@pytest.mark.parametrize("kind", ["wide", "ties", "large", "sharp"])
def test_sample_skip_test_keeps_decisions(sr, kind):
    """The kernel takes the logarithms only for ids that can still win (an exact bound on the uniform); the
    decisions must equal the oracle's full Gumbel-max on spreads where most ids are skipped (wide), on exact ties
    of the top logits (ties: lowest id wins), at large magnitudes (the margin's ulp term) and on a peaked row."""
    rng = np.random.default_rng({"wide": 1, "ties": 2, "large": 3, "sharp": 4}[kind])
    b, V = 48, 128256
    if kind == "wide":
        logits = rng.standard_normal((b, V)) * 8.0
    elif kind == "ties":
        logits = np.round(rng.standard_normal((b, V)) * 2.0)          # many equal values, top ones tied
    elif kind == "large":
        logits = 2.0e4 + rng.standard_normal((b, V)) * 3.0
    else:
        logits = rng.standard_normal((b, V))
        logits[:, rng.integers(0, V, b)] += 12.0
    logits = logits.astype(np.float32)
    ids = rng.integers(0, 4096, b).astype(np.int32)
    steps = rng.integers(0, 3000, b).astype(np.int32)
    seed = int(rng.integers(0, 2 ** 63))
    out = torch.zeros(b, dtype=torch.int32, device="cuda")
    for T in (1.0, 0.7):
        sr.sr_k_sample(dev(logits), V, b, V, dev(ids), dev(steps), seed, T, 1.0, 0, out)
        want = [osamp.sample_token(logits[r], seed, int(ids[r]), int(steps[r]), T, 1.0, 0) for r in range(b)]
        assert out.cpu().numpy().tolist() == want


def test_gumbel_noise_bit_exact(sr):
    """With all logits equal to zero and T = 1 the argmax is the argmax of the noise itself."""
    V, b = 4099, 64
    ids = np.arange(b, dtype=np.int32)
    steps = (np.arange(b) * 7).astype(np.int32)
    out = torch.zeros(b, dtype=torch.int32, device="cuda")
    sr.sr_k_sample(torch.zeros(V, device="cuda"), 0, b, V, dev(ids), dev(steps), 12345, 1.0, 0.0, -1, out)
    want = [int(np.argmax(osamp.gumbel_noise(12345, i, int(steps[i]), V))) for i in range(b)]
    assert out.cpu().numpy().tolist() == want


# ------------------------------------------------------------------------------------------ r_cut
@pytest.mark.parametrize("b", [1, 2, 3, 64, 1000, 1024, 4096])
def test_rcut_bit_exact(sr, b):
    rng = np.random.default_rng(b)
    for trial in range(6):
        if trial % 3 == 0:
            r = rng.integers(-4, 5, b).astype(np.float32)
        elif trial % 3 == 1:
            r = rng.standard_normal(b).astype(np.float32)
            r[: b // 3] = -0.0
        else:
            r = (rng.standard_normal(b) * 10.0 ** rng.uniform(-20, 20, b)).astype(np.float32)
        for alpha in (0.0, 0.3, 0.5, 0.7, 0.999, 1.0):
            rc = torch.zeros(1, device="cuda")
            mask = torch.zeros(b, dtype=torch.uint8, device="cuda")
            sr.sr_k_rcut(dev(r), b, alpha, -1, rc, mask)
            want_rc, want_mask, _ = osel.select_round(r, alpha)
            assert np.float32(rc.item()) == np.float32(want_rc) or (want_rc == 0 and rc.item() == 0)
            assert mask.cpu().numpy().astype(bool).tolist() == want_mask.tolist()


def test_rcut_paper_example(sr):
    r = np.array([2.92, -1.88], np.float32)
    rc = torch.zeros(1, device="cuda")
    mask = torch.zeros(2, dtype=torch.uint8, device="cuda")
    sr.sr_k_rcut(dev(r), 2, 0.5, -1, rc, mask)
    assert np.float32(rc.item()) == np.float32(2.92) and mask.cpu().tolist() == [1, 0]


# ------------------------------------------------------------------------------------------ GEMM
def _bf16(x):
    return torch.from_numpy(x).to(torch.bfloat16)


T16 = {si.DT_BF16: torch.bfloat16, si.DT_F16: torch.float16}


@pytest.mark.parametrize("dt", [si.DT_F16, si.DT_BF16])
# shapes cover all three N-tile widths the launcher picks (64: small tile counts, 128: e.g. 308 x 6144,
# 256: e.g. 1024 x 4096) and ragged M, N and K tails
@pytest.mark.parametrize("M,N,K", [(1, 256, 64), (7, 512, 128), (130, 2304, 768), (300, 288, 1000), (257, 96, 520),
                                   (1024, 4096, 4096), (1, 32000, 768), (2048, 512, 64), (1024, 6144, 520),
                                   (308, 28672, 256), (308, 6144, 512),
                                   # with SR_GEMM_STREAMK=1: shares cut tiles mid-k (48 tiles x 32 k-blocks)
                                   (300, 4096, 2000),
                                   # more M tiles than one raster group (16 M tiles), ragged last group
                                   (4500, 1024, 256)])
def test_gemm_tc_fp32_out(sr, dt, M, N, K):
    g = torch.Generator().manual_seed(M * 7 + N + K)
    A = torch.randn(M, K, generator=g).to(T16[dt])
    W = torch.randn(N, K, generator=g).to(T16[dt])
    ref = A.float() @ W.float().T
    C = torch.zeros(M, N, device="cuda")
    sr.sr_k_gemm(dt, A.cuda(), W.cuda(), C, M, N, K, 0)
    torch.testing.assert_close(C.cpu(), ref, rtol=2e-4, atol=2e-4 * np.sqrt(K))
    # epilogue 1: accumulate into the fp32 output (residual add)
    base = torch.randn(M, N, generator=g)
    C = base.cuda().clone()
    sr.sr_k_gemm(dt, A.cuda(), W.cuda(), C, M, N, K, 1)
    torch.testing.assert_close(C.cpu(), base + ref, rtol=2e-4, atol=2e-4 * np.sqrt(K))


@pytest.mark.parametrize("dt", [si.DT_F16, si.DT_BF16])
@pytest.mark.parametrize("epi", [2, 3, 4, 5])
@pytest.mark.parametrize("M,N,K", [(5, 256, 64), (200, 1024, 512), (129, 512, 4096), (308, 6144, 512),
                                   (1024, 4096, 64), (308, 2048, 4096), (4500, 1024, 256)])
def test_gemm_tc_epilogues(sr, dt, epi, M, N, K):
    g = torch.Generator().manual_seed(epi * 1000 + M)
    A = (torch.randn(M, K, generator=g) / np.sqrt(K)).to(T16[dt])
    W = torch.randn(N, K, generator=g).to(T16[dt])
    acc = A.float() @ W.float().T
    if epi in (3, 4):
        blk = acc.reshape(M, N // 32, 2, 16)
        gate, up = blk[:, :, 0, :].reshape(M, N // 2), blk[:, :, 1, :].reshape(M, N // 2)
        act = torch.nn.functional.silu(gate) if epi == 3 else torch.nn.functional.gelu(gate, approximate="tanh")
        ref = act * up
        C = torch.zeros(M, N // 2, dtype=T16[dt], device="cuda")
    else:
        ref = acc if epi == 2 else torch.nn.functional.gelu(acc, approximate="tanh")
        C = torch.zeros(M, N, dtype=T16[dt], device="cuda")
    sr.sr_k_gemm(dt, A.cuda(), W.cuda(), C, M, N, K, epi)
    tol = 1.6e-2 if dt == si.DT_BF16 else 2e-3
    torch.testing.assert_close(C.float().cpu(), ref.to(T16[dt]).float(), rtol=tol, atol=1e-3)


@pytest.mark.parametrize("M,N,K,epi", [(300, 4096, 2000, 0), (308, 28672, 4096, 3), (1024, 6144, 4096, 0),
                                       (308, 4096, 14336, 1)])
def test_gemm_tc_repeatable(sr, M, N, K, epi):
    """Decode shapes, three calls: the same bits every time.  Split-K partials (the skinny kernel) and stream-K
    shares (SR_GEMM_STREAMK=1) are summed in k order, not in the order the CTAs finish."""
    g = torch.Generator().manual_seed(M + N + K)
    A = (torch.randn(M, K, generator=g) / np.sqrt(K)).half().cuda()
    W = torch.randn(N, K, generator=g).half().cuda()
    shape = (M, N // 2) if epi == 3 else (M, N)
    base = torch.randn(*shape, generator=g).cuda()
    outs = []
    for _ in range(3):
        C = base.clone() if epi == 1 else torch.zeros(*shape, device="cuda", dtype=torch.float16 if epi == 3 else torch.float32)
        sr.sr_k_gemm(si.DT_F16, A, W, C, M, N, K, epi)
        outs.append(C.cpu())
    assert torch.equal(outs[0], outs[1]) and torch.equal(outs[0], outs[2])


@pytest.mark.parametrize("M,N,K", [(1, 64, 16), (33, 200, 77), (128, 512, 128)])
def test_gemm_f32(sr, M, N, K):
    g = torch.Generator().manual_seed(M + N + K)
    A = torch.randn(M, K, generator=g)
    W = torch.randn(N, K, generator=g)
    C = torch.zeros(M, N, device="cuda")
    sr.sr_k_gemm(si.DT_F32, A.cuda(), W.cuda(), C, M, N, K, 0)
    torch.testing.assert_close(C.cpu(), A @ W.T, rtol=1e-5, atol=1e-5 * np.sqrt(K))


# ------------------------------------------------------------------------------------------ attention
def _round16(x, dt=si.DT_F16):
    return torch.from_numpy(x).to(T16[dt]).float().numpy()


@pytest.mark.parametrize("dt,Hq,Hkv,dh,window,lens,shared", [
    (si.DT_F16, 32, 8, 128, 0, [1, 15, 16, 17, 300, 511, 512, 513, 1100, 2000], 0),
    (si.DT_F16, 12, 12, 64, 0, [5, 129, 700], 0),
    (si.DT_F16, 32, 8, 128, 100, [50, 100, 101, 900], 0),
    (si.DT_F16, 16, 2, 128, 0, [33, 64, 600], 0),
    (si.DT_F16, 4, 4, 32, 0, [1, 16, 33, 80], 0),
    (si.DT_BF16, 32, 8, 128, 0, [7, 300, 1300], 0),
    (si.DT_F32, 4, 4, 32, 0, [1, 16, 33, 80], 0),
    # shared prompt pages: the tensor-core prefix pass plus the suffix splits
    (si.DT_F16, 32, 8, 128, 0, [289, 290, 300, 511, 800, 805, 1300] * 10, 288),
    (si.DT_F16, 12, 12, 64, 0, [129, 130, 700], 128),
    (si.DT_F16, 32, 8, 128, 40, [300, 301, 305], 256),
    (si.DT_F16, 32, 8, 128, 0, [17, 18, 600], 16),
    (si.DT_BF16, 32, 8, 128, 0, [300, 900], 272),
    # suffixes of at most 8 pages run one warp per (kv head, slot); 2 kv heads leave two warps idle
    (si.DT_F16, 16, 2, 128, 0, [289, 300, 310, 390], 288),
    (si.DT_F16, 32, 8, 128, 0, [257, 258, 270, 300, 384] * 40, 256),
    # head_dim 128 with 8 kv heads runs the streaming kernel: fewer pages than SMs, group sizes 1, 2 and 8,
    # and a few hundred rows whose pages the per-SM shares cut at many places
    (si.DT_F16, 8, 8, 128, 0, [5, 17, 40], 0),
    (si.DT_F16, 16, 8, 128, 0, [100, 700, 1500], 0),
    (si.DT_F16, 64, 8, 128, 0, [64, 513, 1025], 0),
    (si.DT_F16, 8, 8, 128, 0, [290 + (13 * i) % 200 for i in range(300)], 288),
    (si.DT_BF16, 32, 8, 128, 64, [300 + (3 * i) % 400 for i in range(200)], 128),
])
def test_decode_attention(sr, dt, Hq, Hkv, dh, window, lens, shared):
    rng = np.random.default_rng(dh + len(lens))
    b = len(lens)
    max_pages = max(lens) // 16 + 1
    n_pages = b * max_pages + 3
    pool = rng.standard_normal((n_pages, 2, Hkv, 16, dh)).astype(np.float32)
    q = rng.standard_normal((b, Hq, dh)).astype(np.float32)
    if dt != si.DT_F32:
        pool, q = _round16(pool, dt), _round16(q, dt)
    perm = rng.permutation(n_pages).astype(np.int32)
    ids = rng.permutation(b).astype(np.int32)                       # slot s serves candidate ids[s]
    pt = perm[: b * max_pages].reshape(b, max_pages).copy()         # page table indexed by candidate id
    pt[:, : shared // 16] = pt[0, : shared // 16]                   # the shared prompt pages
    tdt = T16.get(dt, torch.float32)
    out = torch.zeros(b, Hq, dh, dtype=tdt, device="cuda")
    sr.sr_k_decode_attention(dt, dev(q, tdt), dev(pool, tdt), dev(pt), max_pages, dev(ids),
                             dev(np.array(lens, np.int32)), b, Hq, Hkv, dh, window, out, shared_pos=shared)
    got = out.float().cpu().numpy()
    for s in range(b):
        L = lens[s]
        pages = pt[ids[s], : (L + 15) // 16]
        K = pool[pages, 0].transpose(0, 2, 1, 3).reshape(-1, Hkv, dh)[:L]
        Vv = pool[pages, 1].transpose(0, 2, 1, 3).reshape(-1, Hkv, dh)[:L]
        want = otr.attention(q[s][None, None], K[None], Vv[None], np.array([[L - 1]]), np.arange(L)[None], window)
        tol = {si.DT_BF16: 1e-2, si.DT_F16: 2e-3, si.DT_F32: 2e-5}[dt]
        np.testing.assert_allclose(got[s], want[0, 0], rtol=tol, atol=tol)


@pytest.mark.parametrize("dt,Hq,Hkv,dh,n_pre,taus,window", [
    (si.DT_F16, 32, 8, 128, 288, [1, 64, 65, 200, 7], 0),
    (si.DT_F16, 12, 12, 64, 128, [64, 3, 130], 0),
    (si.DT_F16, 8, 8, 256, 100, [70, 1, 128], 0),
    (si.DT_F16, 4, 2, 128, 0, [300], 0),
    (si.DT_F16, 8, 4, 64, 40, [90, 33], 50),
    (si.DT_BF16, 32, 8, 128, 288, [1, 64, 65, 200, 7], 0),
    # head_dim 128 with 8 kv heads runs the tcgen05 kernel: group sizes 1, 2 and 8, a window, a 512-position
    # prefix, and own rows over several 128-key blocks
    (si.DT_F16, 8, 8, 128, 100, [70, 1, 128], 0),
    (si.DT_F16, 16, 8, 128, 0, [300, 17], 0),
    (si.DT_F16, 64, 8, 128, 40, [90, 33], 50),
    (si.DT_F16, 32, 8, 128, 512, [600, 5, 129], 0),
    (si.DT_BF16, 32, 8, 128, 130, [257, 31], 200),
])
def test_prefill_attention(sr, dt, Hq, Hkv, dh, n_pre, taus, window):
    rng = np.random.default_rng(dh + n_pre)
    rows = sum(taus)
    q = _round16(rng.standard_normal((rows, Hq, dh)).astype(np.float32), dt)
    k = _round16(rng.standard_normal((rows, Hkv, dh)).astype(np.float32), dt)
    v = _round16(rng.standard_normal((rows, Hkv, dh)).astype(np.float32), dt)
    kp = _round16(rng.standard_normal((max(n_pre, 1), Hkv, dh)).astype(np.float32), dt)
    vp = _round16(rng.standard_normal((max(n_pre, 1), Hkv, dh)).astype(np.float32), dt)
    off = np.concatenate([[0], np.cumsum(taus)]).astype(np.int32)
    pos0 = n_pre
    t = T16[dt]
    out = torch.zeros(rows, Hq, dh, dtype=t, device="cuda")
    sr.sr_k_prefill_attention(dt, dev(q, t), dev(k, t), dev(v, t), dev(kp, t), dev(vp, t), n_pre, dev(off),
                              len(taus), pos0, Hq, Hkv, dh, window, out)
    got = out.float().cpu().numpy()
    for j, t in enumerate(taus):
        sl = slice(off[j], off[j + 1])
        K = np.concatenate([kp[:n_pre], k[sl]])
        V = np.concatenate([vp[:n_pre], v[sl]])
        kpos = np.concatenate([np.arange(n_pre), pos0 + np.arange(t)])
        want = otr.attention(q[sl][None], K[None], V[None], (pos0 + np.arange(t))[None], kpos[None], window)
        tol = 2e-2 if dt == si.DT_BF16 else 3e-3
        np.testing.assert_allclose(got[sl], want[0], rtol=tol, atol=tol)
