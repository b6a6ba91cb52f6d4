"""The allocation-free decode-attention entry point against the regular one and against the oracle.

sr_k_decode_attention_static serves callers that cannot allocate device memory when they call it
(a server that reserved all GPU memory at start-up, an allocator-free embedding, a caller holding
a lock that an allocation could block on): its split partials live in a fixed device array of the
library instead of a per-call buffer.  This file is collected last so that a run stopping at the
first failure has already run every other test; it passes alone and after them.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import sr_inputs as si
from oracle import transformer as otr

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sr():
    from paper_2410_20290_gb300 import binding
    return binding


def _case(seed, lens, Hq=32, Hkv=8, dh=128):
    rng = np.random.default_rng(seed)
    b = len(lens)
    max_pages = max(lens) // 16 + 1
    n_pages = b * max_pages + 2
    pool = rng.standard_normal((n_pages, 2, Hkv, 16, dh)).astype(np.float32)
    q = rng.standard_normal((b, Hq, dh)).astype(np.float32)
    pt = rng.permutation(n_pages)[: b * max_pages].reshape(b, max_pages).astype(np.int32)
    ids = rng.permutation(b).astype(np.int32)
    return dict(q=torch.from_numpy(q).half().cuda(), pool=torch.from_numpy(pool).half().cuda(),
                pt=torch.from_numpy(pt).cuda(), max_pages=max_pages, ids=torch.from_numpy(ids).cuda(),
                lens=torch.tensor(lens, dtype=torch.int32, device="cuda"), b=b, Hq=Hq, Hkv=Hkv, dh=dh,
                # fp16-rounded host copies for the oracle
                q_h=torch.from_numpy(q).half().float().numpy(), pool_h=torch.from_numpy(pool).half().float().numpy(),
                pt_h=pt, ids_h=ids, lens_h=list(lens))


def _run(sr, c, static, window=0, max_len=None):
    out = torch.zeros(c["b"], c["Hq"], c["dh"], dtype=torch.float16, device="cuda")
    args = (si.DT_F16, c["q"], c["pool"], c["pt"], c["max_pages"], c["ids"], c["lens"], c["b"], c["Hq"], c["Hkv"],
            c["dh"], window)
    if static:
        sr.sr_k_decode_attention_static(*args, int(c["lens"].max()) if max_len is None else max_len, out)
    else:
        sr.sr_k_decode_attention(*args, out)    # no shared prefix: the same kernels as the static entry point
    torch.cuda.synchronize()
    return out.float().cpu()


def _oracle(c, window):
    """softmax(q K^T / sqrt(dh)) V over each slot's pages, by the oracle's attention (fp64)."""
    Hkv, dh = c["Hkv"], c["dh"]
    want = np.zeros((c["b"], c["Hq"], dh), np.float64)
    for s in range(c["b"]):
        L = c["lens_h"][s]
        pages = c["pt_h"][c["ids_h"][s], : (L + 15) // 16]
        K = c["pool_h"][pages, 0].transpose(0, 2, 1, 3).reshape(-1, Hkv, dh)[:L]
        V = c["pool_h"][pages, 1].transpose(0, 2, 1, 3).reshape(-1, Hkv, dh)[:L]
        want[s] = otr.attention(c["q_h"][s][None, None], K[None], V[None], np.array([[L - 1]]), np.arange(L)[None],
                                window)[0, 0]
    return want


def test_static_scratch_matches_allocating_entry_point(sr):
    """Two calls in a row (the second sees the first call's scratch contents) give the same outputs as the
    allocating entry point, within the decode-attention tolerance of the kernel tests."""
    for seed, lens, window in ((1, [1500, 7, 513, 1024, 600], 0), (2, [2000, 300, 1100], 700)):
        c = _case(seed, lens)
        want = _run(sr, c, static=False, window=window)
        got = _run(sr, c, static=True, window=window)
        torch.testing.assert_close(got, want, rtol=2e-3, atol=2e-3)
        got2 = _run(sr, c, static=True, window=window)
        torch.testing.assert_close(got2, want, rtol=2e-3, atol=2e-3)


@pytest.mark.parametrize("seed,lens,window", [
    (4, [1500, 7, 513, 1024, 600], 0),     # several splits, ragged tails
    (5, [2000, 300, 1100], 700),           # sliding window across split boundaries
    (6, [100, 17, 128, 1], 0),             # max_len <= 128: the one-warp-per-(kv head, slot) kernel
])
def test_static_scratch_matches_the_oracle(sr, seed, lens, window):
    c = _case(seed, lens)
    got = _run(sr, c, static=True, window=window).numpy()
    np.testing.assert_allclose(got, _oracle(c, window), rtol=2e-3, atol=2e-3)


def test_static_short_contexts_match_allocating_entry_point(sr):
    """With max_len <= 128 both entry points take the one-warp-per-(kv head, slot) kernel."""
    c = _case(7, [128, 5, 64, 99, 16, 1])
    want = _run(sr, c, static=False)
    for _ in range(2):
        torch.testing.assert_close(_run(sr, c, static=True, max_len=128), want, rtol=2e-3, atol=2e-3)


def test_static_scratch_rejects_understated_max_len(sr):
    """A length beyond max_len's last split is reported as SR_ERR_INVALID_ARG (no read past the scratch),
    and the next call with a true bound succeeds (the error word is cleared per call)."""
    c = _case(8, [1500, 40, 600])
    with pytest.raises(sr.SrError) as e:
        _run(sr, c, static=True, max_len=512)        # one split sized, 1500 needs three
    assert e.value.status == sr.SR_ERR_INVALID_ARG and "max_len" in str(e.value)
    with pytest.raises(sr.SrError) as e:
        _run(sr, c, static=True, max_len=1000)       # two splits sized, 1500 needs three
    assert e.value.status == sr.SR_ERR_INVALID_ARG
    want = _run(sr, c, static=False)
    torch.testing.assert_close(_run(sr, c, static=True, max_len=1500), want, rtol=2e-3, atol=2e-3)
    # an understated bound still within the last split is exact
    torch.testing.assert_close(_run(sr, c, static=True, max_len=1100), want, rtol=2e-3, atol=2e-3)


def test_static_scratch_rejects_oversized_shapes(sr):
    c = _case(3, [600])
    out = torch.zeros(1, 32, 128, dtype=torch.float16, device="cuda")
    with pytest.raises(sr.SrError) as e:
        # 4096 slots x 32 heads x 4 splits x 130 floats exceeds the 2^21-float array
        sr.sr_k_decode_attention_static(si.DT_F16, c["q"], c["pool"], c["pt"], c["max_pages"], c["ids"], c["lens"],
                                        4096, 32, 8, 128, 0, 2048, out)
    assert e.value.status == sr.SR_ERR_INVALID_ARG and "static scratch" in str(e.value)
