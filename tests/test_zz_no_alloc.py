"""The allocation-free decode-attention entry point against the regular one.

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
    pool = torch.from_numpy(rng.standard_normal((n_pages, 2, Hkv, 16, dh)).astype(np.float32)).half().cuda()
    q = torch.from_numpy(rng.standard_normal((b, Hq, dh)).astype(np.float32)).half().cuda()
    pt = torch.from_numpy(rng.permutation(n_pages)[: b * max_pages].reshape(b, max_pages).astype(np.int32)).cuda()
    ids = torch.from_numpy(rng.permutation(b).astype(np.int32)).cuda()
    return dict(q=q, pool=pool, pt=pt, max_pages=max_pages, ids=ids,
                lens=torch.tensor(lens, dtype=torch.int32, device="cuda"), b=b, Hq=Hq, Hkv=Hkv, dh=dh)


def _run(sr, c, static, window=0):
    out = torch.zeros(c["b"], c["Hq"], c["dh"], dtype=torch.float16, device="cuda")
    args = (si.DT_F16, c["q"], c["pool"], c["pt"], c["max_pages"], c["ids"], c["lens"], c["b"], c["Hq"], c["Hkv"],
            c["dh"], window)
    if static:
        sr.sr_k_decode_attention_static(*args, int(c["lens"].max()), out)
    else:
        sr.sr_k_decode_attention(*args, out)    # no shared prefix: the same kernels as the static entry point
    torch.cuda.synchronize()
    return out.float().cpu()


def test_static_scratch_matches_allocating_entry_point(sr):
    """Two calls in a row (the second sees the first call's scratch contents) give the same outputs as the
    allocating entry point, within the decode-attention tolerance of the kernel tests."""
    for seed, lens, window in ((1, [1500, 7, 513, 1024, 600], 0), (2, [2000, 300, 1100], 700)):
        c = _case(seed, lens)
        want = _run(sr, c, static=False, window=window)
        got = _run(sr, c, static=True, window=window)
        torch.testing.assert_close(got, want, rtol=2e-3, atol=2e-3)


def test_static_scratch_rejects_oversized_shapes(sr):
    c = _case(3, [600])
    out = torch.zeros(1, 32, 128, dtype=torch.float16, device="cuda")
    with pytest.raises(sr.SrError) as e:
        # 4096 slots x 32 heads x 4 splits x 130 floats exceeds the 2^21-float array
        sr.sr_k_decode_attention_static(si.DT_F16, c["q"], c["pool"], c["pt"], c["max_pages"], c["ids"], c["lens"],
                                        4096, 32, 8, 128, 0, 2048, out)
    assert e.value.status == sr.SR_ERR_INVALID_ARG and "static scratch" in str(e.value)
