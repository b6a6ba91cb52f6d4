"""Pins of the oracle's transformer against torch library routines and invariants."""
import numpy as np
import pytest
import torch
import torch.nn.functional as tF

import sr_inputs as si
from oracle import transformer as ot


def _t(x):
    return torch.from_numpy(np.asarray(x, np.float64))


def test_norms_and_activations_match_torch():
    rng = np.random.default_rng(0)
    x = rng.standard_normal((7, 48)).astype(np.float32) * 3 + 0.5
    g = rng.standard_normal(48).astype(np.float32)
    b = rng.standard_normal(48).astype(np.float32)
    want = tF.rms_norm(_t(x), (48,), _t(g), eps=1e-5).numpy()
    np.testing.assert_allclose(ot.rms_norm(x, g, 1e-5), want, rtol=2e-5, atol=2e-6)
    want = tF.layer_norm(_t(x), (48,), _t(g), _t(b), eps=1e-5).numpy()
    np.testing.assert_allclose(ot.layer_norm(x, g, b, 1e-5), want, rtol=2e-5, atol=2e-6)
    np.testing.assert_allclose(ot.gelu_tanh(x), tF.gelu(_t(x), approximate="tanh").numpy(), rtol=1e-5, atol=1e-6)
    np.testing.assert_allclose(ot.silu(x), tF.silu(_t(x)).numpy(), rtol=1e-5, atol=1e-6)


@pytest.mark.parametrize("Hq,Hkv,window", [(4, 4, 0), (8, 2, 0), (6, 3, 5)])
def test_attention_matches_sdpa(Hq, Hkv, window):
    rng = np.random.default_rng(1)
    B, T, dh = 2, 11, 16
    q = rng.standard_normal((B, T, Hq, dh)).astype(np.float32)
    k = rng.standard_normal((B, T, Hkv, dh)).astype(np.float32)
    v = rng.standard_normal((B, T, Hkv, dh)).astype(np.float32)
    pos = np.broadcast_to(np.arange(T), (B, T))
    got = ot.attention(q, k, v, pos, pos, window)
    i = np.arange(T)
    mask = i[None, :] <= i[:, None]
    if window:
        mask &= i[None, :] > i[:, None] - window
    want = tF.scaled_dot_product_attention(_t(q).transpose(1, 2), _t(k).transpose(1, 2), _t(v).transpose(1, 2),
                                           attn_mask=torch.from_numpy(mask), enable_gqa=True).transpose(1, 2)
    np.testing.assert_allclose(got, want.numpy(), rtol=1e-4, atol=1e-5)


def test_rope_is_complex_rotation_and_relative():
    rng = np.random.default_rng(2)
    dh, theta = 32, 10000.0
    x = rng.standard_normal((5, 1, dh)).astype(np.float32)
    pos = np.array([0, 1, 7, 100, 2047])
    got = ot.apply_rope(x, pos, theta)
    # rotate-half pairing: dims (i, i + dh/2) form the complex number x_i + j x_{i+dh/2}
    half = dh // 2
    z = x[..., :half].astype(np.float64) + 1j * x[..., half:].astype(np.float64)
    ang = pos[:, None, None] * theta ** (-2.0 * np.arange(half) / dh)
    zr = z * np.exp(1j * ang)
    np.testing.assert_allclose(got, np.concatenate([zr.real, zr.imag], -1), rtol=1e-5, atol=1e-5)
    assert np.array_equal(ot.apply_rope(x[:1], np.array([0]), theta), x[:1])
    # q . k after RoPE depends only on the position difference
    q = rng.standard_normal((1, 1, dh)).astype(np.float32)
    k = rng.standard_normal((1, 1, dh)).astype(np.float32)
    dots = [float(np.sum(ot.apply_rope(q, np.array([p + 9]), theta) * ot.apply_rope(k, np.array([p]), theta)))
            for p in (0, 3, 50, 400)]
    assert np.allclose(dots, dots[0], rtol=1e-4, atol=1e-4)


def _small(norm, act, pos, Hq=4, Hkv=2, window=0):
    return si.ModelDesc(n_layers=2, d_model=32, n_heads=Hq, n_kv_heads=Hkv, head_dim=8, ffn_dim=48, vocab=40,
                        max_pos=64, window=window, norm=norm, act=act, pos=pos, has_lm_head=1, has_scalar_head=1,
                        dtype=si.DT_F32)


MODELS = [
    _small(si.NORM_RMS, si.ACT_SWIGLU, si.POS_ROPE),
    _small(si.NORM_LAYER, si.ACT_GELU, si.POS_LEARNED, Hq=4, Hkv=4),
    _small(si.NORM_RMS, si.ACT_GEGLU, si.POS_ROPE, Hq=2, Hkv=2),
    _small(si.NORM_RMS, si.ACT_SWIGLU, si.POS_ROPE, Hq=4, Hkv=1, window=6),
]


@pytest.mark.parametrize("m", MODELS)
def test_kv_cached_decode_equals_recompute(m):
    w = si.random_weights(m, 11, perturb_norms=True)
    mdl = ot.Transformer(m, w)
    rng = np.random.default_rng(4)
    P, steps = 5, 9
    seqs = rng.integers(1, m.vocab, (3, P + steps))
    full = mdl.forward(seqs)
    dec = ot.Decoder(mdl, 3, P + steps)
    h0 = dec.prefill(seqs[0, :P], [0, 1, 2])
    np.testing.assert_allclose(h0, full[0, :P], rtol=1e-5, atol=1e-5)
    # all three share the prompt only when their prompts are equal: use sequence 0's prompt for all
    seqs[:, :P] = seqs[0, :P]
    full = mdl.forward(seqs)
    for t in range(P, P + steps):
        h = dec.step([0, 1, 2], seqs[:, t], t)
        np.testing.assert_allclose(h, full[:, t], rtol=1e-5, atol=1e-5)


def test_layer_matches_torch_functional():
    """One full forward rebuilt from torch.nn.functional pieces (linear, rms_norm, SDPA with GQA, silu)."""
    m = _small(si.NORM_RMS, si.ACT_SWIGLU, si.POS_ROPE, Hq=4, Hkv=2)
    w = si.weights_as_f32(m, si.random_weights(m, 5, perturb_norms=True))
    mdl = ot.Transformer(m, si.random_weights(m, 5, perturb_norms=True))
    ids = np.array([[3, 9, 1, 22, 7, 30, 2]])
    T = ids.shape[1]
    W = {k: _t(v) for k, v in w.items()}
    x = W["tok_emb"][torch.from_numpy(ids)]
    cos, sin = ot.rope_cos_sin(np.arange(T), m.head_dim, m.rope_theta)
    cos, sin = _t(cos)[None, :, None, :], _t(sin)[None, :, None, :]

    def rope(t):
        h = m.head_dim // 2
        a, b = t[..., :h], t[..., h:]
        return torch.cat([a * cos - b * sin, b * cos + a * sin], -1)

    for l in range(m.n_layers):
        h = tF.rms_norm(x, (m.d_model,), W[f"l{l}.attn_norm_w"], eps=m.norm_eps)
        y = tF.linear(h, W[f"l{l}.wqkv"])
        nq, nk = m.n_heads * m.head_dim, m.n_kv_heads * m.head_dim
        q = rope(y[..., :nq].reshape(1, T, m.n_heads, m.head_dim))
        k = rope(y[..., nq:nq + nk].reshape(1, T, m.n_kv_heads, m.head_dim))
        v = y[..., nq + nk:].reshape(1, T, m.n_kv_heads, m.head_dim)
        a = tF.scaled_dot_product_attention(q.transpose(1, 2), k.transpose(1, 2), v.transpose(1, 2),
                                            is_causal=True, enable_gqa=True).transpose(1, 2).reshape(1, T, -1)
        x = x + tF.linear(a, W[f"l{l}.wo"])
        h = tF.rms_norm(x, (m.d_model,), W[f"l{l}.mlp_norm_w"], eps=m.norm_eps)
        x = x + tF.linear(tF.silu(tF.linear(h, W[f"l{l}.w_gate"])) * tF.linear(h, W[f"l{l}.w_up"]),
                          W[f"l{l}.w_down"])
    hn = tF.rms_norm(x, (m.d_model,), W["final_norm_w"], eps=m.norm_eps)
    got = mdl.forward(ids)
    np.testing.assert_allclose(got, hn.numpy(), rtol=1e-4, atol=1e-4)
    np.testing.assert_allclose(mdl.logits(got), tF.linear(hn, W["lm_head"]).numpy(), rtol=1e-4, atol=1e-4)
    np.testing.assert_allclose(mdl.score(got[0, -1]), float(hn[0, -1] @ W["score_head"]), rtol=1e-4, atol=1e-5)


def test_window_equals_truncated_context():
    m = _small(si.NORM_RMS, si.ACT_SWIGLU, si.POS_ROPE, window=4)
    w = si.random_weights(m, 8)
    rng = np.random.default_rng(6)
    q = rng.standard_normal((1, 1, 4, 8)).astype(np.float32)
    k = rng.standard_normal((1, 10, 2, 8)).astype(np.float32)
    v = rng.standard_normal((1, 10, 2, 8)).astype(np.float32)
    a = ot.attention(q, k, v, np.array([[9]]), np.arange(10)[None], 4)
    b = ot.attention(q, k[:, 6:], v[:, 6:], np.array([[9]]), np.arange(6, 10)[None], 0)
    np.testing.assert_allclose(a, b, rtol=1e-6, atol=1e-7)


def test_bf16_operand_rounding_mode():
    """round_bf16 is torch's float32 -> bfloat16 conversion; the bf16 mode only rounds operands, so KV-cached
    decode still equals recompute in that mode, and an exact-bf16 input passes through unchanged."""
    rng = np.random.default_rng(9)
    x = (rng.standard_normal(100000) * 10.0 ** rng.uniform(-6, 6, 100000)).astype(np.float32)
    want = torch.from_numpy(x).to(torch.bfloat16).float().numpy()
    assert np.array_equal(ot.round_bf16(x), want)
    assert np.array_equal(ot.round_bf16(want), want)
    m = _small(si.NORM_RMS, si.ACT_SWIGLU, si.POS_ROPE).replace(dtype=si.DT_BF16)
    w = si.random_weights(m, 3, perturb_norms=True)
    mdl = ot.Transformer(m, w, operand_rounding="bf16")
    seqs = np.tile(rng.integers(1, m.vocab, (1, 12)), (2, 1))
    seqs[1, 8:] = rng.integers(1, m.vocab, 4)
    full = mdl.forward(seqs)
    dec = ot.Decoder(mdl, 2, 12)
    dec.prefill(seqs[0, :8], [0, 1])
    for t in range(8, 12):
        np.testing.assert_allclose(dec.step([0, 1], seqs[:, t], t), full[:, t], rtol=1e-5, atol=1e-5)
    plain = ot.Transformer(m, w).forward(seqs)
    assert 0 < np.max(np.abs(plain - full)) < 0.1      # rounding changes results, but only slightly
