"""Decoder-only transformer forward (oracle side), float32 NumPy.

The generator p and the reward model s of Section 3 are decoder-only
transformers; the paper uses Llama-3 / Mistral generators and Mistral/Llama
reward models (Section 5).  This module computes, for a model descriptor of
``sr_inputs``:

  x_0       = tok_emb[id] (+ pos_emb[position] for learned positions)
  per layer:
    h       = Norm(x);  [q k v] = h Wqkv^T;  RoPE on q, k (rotate-half pairing)
    a       = softmax(q k^T / sqrt(dh) + causal/window mask) v   (GQA: query head
              j reads kv head j // (Hq / Hkv))
    x       = x + a Wo^T
    h       = Norm(x)
    x       = x + (act(h Wg^T) * (h Wu^T)) Wd^T        (SwiGLU: act = SiLU,
              GeGLU: act = tanh-GELU)  or  x + GELU(h Wfc^T) Wd^T
  out       = Norm_final(x);  logits = out Wlm^T;  reward = out[last] . w_score
Norm is RMSNorm  x / sqrt(mean(x^2) + eps) * g  or LayerNorm
(x - mean) / sqrt(var + eps) * g + b.  RoPE angle for pair i at position p is
p * theta^(-2i/dh), computed in float64 and rounded once.  A sliding window W
lets position t see positions t-W+1 .. t.  Linear layers carry no bias.

Precision: every value is stored as float32 after each operation; every
contraction (matmul, attention scores and weighted sums, norm statistics,
softmax sums) accumulates in float64 before that rounding.  This keeps the
oracle's results independent of how sequences are grouped into batches (a
float32 BLAS call is not), which the exact Best-of-N pins rely on.

Operand precision: with ``operand_rounding="bf16"`` the oracle rounds, to
bfloat16 (round to nearest even), exactly the values a bf16 implementation
feeds to its matrix units and keeps in its KV cache -- the normed inputs of
every projection and of the LM head, q, k and v after RoPE, the attention
output and the MLP hidden activation -- and nothing else; accumulation stays
float64.  This states the arithmetic of "bf16 weights and operands, wide
accumulation" so that a bf16 kernel can be held to a tight tolerance on
rewards; the default (None) is the plain float32 forward.

Two evaluation routes: ``forward`` recomputes a whole sequence with a causal
mask; ``Decoder`` keeps a KV cache and appends one position per call.  Their
agreement, and agreement of the pieces with torch's library routines, is
pinned in tests/test_oracle_transformer.py.
"""
from __future__ import annotations

import numpy as np

import sr_inputs as si

F = np.float32


def round_bf16(x):
    """float32 -> nearest bfloat16 (ties to even), returned as float32."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    r = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16) << 16
    return r.astype(np.uint32).view(np.float32).reshape(np.shape(x))


def mm(x, w64):
    """x @ W^T with float64 accumulation, rounded to float32."""
    return (np.asarray(x, np.float64) @ w64.T).astype(np.float32)


def rms_norm(x, g, eps):
    x = np.asarray(x, np.float64)
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return (x / np.sqrt(ms + eps) * g).astype(np.float32)


def layer_norm(x, g, b, eps):
    x = np.asarray(x, np.float64)
    mu = np.mean(x, axis=-1, keepdims=True)
    var = np.mean((x - mu) ** 2, axis=-1, keepdims=True)
    return ((x - mu) / np.sqrt(var + eps) * g + b).astype(np.float32)


def silu(x):
    return (x / (F(1) + np.exp(-x))).astype(np.float32)


def gelu_tanh(x):
    c = F(np.sqrt(2.0 / np.pi))
    return (F(0.5) * x * (F(1) + np.tanh(c * (x + F(0.044715) * x * x * x)))).astype(np.float32)


def rope_cos_sin(positions, head_dim, theta):
    """cos/sin tables [len(positions), head_dim/2], angles in float64."""
    half = head_dim // 2
    inv = float(theta) ** (-(2.0 * np.arange(half, dtype=np.float64)) / head_dim)
    ang = np.asarray(positions, dtype=np.float64)[..., None] * inv
    return np.cos(ang).astype(np.float32), np.sin(ang).astype(np.float32)


def apply_rope(x, positions, theta):
    """x [..., T, H, dh]; positions broadcastable to [..., T]."""
    dh = x.shape[-1]
    half = dh // 2
    cos, sin = rope_cos_sin(positions, dh, theta)
    cos = cos[..., None, :]
    sin = sin[..., None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * cos - x2 * sin, x2 * cos + x1 * sin], axis=-1).astype(np.float32)


def attention(q, k, v, q_pos, k_pos, window):
    """q [B, Tq, Hq, dh]; k, v [B, Tk, Hkv, dh]; q_pos [B, Tq]; k_pos [B, Tk] -> [B, Tq, Hq, dh]."""
    B, Tq, Hq, dh = q.shape
    Hkv = k.shape[2]
    G = Hq // Hkv
    kk = np.repeat(np.asarray(k, np.float64), G, axis=2)     # query head j uses kv head j // G
    vv = np.repeat(np.asarray(v, np.float64), G, axis=2)
    s = np.einsum("bqhd,bkhd->bhqk", np.asarray(q, np.float64), kk) / np.sqrt(dh)
    qp = np.asarray(q_pos)[:, None, :, None]
    kp = np.asarray(k_pos)[:, None, None, :]
    allowed = kp <= qp
    if window > 0:
        allowed = allowed & (kp > qp - window)
    s = np.where(allowed, s, -np.inf)
    s = s - np.max(s, axis=-1, keepdims=True)
    p = np.exp(s)
    p = p / np.sum(p, axis=-1, keepdims=True)
    return np.einsum("bhqk,bkhd->bqhd", p, vv).astype(np.float32)


class Transformer:
    def __init__(self, m: si.ModelDesc, weights: dict, operand_rounding=None):
        self.m = m
        self.w = si.weights_as_f32(m, weights)
        self._w64 = {}
        assert operand_rounding in (None, "bf16")
        self.op = round_bf16 if operand_rounding == "bf16" else (lambda x: x)

    def W(self, name):
        """float64 copy of a weight matrix (cached) for float64-accumulated products."""
        if name not in self._w64:
            self._w64[name] = self.w[name].astype(np.float64)
        return self._w64[name]

    # -- pieces -----------------------------------------------------------------
    def norm(self, x, prefix):
        m = self.m
        if m.norm == si.NORM_RMS:
            return rms_norm(x, self.w[prefix + "_w"], m.norm_eps)
        return layer_norm(x, self.w[prefix + "_w"], self.w[prefix + "_b"], m.norm_eps)

    def norm_op(self, x, prefix):
        """Norm whose output feeds a projection (an operand of the matrix units)."""
        return self.op(self.norm(x, prefix))

    def embed(self, ids, positions):
        x = self.w["tok_emb"][np.asarray(ids)]
        if self.m.pos == si.POS_LEARNED:
            x = x + self.w["pos_emb"][np.asarray(positions)]
        return x.astype(np.float32)

    def qkv(self, l, x, positions):
        m = self.m
        h = self.norm_op(x, f"l{l}.attn_norm")
        y = mm(h, self.W(f"l{l}.wqkv"))
        nq, nk = m.n_heads * m.head_dim, m.n_kv_heads * m.head_dim
        sh = x.shape[:-1]
        q = y[..., :nq].reshape(*sh, m.n_heads, m.head_dim)
        k = y[..., nq:nq + nk].reshape(*sh, m.n_kv_heads, m.head_dim)
        v = y[..., nq + nk:].reshape(*sh, m.n_kv_heads, m.head_dim)
        if m.pos == si.POS_ROPE:
            q = apply_rope(q, positions, m.rope_theta)
            k = apply_rope(k, positions, m.rope_theta)
        return self.op(q.astype(np.float32)), self.op(k.astype(np.float32)), self.op(v.astype(np.float32))

    def attn_out(self, l, x, a):
        sh = a.shape[:-2]
        return (x + mm(self.op(a.reshape(*sh, -1)), self.W(f"l{l}.wo"))).astype(np.float32)

    def mlp(self, l, x):
        m = self.m
        h = self.norm_op(x, f"l{l}.mlp_norm")
        if m.act == si.ACT_SWIGLU:
            u = silu(mm(h, self.W(f"l{l}.w_gate"))) * mm(h, self.W(f"l{l}.w_up"))
        elif m.act == si.ACT_GEGLU:
            u = gelu_tanh(mm(h, self.W(f"l{l}.w_gate"))) * mm(h, self.W(f"l{l}.w_up"))
        else:
            u = gelu_tanh(mm(h, self.W(f"l{l}.w_fc")))
        return (x + mm(self.op(u.astype(np.float32)), self.W(f"l{l}.w_down"))).astype(np.float32)

    def final(self, x):
        return self.norm(x, "final_norm")

    def logits(self, hn):
        return mm(self.op(hn), self.W("lm_head"))

    def score(self, hn):
        return (np.asarray(hn, np.float64) @ self.W("score_head")).astype(np.float32)

    # -- full recompute -----------------------------------------------------------
    def forward(self, ids):
        """ids [B, T] (positions 0..T-1) -> final-normed hidden [B, T, d]."""
        ids = np.atleast_2d(np.asarray(ids))
        B, T = ids.shape
        pos = np.broadcast_to(np.arange(T), (B, T))
        x = self.embed(ids, pos)
        for l in range(self.m.n_layers):
            q, k, v = self.qkv(l, x, pos)
            x = self.attn_out(l, x, attention(q, k, v, pos, pos, self.m.window))
            x = self.mlp(l, x)
        return self.final(x)


class Decoder:
    """KV-cached decoding for a set of sequences indexed 0..n_seq-1 that share a prompt.

    Cache layout: K[l], V[l] of shape [n_seq, max_len, Hkv, dh].
    """

    def __init__(self, model: Transformer, n_seq: int, max_len: int):
        m = model.m
        self.model = model
        self.K = [np.zeros((n_seq, max_len, m.n_kv_heads, m.head_dim), np.float32) for _ in range(m.n_layers)]
        self.V = [np.zeros_like(k) for k in self.K]

    def prefill(self, prompt, seqs):
        """Run the prompt once; copy its KV into every sequence in ``seqs``; return final-normed hidden [P, d]."""
        mdl = self.model
        P = len(prompt)
        pos = np.arange(P)[None]
        x = mdl.embed(np.asarray(prompt)[None], pos)
        for l in range(mdl.m.n_layers):
            q, k, v = mdl.qkv(l, x, pos)
            self.K[l][seqs, :P] = k[0]
            self.V[l][seqs, :P] = v[0]
            x = mdl.attn_out(l, x, attention(q, k, v, pos, pos, mdl.m.window))
            x = mdl.mlp(l, x)
        return mdl.final(x)[0]

    def step(self, seqs, tokens, position):
        """Append one token per sequence at ``position`` (same for all); return final-normed hidden [b, d]."""
        mdl = self.model
        seqs = np.asarray(seqs)
        b = len(seqs)
        pos = np.full((b, 1), position)
        x = mdl.embed(np.asarray(tokens)[:, None], pos)
        kpos = np.broadcast_to(np.arange(position + 1), (b, position + 1))
        for l in range(mdl.m.n_layers):
            q, k, v = mdl.qkv(l, x, pos)
            self.K[l][seqs, position] = k[:, 0]
            self.V[l][seqs, position] = v[:, 0]
            kk = self.K[l][seqs, :position + 1]
            vv = self.V[l][seqs, :position + 1]
            x = mdl.attn_out(l, x, attention(q, kk, vv, pos, kpos, mdl.m.window))
            x = mdl.mlp(l, x)
        return mdl.final(x)[:, 0]
