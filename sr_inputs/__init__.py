"""Seeded synthetic inputs shared by the oracle, the tests and the benchmark.

This module only draws random numbers and lays them out in memory: model
descriptors for the five synthetic workloads, random-init weights, random
prompts and the flat weight blob that both the CPU oracle and the CUDA library
read.  It contains none of the method's arithmetic (no forward pass, no
sampling, no reward, no selection) and imports neither ``oracle`` nor the CUDA
package.

Workloads stand in for the paper's AlpacaFarm-Eval prompts and trained
Llama-3 / Mistral / reward-model checkpoints (Section 5, "Setup"), none of which
are available: weights are i.i.d. N(0, 0.02^2) random-init and prompt ids are
uniform on [1, V) so that no prompt token is the EOS id 0.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Tuple

import numpy as np

# enum values mirrored by include/sr.h
NORM_RMS, NORM_LAYER = 0, 1
ACT_SWIGLU, ACT_GELU, ACT_GEGLU = 0, 1, 2
POS_ROPE, POS_LEARNED = 0, 1
DT_F32, DT_BF16, DT_F16 = 0, 1, 2
SCHED_FIXED, SCHED_POOL_FULL = 0, 1


@dataclasses.dataclass(frozen=True)
class ModelDesc:
    """Shape of one decoder-only transformer (generator or reward model)."""
    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    ffn_dim: int
    vocab: int
    max_pos: int
    window: int = 0            # sliding attention window in tokens, 0 = none
    norm: int = NORM_RMS
    act: int = ACT_SWIGLU
    pos: int = POS_ROPE
    rope_theta: float = 10000.0
    norm_eps: float = 1e-5
    has_lm_head: int = 1
    has_scalar_head: int = 0
    dtype: int = DT_BF16

    @property
    def gated(self) -> bool:
        return self.act in (ACT_SWIGLU, ACT_GEGLU)

    @property
    def qkv_dim(self) -> int:
        return (self.n_heads + 2 * self.n_kv_heads) * self.head_dim

    def replace(self, **kw) -> "ModelDesc":
        return dataclasses.replace(self, **kw)


def weight_layout(m: ModelDesc) -> List[Tuple[str, Tuple[int, ...]]]:
    """Ordered (name, shape) list of the tensors in a weight blob.

    Matrices are stored [out_features, in_features] row-major, so a linear
    layer computes y = x @ W.T.  The order here is the blob format documented
    in include/sr.h.
    """
    d, F = m.d_model, m.ffn_dim
    out: List[Tuple[str, Tuple[int, ...]]] = [("tok_emb", (m.vocab, d))]
    if m.pos == POS_LEARNED:
        out.append(("pos_emb", (m.max_pos, d)))
    for l in range(m.n_layers):
        p = f"l{l}."
        out.append((p + "attn_norm_w", (d,)))
        if m.norm == NORM_LAYER:
            out.append((p + "attn_norm_b", (d,)))
        out.append((p + "wqkv", (m.qkv_dim, d)))
        out.append((p + "wo", (d, m.n_heads * m.head_dim)))
        out.append((p + "mlp_norm_w", (d,)))
        if m.norm == NORM_LAYER:
            out.append((p + "mlp_norm_b", (d,)))
        if m.gated:
            out.append((p + "w_gate", (F, d)))
            out.append((p + "w_up", (F, d)))
        else:
            out.append((p + "w_fc", (F, d)))
        out.append((p + "w_down", (d, F)))
    out.append(("final_norm_w", (d,)))
    if m.norm == NORM_LAYER:
        out.append(("final_norm_b", (d,)))
    if m.has_lm_head:
        out.append(("lm_head", (m.vocab, d)))
    if m.has_scalar_head:
        out.append(("score_head", (d,)))
    return out


def n_params(m: ModelDesc) -> int:
    return sum(int(np.prod(s)) for _, s in weight_layout(m))


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even float32 -> bfloat16 bit patterns (uint16)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    rounded = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return rounded.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def random_weights(m: ModelDesc, seed: int, model_index: int = 0, std: float = 0.02,
                   perturb_norms: bool = False) -> Dict[str, np.ndarray]:
    """Random-init weights as a dict of arrays in the model's storage dtype.

    float32 models give float32 arrays; bf16 models give uint16 bf16 bit
    patterns.  Matrices and embeddings are N(0, std^2).  Norm gains are 1 and
    norm biases 0 (the usual init), unless ``perturb_norms`` is set, in which
    case gains are 1 + N(0, 0.1^2) and biases N(0, 0.02^2) so that parity tests
    also exercise those terms.  ``model_index`` separates the generator (0) and
    reward model (1) streams drawn from the same seed.
    """
    rng = np.random.default_rng([seed, model_index])
    out: Dict[str, np.ndarray] = {}
    for name, shape in weight_layout(m):
        base = name.split(".")[-1]
        if base.endswith("norm_w"):
            a = np.ones(shape, np.float32)
            if perturb_norms:
                a += rng.standard_normal(shape, dtype=np.float32) * np.float32(0.1)
        elif base.endswith("norm_b"):
            a = np.zeros(shape, np.float32)
            if perturb_norms:
                a += rng.standard_normal(shape, dtype=np.float32) * np.float32(0.02)
        else:
            a = rng.standard_normal(shape, dtype=np.float32) * np.float32(std)
        out[name] = a if m.dtype == DT_F32 else f32_to_bf16_bits(a)
    return out


def weights_as_f32(m: ModelDesc, w: Dict[str, np.ndarray]) -> Dict[str, np.ndarray]:
    """Upcast a weight dict to float32 (bf16 bit patterns are widened exactly)."""
    if m.dtype == DT_F32:
        return {k: np.asarray(v, np.float32) for k, v in w.items()}
    return {k: bf16_bits_to_f32(v) for k, v in w.items()}


def pack_blob(m: ModelDesc, w: Dict[str, np.ndarray]) -> np.ndarray:
    """Concatenate the tensors in ``weight_layout`` order, densely packed."""
    parts = []
    dt = np.float32 if m.dtype == DT_F32 else np.uint16
    for name, shape in weight_layout(m):
        a = np.ascontiguousarray(w[name], dtype=dt)
        assert a.shape == tuple(shape), (name, a.shape, shape)
        parts.append(a.reshape(-1))
    return np.concatenate(parts)


def unpack_blob(m: ModelDesc, blob: np.ndarray) -> Dict[str, np.ndarray]:
    out, off = {}, 0
    for name, shape in weight_layout(m):
        n = int(np.prod(shape))
        out[name] = blob[off:off + n].reshape(shape)
        off += n
    assert off == blob.size
    return out


def random_prompt(vocab: int, length: int, seed: int) -> np.ndarray:
    """Uniform token ids on [1, vocab); id 0 is the EOS id of every workload."""
    rng = np.random.default_rng([seed, 7919])
    return rng.integers(1, vocab, size=length, dtype=np.int64).astype(np.int32)


def device_weight_blob(m: ModelDesc, seed: int, model_index: int = 0, device="cuda", std: float = 0.02):
    """Same recipe as ``random_weights`` but drawn on the GPU with torch's
    generator, for the 7-8B-parameter workloads where a host draw is too slow.
    Returns a flat bf16 torch tensor in blob order.  (Not bit-identical to the
    host draw; workloads using it read weights back from the device when an
    oracle comparison needs them.)"""
    import torch
    assert m.dtype == DT_BF16
    g = torch.Generator(device=device)
    g.manual_seed(int(seed) * 1000003 + int(model_index))
    total = n_params(m)
    blob = torch.empty(total, dtype=torch.bfloat16, device=device)
    off = 0
    for name, shape in weight_layout(m):
        n = int(np.prod(shape))
        base = name.split(".")[-1]
        view = blob[off:off + n]
        if base.endswith("norm_w"):
            view.fill_(1.0)
        elif base.endswith("norm_b"):
            view.zero_()
        else:
            # draw in fp32 chunks to bound temporary memory, then round to bf16
            step = 1 << 28
            for s in range(0, n, step):
                e = min(n, s + step)
                view[s:e].copy_(torch.randn(e - s, generator=g, device=device, dtype=torch.float32) * std)
        off += n
    return blob


# ---------------------------------------------------------------------------
# The five synthetic workloads.
# ---------------------------------------------------------------------------

def _llama8b(max_pos: int, lm: bool) -> ModelDesc:
    return ModelDesc(n_layers=32, d_model=4096, n_heads=32, n_kv_heads=8, head_dim=128, ffn_dim=14336,
                     vocab=128256, max_pos=max_pos, norm=NORM_RMS, act=ACT_SWIGLU, pos=POS_ROPE,
                     rope_theta=500000.0, has_lm_head=int(lm), has_scalar_head=int(not lm), dtype=DT_BF16)


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    gen: ModelDesc
    rm: ModelDesc
    prompt_len: int                 # fixed length, or upper bound when prompt_len_min > 0
    N: int
    alpha: float
    sched_kind: int
    taus: Tuple[int, ...]
    max_new: int
    temperature: float
    eos_bias: float
    eos_id: int = 0
    pool_bytes: int = 0             # 0: sized so that all N fit to max_new
    prompt_len_min: int = 0
    n_prompts: int = 1
    weight_seed: int = 0

    def prompt(self, i: int = 0) -> np.ndarray:
        """Prompt i (its seed is i); length uniform on [prompt_len_min, prompt_len] when a range is set."""
        if self.prompt_len_min:
            rng = np.random.default_rng([i, 104729])
            P = int(rng.integers(self.prompt_len_min, self.prompt_len + 1))
        else:
            P = self.prompt_len
        return random_prompt(self.gen.vocab, P, i)

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


def _tiny() -> Workload:
    g = ModelDesc(n_layers=2, d_model=128, n_heads=4, n_kv_heads=4, head_dim=32, ffn_dim=512, vocab=512,
                  max_pos=16 + 64, norm=NORM_RMS, act=ACT_SWIGLU, pos=POS_ROPE, rope_theta=10000.0,
                  has_lm_head=1, has_scalar_head=0, dtype=DT_F32)
    rm = g.replace(has_lm_head=0, has_scalar_head=1)
    return Workload("tiny", g, rm, prompt_len=16, N=8, alpha=0.5, sched_kind=SCHED_FIXED, taus=(16,),
                    max_new=64, temperature=1.0, eos_bias=0.0)


def _gpt2() -> Workload:
    g = ModelDesc(n_layers=12, d_model=768, n_heads=12, n_kv_heads=12, head_dim=64, ffn_dim=3072, vocab=32000,
                  max_pos=1024, norm=NORM_LAYER, act=ACT_GELU, pos=POS_LEARNED, has_lm_head=1,
                  has_scalar_head=0, dtype=DT_BF16)
    rm = g.replace(has_lm_head=0, has_scalar_head=1)
    return Workload("gpt2", g, rm, prompt_len=128, N=128, alpha=0.5, sched_kind=SCHED_FIXED, taus=(64,),
                    max_new=256, temperature=1.0, eos_bias=0.0)


def _llama_n256() -> Workload:
    return Workload("llama8b_n256", _llama8b(256 + 1024, True), _llama8b(256 + 1024, False), prompt_len=256,
                    N=256, alpha=0.5, sched_kind=SCHED_FIXED, taus=(128,), max_new=1024, temperature=0.8,
                    eos_bias=2.0)


def _llama_n1024() -> Workload:
    return Workload("llama8b_n1024", _llama8b(512 + 1024, True), _llama8b(512 + 1024, False), prompt_len=512,
                    prompt_len_min=64, n_prompts=8, N=1024, alpha=0.7, sched_kind=SCHED_POOL_FULL, taus=(),
                    max_new=1024, temperature=1.0, eos_bias=1.0, pool_bytes=60 * 10**9)


def _mistral_2b() -> Workload:
    g = ModelDesc(n_layers=32, d_model=4096, n_heads=32, n_kv_heads=8, head_dim=128, ffn_dim=14336, vocab=32000,
                  max_pos=512 + 2048, window=4096, norm=NORM_RMS, act=ACT_SWIGLU, pos=POS_ROPE,
                  rope_theta=10000.0, has_lm_head=1, has_scalar_head=0, dtype=DT_BF16)
    rm = ModelDesc(n_layers=18, d_model=2048, n_heads=8, n_kv_heads=8, head_dim=256, ffn_dim=16384, vocab=32000,
                   max_pos=512 + 2048, norm=NORM_RMS, act=ACT_GEGLU, pos=POS_ROPE, rope_theta=10000.0,
                   has_lm_head=0, has_scalar_head=1, dtype=DT_BF16)
    return Workload("mistral7b_rm2b", g, rm, prompt_len=512, N=2048, alpha=0.5, sched_kind=SCHED_POOL_FULL,
                    taus=(), max_new=2048, temperature=1.0, eos_bias=0.0, pool_bytes=60 * 10**9)


WORKLOADS: Dict[str, Workload] = {w.name: w for w in (_tiny(), _gpt2(), _llama_n256(), _llama_n1024(), _mistral_2b())}
MISTRAL_ALPHAS = (0.3, 0.5, 0.7, 0.9)


def kv_bytes_per_token(m: ModelDesc) -> int:
    elt = 4 if m.dtype == DT_F32 else 2
    return m.n_layers * 2 * m.n_kv_heads * m.head_dim * elt


def shrink(w: Workload, n_layers: int = 2, **kw) -> Workload:
    """Same widths with fewer layers (parity cases the oracle can run quickly)."""
    g = w.gen.replace(n_layers=n_layers)
    rm = w.rm.replace(n_layers=n_layers)
    return w.replace(gen=g, rm=rm, **kw)
