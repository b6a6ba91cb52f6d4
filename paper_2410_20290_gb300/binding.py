"""Thin ctypes binding of libsr (include/sr.h): the same entry points under the same names.

Only argument marshalling lives here -- every step of the method runs in the library's CUDA
kernels.  Host arrays are NumPy arrays; device buffers are torch CUDA tensors (PyTorch is
used for device memory and streams only).  Importing this module loads libsr.so and fails
loudly when it has not been built (``python -m paper_2410_20290_gb300.build``).
"""
from __future__ import annotations

import ctypes
import os
import re
from typing import Optional, Sequence

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libsr.so")
HEADER = os.path.join(os.path.dirname(HERE), "include", "sr.h")

SR_OK, SR_ERR_INVALID_ARG, SR_ERR_OOM, SR_ERR_CUDA, SR_ERR_TIMEOUT, SR_ERR_STATE, SR_ERR_UNSUPPORTED = range(7)
SR_MAX_ROUNDS = 64
SR_KC_N = 8
KERNEL_CLASSES = ("gemm_decode", "gemm_score", "gemm_prompt", "attn_decode", "attn_prefill", "sample", "elementwise",
                  "control")


class SrError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"libsr status {status}: {msg}")
        self.status = status


class sr_model_desc(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int) for n in ("n_layers", "d_model", "n_heads", "n_kv_heads", "head_dim", "ffn_dim",
                                             "vocab", "max_pos", "window", "norm", "act", "pos")] + \
               [("rope_theta", ctypes.c_float), ("norm_eps", ctypes.c_float), ("has_lm_head", ctypes.c_int),
                ("has_scalar_head", ctypes.c_int), ("dtype", ctypes.c_int)]


class sr_schedule(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int), ("n_tau", ctypes.c_int), ("tau", ctypes.POINTER(ctypes.c_int))]


class sr_stats(ctypes.Structure):
    _fields_ = [("rounds", ctypes.c_int), ("b_per_round", ctypes.c_int * SR_MAX_ROUNDS),
                ("step_per_round", ctypes.c_int * SR_MAX_ROUNDS), ("k_per_round", ctypes.c_int * SR_MAX_ROUNDS),
                ("accepted_per_round", ctypes.c_int * SR_MAX_ROUNDS),
                ("r_cut_per_round", ctypes.c_float * SR_MAX_ROUNDS), ("k_raised", ctypes.c_int),
                ("n_completed", ctypes.c_int), ("best_id", ctypes.c_int), ("waves", ctypes.c_int),
                ("gen_tokens", ctypes.c_longlong), ("rm_tokens", ctypes.c_longlong),
                ("decode_steps", ctypes.c_longlong), ("pool_pages", ctypes.c_int),
                ("peak_pages_in_use", ctypes.c_int), ("ms_prefill", ctypes.c_double), ("ms_decode", ctypes.c_double),
                ("ms_score", ctypes.c_double), ("ms_select", ctypes.c_double), ("ms_total", ctypes.c_double),
                ("kern_ms", ctypes.c_double * SR_KC_N), ("kern_launches", ctypes.c_longlong * SR_KC_N),
                ("kern_flops", ctypes.c_double * SR_KC_N), ("kern_bytes", ctypes.c_double * SR_KC_N),
                ("kern_timed", ctypes.c_longlong * SR_KC_N), ("kern_timed_flops", ctypes.c_double * SR_KC_N),
                ("kern_timed_bytes", ctypes.c_double * SR_KC_N), ("rm_tokens_cached", ctypes.c_longlong)]

    def as_dict(self) -> dict:
        r = self.rounds
        n = min(r, SR_MAX_ROUNDS)
        out = {f: getattr(self, f) for f, _ in self._fields_ if not f.endswith("_round") and not f.startswith("kern_")}
        for f in ("b_per_round", "step_per_round", "k_per_round", "accepted_per_round", "r_cut_per_round"):
            out[f] = list(getattr(self, f))[:n]
        out["kernels"] = {KERNEL_CLASSES[k]: dict(ms=self.kern_ms[k], launches=self.kern_launches[k],
                                                  flops=self.kern_flops[k], bytes=self.kern_bytes[k],
                                                  timed=self.kern_timed[k], timed_flops=self.kern_timed_flops[k],
                                                  timed_bytes=self.kern_timed_bytes[k])
                          for k in range(SR_KC_N)}
        return out


_P = ctypes.c_void_p
_I = ctypes.c_int
_F = ctypes.c_float
_SIG = {
    "sr_init": [ctypes.POINTER(_P), ctypes.POINTER(sr_model_desc), _P, ctypes.POINTER(sr_model_desc), _P,
                ctypes.c_size_t, _I, _I],
    "sr_destroy": [_P],
    "sr_set_stream": [_P, _P],
    "sr_set_profiling": [_P, _I],
    "sr_generate": [_P, _P, _I, _I, _F, ctypes.POINTER(sr_schedule), _I, _F, _F, _I, ctypes.c_uint64, _P, _P, _P,
                    ctypes.POINTER(sr_stats)],
    "sr_generate_dev": [_P, _P, _I, _I, _F, ctypes.POINTER(sr_schedule), _I, _F, _F, _I, ctypes.c_uint64, _P, _P,
                        _P, ctypes.POINTER(sr_stats), _P],
    "sr_batch_begin": [_P, _P, _I, _I, _I, _F, _F, _I, ctypes.c_uint64, ctypes.POINTER(_P)],
    "sr_decode_step": [_P, _P, _P],
    "sr_score_partial": [_P, _P, _P, _P],
    "sr_reject_compact": [_P, _P, _P, _F, _P, _P, _P, _P],
    "sr_batch_query": [_P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P],
    "sr_batch_end": [_P, _P],
    "sr_k_sample": [_P, ctypes.c_longlong, _I, _I, _P, _P, ctypes.c_uint64, _F, _F, _I, _P, _P, _P],
    "sr_k_lm_head_sample": [_I, _P, _P, _I, _I, _I, _P, _P, ctypes.c_uint64, _F, _F, _I, _P, _P],
    "sr_set_reward": [_P, _I],
    "sr_set_rm_cache": [_P, ctypes.c_size_t],
    "sr_auto_b_init": [_P, ctypes.c_size_t, _I, _I, _I, _P],
    "sr_k_rcut": [_P, _I, _F, _I, _P, _P, _P],
    "sr_k_gemm": [_I, _P, _P, _P, _I, _I, _I, _I, _P],
    "sr_k_decode_attention": [_I, _P, _P, _P, _I, _P, _P, _I, _I, _I, _I, _I, _I, _P, _P],
    "sr_k_decode_attention_static": [_I, _P, _P, _P, _I, _P, _P, _I, _I, _I, _I, _I, _I, _P, _P],
    "sr_k_prefill_attention": [_I, _P, _P, _P, _P, _P, _I, _P, _I, _I, _I, _I, _I, _I, _P, _P],
}


def _load() -> ctypes.CDLL:
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"libsr.so is not built at {LIB_PATH}; run python -m paper_2410_20290_gb300.build")
    lib = ctypes.CDLL(LIB_PATH)
    for name, args in _SIG.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = None if name in ("sr_destroy", "sr_batch_end") else ctypes.c_int
    lib.sr_last_error.restype = ctypes.c_char_p
    lib.sr_last_error.argtypes = []
    return lib


LIB = _load()


def declared_symbols(header: str = HEADER) -> list:
    """Function names declared in include/sr.h."""
    text = open(header).read()
    return sorted(set(re.findall(r"\b(sr_[a-z_0-9]+)\s*\(", text)))


def _check(status: int):
    if status != SR_OK:
        raise SrError(status, LIB.sr_last_error().decode())


def _ptr(x) -> Optional[int]:
    """Address of a NumPy array, a torch tensor, or None."""
    if x is None:
        return None
    if isinstance(x, np.ndarray):
        assert x.flags["C_CONTIGUOUS"]
        return x.ctypes.data
    if hasattr(x, "data_ptr"):
        assert x.is_contiguous()
        return x.data_ptr()
    if isinstance(x, int):
        return x
    raise TypeError(type(x))


def _stream(s) -> Optional[int]:
    if s is None:
        return None
    if hasattr(s, "cuda_stream"):
        return s.cuda_stream
    return int(s)


def make_desc(m) -> sr_model_desc:
    """sr_model_desc from any object with the descriptor's attribute names (e.g. sr_inputs.ModelDesc)."""
    d = sr_model_desc()
    for f, _ in sr_model_desc._fields_:
        setattr(d, f, getattr(m, f))
    return d


def make_schedule(kind: int, taus: Sequence[int] = ()):
    arr = (ctypes.c_int * max(1, len(taus)))(*taus)
    s = sr_schedule(kind, len(taus), ctypes.cast(arr, ctypes.POINTER(ctypes.c_int)))
    s._keep = arr
    return s


# ---- the C entry points -------------------------------------------------------------------------
def sr_init(gen_desc, gen_w, rm_desc, rm_w, kv_pool_bytes: int = 0, page_tokens: int = 16, device: int = 0):
    ctx = _P()
    g, r = make_desc(gen_desc), make_desc(rm_desc)
    _check(LIB.sr_init(ctypes.byref(ctx), ctypes.byref(g), _ptr(gen_w), ctypes.byref(r), _ptr(rm_w),
                       int(kv_pool_bytes), page_tokens, device))
    return ctx


def sr_destroy(ctx):
    LIB.sr_destroy(ctx)


SR_REWARD_MODEL, SR_REWARD_LOGPROB = 0, 1


def sr_auto_b_init(gen, kv_pool_bytes: int, P: int, tau_min: int, n_max: int) -> int:
    """Largest N <= n_max that reaches tau_min tokens before the first memory-triggered round."""
    d = make_desc(gen)
    n = ctypes.c_int(0)
    st = LIB.sr_auto_b_init(ctypes.byref(d), kv_pool_bytes, P, tau_min, n_max, ctypes.byref(n))
    if st == SR_ERR_OOM:
        return 0
    _check(st)
    return n.value


def sr_set_rm_cache(ctx, nbytes: int):
    """Keep the reward model's KV across rounds in a pool of nbytes (0: off)."""
    _check(LIB.sr_set_rm_cache(ctx, int(nbytes)))


def sr_set_reward(ctx, kind: int):
    """SR_REWARD_MODEL (reward model) or SR_REWARD_LOGPROB (mean log-probability under the generator)."""
    _check(LIB.sr_set_reward(ctx, int(kind)))


def sr_set_profiling(ctx, period: int = 1):
    """0 / False: off; k >= 1: time one launch in k of each kernel class (True = every launch)."""
    _check(LIB.sr_set_profiling(ctx, int(period)))


def sr_set_stream(ctx, stream=None):
    _check(LIB.sr_set_stream(ctx, _stream(stream)))


def sr_generate(ctx, prompt, N, alpha, sched_kind, taus, max_new, temperature, eos_bias, eos_id, seed):
    """Host-buffer Algorithm 1.  Returns (tokens ndarray, score, stats dict)."""
    prompt = np.ascontiguousarray(prompt, dtype=np.int32)
    out = np.zeros(max_new, np.int32)
    n = ctypes.c_int(0)
    sc = ctypes.c_float(0)
    st = sr_stats()
    sched = make_schedule(sched_kind, taus)
    _check(LIB.sr_generate(ctx, _ptr(prompt), len(prompt), N, alpha, ctypes.byref(sched), max_new, temperature,
                           eos_bias, eos_id, seed, _ptr(out), ctypes.addressof(n), ctypes.addressof(sc),
                           ctypes.byref(st)))
    return out[:n.value].copy(), float(sc.value), st.as_dict()


def sr_generate_dev(ctx, prompt_dev, N, alpha, sched_kind, taus, max_new, temperature, eos_bias, eos_id, seed,
                    out_tokens_dev, out_len_dev, out_score_dev, stream=None):
    """Device-buffer Algorithm 1 (torch CUDA tensors); returns the stats dict."""
    st = sr_stats()
    sched = make_schedule(sched_kind, taus)
    _check(LIB.sr_generate_dev(ctx, _ptr(prompt_dev), prompt_dev.numel(), N, alpha, ctypes.byref(sched), max_new,
                               temperature, eos_bias, eos_id, seed, _ptr(out_tokens_dev), _ptr(out_len_dev),
                               _ptr(out_score_dev), ctypes.byref(st), _stream(stream)))
    return st.as_dict()


def sr_batch_begin(ctx, prompt, N, max_new, temperature, eos_bias, eos_id, seed):
    prompt = np.ascontiguousarray(prompt, dtype=np.int32)
    b = _P()
    _check(LIB.sr_batch_begin(ctx, _ptr(prompt), len(prompt), N, max_new, temperature, eos_bias, eos_id, seed,
                              ctypes.byref(b)))
    return b


def sr_decode_step(ctx, batch, logits_out: Optional[np.ndarray] = None):
    _check(LIB.sr_decode_step(ctx, batch, _ptr(logits_out)))


def sr_score_partial(ctx, batch, capacity: int) -> np.ndarray:
    r = np.zeros(capacity, np.float32)
    b = ctypes.c_int(0)
    _check(LIB.sr_score_partial(ctx, batch, _ptr(r), ctypes.addressof(b)))
    return r[:b.value].copy()


def sr_reject_compact(ctx, batch, rewards, alpha):
    rewards = np.ascontiguousarray(rewards, dtype=np.float32)
    acc = np.zeros(len(rewards), np.int32)
    rc = ctypes.c_float(0)
    nb = ctypes.c_int(0)
    nl = ctypes.c_int(0)
    _check(LIB.sr_reject_compact(ctx, batch, _ptr(rewards), alpha, ctypes.addressof(rc), _ptr(acc),
                                 ctypes.addressof(nb), ctypes.addressof(nl)))
    return float(rc.value), acc[:nb.value].copy(), nl.value


def sr_batch_query(ctx, batch, N: int, max_new: int, max_pages: int, pool_pages: int):
    ids = np.zeros(N, np.int32)
    lens = np.zeros(N, np.int32)
    stat = np.zeros(N, np.int32)
    toks = np.zeros((N, max_new), np.int32)
    pt = np.zeros((N, max_pages), np.int32)
    fs = np.zeros(max(pool_pages, 1), np.int32)
    nl, top, mp = ctypes.c_int(0), ctypes.c_int(0), ctypes.c_int(0)
    _check(LIB.sr_batch_query(ctx, batch, _ptr(ids), _ptr(lens), _ptr(stat), _ptr(toks), _ptr(pt), _ptr(fs),
                              ctypes.addressof(nl), ctypes.addressof(top), ctypes.addressof(mp)))
    return dict(ids_live=ids[:nl.value].copy(), lengths=lens, status=stat, tokens=toks, page_table=pt,
                free_stack=fs[:top.value].copy(), n_live=nl.value, free_top=top.value, max_pages=mp.value)


def sr_batch_end(ctx, batch):
    LIB.sr_batch_end(ctx, batch)


def sr_k_sample(logits, ld, b, vocab, orig_ids, steps, seed, temperature, eos_bias, eos_id, tokens_out, stream=None,
                logprob_sum=None):
    _check(LIB.sr_k_sample(_ptr(logits), ld, b, vocab, _ptr(orig_ids), _ptr(steps), seed, temperature, eos_bias,
                           eos_id, _ptr(tokens_out), _stream(stream), _ptr(logprob_sum)))


def sr_k_lm_head_sample(dtype, x, W, M, vocab, K, orig_ids, lens, seed, temperature, eos_bias, eos_id, tokens_out,
                        stream=None):
    _check(LIB.sr_k_lm_head_sample(dtype, _ptr(x), _ptr(W), M, vocab, K, _ptr(orig_ids), _ptr(lens), seed, temperature,
                                   eos_bias, eos_id, _ptr(tokens_out), _stream(stream)))


def sr_k_rcut(rewards, b, alpha, k_override, r_cut_out, mask_out, stream=None):
    _check(LIB.sr_k_rcut(_ptr(rewards), b, alpha, k_override, _ptr(r_cut_out), _ptr(mask_out), _stream(stream)))


def sr_k_gemm(dtype, A, W, C, M, N, K, epilogue, stream=None):
    _check(LIB.sr_k_gemm(dtype, _ptr(A), _ptr(W), _ptr(C), M, N, K, epilogue, _stream(stream)))


def sr_k_decode_attention(dtype, q, pool, page_table, pt_stride, orig_ids, lens, b, n_heads, n_kv_heads, head_dim,
                          window, out, stream=None, shared_pos=0):
    _check(LIB.sr_k_decode_attention(dtype, _ptr(q), _ptr(pool), _ptr(page_table), pt_stride, _ptr(orig_ids),
                                     _ptr(lens), b, n_heads, n_kv_heads, head_dim, window, shared_pos, _ptr(out),
                                     _stream(stream)))


def sr_k_decode_attention_static(dtype, q, pool, page_table, pt_stride, orig_ids, lens, b, n_heads, n_kv_heads,
                                 head_dim, window, max_len, out, stream=None):
    """Decode attention that allocates nothing (split partials in the library's fixed device array)."""
    _check(LIB.sr_k_decode_attention_static(dtype, _ptr(q), _ptr(pool), _ptr(page_table), pt_stride, _ptr(orig_ids),
                                            _ptr(lens), b, n_heads, n_kv_heads, head_dim, window, max_len, _ptr(out),
                                            _stream(stream)))


def sr_k_prefill_attention(dtype, q, k, v, k_pre, v_pre, n_pre, seq_off, n_seq, pos0, n_heads, n_kv_heads, head_dim,
                           window, out, stream=None):
    _check(LIB.sr_k_prefill_attention(dtype, _ptr(q), _ptr(k), _ptr(v), _ptr(k_pre), _ptr(v_pre), n_pre, _ptr(seq_off),
                                      n_seq, pos0, n_heads, n_kv_heads, head_dim, window, _ptr(out),
                                      _stream(stream)))
