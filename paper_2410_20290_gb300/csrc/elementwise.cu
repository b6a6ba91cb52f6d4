// Row-wise transformer pieces: embedding, RMSNorm / LayerNorm (fused with the cast to the GEMM
// operand type), RoPE (rotate-half pairing) fused with the KV-cache append into the paged pool,
// the fp32-path activations, the reward model's scalar head and page copies.
//
// These compute the per-position parts of the generator and reward model of Section 3; the KV
// append is the paged cache of the Section 5 engine ("pre-allocates the corresponding KV cache").
#include <algorithm>
#include <cstdint>
#include <type_traits>

#include "common.cuh"

namespace sr {
namespace {

template <typename T>
__global__ void k_embed(const T* __restrict__ tok_emb, const T* __restrict__ pos_emb, const int* __restrict__ tokens,
                        const int* __restrict__ positions, int d, float* __restrict__ x) {
  pdl_entry();
  const int r = blockIdx.x;
  const T* te = tok_emb + (size_t)tokens[r] * d;
  const T* pe = pos_emb ? pos_emb + (size_t)positions[r] * d : nullptr;
  float* xr = x + (size_t)r * d;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    float v = to_f(te[c]);
    if (pe) v += to_f(pe[c]);
    xr[c] = v;
  }
}

template <typename T>
__global__ void k_norm(const float* __restrict__ x, const T* __restrict__ w, const T* __restrict__ b, float eps,
                       int d, int layer_norm, T* __restrict__ out) {
  pdl_entry();
  __shared__ float red[32];
  const int r = blockIdx.x;
  const float* xr = x + (size_t)r * d;
  float mean = 0.f;
  if (layer_norm) {
    float s = 0.f;
    for (int c = threadIdx.x; c < d; c += blockDim.x) s += xr[c];
    mean = block_sum(s, red) / (float)d;
  }
  float ss = 0.f;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    const float v = xr[c] - mean;
    ss += v * v;
  }
  const float rstd = rsqrtf(block_sum(ss, red) / (float)d + eps);
  T* orow = out + (size_t)r * d;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    float v = (xr[c] - mean) * rstd * to_f(w[c]);
    if (layer_norm) v += to_f(b[c]);
    orow[c] = f_to<T>(v);
  }
}

// Vectorised form for d % 4 == 0 and d <= 16 * blockDim.x: the row stays in registers (up to four
// float4 per thread, consecutive float4 across a warp), one pass over x.
template <typename T>
__device__ __forceinline__ void store4(T* p, float a, float b, float c, float d) {
  if constexpr (std::is_same<T, float>::value) {
    *reinterpret_cast<float4*>(p) = make_float4(a, b, c, d);
  } else {
    T h[4] = {f_to<T>(a), f_to<T>(b), f_to<T>(c), f_to<T>(d)};
    *reinterpret_cast<uint2*>(p) = *reinterpret_cast<const uint2*>(h);
  }
}
template <typename T>
__device__ __forceinline__ float4 load4(const T* p) {
  if constexpr (std::is_same<T, float>::value) {
    return *reinterpret_cast<const float4*>(p);
  } else {
    const uint2 u = *reinterpret_cast<const uint2*>(p);
    const T* h = reinterpret_cast<const T*>(&u);
    return make_float4(to_f(h[0]), to_f(h[1]), to_f(h[2]), to_f(h[3]));
  }
}

template <typename T>
__global__ void __launch_bounds__(1024) k_norm_v(const float* __restrict__ x, const T* __restrict__ w,
                                                 const T* __restrict__ b, float eps, int d, int layer_norm,
                                                 T* __restrict__ out) {
  pdl_entry();
  __shared__ float red[32];
  const int r = blockIdx.x, n4 = d >> 2, nt = blockDim.x;
  const float4* xr = reinterpret_cast<const float4*>(x + (size_t)r * d);
  float4 v[4];
  float sum = 0.f;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int i = threadIdx.x + k * nt;
    v[k] = i < n4 ? xr[i] : make_float4(0.f, 0.f, 0.f, 0.f);
    sum += (v[k].x + v[k].y) + (v[k].z + v[k].w);
  }
  const float mean = layer_norm ? block_sum(sum, red) / (float)d : 0.f;
  float ss = 0.f;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    if (threadIdx.x + k * nt < n4) {
      const float a = v[k].x - mean, bb = v[k].y - mean, c = v[k].z - mean, e = v[k].w - mean;
      ss += (a * a + bb * bb) + (c * c + e * e);
    }
  }
  const float rstd = rsqrtf(block_sum(ss, red) / (float)d + eps);
  T* orow = out + (size_t)r * d;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int i = threadIdx.x + k * nt;
    if (i < n4) {
      const float4 wv = load4(w + 4 * i);
      float4 o = make_float4((v[k].x - mean) * rstd * wv.x, (v[k].y - mean) * rstd * wv.y,
                             (v[k].z - mean) * rstd * wv.z, (v[k].w - mean) * rstd * wv.w);
      if (layer_norm) {
        const float4 bv = load4(b + 4 * i);
        o.x += bv.x, o.y += bv.y, o.z += bv.z, o.w += bv.w;
      }
      store4(orow + 4 * i, o.x, o.y, o.z, o.w);
    }
  }
}

// cos/sin of p * theta^(-2i/dh), evaluated in double precision and rounded once.
__global__ void k_rope_table(float2* tab, int max_pos, int half, int dh, double theta) {
  pdl_entry();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= max_pos * half) return;
  const int p = i / half, j = i % half;
  const double inv = pow(theta, -2.0 * (double)j / (double)dh);
  const double a = (double)p * inv;
  tab[i] = make_float2((float)cos(a), (float)sin(a));
}

// One block per input row: rotate q and k, write q / k / v rows and append k, v to the pool page
// holding the row's position.
template <typename T>
__global__ void k_rope_store(const float* __restrict__ qkv, const int* __restrict__ positions,
                             const float2* __restrict__ rope, int Hq, int Hkv, int dh, T* __restrict__ q_out,
                             T* __restrict__ k_out, T* __restrict__ v_out, KvSink sink) {
  pdl_entry();
  const int r = blockIdx.x;
  const int pos = positions[r];
  const int half = dh / 2;
  const int W = (Hq + 2 * Hkv) * dh;
  const float* row = qkv + (size_t)r * W;
  T* pk = nullptr;
  T* pv = nullptr;
  if (sink.pool_layer && (!sink.n_rows || r < *sink.n_rows)) {
    const int seq = sink.row_seq ? sink.row_seq[r] : 0;
    if (seq >= 0) {
      const int pp = pos - sink.pos_base;
      const int page = sink.page_table[(size_t)seq * sink.pt_stride + pp / PAGE];
      T* base = reinterpret_cast<T*>(sink.pool_layer) + (size_t)page * 2 * Hkv * PAGE * dh + (size_t)(pp % PAGE) * dh;
      pk = base;
      pv = base + (size_t)Hkv * PAGE * dh;
    }
  }
  // rotated heads: Hq query heads then Hkv key heads, pairs (i, i + half)
  for (int idx = threadIdx.x; idx < (Hq + Hkv) * half; idx += blockDim.x) {
    const int h = idx / half, i = idx % half;
    const float* src = row + h * dh;
    float y1 = src[i], y2 = src[i + half];
    if (rope) {
      const float2 cs = rope[(size_t)pos * half + i];
      const float x1 = y1, x2 = y2;
      y1 = x1 * cs.x - x2 * cs.y;
      y2 = x2 * cs.x + x1 * cs.y;
    }
    if (h < Hq) {
      T* q = q_out + (size_t)r * Hq * dh + h * dh;
      q[i] = f_to<T>(y1);
      q[i + half] = f_to<T>(y2);
    } else {
      const int kh = h - Hq;
      if (k_out) {
        T* k = k_out + (size_t)r * Hkv * dh + kh * dh;
        k[i] = f_to<T>(y1);
        k[i + half] = f_to<T>(y2);
      }
      if (pk) {
        T* k = pk + (size_t)kh * PAGE * dh;
        k[i] = f_to<T>(y1);
        k[i + half] = f_to<T>(y2);
      }
    }
  }
  for (int idx = threadIdx.x; idx < Hkv * dh; idx += blockDim.x) {
    const int h = idx / dh, c = idx % dh;
    const T v = f_to<T>(row[(Hq + Hkv) * dh + idx]);
    if (v_out) v_out[(size_t)r * Hkv * dh + idx] = v;
    if (pv) pv[(size_t)h * PAGE * dh + c] = v;
  }
}

// Vectorised form for dh % 8 == 0: each thread rotates four consecutive pairs (i .. i+3, i+half ..
// i+half+3) of one head with float4 loads and 4-element stores.
template <typename T>
__global__ void __launch_bounds__(256) k_rope_store_v(const float* __restrict__ qkv, const int* __restrict__ positions,
                                                      const float2* __restrict__ rope, int Hq, int Hkv, int dh,
                                                      T* __restrict__ q_out, T* __restrict__ k_out,
                                                      T* __restrict__ v_out, KvSink sink) {
  pdl_entry();
  const int r = blockIdx.x;
  const int pos = positions[r];
  const int half = dh / 2, gph = half / 4;  // 4-pair groups per head
  const float* row = qkv + (size_t)r * (Hq + 2 * Hkv) * dh;
  T* pk = nullptr;
  T* pv = nullptr;
  if (sink.pool_layer && (!sink.n_rows || r < *sink.n_rows)) {
    const int seq = sink.row_seq ? sink.row_seq[r] : 0;
    if (seq >= 0) {
      const int pp = pos - sink.pos_base;
      const int page = sink.page_table[(size_t)seq * sink.pt_stride + pp / PAGE];
      T* base = reinterpret_cast<T*>(sink.pool_layer) + (size_t)page * 2 * Hkv * PAGE * dh + (size_t)(pp % PAGE) * dh;
      pk = base;
      pv = base + (size_t)Hkv * PAGE * dh;
    }
  }
  for (int idx = threadIdx.x; idx < (Hq + Hkv) * gph; idx += blockDim.x) {
    const int h = idx / gph, i = (idx % gph) * 4;
    const float* src = row + h * dh;
    float4 y1 = *reinterpret_cast<const float4*>(src + i), y2 = *reinterpret_cast<const float4*>(src + i + half);
    if (rope) {
      const float4 c01 = *reinterpret_cast<const float4*>(rope + (size_t)pos * half + i);      // cos, sin of i, i+1
      const float4 c23 = *reinterpret_cast<const float4*>(rope + (size_t)pos * half + i + 2);  // of i+2, i+3
      const float4 x1 = y1, x2 = y2;
      y1 = make_float4(x1.x * c01.x - x2.x * c01.y, x1.y * c01.z - x2.y * c01.w, x1.z * c23.x - x2.z * c23.y,
                       x1.w * c23.z - x2.w * c23.w);
      y2 = make_float4(x2.x * c01.x + x1.x * c01.y, x2.y * c01.z + x1.y * c01.w, x2.z * c23.x + x1.z * c23.y,
                       x2.w * c23.z + x1.w * c23.w);
    }
    T* dsts[2] = {nullptr, nullptr};
    if (h < Hq) {
      dsts[0] = q_out + ((size_t)r * Hq + h) * dh;
    } else {
      const int kh = h - Hq;
      if (k_out) dsts[0] = k_out + ((size_t)r * Hkv + kh) * dh;
      if (pk) dsts[1] = pk + (size_t)kh * PAGE * dh;
    }
#pragma unroll
    for (int t = 0; t < 2; ++t) {
      if (!dsts[t]) continue;
      store4(dsts[t] + i, y1.x, y1.y, y1.z, y1.w);
      store4(dsts[t] + i + half, y2.x, y2.y, y2.z, y2.w);
    }
  }
  const float* vrow = row + (Hq + Hkv) * dh;
  for (int idx = threadIdx.x; idx < Hkv * dh / 4; idx += blockDim.x) {
    const int h = (4 * idx) / dh, c = (4 * idx) % dh;
    const float4 v = *reinterpret_cast<const float4*>(vrow + 4 * idx);
    if (v_out) store4(v_out + (size_t)r * Hkv * dh + 4 * idx, v.x, v.y, v.z, v.w);
    if (pv) store4(pv + (size_t)h * PAGE * dh + c, v.x, v.y, v.z, v.w);
  }
}

__device__ __forceinline__ float silu_d(float x) { return x / (1.f + expf(-x)); }
__device__ __forceinline__ float gelu_d(float x) {
  return 0.5f * x * (1.f + tanhf(0.7978845608028654f * (x + 0.044715f * x * x * x)));
}

// fp32 path: gated activations read gate/up interleaved in blocks of 16 columns.
template <typename T>
__global__ void k_act(const float* __restrict__ in, int F, int act, T* __restrict__ out) {
  pdl_entry();
  const int r = blockIdx.x;
  for (int j = threadIdx.x; j < F; j += blockDim.x) {
    float v;
    if (act == SR_ACT_GELU) {
      v = gelu_d(in[(size_t)r * F + j]);
    } else {
      const float* row = in + (size_t)r * 2 * F;
      const int blk = j / 16, o = j % 16;
      const float g = row[blk * 32 + o], u = row[blk * 32 + 16 + o];
      v = (act == SR_ACT_SWIGLU ? silu_d(g) : gelu_d(g)) * u;
    }
    out[(size_t)r * F + j] = f_to<T>(v);
  }
}

// reward[j] = Norm_final(x[rows[j]]) . head   (the scalar head on each sequence's last position)
template <typename T>
__global__ void k_score_head(const float* __restrict__ x, const int* __restrict__ rows, const T* __restrict__ w,
                             const T* __restrict__ b, float eps, int layer_norm, const T* __restrict__ head, int d,
                             float* __restrict__ rewards) {
  pdl_entry();
  __shared__ float red[32];
  const float* xr = x + (size_t)rows[blockIdx.x] * d;
  float mean = 0.f;
  if (layer_norm) {
    float s = 0.f;
    for (int c = threadIdx.x; c < d; c += blockDim.x) s += xr[c];
    mean = block_sum(s, red) / (float)d;
  }
  float ss = 0.f;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    const float v = xr[c] - mean;
    ss += v * v;
  }
  const float rstd = rsqrtf(block_sum(ss, red) / (float)d + eps);
  float dot = 0.f;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    float v = (xr[c] - mean) * rstd * to_f(w[c]);
    if (layer_norm) v += to_f(b[c]);
    dot += v * to_f(head[c]);
  }
  dot = block_sum(dot, red);
  if (threadIdx.x == 0) rewards[blockIdx.x] = dot;
}

// Copy page `src` to pages dst[0..n) in every layer (prompt-tail KV into each candidate's page).
template <typename T>
__global__ void k_copy_page(T* pool, long long layer_stride, int page_elems, int src, const int* __restrict__ dst) {
  pdl_entry();
  const int l = blockIdx.y, j = blockIdx.x;
  const T* s = pool + (size_t)l * layer_stride + (size_t)src * page_elems;
  T* t = pool + (size_t)l * layer_stride + (size_t)dst[j] * page_elems;
  for (int i = threadIdx.x; i < page_elems; i += blockDim.x) t[i] = s[i];
}

// bf16 bit patterns -> fp16 bit patterns, in place (exact for |x| in [2^-17, 65504]; smaller
// magnitudes round to the fp16 subnormal grid, larger ones saturate)
__global__ void k_bf16_to_f16(uint16_t* p, size_t n) {
  pdl_entry();
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
    const float v = __uint_as_float((uint32_t)p[i] << 16);
    const f16 h = f_to<f16>(v);
    p[i] = *reinterpret_cast<const uint16_t*>(&h);
  }
}

int threads_for(int d) { return d >= 1024 ? 256 : (d >= 256 ? 128 : 64); }

}  // namespace

sr_status launch_embed(int et, const void* tok_emb, const void* pos_emb, const int* tokens, const int* positions,
                       int M, int d, float* x, cudaStream_t st) {
  if (M == 0) return SR_OK;
  SR_DISPATCH_ET(et, T, (launch_k(k_embed<T>, M, threads_for(d), 0, st, (const T*)tok_emb, (const T*)pos_emb, tokens,
                                                                  positions, d, x)));
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_norm(int et, int norm, const float* x, const void* w, const void* b, float eps, int M, int d,
                      void* out, cudaStream_t st) {
  if (M == 0) return SR_OK;
  const int ln = norm == SR_NORM_LAYER;
  const bool aligned = ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(w) |
                         reinterpret_cast<uintptr_t>(b) | reinterpret_cast<uintptr_t>(out)) & 15) == 0;
  if (d % 4 == 0 && d <= 16 * 1024 && aligned) {
    const int nt = std::max(32, ((d / 16 + 31) / 32) * 32);  // up to four float4 per thread
    SR_DISPATCH_ET(et, T, (launch_k(k_norm_v<T>, M, nt, 0, st, x, (const T*)w, (const T*)b, eps, d, ln, (T*)out)));
  } else {
    SR_DISPATCH_ET(et, T, (launch_k(k_norm<T>, M, threads_for(d), 0, st, x, (const T*)w, (const T*)b, eps, d, ln, (T*)out)));
  }
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_rope_table(float2* tab, int max_pos, int head_dim, double theta, cudaStream_t st) {
  const int n = max_pos * (head_dim / 2);
  launch_k(k_rope_table, (n + 255) / 256, 256, 0, st, tab, max_pos, head_dim / 2, head_dim, theta);
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_rope_store(int et, const float* qkv, int M, const int* positions, const float2* rope, int Hq,
                            int Hkv, int dh, void* q_out, void* k_out, void* v_out, KvSink sink, cudaStream_t st) {
  if (M == 0) return SR_OK;
  const bool aligned = ((reinterpret_cast<uintptr_t>(qkv) | reinterpret_cast<uintptr_t>(rope) |
                         reinterpret_cast<uintptr_t>(q_out) | reinterpret_cast<uintptr_t>(k_out) |
                         reinterpret_cast<uintptr_t>(v_out) | reinterpret_cast<uintptr_t>(sink.pool_layer)) & 15) == 0;
  if (dh % 8 == 0 && aligned) {
    SR_DISPATCH_ET(et, T, (launch_k(k_rope_store_v<T>, M, 256, 0, st, qkv, positions, rope, Hq, Hkv, dh, (T*)q_out,
                                                                (T*)k_out, (T*)v_out, sink)));
  } else {
    SR_DISPATCH_ET(et, T, (launch_k(k_rope_store<T>, M, 128, 0, st, qkv, positions, rope, Hq, Hkv, dh, (T*)q_out,
                                                              (T*)k_out, (T*)v_out, sink)));
  }
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_act(int et, int act, const float* in, int M, int F, void* out, cudaStream_t st) {
  if (M == 0) return SR_OK;
  SR_DISPATCH_ET(et, T, (launch_k(k_act<T>, M, 128, 0, st, in, F, act, (T*)out)));
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_score_head(int et, int norm, const float* x, const int* rows, int n, const void* w, const void* b,
                            float eps, const void* head, int d, float* rewards, cudaStream_t st) {
  if (n == 0) return SR_OK;
  const int ln = norm == SR_NORM_LAYER;
  SR_DISPATCH_ET(et, T, (launch_k(k_score_head<T>, n, threads_for(d), 0, st, x, rows, (const T*)w, (const T*)b, eps, ln,
                                                                       (const T*)head, d, rewards)));
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_copy_page(int et, void* pool, long long layer_stride, int n_layers, int page_elems, int src,
                           const int* dst, int n_dst, cudaStream_t st) {
  if (n_dst == 0) return SR_OK;
  dim3 grid(n_dst, n_layers);
  SR_DISPATCH_ET(et, T, (launch_k(k_copy_page<T>, grid, 256, 0, st, (T*)pool, layer_stride, page_elems, src, dst)));
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_bf16_to_f16(void* p, size_t n, cudaStream_t st) {
  if (n == 0) return SR_OK;
  const size_t blocks = std::min<size_t>((n + 255) / 256, 65535 * 8);
  launch_k(k_bf16_to_f16, (unsigned)blocks, 256, 0, st, reinterpret_cast<uint16_t*>(p), n);
  SR_LAUNCH();
  return SR_OK;
}

}  // namespace sr
