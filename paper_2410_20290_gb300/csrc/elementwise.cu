// Row-wise transformer pieces: embedding, RMSNorm / LayerNorm (fused with the cast to the GEMM
// operand type), RoPE (rotate-half pairing) fused with the KV-cache append into the paged pool,
// the fp32-path activations, the reward model's scalar head and page copies.
//
// These compute the per-position parts of the generator and reward model of Section 3; the KV
// append is the paged cache of the Section 5 engine ("pre-allocates the corresponding KV cache").
#include <algorithm>

#include "common.cuh"

namespace sr {
namespace {

template <typename T>
__global__ void k_embed(const T* __restrict__ tok_emb, const T* __restrict__ pos_emb, const int* __restrict__ tokens,
                        const int* __restrict__ positions, int d, float* __restrict__ x) {
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

// cos/sin of p * theta^(-2i/dh), evaluated in double precision and rounded once.
__global__ void k_rope_table(float2* tab, int max_pos, int half, int dh, double theta) {
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
  const int r = blockIdx.x;
  const int pos = positions[r];
  const int half = dh / 2;
  const int W = (Hq + 2 * Hkv) * dh;
  const float* row = qkv + (size_t)r * W;
  T* pk = nullptr;
  T* pv = nullptr;
  if (sink.pool_layer) {
    const int seq = sink.row_seq ? sink.row_seq[r] : 0;
    const int page = sink.page_table[(size_t)seq * sink.pt_stride + pos / PAGE];
    T* base = reinterpret_cast<T*>(sink.pool_layer) + (size_t)page * 2 * Hkv * PAGE * dh + (size_t)(pos % PAGE) * dh;
    pk = base;
    pv = base + (size_t)Hkv * PAGE * dh;
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

__device__ __forceinline__ float silu_d(float x) { return x / (1.f + expf(-x)); }
__device__ __forceinline__ float gelu_d(float x) {
  return 0.5f * x * (1.f + tanhf(0.7978845608028654f * (x + 0.044715f * x * x * x)));
}

// fp32 path: gated activations read gate/up interleaved in blocks of 32 columns.
template <typename T>
__global__ void k_act(const float* __restrict__ in, int F, int act, T* __restrict__ out) {
  const int r = blockIdx.x;
  for (int j = threadIdx.x; j < F; j += blockDim.x) {
    float v;
    if (act == SR_ACT_GELU) {
      v = gelu_d(in[(size_t)r * F + j]);
    } else {
      const float* row = in + (size_t)r * 2 * F;
      const int blk = j / 32, o = j % 32;
      const float g = row[blk * 64 + o], u = row[blk * 64 + 32 + o];
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
  const int l = blockIdx.y, j = blockIdx.x;
  const T* s = pool + (size_t)l * layer_stride + (size_t)src * page_elems;
  T* t = pool + (size_t)l * layer_stride + (size_t)dst[j] * page_elems;
  for (int i = threadIdx.x; i < page_elems; i += blockDim.x) t[i] = s[i];
}

// bf16 bit patterns -> fp16 bit patterns, in place (exact for |x| in [2^-17, 65504]; smaller
// magnitudes round to the fp16 subnormal grid, larger ones saturate)
__global__ void k_bf16_to_f16(uint16_t* p, size_t n) {
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
  SR_DISPATCH_ET(et, T, (k_embed<T><<<M, threads_for(d), 0, st>>>((const T*)tok_emb, (const T*)pos_emb, tokens,
                                                                  positions, d, x)));
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_norm(int et, int norm, const float* x, const void* w, const void* b, float eps, int M, int d,
                      void* out, cudaStream_t st) {
  if (M == 0) return SR_OK;
  const int ln = norm == SR_NORM_LAYER;
  SR_DISPATCH_ET(et, T, (k_norm<T><<<M, threads_for(d), 0, st>>>(x, (const T*)w, (const T*)b, eps, d, ln, (T*)out)));
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_rope_table(float2* tab, int max_pos, int head_dim, double theta, cudaStream_t st) {
  const int n = max_pos * (head_dim / 2);
  k_rope_table<<<(n + 255) / 256, 256, 0, st>>>(tab, max_pos, head_dim / 2, head_dim, theta);
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_rope_store(int et, const float* qkv, int M, const int* positions, const float2* rope, int Hq,
                            int Hkv, int dh, void* q_out, void* k_out, void* v_out, KvSink sink, cudaStream_t st) {
  if (M == 0) return SR_OK;
  SR_DISPATCH_ET(et, T, (k_rope_store<T><<<M, 128, 0, st>>>(qkv, positions, rope, Hq, Hkv, dh, (T*)q_out, (T*)k_out,
                                                            (T*)v_out, sink)));
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_act(int et, int act, const float* in, int M, int F, void* out, cudaStream_t st) {
  if (M == 0) return SR_OK;
  SR_DISPATCH_ET(et, T, (k_act<T><<<M, 128, 0, st>>>(in, F, act, (T*)out)));
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_score_head(int et, int norm, const float* x, const int* rows, int n, const void* w, const void* b,
                            float eps, const void* head, int d, float* rewards, cudaStream_t st) {
  if (n == 0) return SR_OK;
  const int ln = norm == SR_NORM_LAYER;
  SR_DISPATCH_ET(et, T, (k_score_head<T><<<n, threads_for(d), 0, st>>>(x, rows, (const T*)w, (const T*)b, eps, ln,
                                                                       (const T*)head, d, rewards)));
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_copy_page(int et, void* pool, long long layer_stride, int n_layers, int page_elems, int src,
                           const int* dst, int n_dst, cudaStream_t st) {
  if (n_dst == 0) return SR_OK;
  dim3 grid(n_dst, n_layers);
  SR_DISPATCH_ET(et, T, (k_copy_page<T><<<grid, 256, 0, st>>>((T*)pool, layer_stride, page_elems, src, dst)));
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_bf16_to_f16(void* p, size_t n, cudaStream_t st) {
  if (n == 0) return SR_OK;
  const size_t blocks = std::min<size_t>((n + 255) / 256, 65535 * 8);
  k_bf16_to_f16<<<(unsigned)blocks, 256, 0, st>>>(reinterpret_cast<uint16_t*>(p), n);
  SR_LAUNCH();
  return SR_OK;
}

}  // namespace sr
