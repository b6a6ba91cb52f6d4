// Row-wise transformer pieces: embedding, RMSNorm / LayerNorm (fused with the cast to the GEMM
// operand type), RoPE (rotate-half pairing) fused with the KV-cache append into the paged pool,
// the fp32-path activations, the reward model's scalar head and page copies.
//
// These compute the per-position parts of the generator and reward model of Section 3; the KV
// append is the paged cache of the Section 5 engine ("pre-allocates the corresponding KV cache").
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

int threads_for(int d) { return d >= 1024 ? 256 : (d >= 256 ? 128 : 64); }

}  // namespace

sr_status launch_embed(int dtype, const void* tok_emb, const void* pos_emb, const int* tokens, const int* positions,
                       int M, int d, float* x, cudaStream_t st) {
  if (M == 0) return SR_OK;
  if (dtype == SR_DT_BF16)
    k_embed<bf16><<<M, threads_for(d), 0, st>>>((const bf16*)tok_emb, (const bf16*)pos_emb, tokens, positions, d, x);
  else
    k_embed<float><<<M, threads_for(d), 0, st>>>((const float*)tok_emb, (const float*)pos_emb, tokens, positions, d,
                                                 x);
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_norm(int dtype, int norm, const float* x, const void* w, const void* b, float eps, int M, int d,
                      void* out, cudaStream_t st) {
  if (M == 0) return SR_OK;
  const int ln = norm == SR_NORM_LAYER;
  if (dtype == SR_DT_BF16)
    k_norm<bf16><<<M, threads_for(d), 0, st>>>(x, (const bf16*)w, (const bf16*)b, eps, d, ln, (bf16*)out);
  else
    k_norm<float><<<M, threads_for(d), 0, st>>>(x, (const float*)w, (const float*)b, eps, d, ln, (float*)out);
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_rope_table(float2* tab, int max_pos, int head_dim, double theta, cudaStream_t st) {
  const int n = max_pos * (head_dim / 2);
  k_rope_table<<<(n + 255) / 256, 256, 0, st>>>(tab, max_pos, head_dim / 2, head_dim, theta);
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_rope_store(int dtype, const float* qkv, int M, const int* positions, const float2* rope, int Hq,
                            int Hkv, int dh, void* q_out, void* k_out, void* v_out, KvSink sink, cudaStream_t st) {
  if (M == 0) return SR_OK;
  if (dtype == SR_DT_BF16)
    k_rope_store<bf16><<<M, 128, 0, st>>>(qkv, positions, rope, Hq, Hkv, dh, (bf16*)q_out, (bf16*)k_out,
                                          (bf16*)v_out, sink);
  else
    k_rope_store<float><<<M, 128, 0, st>>>(qkv, positions, rope, Hq, Hkv, dh, (float*)q_out, (float*)k_out,
                                           (float*)v_out, sink);
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_act(int dtype, int act, const float* in, int M, int F, void* out, cudaStream_t st) {
  if (M == 0) return SR_OK;
  if (dtype == SR_DT_BF16)
    k_act<bf16><<<M, 128, 0, st>>>(in, F, act, (bf16*)out);
  else
    k_act<float><<<M, 128, 0, st>>>(in, F, act, (float*)out);
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_score_head(int dtype, int norm, const float* x, const int* rows, int n, const void* w,
                            const void* b, float eps, const void* head, int d, float* rewards, cudaStream_t st) {
  if (n == 0) return SR_OK;
  const int ln = norm == SR_NORM_LAYER;
  if (dtype == SR_DT_BF16)
    k_score_head<bf16><<<n, threads_for(d), 0, st>>>(x, rows, (const bf16*)w, (const bf16*)b, eps, ln,
                                                     (const bf16*)head, d, rewards);
  else
    k_score_head<float><<<n, threads_for(d), 0, st>>>(x, rows, (const float*)w, (const float*)b, eps, ln,
                                                      (const float*)head, d, rewards);
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_copy_page(int dtype, void* pool, long long layer_stride, int n_layers, int page_elems, int src,
                           const int* dst, int n_dst, cudaStream_t st) {
  if (n_dst == 0) return SR_OK;
  dim3 grid(n_dst, n_layers);
  if (dtype == SR_DT_BF16)
    k_copy_page<bf16><<<grid, 256, 0, st>>>((bf16*)pool, layer_stride, page_elems, src, dst);
  else
    k_copy_page<float><<<grid, 256, 0, st>>>((float*)pool, layer_stride, page_elems, src, dst);
  SR_LAUNCH();
  return SR_OK;
}

}  // namespace sr
