// Next-token sampling (Section 3, Eq. auto-regressive) by the Gumbel-max trick; the noise, the logarithm and the
// per-id step are in sampling.cuh.
//
// k_sample: one block per row of materialised logits; each thread handles groups of 4 consecutive vocabulary ids
// (one Philox call per group); block argmax with ties to the lowest id; NaN logits count as -inf.  The two
// logarithms are taken only for ids that can still beat the thread's running maximum (gumbel_step's exact
// test on the uniform), which after the first few ids of a thread is a small fraction.
//
// k_sample_reduce: the same decision from the per-64-id records the LM-head GEMM's sampling epilogue writes
// (best perturbed logit, its id and raw logit, log-sum-exp partial), reduced in id order.
//
// With `lp_sum` set, the same pass also takes ln sum_v exp(logit_v) of the raw logits (online max / rescaled
// sum) and adds ln p(token) = logit_token - that to lp_sum[candidate id]: the running ln p(Y | X) of the
// self-likelihood reward of Section 5.3 (temperature 1, no EOS bias).
#include "common.cuh"
#include "sampling.cuh"

namespace sr {
namespace {

constexpr int THREADS = 512;

__global__ void __launch_bounds__(THREADS) k_sample(const float* __restrict__ logits, long long ld, int V,
                                                    const int* __restrict__ orig_ids, const int* __restrict__ steps,
                                                    uint32_t k0, uint32_t k1, float temperature, float eos_bias,
                                                    int eos_id, int* __restrict__ tokens_out, int* tok_hist,
                                                    int max_new, int* lens, int* status, double* lp_sum,
                                                    const int* __restrict__ n_rows) {
  pdl_entry();
  if (n_rows && (int)blockIdx.x >= *n_rows) return;  // a slot past the live count the step started with
  __shared__ float s_best[THREADS / 32];
  __shared__ int s_idx[THREADS / 32];
  __shared__ float s_m[THREADS / 32], s_s[THREADS / 32];
  float lm = -__int_as_float(0x7f800000), ls = 0.f;  // running max and sum exp(l - max) of the raw logits
  const int r = blockIdx.x;
  const int id = orig_ids[r];
  const int step = steps ? steps[r] : lens[id];
  const float* row = logits + (size_t)r * ld;
  const GumbelParams gp{k0, k1, __fdiv_rn(1.0f, temperature), eos_bias, eos_id};
  float best = -__int_as_float(0x7f800000);
  int best_v = 0x7fffffff;
  const int groups = (V + 3) / 4;
  const bool vec = ((reinterpret_cast<uintptr_t>(row) & 15) == 0) && (V % 4 == 0);
  for (int gi = threadIdx.x; gi < groups; gi += THREADS) {
    const int v0 = gi * 4;
    float l[4];
    if (vec) {
      const float4 t = reinterpret_cast<const float4*>(row)[gi];
      l[0] = t.x, l[1] = t.y, l[2] = t.z, l[3] = t.w;
    } else {
#pragma unroll
      for (int j = 0; j < 4; ++j) l[j] = (v0 + j < V) ? row[v0 + j] : 0.f;
    }
    const uint4 w = philox4x32_10(make_uint4((uint32_t)gi, (uint32_t)id, (uint32_t)step, 0u), k0, k1);
    const uint32_t words[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int v = v0 + j;
      if (v >= V) break;
      if (lp_sum) lse_step(l[j], lm, ls);
      gumbel_step(l[j], v, words[j], gp, best, best_v);  // v increases per thread: ties keep the lowest id
    }
  }
  // block argmax, ties to the lowest id
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ob = __shfl_xor_sync(0xffffffffu, best, o);
    const int ov = __shfl_xor_sync(0xffffffffu, best_v, o);
    if (ob > best || (ob == best && ov < best_v)) best = ob, best_v = ov;
  }
  if ((threadIdx.x & 31) == 0) s_best[threadIdx.x >> 5] = best, s_idx[threadIdx.x >> 5] = best_v;
  if (lp_sum) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float om = __shfl_xor_sync(0xffffffffu, lm, o), os = __shfl_xor_sync(0xffffffffu, ls, o);
      lse_merge(lm, ls, om, os);
    }
    if ((threadIdx.x & 31) == 0) s_m[threadIdx.x >> 5] = lm, s_s[threadIdx.x >> 5] = ls;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < THREADS / 32; ++w)
      if (s_best[w] > best || (s_best[w] == best && s_idx[w] < best_v)) best = s_best[w], best_v = s_idx[w];
    if (best_v == 0x7fffffff) best_v = 0;  // every perturbed logit was -inf / NaN: id 0
    if (lp_sum) {
      float M = s_m[0], S = s_s[0];
      for (int w = 1; w < THREADS / 32; ++w) lse_merge(M, S, s_m[w], s_s[w]);
      const float lt = row[best_v];
      const double lp = (lt != lt || M == -__int_as_float(0x7f800000)) ? -INFINITY
                                                                         : (double)lt - ((double)M + log((double)S));
      lp_sum[id] += lp;
    }
    if (tokens_out) tokens_out[r] = best_v;
    if (tok_hist) {
      tok_hist[(size_t)id * max_new + step] = best_v;
      lens[id] = step + 1;
      if (best_v == eos_id || step + 1 >= max_new) status[id] = 1;  // completed, not yet scored
    }
  }
}

constexpr int RTHREADS = 256;

// One block per row: the records of the row's vocabulary chunks in increasing id order per thread, then the
// block; ties of the perturbed maximum go to the lowest id, as in k_sample.
__global__ void __launch_bounds__(RTHREADS) k_sample_reduce(const SampleRec* __restrict__ rec, int n_chunks,
                                                            const int* __restrict__ orig_ids, int eos_id,
                                                            int* __restrict__ tokens_out, int* tok_hist, int max_new,
                                                            int* lens, int* status, double* lp_sum,
                                                            const int* __restrict__ n_rows) {
  pdl_entry();
  if (n_rows && (int)blockIdx.x >= *n_rows) return;
  __shared__ float s_best[RTHREADS / 32], s_a[RTHREADS / 32], s_m[RTHREADS / 32], s_s[RTHREADS / 32];
  __shared__ int s_idx[RTHREADS / 32];
  const int r = blockIdx.x;
  const int id = orig_ids[r];
  const int step = lens[id];
  const SampleRec* row = rec + (size_t)r * n_chunks;
  float best = -__int_as_float(0x7f800000), best_a = 0.f, m = -__int_as_float(0x7f800000), s = 0.f;
  int best_v = 0x7fffffff;
  for (int c = threadIdx.x; c < n_chunks; c += RTHREADS) {
    const float4 r0 = reinterpret_cast<const float4*>(row + c)[0];
    const float4 r1 = reinterpret_cast<const float4*>(row + c)[1];
    const int v = __float_as_int(r0.y);
    if (r0.x > best || (r0.x == best && v < best_v)) best = r0.x, best_v = v, best_a = r0.z;
    if (lp_sum) lse_merge(m, s, r0.w, r1.x);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ob = __shfl_xor_sync(0xffffffffu, best, o), oa = __shfl_xor_sync(0xffffffffu, best_a, o);
    const int ov = __shfl_xor_sync(0xffffffffu, best_v, o);
    if (ob > best || (ob == best && ov < best_v)) best = ob, best_v = ov, best_a = oa;
    if (lp_sum) {
      const float om = __shfl_xor_sync(0xffffffffu, m, o), os = __shfl_xor_sync(0xffffffffu, s, o);
      lse_merge(m, s, om, os);
    }
  }
  const int warp = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) s_best[warp] = best, s_idx[warp] = best_v, s_a[warp] = best_a, s_m[warp] = m, s_s[warp] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < RTHREADS / 32; ++w) {
      if (s_best[w] > best || (s_best[w] == best && s_idx[w] < best_v)) best = s_best[w], best_v = s_idx[w], best_a = s_a[w];
      if (lp_sum) lse_merge(m, s, s_m[w], s_s[w]);
    }
    if (best_v == 0x7fffffff) best_v = 0, best_a = row[0].a0;  // every perturbed logit was -inf / NaN: id 0
    if (lp_sum) {
      const float lt = best_a;
      const double lp = (lt != lt || m == -__int_as_float(0x7f800000)) ? -INFINITY
                                                                         : (double)lt - ((double)m + log((double)s));
      lp_sum[id] += lp;
    }
    if (tokens_out) tokens_out[r] = best_v;
    if (tok_hist) {
      tok_hist[(size_t)id * max_new + step] = best_v;
      lens[id] = step + 1;
      if (best_v == eos_id || step + 1 >= max_new) status[id] = 1;  // completed, not yet scored
    }
  }
}

}  // namespace

sr_status launch_sample_reduce(const SampleRec* rec, int n_chunks, int b, const int* orig_ids, int eos_id,
                               int* tokens_out, int* tok_hist, int max_new, int* lens, int* status, cudaStream_t st,
                               double* lp_sum, const int* n_rows) {
  if (b == 0) return SR_OK;
  launch_k(k_sample_reduce, b, RTHREADS, 0, st, rec, n_chunks, orig_ids, eos_id, tokens_out, tok_hist, max_new, lens,
           status, lp_sum, n_rows);
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_sample(const float* logits, long long ld, int b, int V, const int* orig_ids, const int* steps,
                        uint64_t seed, float temperature, float eos_bias, int eos_id, int* tokens_out, int* tok_hist,
                        int max_new, int* lens, int* status, cudaStream_t st, double* lp_sum, const int* n_rows) {
  if (b == 0) return SR_OK;
  if (!(temperature > 0.f)) return set_err(SR_ERR_INVALID_ARG, "temperature must be > 0");
  launch_k(k_sample, b, THREADS, 0, st, logits, ld, V, orig_ids, steps, (uint32_t)(seed & 0xFFFFFFFFu),
                                  (uint32_t)(seed >> 32), temperature, eos_bias, eos_id, tokens_out, tok_hist, max_new,
                                  lens, status, lp_sum, n_rows);
  SR_LAUNCH();
  return SR_OK;
}

}  // namespace sr
