// Next-token sampling (Section 3, Eq. auto-regressive) by the Gumbel-max trick:
//   y = argmax_v  (logit_v + eos_bias [v == eos]) * (1/T) + g_v,   g_v = -ln(-ln u_v),
// which draws y from softmax((logit + eos_bias e_eos) / T).  The uniforms come from
// Philox4x32-10 (Salmon et al., SC'11) keyed (seed_lo, seed_hi) with counter
// (v / 4, candidate id, token index, 0), word v % 4, so a candidate's draws do not depend on
// its batch slot.  u = ((word >> 9) + 1/2) 2^-23 is exact in float32.
//
// The logarithm is this file's own: Cody-Waite reduction x = m 2^e, m in [sqrt(1/2), sqrt(2)],
// and ln m = 2 atanh(s), s = (m-1)/(m+1), as the odd series through s^13, evaluated with one
// IEEE round-to-nearest operation per step (__fadd_rn / __fmul_rn / __fdiv_rn, no contraction)
// so its bits are fixed by the method, not by the compiler.
//
// One block per row; each thread handles groups of 4 consecutive vocabulary ids (one Philox
// call per group); block argmax with ties to the lowest id; NaN logits count as -inf.  The two
// logarithms are taken only for ids that can still beat the thread's running maximum (an exact
// test on the uniform, see k_sample), which after the first few ids of a thread is a small fraction.
//
// With `lp_sum` set, the same pass also takes ln sum_v exp(logit_v) of the raw logits (online
// max / rescaled sum) and adds ln p(token) = logit_token - that to lp_sum[candidate id]: the running
// ln p(Y | X) of the self-likelihood reward of Section 5.3 (temperature 1, no EOS bias).
#include "common.cuh"

namespace sr {
namespace {

__device__ __forceinline__ uint32_t mulhi32(uint32_t a, uint32_t b) { return __umulhi(a, b); }

__device__ __forceinline__ uint4 philox(uint4 c, uint32_t k0, uint32_t k1) {
  const uint32_t M0 = 0xD2511F53u, M1 = 0xCD9E8D57u;
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r) k0 += 0x9E3779B9u, k1 += 0xBB67AE85u;
    const uint32_t hi0 = mulhi32(M0, c.x), lo0 = M0 * c.x;
    const uint32_t hi1 = mulhi32(M1, c.z), lo1 = M1 * c.z;
    c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
  }
  return c;
}

// ln x for positive normal float32 x (see the file header for the method)
__device__ __forceinline__ float series_log(float x) {
  const uint32_t bits = __float_as_uint(x);
  int e = (int)(bits >> 23) - 127;
  uint32_t mb = (bits & 0x7FFFFFu) | 0x3F800000u;
  float m = __uint_as_float(mb);
  if (mb > 0x3FB504F3u) {  // m > sqrt(2): halve (exact)
    m = __fmul_rn(m, 0.5f);
    e += 1;
  }
  const float s = __fdiv_rn(__fadd_rn(m, -1.0f), __fadd_rn(m, 1.0f));
  const float z = __fmul_rn(s, s);
  float p = 0x1.3b13b2p-3f;                         // 2/13
  p = __fadd_rn(0x1.745d18p-3f, __fmul_rn(z, p));   // 2/11
  p = __fadd_rn(0x1.c71c72p-3f, __fmul_rn(z, p));   // 2/9
  p = __fadd_rn(0x1.24924ap-2f, __fmul_rn(z, p));   // 2/7
  p = __fadd_rn(0x1.99999ap-2f, __fmul_rn(z, p));   // 2/5
  p = __fadd_rn(0x1.555556p-1f, __fmul_rn(z, p));   // 2/3
  const float r = __fmul_rn(z, p);
  const float lnm = __fadd_rn(__fadd_rn(s, s), __fmul_rn(s, r));
  const float ef = (float)e;
  return __fadd_rn(__fmul_rn(ef, 0x1.62e4p-1f), __fadd_rn(__fmul_rn(ef, 0x1.7f7d1cp-20f), lnm));
}

__device__ __forceinline__ float gumbel_of(uint32_t word) {
  const float u = __fmul_rn(__fadd_rn((float)(word >> 9), 0.5f), 0x1p-23f);
  const float l1 = series_log(u);
  return -series_log(-l1);
}

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
  const float inv_t = __fdiv_rn(1.0f, temperature);
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
    const uint4 w = philox(make_uint4((uint32_t)gi, (uint32_t)id, (uint32_t)step, 0u), k0, k1);
    const uint32_t words[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int v = v0 + j;
      if (v >= V) break;
      float a = l[j];
      if (lp_sum && a == a) {
        if (a > lm) {
          ls = ls * expf(lm - a) + 1.f;
          lm = a;
        } else {
          ls += expf(a - lm);
        }
      }
      if (v == eos_id) a = __fadd_rn(a, eos_bias);
      if (a != a) a = -__int_as_float(0x7f800000);
      const float ap = __fmul_rn(a, inv_t);
      // Exact skip of ids that cannot win.  g(u) = -ln(-ln u) reaches best - ap only if -ln u <= exp(ap - best),
      // and -ln u >= 1 - u, so 1 - u > exp(ap - best + margin) proves g(u) < best - ap - margin.  The margin
      // (1e-4 + 5 ulp of best) exceeds the error of the two series logarithms (< 1e-5 for |g| <= 17, checked
      // over all 2^23 uniforms) plus the roundings of ap - best and of z, so a skipped id's z is strictly below
      // this thread's best and below the row's maximum; 1 - u is exact in float32 and the 1.001 factor covers
      // __expf's error.
      const float one_minus_u = __fmul_rn((float)(0x7FFFFFu - (words[j] >> 9)) + 0.5f, 0x1p-23f);
      if (one_minus_u > __expf(ap - best + (1e-4f + fabsf(best) * 6e-7f)) * 1.001f) continue;
      const float z = __fadd_rn(ap, gumbel_of(words[j]));
      if (z > best) best = z, best_v = v;  // v increases per thread, so ">" keeps the lowest id
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
      const float mn = fmaxf(lm, om);
      ls = (mn == -__int_as_float(0x7f800000)) ? 0.f : ls * expf(lm - mn) + os * expf(om - mn);
      lm = mn;
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
      for (int w = 1; w < THREADS / 32; ++w) {
        const float mn = fmaxf(M, s_m[w]);
        S = (mn == -__int_as_float(0x7f800000)) ? 0.f : S * expf(M - mn) + s_s[w] * expf(s_m[w] - mn);
        M = mn;
      }
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

}  // namespace

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
