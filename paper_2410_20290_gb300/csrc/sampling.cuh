// Next-token sampling arithmetic shared by the sampling kernel and the LM-head GEMM's sampling epilogue
// (Section 3, Eq. auto-regressive): Gumbel-max over temperature-scaled logits,
//   y = argmax_v  (logit_v + eos_bias [v == eos]) * (1/T) + g_v,   g_v = -ln(-ln u_v),
// which draws y from softmax((logit + eos_bias e_eos) / T).  The uniforms come from Philox4x32-10
// (Salmon et al., SC'11) keyed (seed_lo, seed_hi) with counter (v / 4, candidate id, token index, 0),
// word v % 4, so a candidate's draws do not depend on its batch slot.  u = ((word >> 9) + 1/2) 2^-23
// is exact in float32.
//
// The logarithm is this file's own: Cody-Waite reduction x = m 2^e, m in [sqrt(1/2), sqrt(2)], and
// ln m = 2 atanh(s), s = (m-1)/(m+1), as the odd series through s^13, evaluated with one IEEE
// round-to-nearest operation per step (__fadd_rn / __fmul_rn / __fdiv_rn, no contraction) so its bits
// are fixed by the method, not by the compiler.
#pragma once

#include <cstdint>

namespace sr {

__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1) {
  const uint32_t M0 = 0xD2511F53u, M1 = 0xCD9E8D57u;
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r) k0 += 0x9E3779B9u, k1 += 0xBB67AE85u;
    const uint32_t hi0 = __umulhi(M0, c.x), lo0 = M0 * c.x;
    const uint32_t hi1 = __umulhi(M1, c.z), lo1 = M1 * c.z;
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

struct GumbelParams {
  uint32_t k0, k1;  // Philox key: the seed's low and high words
  float inv_t;      // 1 / T, rounded once
  float eos_bias;
  int eos_id;
};

// The perturbed logit of an id that passed the skip test (out of line: the logarithms are taken for a few ids per
// row, and inlining them at every id of an unrolled scan would only grow the code the SM has to fetch).
static __device__ __noinline__ float gumbel_z(float ap, uint32_t word) { return __fadd_rn(ap, gumbel_of(word)); }

// One id of a Gumbel-max scan in increasing id order: raises (best, best_v) when the perturbed logit of v is
// larger (">" keeps the lowest id on ties) and returns whether it did.  NaN logits count as -inf.
//
// Exact skip of ids that cannot win: g(u) = -ln(-ln u) reaches best - ap only if -ln u <= exp(ap - best), and
// -ln u >= 1 - u, so 1 - u > exp(ap - best + margin) proves g(u) < best - ap - margin.  The margin (1e-4 + 5 ulp
// of best) exceeds the error of the two series logarithms (< 1e-5 for |g| <= 17, checked over all 2^23
// uniforms) plus the roundings of ap - best and of z, so a skipped id's z is strictly below the running best and
// below the row's maximum; 1 - u is exact in float32 and the 1.001 factor covers __expf's error.
__device__ __forceinline__ bool gumbel_step(float a, int v, uint32_t word, const GumbelParams& p, float& best,
                                            int& best_v) {
  if (v == p.eos_id) a = __fadd_rn(a, p.eos_bias);
  if (a != a) a = -__int_as_float(0x7f800000);
  const float ap = __fmul_rn(a, p.inv_t);
  const float one_minus_u = __fmul_rn((float)(0x7FFFFFu - (word >> 9)) + 0.5f, 0x1p-23f);
  if (one_minus_u > __expf(ap - best + (1e-4f + fabsf(best) * 6e-7f)) * 1.001f) return false;
  const float z = gumbel_z(ap, word);
  if (z > best) {
    best = z, best_v = v;
    return true;
  }
  return false;
}

// The skip test of gumbel_step alone, against a threshold `ref` at most the running best (a snapshot taken
// before a run of ids, so the tests of the run do not wait on one another): true = the id cannot win.
__device__ __forceinline__ bool gumbel_skip(float a, int v, uint32_t word, const GumbelParams& p, float ref) {
  if (v == p.eos_id) a = __fadd_rn(a, p.eos_bias);
  if (a != a) return true;
  const float ap = __fmul_rn(a, p.inv_t);
  const float one_minus_u = __fmul_rn((float)(0x7FFFFFu - (word >> 9)) + 0.5f, 0x1p-23f);
  return one_minus_u > __expf(ap - ref + (1e-4f + fabsf(ref) * 6e-7f)) * 1.001f;
}

// Online log-sum-exp of raw logits (NaN skipped): running maximum m and sum s of exp(a - m).
__device__ __forceinline__ void lse_step(float a, float& m, float& s) {
  if (a != a) return;
  if (a > m) {
    s = s * expf(m - a) + 1.f;
    m = a;
  } else {
    s += expf(a - m);
  }
}

__device__ __forceinline__ void lse_merge(float& m, float& s, float om, float os) {
  const float mn = fmaxf(m, om);
  s = (mn == -__int_as_float(0x7f800000)) ? 0.f : s * expf(m - mn) + os * expf(om - mn);
  m = mn;
}

}  // namespace sr
