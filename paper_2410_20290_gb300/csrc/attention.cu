// Attention for the generator's decode steps and for reward-model / prompt prefill.
//
// softmax(q k^T / sqrt(dh)) v per query head, GQA (query head j reads kv head j / (Hq / Hkv)),
// causal, optional sliding window -- the attention of the decoder-only models of Section 3.
//
// Decode (k_decode_attn): one CTA per (kv head, slot, KV split of 512 positions); the CTA serves
// the G query heads of its kv head, so each K/V byte is read once per group.  A token's K (and V)
// row of dh elements is read by dh*size/16 threads with one 16-byte load each (fully coalesced
// within the 4 KB (bf16, dh 128) page block of that head); token groups stride over the split;
// scores are reduced with warp shuffles and folded into per-group online-softmax state, merged
// through shared memory at the end.  Splits are a fixed number of positions, so a candidate's
// result does not depend on the batch it is in; a combine kernel merges split partials.
//
// Prefill (k_prefill_attn): flash-attention style over packed variable-length sequences with a
// shared prefix (the prompt's KV) -- 64 query rows x one head per CTA, 64-key blocks staged by
// cp.async, bf16 mma.sync m16n8k16 with fp32 accumulation, online softmax in registers.
#include <algorithm>
#include <mutex>
#include <type_traits>

#include "common.cuh"

namespace sr {
namespace {

constexpr int SPLIT = 512;  // KV positions per decode split

// A row's split count, limited to the `slots` partial slots the launch provides per (row, head).  A
// row needing more (its length exceeds the bound the launch was sized for) keeps only its first `slots`
// splits, and `err` (when given) records the overrun, so no read or write leaves the row's slots.
__device__ __forceinline__ int clamp_splits(int nsplit, int slots, int* err) {
  if (nsplit <= slots) return nsplit;
  if (err) atomicExch(err, 1);
  return slots;
}

template <typename T, int DH, int G>
__global__ void __launch_bounds__(128) k_decode_attn(const T* __restrict__ q, const T* __restrict__ pool,
                                                     const int* __restrict__ pt, int pt_stride,
                                                     const int* __restrict__ slot_ids, const int* __restrict__ lens,
                                                     int Hkv, float scale_log2, int window, int max_splits,
                                                     T* __restrict__ out, float* __restrict__ part,
                                                     int* __restrict__ err) {
  pdl_entry();
  constexpr int VE = 16 / sizeof(T);  // elements per 16-byte vector
  constexpr int TPT = DH / VE;        // threads per token
  constexpr int NG = 128 / TPT;       // token groups per CTA
  static_assert(TPT >= 1 && TPT <= 32 && 32 % TPT == 0, "head_dim / dtype combination");
  __shared__ float s_m[NG][G], s_l[NG][G];
  __shared__ float s_acc[NG][G][DH];

  const int h = blockIdx.x, s = blockIdx.y, split = blockIdx.z;
  const int Hq = Hkv * G;
  const int L = lens[s];
  const int t_lo = window > 0 ? max(0, L - window) : 0;
  const int nsplit = clamp_splits((L - t_lo + SPLIT - 1) / SPLIT, max_splits, err);
  if (split >= nsplit) return;
  const int t_begin = t_lo + split * SPLIT, t_end = min(L, t_begin + SPLIT);
  const int tid = threadIdx.x, grp = tid / TPT, sub = tid % TPT, d0 = sub * VE;
  const int id = slot_ids[s];

  float qv[G][VE];
#pragma unroll
  for (int g = 0; g < G; ++g) {
    const T* qp = q + ((size_t)s * Hq + h * G + g) * DH + d0;
    const uint4 raw = *reinterpret_cast<const uint4*>(qp);
    const T* e = reinterpret_cast<const T*>(&raw);
#pragma unroll
    for (int i = 0; i < VE; ++i) qv[g][i] = to_f(e[i]) * scale_log2;
  }
  float m[G], l[G], acc[G][VE];
#pragma unroll
  for (int g = 0; g < G; ++g) {
    m[g] = -INFINITY;
    l[g] = 0.f;
#pragma unroll
    for (int i = 0; i < VE; ++i) acc[g][i] = 0.f;
  }
  const int* ptrow = pt + (size_t)id * pt_stride;
  const size_t page_elems = (size_t)2 * Hkv * PAGE * DH;
  const size_t v_off = (size_t)Hkv * PAGE * DH;

  // The trip count is the same for every thread of the CTA (base is block-uniform), so the
  // full-warp shuffles below always see all 32 lanes; a group past the end masks its update.
  for (int base = t_begin; base < t_end; base += NG) {
    const int t = base + grp;
    const bool valid = t < t_end;
    float kf[VE], vf[VE];
    if (valid) {
      const int page = ptrow[t / PAGE];
      const T* kp = pool + (size_t)page * page_elems + ((size_t)h * PAGE + (t % PAGE)) * DH + d0;
      const uint4 kr = *reinterpret_cast<const uint4*>(kp);
      const uint4 vr = *reinterpret_cast<const uint4*>(kp + v_off);
      const T* ke = reinterpret_cast<const T*>(&kr);
      const T* ve = reinterpret_cast<const T*>(&vr);
#pragma unroll
      for (int i = 0; i < VE; ++i) kf[i] = to_f(ke[i]), vf[i] = to_f(ve[i]);
    } else {
#pragma unroll
      for (int i = 0; i < VE; ++i) kf[i] = 0.f, vf[i] = 0.f;
    }
#pragma unroll
    for (int g = 0; g < G; ++g) {
      float sc = 0.f;
#pragma unroll
      for (int i = 0; i < VE; ++i) sc = fmaf(qv[g][i], kf[i], sc);
#pragma unroll
      for (int o = TPT / 2; o > 0; o >>= 1) sc += __shfl_xor_sync(0xffffffffu, sc, o);
      if (!valid) continue;
      const float mn = fmaxf(m[g], sc);
      const float corr = exp2f(m[g] - mn);
      const float p = exp2f(sc - mn);
      l[g] = l[g] * corr + p;
#pragma unroll
      for (int i = 0; i < VE; ++i) acc[g][i] = fmaf(acc[g][i], corr, p * vf[i]);
      m[g] = mn;
    }
  }
#pragma unroll
  for (int g = 0; g < G; ++g) {
    if (sub == 0) s_m[grp][g] = m[g], s_l[grp][g] = l[g];
#pragma unroll
    for (int i = 0; i < VE; ++i) s_acc[grp][g][d0 + i] = acc[g][i];
  }
  __syncthreads();
  for (int idx = tid; idx < G * DH; idx += 128) {
    const int g = idx / DH, d = idx % DH;
    float M = -INFINITY;
#pragma unroll
    for (int j = 0; j < NG; ++j) M = fmaxf(M, s_m[j][g]);
    float Lsum = 0.f, O = 0.f;
#pragma unroll
    for (int j = 0; j < NG; ++j) {
      const float w = (s_m[j][g] == -INFINITY) ? 0.f : exp2f(s_m[j][g] - M);
      Lsum += s_l[j][g] * w;
      O += s_acc[j][g][d] * w;
    }
    const int hq = h * G + g;
    if (nsplit == 1) {
      out[((size_t)s * Hq + hq) * DH + d] = f_to<T>(O / Lsum);
    } else {
      float* pp = part + (((size_t)s * Hq + hq) * max_splits + split) * (DH + 2);
      pp[d] = O;
      if (d == 0) pp[DH] = M, pp[DH + 1] = Lsum;
    }
  }
}

// Merges the partial (O, m, l) of each split; with a shared-prefix pass, partial slot 0 holds the
// prefix and the position splits start at slot 1 (sbase = 1, suffix positions from t_min).
template <typename T, int DH>
__global__ void k_decode_combine(const float* __restrict__ part, const int* __restrict__ lens, int Hq, int window,
                                 int max_splits, int t_min, int sbase, T* __restrict__ out, int* __restrict__ err) {
  pdl_entry();
  const int hq = blockIdx.x, s = blockIdx.y, d = threadIdx.x;
  const int L = lens[s];
  const int t_lo = max(t_min, window > 0 ? max(0, L - window) : 0);
  const int nsplit = clamp_splits((L - t_lo + SPLIT - 1) / SPLIT, max_splits - sbase, err);
  if (nsplit <= 1 && (sbase == 0 || nsplit == 1)) return;  // written directly by the attention kernel
  const int total = sbase + nsplit;
  const float* pp = part + ((size_t)s * Hq + hq) * max_splits * (DH + 2);
  float M = -INFINITY;
  for (int j = 0; j < total; ++j) M = fmaxf(M, pp[j * (DH + 2) + DH]);
  float Lsum = 0.f, O = 0.f;
  for (int j = 0; j < total; ++j) {
    const float mj = pp[j * (DH + 2) + DH];
    const float w = (mj == -INFINITY) ? 0.f : exp2f(mj - M);
    Lsum += pp[j * (DH + 2) + DH + 1] * w;
    O += pp[j * (DH + 2) + d] * w;
  }
  out[((size_t)s * Hq + hq) * DH + d] = f_to<T>(O / Lsum);
}

// ------------------------------------------------------------------------------------------------
// prefill attention
// ------------------------------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void cp_async16(void* dst, const void* src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_addr(dst)), "l"(src), "r"(valid ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\ncp.async.wait_group 0;" ::: "memory");
}
__device__ __forceinline__ void ldm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
template <typename T>
__device__ __forceinline__ void mma16816(float* c, uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t b0,
                                         uint32_t b1) {
  if constexpr (std::is_same<T, bf16>::value)
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
  else
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// (a, b) -> packed 16-bit pair (hi) and the packed rounding of the remainders (lo)
template <typename T>
__device__ __forceinline__ void split16(float a, float b, uint32_t& hi, uint32_t& lo) {
  if constexpr (std::is_same<T, bf16>::value) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    const float2 hf = __bfloat1622float2(h);
    const __nv_bfloat162 l = __floats2bfloat162_rn(a - hf.x, b - hf.y);
    hi = *reinterpret_cast<const uint32_t*>(&h);
    lo = *reinterpret_cast<const uint32_t*>(&l);
  } else {
    const __half2 h = __floats2half2_rn(a, b);
    const float2 hf = __half22float2(h);
    const __half2 l = __floats2half2_rn(a - hf.x, b - hf.y);
    hi = *reinterpret_cast<const uint32_t*>(&h);
    lo = *reinterpret_cast<const uint32_t*>(&l);
  }
}
template <typename T>
__device__ __forceinline__ uint32_t pack2(float a, float b) {
  if constexpr (std::is_same<T, bf16>::value) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<const uint32_t*>(&h);
  } else {
    const __half2 h = __floats2half2_rn(fminf(fmaxf(a, -65504.f), 65504.f), fminf(fmaxf(b, -65504.f), 65504.f));
    return *reinterpret_cast<const uint32_t*>(&h);
  }
}


// Tensor-core paged decode attention for 16-bit KV (G <= 8 query heads per kv head).
// One CTA per (kv head, slot, split); warp w takes pages w, w+4, ... of the split.  Each page's K and V
// blocks (16 positions x dh, contiguous in the pool) are copied by a 2-deep per-warp cp.async pipeline
// into padded shared memory; S^T = K Q^T is one m16n8 tile per page (16 positions x 8 head columns,
// the G real heads plus zero padding), the online softmax runs per head column across the 8 lanes
// holding its 16 positions, and O^T += V^T P^T adds dh/16 tiles with P carried as an fp16/bf16
// hi + lo pair.  Warps merge their (m, l, O) through shared memory at the end.
// WPH = 1 (short suffixes): the CTA's four warps take four kv heads of the slot instead, each warp walks
// all pages of its head and writes its result itself -- a quarter of the CTAs, for suffixes of a few pages
// where one CTA per (head, slot) would be mostly launch and merge latency.
template <typename T, int DH, int G, int WPH>
__global__ void __launch_bounds__(128) k_decode_attn_tc(const T* __restrict__ q, const T* __restrict__ pool,
                                                        const int* __restrict__ pt, int pt_stride,
                                                        const int* __restrict__ slot_ids,
                                                        const int* __restrict__ lens, int Hkv, float scale_log2,
                                                        int window, int t_min, int sbase, int max_splits,
                                                        T* __restrict__ out, float* __restrict__ part,
                                                        int* __restrict__ err) {
  pdl_entry();
  static_assert(G >= 1 && G <= 8 && DH % 16 == 0, "shape");
  constexpr int LDS = DH + 8;                  // padded smem row (elements): conflict-free ldmatrix
  constexpr int BLK = PAGE * LDS;              // one K or V page block in smem
  constexpr int WARP_ELEMS = 2 * 2 * BLK + 2 * 8 * PAGE;  // 2 stages x (K, V) + P hi / lo [8][16]
  constexpr int KS = DH / 16;
  extern __shared__ __align__(16) uint8_t smem_raw[];
  T* sw = reinterpret_cast<T*>(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t4 = lane & 3;
  T* wbase = sw + warp * WARP_ELEMS;
  uint16_t* sPh = reinterpret_cast<uint16_t*>(wbase + 4 * BLK);
  uint16_t* sPl = sPh + 8 * PAGE;

  static_assert(WPH == 4 || WPH == 1, "warps per head");
  const int h_raw = WPH == 4 ? (int)blockIdx.x : (int)blockIdx.x * 4 + warp;
  const bool hvalid = h_raw < Hkv;
  const int h = hvalid ? h_raw : 0;
  const int s = blockIdx.y, split = blockIdx.z;
  const int pw = WPH == 4 ? warp : 0;  // this warp's first page of the split; pages step by WPH
  const int Hq = Hkv * G;
  const int L = lens[s];
  const int t_lo = max(t_min, window > 0 ? max(0, L - window) : 0);
  const int nsplit = clamp_splits((L - t_lo + SPLIT - 1) / SPLIT, max_splits - sbase, err);
  if (split >= nsplit) return;
  const int t_begin = t_lo + split * SPLIT, t_end = min(L, t_begin + SPLIT);
  const int p_first = t_begin / PAGE, n_pages = (t_end - 1) / PAGE - p_first + 1;
  const int my_pages = (hvalid && n_pages > pw) ? (n_pages - pw + WPH - 1) / WPH : 0;
  const int* ptrow = pt + (size_t)slot_ids[s] * pt_stride;
  const size_t page_elems = (size_t)2 * Hkv * PAGE * DH;
  const size_t v_off = (size_t)Hkv * PAGE * DH;

  // B fragments of Q^T (k = dim, n = head): lane holds head g (zero when g >= G)
  uint32_t qb[KS][2];
  {
    const T* qh = q + ((size_t)s * Hq + h * G + (g < G ? g : 0)) * DH;
#pragma unroll
    for (int k = 0; k < KS; ++k) {
      qb[k][0] = g < G ? *reinterpret_cast<const uint32_t*>(qh + k * 16 + 2 * t4) : 0u;
      qb[k][1] = g < G ? *reinterpret_cast<const uint32_t*>(qh + k * 16 + 8 + 2 * t4) : 0u;
    }
  }
  auto issue = [&](int i, int stage) {
    const int page = ptrow[p_first + pw + WPH * i];
    const T* srcK = pool + (size_t)page * page_elems + (size_t)h * PAGE * DH;
    const T* srcV = srcK + v_off;
    T* dK = wbase + stage * 2 * BLK;
    T* dV = dK + BLK;
#pragma unroll
    for (int c = lane; c < PAGE * DH / 8; c += 32) {
      const int row = c / (DH / 8), col = (c % (DH / 8)) * 8;
      cp_async16(dK + row * LDS + col, srcK + row * DH + col, true);
      cp_async16(dV + row * LDS + col, srcV + row * DH + col, true);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };

  float m[2] = {-INFINITY, -INFINITY}, l[2] = {0.f, 0.f};
  float o[KS][4];
#pragma unroll
  for (int i = 0; i < KS; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;

  if (my_pages > 0) issue(0, 0);
  if (my_pages > 1) issue(1, 1);
  for (int i = 0; i < my_pages; ++i) {
    const int stage = i & 1;
    if (i + 1 < my_pages) asm volatile("cp.async.wait_group 1;" ::: "memory");
    else asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncwarp();
    const T* sK = wbase + stage * 2 * BLK;
    const T* sV = sK + BLK;
    // S^T = K Q^T : 16 positions x 8 head columns
    float sc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int k = 0; k < KS; ++k) {
      uint32_t a0, a1, a2, a3;
      ldm_x4(smem_addr(sK + (lane & 15) * LDS + k * 16 + (lane >> 4) * 8), a0, a1, a2, a3);
      mma16816<T>(sc, a0, a1, a2, a3, qb[k][0], qb[k][1]);
    }
    const int tok0 = (p_first + pw + WPH * i) * PAGE + g;
    const bool v0 = tok0 >= t_begin && tok0 < t_end, v1 = tok0 + 8 >= t_begin && tok0 + 8 < t_end;
    float corr[2];
#pragma unroll
    for (int j = 0; j < 2; ++j) {      // head columns 2 t4 + j
      const float x0 = v0 ? sc[j] * scale_log2 : -INFINITY;
      const float x1 = v1 ? sc[2 + j] * scale_log2 : -INFINITY;
      float bm = fmaxf(x0, x1);
      bm = fmaxf(bm, __shfl_xor_sync(0xffffffffu, bm, 4));
      bm = fmaxf(bm, __shfl_xor_sync(0xffffffffu, bm, 8));
      bm = fmaxf(bm, __shfl_xor_sync(0xffffffffu, bm, 16));
      const float mn = fmaxf(m[j], bm);
      const float base = (mn == -INFINITY) ? 0.f : mn;
      corr[j] = exp2f(m[j] - base);
      const float p0 = exp2f(x0 - base), p1 = exp2f(x1 - base);
      float ps = p0 + p1;
      ps += __shfl_xor_sync(0xffffffffu, ps, 4);
      ps += __shfl_xor_sync(0xffffffffu, ps, 8);
      ps += __shfl_xor_sync(0xffffffffu, ps, 16);
      l[j] = l[j] * corr[j] + ps;
      m[j] = mn;
      // P[head][position] as hi + lo 16-bit values
      const int hc = 2 * t4 + j;
      uint32_t hi, lo = 0u;
      if constexpr (std::is_same<T, bf16>::value) split16<T>(p0, p1, hi, lo);
      else hi = pack2<T>(p0, p1);
      sPh[hc * PAGE + g] = (uint16_t)(hi & 0xFFFFu);
      sPh[hc * PAGE + g + 8] = (uint16_t)(hi >> 16);
      sPl[hc * PAGE + g] = (uint16_t)(lo & 0xFFFFu);
      sPl[hc * PAGE + g + 8] = (uint16_t)(lo >> 16);
    }
#pragma unroll
    for (int mt = 0; mt < KS; ++mt) {
      o[mt][0] *= corr[0], o[mt][1] *= corr[1];
      o[mt][2] *= corr[0], o[mt][3] *= corr[1];
    }
    __syncwarp();
    // B fragments of P^T (k = position, n = head g)
    const uint32_t bh0 = *reinterpret_cast<const uint32_t*>(sPh + g * PAGE + 2 * t4);
    const uint32_t bh1 = *reinterpret_cast<const uint32_t*>(sPh + g * PAGE + 8 + 2 * t4);
    const uint32_t bl0 = *reinterpret_cast<const uint32_t*>(sPl + g * PAGE + 2 * t4);
    const uint32_t bl1 = *reinterpret_cast<const uint32_t*>(sPl + g * PAGE + 8 + 2 * t4);
    // O^T += V^T P^T : dims in m16 tiles
#pragma unroll
    for (int mt = 0; mt < KS; ++mt) {
      uint32_t a0, a1, a2, a3;
      const int mi = lane >> 3, r = lane & 7;
      ldm_x4_t(smem_addr(sV + (r + ((mi >> 1) << 3)) * LDS + mt * 16 + (mi & 1) * 8), a0, a1, a2, a3);
      mma16816<T>(o[mt], a0, a1, a2, a3, bh0, bh1);
      if constexpr (std::is_same<T, bf16>::value) mma16816<T>(o[mt], a0, a1, a2, a3, bl0, bl1);
    }
    __syncwarp();
    if (i + 2 < my_pages) issue(i + 2, stage);
  }
  // final (O, m, l) of head column j, dim d: the output when the row has one split (after folding in the
  // shared-prefix partial), else the split's partial
  auto emit = [&](int j, int d, float M, float Lsum, float O) {
    const int hq = h * G + j;
    if (nsplit == 1) {
      if (sbase) {  // fold in the shared-prefix pass (partial slot 0, written by the preceding launch)
        const float* p0 = part + ((size_t)s * Hq + hq) * max_splits * (DH + 2);
        const float m0 = p0[DH], Mn = fmaxf(M, m0);
        const float w0 = (m0 == -INFINITY) ? 0.f : exp2f(m0 - Mn), w1 = (M == -INFINITY) ? 0.f : exp2f(M - Mn);
        O = O * w1 + p0[d] * w0;
        Lsum = Lsum * w1 + p0[DH + 1] * w0;
      }
      out[((size_t)s * Hq + hq) * DH + d] = f_to<T>(O / Lsum);
    } else {
      float* pp = part + (((size_t)s * Hq + hq) * max_splits + sbase + split) * (DH + 2);
      pp[d] = O;
      if (d == 0) pp[DH] = M, pp[DH + 1] = Lsum;
    }
  };
  if constexpr (WPH == 1) {
    // the warp's own stage buffers are idle now (every copy was waited for): stage (m, l, O^T) there
    float* wm = reinterpret_cast<float*>(wbase);  // [8] maxima, [8] sums, [DH][8] O^T
    float* wl = wm + 8;
    float* wo = wl + 8;
    if (g == 0) {
#pragma unroll
      for (int j = 0; j < 2; ++j) wm[2 * t4 + j] = m[j], wl[2 * t4 + j] = l[j];
    }
#pragma unroll
    for (int mt = 0; mt < KS; ++mt) {
      wo[(mt * 16 + g) * 8 + 2 * t4] = o[mt][0];
      wo[(mt * 16 + g) * 8 + 2 * t4 + 1] = o[mt][1];
      wo[(mt * 16 + g + 8) * 8 + 2 * t4] = o[mt][2];
      wo[(mt * 16 + g + 8) * 8 + 2 * t4 + 1] = o[mt][3];
    }
    __syncwarp();
    if (!hvalid) return;
    for (int idx = lane; idx < G * DH; idx += 32) {
      const int j = idx / DH, d = idx % DH;
      emit(j, d, wm[j], wl[j], wo[d * 8 + j]);
    }
    return;
  }
  // merge the 4 warps' partial softmax states
  __syncthreads();
  float* sm = reinterpret_cast<float*>(smem_raw);            // [4][8] maxima
  float* sl = sm + 32;                                       // [4][8] sums
  float* so = sl + 32;                                       // [4][DH][8] O^T
  if (g == 0) {
#pragma unroll
    for (int j = 0; j < 2; ++j) sm[warp * 8 + 2 * t4 + j] = m[j], sl[warp * 8 + 2 * t4 + j] = l[j];
  }
#pragma unroll
  for (int mt = 0; mt < KS; ++mt) {
    float* ow = so + (size_t)warp * DH * 8;
    ow[(mt * 16 + g) * 8 + 2 * t4] = o[mt][0];
    ow[(mt * 16 + g) * 8 + 2 * t4 + 1] = o[mt][1];
    ow[(mt * 16 + g + 8) * 8 + 2 * t4] = o[mt][2];
    ow[(mt * 16 + g + 8) * 8 + 2 * t4 + 1] = o[mt][3];
  }
  __syncthreads();
  for (int idx = threadIdx.x; idx < G * DH; idx += 128) {
    const int j = idx / DH, d = idx % DH;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < 4; ++w) M = fmaxf(M, sm[w * 8 + j]);
    float Lsum = 0.f, O = 0.f;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const float wt = (sm[w * 8 + j] == -INFINITY) ? 0.f : exp2f(sm[w * 8 + j] - M);
      Lsum += sl[w * 8 + j] * wt;
      O += so[((size_t)w * DH + d) * 8 + j] * wt;
    }
    emit(j, d, M, Lsum, O);
  }
}

// O[16 x 16*NDP] += P[16 x 64] V[64 x 16*NDP] for one warp: P comes from the S accumulators (C layout of
// m16n8k16), V rows are read transposed from shared memory.  fp16 P is used as is (11-bit significand);
// bf16 P is split into hi + lo pairs (two MMAs) to keep ~16 significand bits.
template <typename T, int NDP>
__device__ __forceinline__ void pv_accumulate(const float (*sc)[4], const T* sV, int ldv, int lane, float (*o)[4]) {
#pragma unroll
  for (int kk = 0; kk < 4; ++kk) {
    uint32_t ah[4], al[4];
    if constexpr (std::is_same<T, bf16>::value) {
      split16<T>(sc[2 * kk][0], sc[2 * kk][1], ah[0], al[0]);
      split16<T>(sc[2 * kk][2], sc[2 * kk][3], ah[1], al[1]);
      split16<T>(sc[2 * kk + 1][0], sc[2 * kk + 1][1], ah[2], al[2]);
      split16<T>(sc[2 * kk + 1][2], sc[2 * kk + 1][3], ah[3], al[3]);
    } else {
      ah[0] = pack2<T>(sc[2 * kk][0], sc[2 * kk][1]);
      ah[1] = pack2<T>(sc[2 * kk][2], sc[2 * kk][3]);
      ah[2] = pack2<T>(sc[2 * kk + 1][0], sc[2 * kk + 1][1]);
      ah[3] = pack2<T>(sc[2 * kk + 1][2], sc[2 * kk + 1][3]);
    }
#pragma unroll
    for (int dp = 0; dp < NDP; ++dp) {
      uint32_t b0, b1, b2, b3;
      ldm_x4_t(smem_addr(sV + (kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8) * ldv + dp * 16 + (lane >> 4) * 8), b0,
               b1, b2, b3);
      mma16816<T>(o[2 * dp], ah[0], ah[1], ah[2], ah[3], b0, b1);
      mma16816<T>(o[2 * dp + 1], ah[0], ah[1], ah[2], ah[3], b2, b3);
      if constexpr (std::is_same<T, bf16>::value) {
        mma16816<T>(o[2 * dp], al[0], al[1], al[2], al[3], b0, b1);
        mma16816<T>(o[2 * dp + 1], al[0], al[1], al[2], al[3], b2, b3);
      }
    }
  }
}

constexpr int BQ = 64, BKV = 64;

template <typename T, int DH, int DV>
__global__ void __launch_bounds__(128) k_prefill_attn(const T* __restrict__ q, const T* __restrict__ k,
                                                      const T* __restrict__ v, const T* __restrict__ kpre,
                                                      const T* __restrict__ vpre, int npre,
                                                      const int* __restrict__ seq_off,
                                                      const int* __restrict__ tile_seq,
                                                      const int* __restrict__ tile_q0, int pos0, int Hq, int Hkv,
                                                      float scale_log2, int window, T* __restrict__ out,
                                                      CachedKeys ck) {
  pdl_entry();
  constexpr int LD = DH + 8, LDV = DV + 8;
  extern __shared__ __align__(16) uint8_t smem_raw[];
  T* sQ = reinterpret_cast<T*>(smem_raw);
  T* sK = sQ + BQ * LD;
  T* sV = sK + BKV * LD;

  const int tile = blockIdx.x, hq = blockIdx.y, dvo = blockIdx.z * DV;
  const int j = tile_seq[tile], q0 = tile_q0[tile];
  const int r0 = seq_off[j], nrows = seq_off[j + 1] - r0;
  const int hk = hq / (Hq / Hkv);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, g = lane >> 2, t4 = lane & 3;
  const size_t qstride = (size_t)Hq * DH, kstride = (size_t)Hkv * DH;

  // Q tile
  for (int c = tid; c < BQ * (DH / 8); c += 128) {
    const int row = c / (DH / 8), col = (c % (DH / 8)) * 8;
    const bool ok = q0 + row < nrows;
    const T* src = ok ? q + (size_t)(r0 + q0 + row) * qstride + (size_t)hq * DH + col : q;
    cp_async16(sQ + row * LD + col, src, ok);
  }

  float o[DV / 8][4];
#pragma unroll
  for (int i = 0; i < DV / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.f, 0.f};
  // cached keys of this sequence (positions pos0 .. pos0 + ncache - 1, paged); its own rows follow them
  const int ncache = ck.pool ? ck.seq_cached[j] : 0;
  const int* cpt = ck.pool ? ck.page_table + (size_t)ck.seq_cand[j] * ck.pt_stride : nullptr;
  const int opos0 = pos0 + ncache;      // position of own row 0
  const int qi_a = q0 + warp * 16 + g;  // query index within the sequence (rows g and g + 8)
  const int qpos[2] = {opos0 + qi_a, opos0 + qi_a + 8};
  const int qpos_min = opos0 + q0;
  const int qpos_max = opos0 + min(nrows, q0 + BQ) - 1;

  const int nb_pre = (npre + BKV - 1) / BKV;
  const int nb_c = (ncache + BKV - 1) / BKV;
  const int own_keys = min(nrows, q0 + BQ);
  const int nb_own = (own_keys + BKV - 1) / BKV;
  const size_t cpage = (size_t)2 * Hkv * PAGE * DH;  // elements per cached page (K and V of every kv head)

  for (int kb = 0; kb < nb_pre + nb_c + nb_own; ++kb) {
    const int seg = kb < nb_pre ? 0 : (kb < nb_pre + nb_c ? 1 : 2);  // prefix, cached, own
    const int kbase = seg == 0 ? kb * BKV : (seg == 1 ? (kb - nb_pre) * BKV : (kb - nb_pre - nb_c) * BKV);
    const int kcount = min(BKV, (seg == 0 ? npre : (seg == 1 ? ncache : own_keys)) - kbase);
    const int kpos0 = seg == 0 ? kbase : (seg == 1 ? pos0 + kbase : opos0 + kbase);
    if (window > 0 && kpos0 + kcount - 1 <= qpos_min - window) continue;  // whole block left of every window
    if (kpos0 > qpos_max) continue;
    __syncthreads();  // previous block's smem reads are done
    if (seg == 1) {
      const T* cpool = reinterpret_cast<const T*>(ck.pool);
      for (int c = tid; c < BKV * (DH / 8); c += 128) {
        const int row = c / (DH / 8), col = (c % (DH / 8)) * 8;
        const bool ok = row < kcount;
        const int t = kbase + row;
        const T* src = ok ? cpool + (size_t)cpt[t / PAGE] * cpage + ((size_t)hk * PAGE + t % PAGE) * DH + col : cpool;
        cp_async16(sK + row * LD + col, src, ok);
      }
      for (int c = tid; c < BKV * (DV / 8); c += 128) {
        const int row = c / (DV / 8), col = (c % (DV / 8)) * 8;
        const bool ok = row < kcount;
        const int t = kbase + row;
        const T* src = ok ? cpool + (size_t)cpt[t / PAGE] * cpage + ((size_t)(Hkv + hk) * PAGE + t % PAGE) * DH + dvo +
                                col
                          : cpool;
        cp_async16(sV + row * LDV + col, src, ok);
      }
    } else {
      const bool is_pre = seg == 0;
      const T* ksrc = is_pre ? kpre : k + (size_t)r0 * kstride;
      const T* vsrc = is_pre ? vpre : v + (size_t)r0 * kstride;
      for (int c = tid; c < BKV * (DH / 8); c += 128) {
        const int row = c / (DH / 8), col = (c % (DH / 8)) * 8;
        const bool ok = row < kcount;
        const T* src = ok ? ksrc + (size_t)(kbase + row) * kstride + (size_t)hk * DH + col : ksrc;
        cp_async16(sK + row * LD + col, src, ok);
      }
      for (int c = tid; c < BKV * (DV / 8); c += 128) {
        const int row = c / (DV / 8), col = (c % (DV / 8)) * 8;
        const bool ok = row < kcount;
        const T* src = ok ? vsrc + (size_t)(kbase + row) * kstride + (size_t)hk * DH + dvo + col : vsrc;
        cp_async16(sV + row * LDV + col, src, ok);
      }
    }
    cp_async_wait_all();
    __syncthreads();

    // S = Q K^T for this warp's 16 rows x 64 keys
    float sc[BKV / 8][4];
#pragma unroll
    for (int i = 0; i < BKV / 8; ++i) sc[i][0] = sc[i][1] = sc[i][2] = sc[i][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < DH / 16; ++kk) {
      uint32_t a0, a1, a2, a3;
      ldm_x4(smem_addr(sQ + (warp * 16 + (lane & 15)) * LD + kk * 16 + (lane >> 4) * 8), a0, a1, a2, a3);
#pragma unroll
      for (int np = 0; np < BKV / 16; ++np) {
        uint32_t b0, b1, b2, b3;
        ldm_x4(smem_addr(sK + (np * 16 + (lane & 7) + ((lane >> 4) << 3)) * LD + kk * 16 + ((lane >> 3) & 1) * 8), b0,
               b1, b2, b3);
        mma16816<T>(sc[2 * np], a0, a1, a2, a3, b0, b1);
        mma16816<T>(sc[2 * np + 1], a0, a1, a2, a3, b2, b3);
      }
    }
    // mask, scale, online softmax
    float bmax[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int nt = 0; nt < BKV / 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int kidx = nt * 8 + 2 * t4 + (e & 1);
        const int r = e >> 1;
        const int kpos = kpos0 + kidx;
        bool ok = kidx < kcount && kpos <= qpos[r];
        if (window > 0) ok = ok && kpos > qpos[r] - window;
        const float x = ok ? sc[nt][e] * scale_log2 : -INFINITY;
        sc[nt][e] = x;
        bmax[r] = fmaxf(bmax[r], x);
      }
    }
    float corr[2], base[2];
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      bmax[r] = fmaxf(bmax[r], __shfl_xor_sync(0xffffffffu, bmax[r], 1));
      bmax[r] = fmaxf(bmax[r], __shfl_xor_sync(0xffffffffu, bmax[r], 2));
      const float mn = fmaxf(mrow[r], bmax[r]);
      base[r] = (mn == -INFINITY) ? 0.f : mn;
      corr[r] = exp2f(mrow[r] - base[r]);
      mrow[r] = mn;
    }
    float psum[2] = {0.f, 0.f};
#pragma unroll
    for (int nt = 0; nt < BKV / 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float p = exp2f(sc[nt][e] - base[e >> 1]);
        sc[nt][e] = p;
        psum[e >> 1] += p;
      }
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) lrow[r] = lrow[r] * corr[r] + psum[r];
#pragma unroll
    for (int i = 0; i < DV / 8; ++i) {
      o[i][0] *= corr[0], o[i][1] *= corr[0];
      o[i][2] *= corr[1], o[i][3] *= corr[1];
    }
    // O += P V (bf16 carries P as a hi + lo pair so the probabilities are not the coarsest operand)
    pv_accumulate<T, DV / 16>(sc, sV, LDV, lane, o);
  }
  // finish: full row sums across the quad, normalise, store
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 1);
    lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 2);
  }
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int qi = qi_a + 8 * r;
    if (qi >= nrows) continue;
    const float inv = lrow[r] > 0.f ? 1.f / lrow[r] : 0.f;
    T* dst = out + (size_t)(r0 + qi) * qstride + (size_t)hq * DH + dvo;
#pragma unroll
    for (int nt = 0; nt < DV / 8; ++nt)
      *reinterpret_cast<uint32_t*>(dst + nt * 8 + 2 * t4) = pack2<T>(o[nt][2 * r] * inv, o[nt][2 * r + 1] * inv);
  }
}


// Shared-prompt prefix of decode attention.  Positions [0, S) sit in pages every live candidate shares
// (the prompt's full pages), so instead of each candidate re-reading them, one CTA takes the queries of
// several candidates for up to 4 query heads of one kv head (NW warps of 16 query rows each) and runs
// flash attention over the prefix keys with mma.sync; each 64-position K/V block is loaded once per CTA
// through a 2-stage cp.async pipeline.  The result is written unnormalised as partial slot 0 (O, m, l in
// the decode kernels' log2-scaled convention); the suffix kernel folds it into its result when a row's
// suffix is one split, k_decode_combine merges it with the split partials otherwise.
// No causal mask is needed (every prefix position precedes the query); a window masks per row.
template <typename T, int DH, int G, int NW>
__global__ void __launch_bounds__(NW * 32, 2) k_prefix_attn(const T* __restrict__ q, const T* __restrict__ pool,
                                                     const int* __restrict__ pt, int pt_stride,
                                                     const int* __restrict__ slot_ids,
                                                     const int* __restrict__ lens, int n, int S, int Hkv,
                                                     float scale_log2, int window, int max_splits,
                                                     float* __restrict__ part) {
  pdl_entry();
  constexpr int HPC = G < 4 ? G : 4;       // query heads per CTA
  constexpr int CPC = NW / HPC;            // 16-candidate blocks per CTA (one warp per 16 rows)
  constexpr int NT = NW * 32;
  constexpr int LD = DH + 8;
  extern __shared__ __align__(16) uint8_t smem_raw[];
  T* sQ = reinterpret_cast<T*>(smem_raw);
  T* sKV = sQ + 16 * NW * LD;              // [stage][K | V][64][LD]
  const int Hq = Hkv * G;
  const int h = blockIdx.y / (G / HPC), hg0 = (blockIdx.y % (G / HPC)) * HPC;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, g = lane >> 2, t4 = lane & 3;
  const int wh = warp % HPC, wc = warp / HPC;
  const int hq = h * G + hg0 + wh;
  const int s0 = blockIdx.x * 16 * CPC + wc * 16;       // this warp's first candidate row
  const int* prow = pt + (size_t)slot_ids[0] * pt_stride;   // the prompt pages, identical in every row
  const size_t page_elems = (size_t)2 * Hkv * PAGE * DH;
  const size_t v_off = (size_t)Hkv * PAGE * DH;

  // Q rows: warp w's 16 rows are (candidates s0 .. s0 + 15, head hq)
  for (int c = lane; c < 16 * (DH / 8); c += 32) {
    const int row = c / (DH / 8), col = (c % (DH / 8)) * 8;
    const bool ok = s0 + row < n;
    const T* src = ok ? q + ((size_t)(s0 + row) * Hq + hq) * DH + col : q;
    cp_async16(sQ + (warp * 16 + row) * LD + col, src, ok);
  }
  const int nb = (S + BKV - 1) / BKV;
  auto issue = [&](int kb) {
    T* dK = sKV + (size_t)(kb & 1) * 2 * BKV * LD;
    T* dV = dK + BKV * LD;
    const int kbase = kb * BKV, kcount = min(BKV, S - kbase);
    for (int c = tid; c < BKV * (DH / 8); c += NT) {
      const int row = c / (DH / 8), col = (c % (DH / 8)) * 8;
      const bool ok = row < kcount;
      const int key = kbase + row;
      const T* src = ok ? pool + (size_t)prow[key / PAGE] * page_elems + ((size_t)h * PAGE + key % PAGE) * DH + col
                        : pool;
      cp_async16(dK + row * LD + col, src, ok);
      cp_async16(dV + row * LD + col, ok ? src + v_off : pool, ok);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };

  float o[DH / 8][4];
#pragma unroll
  for (int i = 0; i < DH / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.f, 0.f};
  int qpos[2];
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int row = s0 + g + 8 * r;
    qpos[r] = row < n ? lens[row] - 1 : 0;
  }
  issue(0);  // also completes the Q copies (same commit group)
  for (int kb = 0; kb < nb; ++kb) {
    if (kb + 1 < nb) {
      issue(kb + 1);
      asm volatile("cp.async.wait_group 1;" ::: "memory");
    } else {
      asm volatile("cp.async.wait_group 0;" ::: "memory");
    }
    __syncthreads();
    const T* sK = sKV + (size_t)(kb & 1) * 2 * BKV * LD;
    const T* sV = sK + BKV * LD;
    const int kbase = kb * BKV, kcount = min(BKV, S - kbase);
    float sc[BKV / 8][4];
#pragma unroll
    for (int i = 0; i < BKV / 8; ++i) sc[i][0] = sc[i][1] = sc[i][2] = sc[i][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < DH / 16; ++kk) {
      uint32_t a0, a1, a2, a3;
      ldm_x4(smem_addr(sQ + (warp * 16 + (lane & 15)) * LD + kk * 16 + (lane >> 4) * 8), a0, a1, a2, a3);
#pragma unroll
      for (int np = 0; np < BKV / 16; ++np) {
        uint32_t b0, b1, b2, b3;
        ldm_x4(smem_addr(sK + (np * 16 + (lane & 7) + ((lane >> 4) << 3)) * LD + kk * 16 + ((lane >> 3) & 1) * 8), b0,
               b1, b2, b3);
        mma16816<T>(sc[2 * np], a0, a1, a2, a3, b0, b1);
        mma16816<T>(sc[2 * np + 1], a0, a1, a2, a3, b2, b3);
      }
    }
    float bmax[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int nt = 0; nt < BKV / 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int kidx = nt * 8 + 2 * t4 + (e & 1);
        const int r = e >> 1;
        bool ok = kidx < kcount;
        if (window > 0) ok = ok && kbase + kidx > qpos[r] - window;
        const float x = ok ? sc[nt][e] * scale_log2 : -INFINITY;
        sc[nt][e] = x;
        bmax[r] = fmaxf(bmax[r], x);
      }
    }
    float corr[2], base[2];
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      bmax[r] = fmaxf(bmax[r], __shfl_xor_sync(0xffffffffu, bmax[r], 1));
      bmax[r] = fmaxf(bmax[r], __shfl_xor_sync(0xffffffffu, bmax[r], 2));
      const float mn = fmaxf(mrow[r], bmax[r]);
      base[r] = (mn == -INFINITY) ? 0.f : mn;
      corr[r] = exp2f(mrow[r] - base[r]);
      mrow[r] = mn;
    }
    float psum[2] = {0.f, 0.f};
#pragma unroll
    for (int nt = 0; nt < BKV / 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float p = exp2f(sc[nt][e] - base[e >> 1]);
        sc[nt][e] = p;
        psum[e >> 1] += p;
      }
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) lrow[r] = lrow[r] * corr[r] + psum[r];
#pragma unroll
    for (int i = 0; i < DH / 8; ++i) {
      o[i][0] *= corr[0], o[i][1] *= corr[0];
      o[i][2] *= corr[1], o[i][3] *= corr[1];
    }
    pv_accumulate<T, DH / 16>(sc, sV, LD, lane, o);
    __syncthreads();  // this stage is refilled by the next iteration's issue
  }
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 1);
    lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 2);
  }
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int row = s0 + g + 8 * r;
    if (row >= n) continue;
    float* pp = part + ((size_t)row * Hq + hq) * max_splits * (DH + 2);   // partial slot 0
#pragma unroll
    for (int nt = 0; nt < DH / 8; ++nt) {
      pp[nt * 8 + 2 * t4] = o[nt][2 * r];
      pp[nt * 8 + 2 * t4 + 1] = o[nt][2 * r + 1];
    }
    if (t4 == 0) pp[DH] = mrow[r], pp[DH + 1] = lrow[r];
  }
}

// fp32 models: straightforward prefill attention, one block per (query row, head); scores of the
// row's visible keys live in shared memory.
__global__ void k_prefill_attn_f32(const float* __restrict__ q, const float* __restrict__ k,
                                   const float* __restrict__ v, const float* __restrict__ kpre,
                                   const float* __restrict__ vpre, int npre, const int* __restrict__ seq_off,
                                   int n_seq, int pos0, int Hq, int Hkv, int dh, float scale, int window,
                                   float* __restrict__ out, CachedKeys ck) {
  pdl_entry();
  extern __shared__ float sc[];
  __shared__ float red[32];
  const int r = blockIdx.x, hq = blockIdx.y, hk = hq / (Hq / Hkv);
  int j = 0;
  while (j + 1 < n_seq && seq_off[j + 1] <= r) ++j;
  // keys: npre prefix keys, ncache cached keys (paged, positions pos0 ..), then the sequence's own rows
  const int ncache = ck.pool ? ck.seq_cached[j] : 0;
  const int* cpt = ck.pool ? ck.page_table + (size_t)ck.seq_cand[j] * ck.pt_stride : nullptr;
  const float* cpool = reinterpret_cast<const float*>(ck.pool);
  const size_t cpage = (size_t)2 * Hkv * PAGE * dh;
  const int r0 = seq_off[j], qi = r - r0, qpos = pos0 + ncache + qi;
  const int nk = npre + ncache + qi + 1;
  auto key_row = [&](int t, int which) -> const float* {  // which 0: K, 1: V
    if (t < npre) return (which ? vpre : kpre) + ((size_t)t * Hkv + hk) * dh;
    if (t < npre + ncache) {
      const int c = t - npre;
      return cpool + (size_t)cpt[c / PAGE] * cpage + ((size_t)(which * Hkv + hk) * PAGE + c % PAGE) * dh;
    }
    return (which ? v : k) + ((size_t)(r0 + t - npre - ncache) * Hkv + hk) * dh;
  };
  const float* qr = q + ((size_t)r * Hq + hq) * dh;
  float mx = -INFINITY;
  for (int t = threadIdx.x; t < nk; t += blockDim.x) {
    const int kpos = t < npre ? t : pos0 + (t - npre);
    const float* kr = key_row(t, 0);
    float s = 0.f;
    for (int d = 0; d < dh; ++d) s = fmaf(qr[d], kr[d], s);
    s *= scale;
    if (window > 0 && kpos <= qpos - window) s = -INFINITY;
    sc[t] = s;
    mx = fmaxf(mx, s);
  }
  mx = warp_max(mx);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = mx;
  __syncthreads();
  mx = -INFINITY;
  for (int w = 0; w < (int)(blockDim.x >> 5); ++w) mx = fmaxf(mx, red[w]);
  float sum = 0.f;
  for (int t = threadIdx.x; t < nk; t += blockDim.x) {
    const float p = expf(sc[t] - mx);
    sc[t] = p;
    sum += p;
  }
  sum = block_sum(sum, red);
  for (int d = threadIdx.x; d < dh; d += blockDim.x) {
    float o = 0.f;
    for (int t = 0; t < nk; ++t) o = fmaf(sc[t], key_row(t, 1)[d], o);
    out[((size_t)r * Hq + hq) * dh + d] = o / sum;
  }
}

template <typename T, int DH, int G>
sr_status decode_attn_tc_t(const void* q, const void* pool, const int* pt, int pt_stride, const int* ids,
                           const int* lens, int b, int Hkv, int window, void* out, float* part, int max_splits,
                           int shared_pos, int max_len, cudaStream_t st, int* err) {
  // with a shared prefix: slot 0 of the partials is the prefix pass, position splits follow
  const int sbase = shared_pos > 0 ? 1 : 0;
  const int t_min = shared_pos;
  if (sbase) {
    if (!part) return set_err(SR_ERR_INVALID_ARG, "decode attention: partial buffer missing for the prefix pass");
    // eight warps (128 query rows) per CTA share each staged K/V block
    constexpr int NW = 8, HPC = G < 4 ? G : 4, CPC = NW / HPC;
    const size_t psmem = (size_t)(16 * NW + 4 * BKV) * (DH + 8) * sizeof(T);
    static bool pattr = false;
    if (!pattr) {
      SR_CUDA(cudaFuncSetAttribute(k_prefix_attn<T, DH, G, NW>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)psmem));
      pattr = true;
    }
    launch_k(k_prefix_attn<T, DH, G, NW>, dim3((b + 16 * CPC - 1) / (16 * CPC), Hkv * (G / HPC)), NW * 32, psmem, st, 
        (const T*)q, (const T*)pool, pt, pt_stride, ids, lens, b, shared_pos, Hkv,
        1.4426950408889634f / sqrtf((float)DH), window, max_splits, part);
    SR_LAUNCH();
  }
  constexpr int LDS = DH + 8;
  const size_t smem = std::max<size_t>((size_t)4 * (2 * 2 * PAGE * LDS + 2 * 8 * PAGE) * sizeof(T),
                                       (size_t)(64 + 4 * DH * 8) * sizeof(float));
  static bool attr_set = false;
  if (!attr_set) {
    SR_CUDA(cudaFuncSetAttribute(k_decode_attn_tc<T, DH, G, 4>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    SR_CUDA(cudaFuncSetAttribute(k_decode_attn_tc<T, DH, G, 1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    attr_set = true;
  }
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)DH);
  // suffixes of at most 8 pages: one warp per (kv head, slot)
  int span = max_len - t_min;
  if (window > 0) span = std::min(span, window);
  if (max_len > 0 && span <= 8 * PAGE && max_splits - sbase == 1) {
    dim3 grid((Hkv + 3) / 4, b, 1);
    launch_k(k_decode_attn_tc<T, DH, G, 1>, grid, 128, smem, st, (const T*)q, (const T*)pool, pt, pt_stride, ids, lens,
             Hkv, scale_log2, window, t_min, sbase, max_splits, (T*)out, part, err);
  } else {
    dim3 grid(Hkv, b, max_splits - sbase);
    launch_k(k_decode_attn_tc<T, DH, G, 4>, grid, 128, smem, st, (const T*)q, (const T*)pool, pt, pt_stride, ids, lens,
             Hkv, scale_log2, window, t_min, sbase, max_splits, (T*)out, part, err);
  }
  SR_LAUNCH();
  if (max_splits - sbase > 1) {  // some row has several position splits (a lone split merges the prefix itself)
    launch_k(k_decode_combine<T, DH>, dim3(Hkv * G, b), DH, 0, st, part, lens, Hkv * G, window, max_splits, t_min, sbase,
             (T*)out, err);
    SR_LAUNCH();
  }
  return SR_OK;
}

template <typename T, int DH, int G>
sr_status decode_attn_t(const void* q, const void* pool, const int* pt, int pt_stride, const int* ids,
                        const int* lens, int b, int Hkv, int window, void* out, float* part, int max_splits,
                        cudaStream_t st, int* err) {
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)DH);
  dim3 grid(Hkv, b, max_splits);
  launch_k(k_decode_attn<T, DH, G>, grid, 128, 0, st, (const T*)q, (const T*)pool, pt, pt_stride, ids, lens, Hkv,
           scale_log2, window, max_splits, (T*)out, part, err);
  SR_LAUNCH();
  if (max_splits > 1) {
    launch_k(k_decode_combine<T, DH>, dim3(Hkv * G, b), DH, 0, st, part, lens, Hkv * G, window, max_splits, 0, 0,
             (T*)out, err);
    SR_LAUNCH();
  }
  return SR_OK;
}

template <typename T, int DH, int DV>
sr_status prefill_t(const void* q, const void* k, const void* v, const void* kpre, const void* vpre, int npre,
                    const int* seq_off, const int* tile_seq, const int* tile_q0, int n_tiles, int pos0, int Hq,
                    int Hkv, int window, void* out, cudaStream_t st, CachedKeys ck) {
  const size_t smem = (size_t)(BQ * (DH + 8) + BKV * (DH + 8) + BKV * (DV + 8)) * sizeof(T);
  static bool attr_set = false;
  if (!attr_set) {
    SR_CUDA(cudaFuncSetAttribute(k_prefill_attn<T, DH, DV>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    attr_set = true;
  }
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)DH);
  dim3 grid(n_tiles, Hq, DH / DV);
  launch_k(k_prefill_attn<T, DH, DV>, grid, 128, smem, st, (const T*)q, (const T*)k, (const T*)v, (const T*)kpre,
           (const T*)vpre, npre, seq_off, tile_seq, tile_q0, pos0, Hq, Hkv, scale_log2, window, (T*)out, ck);
  SR_LAUNCH();
  return SR_OK;
}

}  // namespace

int decode_attention_max_splits(int max_len) { return max_len <= 0 ? 1 : (max_len + SPLIT - 1) / SPLIT; }
int decode_attention_slots(int max_len, int window, int shared_pos) {
  const int lo = shared_pos > 0 ? shared_pos : 0;
  const int span = window > 0 ? std::min(max_len - lo, window) : max_len - lo;
  return (shared_pos > 0 ? 1 : 0) + decode_attention_max_splits(span);
}
size_t decode_attention_part_floats(int b, int Hq, int dh, int max_splits) {
  return (size_t)b * Hq * max_splits * (dh + 2);
}

sr_status launch_decode_attention(int et, const void* q, const void* pool_layer, const int* pt, int pt_stride,
                                  const int* ids, const int* lens, int b, int Hq, int Hkv, int dh, int window,
                                  void* out, float* part, int max_splits, cudaStream_t st, int shared_pos,
                                  int max_len, int* err) {
  if (b == 0) return SR_OK;
  const int G = Hq / Hkv;
  if (Hq % Hkv) return set_err(SR_ERR_UNSUPPORTED, "decode attention: n_heads %% n_kv_heads != 0");
  if (max_splits > 1 && !part) return set_err(SR_ERR_INVALID_ARG, "decode attention: split partial buffer missing");
#define SR_DEC(T, D, GG)                                                                                          \
  if (dh == D && G == GG)                                                                                         \
    return decode_attn_t<T, D, GG>(q, pool_layer, pt, pt_stride, ids, lens, b, Hkv, window, out, part, max_splits, \
                                   st, err);
#define SR_DECT(T, D, GG)                                                                                          \
  if (dh == D && G == GG)                                                                                            \
    return decode_attn_tc_t<T, D, GG>(q, pool_layer, pt, pt_stride, ids, lens, b, Hkv, window, out, part, max_splits, \
                                      shared_pos, max_len, st, err);
  if (et == SR_DT_F16) {
    SR_DECT(f16, 128, 4) SR_DECT(f16, 128, 1) SR_DECT(f16, 128, 2) SR_DECT(f16, 128, 8)
    SR_DECT(f16, 64, 1) SR_DECT(f16, 64, 4) SR_DECT(f16, 32, 1)
  } else if (et == SR_DT_BF16) {
    SR_DECT(bf16, 128, 4) SR_DECT(bf16, 128, 1) SR_DECT(bf16, 64, 1)
  } else {
    if (shared_pos > 0) return set_err(SR_ERR_UNSUPPORTED, "decode attention: shared-prefix pass needs 16-bit KV");
    SR_DEC(float, 32, 1) SR_DEC(float, 32, 2) SR_DEC(float, 32, 4) SR_DEC(float, 64, 1) SR_DEC(float, 128, 1)
    SR_DEC(float, 8, 1) SR_DEC(float, 8, 2) SR_DEC(float, 8, 4)
  }
#undef SR_DEC
#undef SR_DECT
  return set_err(SR_ERR_UNSUPPORTED, "decode attention: head_dim %d with group %d (type %d) not built", dh, G, et);
}

sr_status launch_prefill_attention_f32(const float* q, const float* k, const float* v, const float* kpre,
                                       const float* vpre, int npre, const int* seq_off, int n_seq, int rows, int pos0,
                                       int Hq, int Hkv, int dh, int window, float* out, cudaStream_t st,
                                       CachedKeys ck, int max_cached) {
  if (rows == 0) return SR_OK;
  const int max_keys = npre + max_cached + rows;
  const size_t smem = (size_t)max_keys * sizeof(float);
  if (smem > 200 * 1024) return set_err(SR_ERR_UNSUPPORTED, "fp32 prefill attention: %d keys too many", max_keys);
  static size_t attr = 48 * 1024;
  if (smem > attr) {
    SR_CUDA(cudaFuncSetAttribute(k_prefill_attn_f32, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    attr = smem;
  }
  launch_k(k_prefill_attn_f32, dim3(rows, Hq), 128, smem, st, q, k, v, kpre, vpre, npre, seq_off, n_seq, pos0, Hq, Hkv, dh,
           1.f / sqrtf((float)dh), window, out, ck);
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_prefill_attention(int et, const void* q, const void* k, const void* v, const void* kpre,
                                   const void* vpre, int npre, const int* seq_off, int n_seq, const int* tile_seq,
                                   const int* tile_q0, int n_tiles, int pos0, int Hq, int Hkv, int dh, int window,
                                   void* out, cudaStream_t st, CachedKeys ck) {
  (void)n_seq;
  if (n_tiles == 0) return SR_OK;
  if (Hq % Hkv) return set_err(SR_ERR_UNSUPPORTED, "prefill attention: n_heads %% n_kv_heads != 0");
  if (et != SR_DT_F16 && et != SR_DT_BF16) return set_err(SR_ERR_INVALID_ARG, "prefill attention: 16-bit types only");
#define SR_PRE(T)                                                                                                      \
  switch (dh) {                                                                                                        \
    case 32: return prefill_t<T, 32, 32>(q, k, v, kpre, vpre, npre, seq_off, tile_seq, tile_q0, n_tiles, pos0, Hq, Hkv, \
                                         window, out, st, ck);                                                            \
    case 64: return prefill_t<T, 64, 64>(q, k, v, kpre, vpre, npre, seq_off, tile_seq, tile_q0, n_tiles, pos0, Hq, Hkv, \
                                         window, out, st, ck);                                                            \
    case 128: return prefill_t<T, 128, 128>(q, k, v, kpre, vpre, npre, seq_off, tile_seq, tile_q0, n_tiles, pos0, Hq, \
                                            Hkv, window, out, st, ck);                                                    \
    case 256: return prefill_t<T, 256, 128>(q, k, v, kpre, vpre, npre, seq_off, tile_seq, tile_q0, n_tiles, pos0, Hq, \
                                            Hkv, window, out, st, ck);                                                    \
  }
  if (et == SR_DT_F16) {
    SR_PRE(f16)
  } else {
    SR_PRE(bf16)
  }
#undef SR_PRE
  return set_err(SR_ERR_UNSUPPORTED, "prefill attention: head_dim %d not built", dh);
}

}  // namespace sr

// -------------------------------------------------------------------------------------------------
// Decode attention without allocation.
//
// Some callers cannot allocate device memory at call time: code running inside a pre-sized memory
// budget (an inference server that reserves all of the GPU's memory up front), allocator-free
// embeddings, or callers holding locks under which an allocation could block.  For them the split
// partials of decode attention live in this fixed device array instead of a buffer allocated per
// call, next to one int the kernels set when a row is longer than the caller's bound.  Every GPU
// that loads the library holds the array (8 MiB) until the process exits.
// -------------------------------------------------------------------------------------------------
namespace sr {
namespace {

constexpr size_t kStaticPartFloats = (size_t)1 << 21;  // 8 MiB of fp32 split partials
static __device__ __align__(256) float g_static_part[kStaticPartFloats];
static __device__ __align__(256) int g_static_err;      // 1 after a row needed more splits than max_len allows

constexpr int kMaxDevices = 64;
std::mutex g_static_mu;
struct StaticScratch {
  float* part = nullptr;  // device address of g_static_part
  int* err = nullptr;     // device address of g_static_err
};
StaticScratch g_static[kMaxDevices];  // per device ordinal

// In host code `g_static_part` and `g_static_err` name host-side stand-ins, not device memory, so
// their device addresses are looked up once per device (with that device current) and cached.
sr_status static_scratch(StaticScratch* out) {
  int dev = 0;
  SR_CUDA(cudaGetDevice(&dev));
  if (dev < 0 || dev >= kMaxDevices) return set_err(SR_ERR_UNSUPPORTED, "device ordinal %d out of range", dev);
  std::lock_guard<std::mutex> lock(g_static_mu);
  if (!g_static[dev].part) {
    void *p = nullptr, *e = nullptr;
    cudaError_t r = cudaGetSymbolAddress(&p, g_static_part);
    if (r == cudaSuccess) r = cudaGetSymbolAddress(&e, g_static_err);
    if (r != cudaSuccess)
      return set_err(SR_ERR_CUDA, "cudaGetSymbolAddress(static decode-attention scratch): %s", cudaGetErrorString(r));
    g_static[dev].part = static_cast<float*>(p);
    g_static[dev].err = static_cast<int*>(e);
  }
  *out = g_static[dev];
  return SR_OK;
}

}  // namespace
}  // namespace sr

extern "C" sr_status sr_k_decode_attention_static(int dtype, const void* q, const void* pool,
                                                  const int32_t* page_table, int pt_stride, const int32_t* orig_ids,
                                                  const int32_t* lens, int b, int n_heads, int n_kv_heads,
                                                  int head_dim, int window, int max_len, void* out, void* stream) {
  using namespace sr;
  if (!q || !pool || !page_table || !orig_ids || !lens || !out)
    return set_err(SR_ERR_INVALID_ARG, "sr_k_decode_attention_static: null argument");
  if (b < 0 || n_kv_heads < 1 || n_heads < 1 || head_dim < 1 || max_len < 1)
    return set_err(SR_ERR_INVALID_ARG, "sr_k_decode_attention_static: bad shape");
  const int splits = decode_attention_max_splits(window > 0 ? std::min(max_len, window) : max_len);
  const size_t need = splits > 1 ? decode_attention_part_floats(b, n_heads, head_dim, splits) : 0;
  if (need > kStaticPartFloats)
    return set_err(SR_ERR_INVALID_ARG,
                   "sr_k_decode_attention_static: %zu scratch floats needed (b=%d, heads=%d, head_dim=%d, %d "
                   "splits of %d positions) but the static scratch holds %zu",
                   need, b, n_heads, head_dim, splits, SPLIT, kStaticPartFloats);
  if (b == 0) return SR_OK;
  StaticScratch sc;
  SR_TRY(static_scratch(&sc));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // the error word keeps the last call's value: clear it before the kernels run
  SR_CUDA(cudaMemsetAsync(sc.err, 0, sizeof(int), st));
  SR_TRY(launch_decode_attention(dtype, q, pool, page_table, pt_stride, orig_ids, lens, b, n_heads, n_kv_heads,
                                 head_dim, window, out, splits > 1 ? sc.part : nullptr, splits, st, 0, max_len,
                                 sc.err));
  // lens[] lives on the device, so whether every length was within max_len is known only once the
  // kernels ran: read their flag back (this synchronises `stream`)
  int h_err = 0;
  SR_CUDA(cudaMemcpyAsync(&h_err, sc.err, sizeof(int), cudaMemcpyDeviceToHost, st));
  SR_CUDA(cudaStreamSynchronize(st));
  if (h_err)
    return set_err(SR_ERR_INVALID_ARG,
                   "sr_k_decode_attention_static: a length in lens[] exceeds max_len = %d by more than its last "
                   "512-position split; the rows concerned kept only their first %d split(s) and `out` is not valid",
                   max_len, splits);
  return SR_OK;
}
