// Attention for the generator's decode steps and for reward-model / prompt prefill.
//
// softmax(q k^T / sqrt(dh)) v per query head, GQA (query head j reads kv head j / (Hq / Hkv)),
// causal, optional sliding window -- the attention of the decoder-only models of Section 3.
//
// Decode, default for 16-bit KV with head_dim 128 and 8 kv heads: k_prefix_attn reads the prompt pages every
// candidate shares once per 128 query rows (mma.sync, partial slot 0), then k_decode_stream -- one persistent
// CTA per SM, each streaming an equal share of all (row, page) work through a TMA-fed ring of whole pages,
// one mma.sync consumer warp per kv head, rows cut by a share boundary merged in CTA order by their last
// finisher (no inter-CTA wait) -- folds the prefix partial into each row's result.
//
// Decode, other shapes and SR_ATTN_STREAM=0 (k_decode_attn_tc for 16-bit KV with mma.sync, k_decode_attn for
// fp32 KV): one CTA per (kv head, slot, KV split of 512 positions); the CTA serves
// the G query heads of its kv head, so each K/V byte is read once per group.  A token's K (and V)
// row of dh elements is read by dh*size/16 threads with one 16-byte load each (fully coalesced
// within the 4 KB (bf16, dh 128) page block of that head); token groups stride over the split;
// scores are reduced with warp shuffles and folded into per-group online-softmax state, merged
// through shared memory at the end.  Splits are a fixed number of positions, so a candidate's
// result does not depend on the batch it is in; a combine kernel merges split partials.
//
// Prefill (k_prefill_attn): flash-attention style over packed variable-length sequences with a
// shared prefix (the prompt's KV) and, for the reward model with its cache, cached keys read from pages --
// 64 query rows x one head per CTA, 64-key blocks staged by cp.async, 16-bit mma.sync m16n8k16 with fp32
// accumulation, online softmax in registers.  Opt-in tcgen05 forms of the prefix pass and the prefill
// (SR_PREFIX_TC=1, SR_PREFILL_TC=1) keep S and O in TMEM; they are parity-tested and measured slower.
#include <algorithm>
#include <mutex>
#include <type_traits>

#include "common.cuh"
#include "tma.cuh"

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

// ------------------------------------------------------------------------------------------------
// Streaming paged decode attention (16-bit KV, head_dim 128, 8 kv heads, G query heads per kv head).
//
// All (row, page) work of one launch is laid out row by row (row s contributes the pages of its positions
// [t_lo, L)) and cut into gridDim.x contiguous shares of (almost) equal page counts; one persistent CTA per
// SM walks its share in order, so short and long rows alike keep every SM's copy stream full and no row
// pays a launch or pipeline fill of its own.  Warp 8 (one lane) is the producer: per page it issues four
// 128-byte-swizzled TMA copies (K and V of all 8 kv heads, each as two 64-column halves, 64 KB) into a
// 3-stage ring.  Warps 0..7 are the consumers, warp h serving kv head h: S^T = K Q^T per page with
// mma.sync (16 positions x 8 head columns: the G query heads, zero-padded), the online softmax over the
// 8 lanes holding a head column, and O^T += V^T P^T, exactly as the per-row kernel does.  A row whose pages
// lie inside the share is finalised by the CTA (folding in the shared-prefix partial when there is one).
// A row cut by a share boundary leaves (O, m, l) partials, at most two per CTA (its first and last
// segment); each consumer warp counts its finished segment on a per-(row, kv head) counter and the last
// one merges the row's partials in a fixed order (prefix, then the CTAs in order), so the result does not
// depend on which CTA finishes last, and resets the counter.  No CTA waits on another.
constexpr int ST_HKV = 8, ST_DH = 128, ST_STAGES = 3;
constexpr int ST_TILE = ST_HKV * PAGE * 64 * 2;  // one 64-column half of a page's K or V: 16 KB
constexpr int ST_STAGE = 4 * ST_TILE;             // K lo, K hi, V lo, V hi
constexpr int ST_THREADS = (ST_HKV + 1) * 32;
constexpr int ST_ROWS_MAX = MAX_BATCH;
constexpr size_t ST_SMEM = 1024 + (size_t)ST_STAGES * ST_STAGE + (ST_ROWS_MAX + 4) * sizeof(int) +
                           (size_t)ST_HKV * 2 * 8 * PAGE * sizeof(uint16_t) + 2 * ST_STAGES * sizeof(uint64_t) + 16;

struct StreamArgs {
  const int* pt;
  int pt_stride;
  const int* slot_ids;
  const int* lens;
  int b, window, t_min, max_splits;
  float scale_log2;
  const float* prefix_part;  // prefix partials (slot 0 of [b][Hq][max_splits][DH + 2]) or nullptr
  float* seg_part;           // [gridDim.x][2][Hq][DH + 2]
  int* seg_cnt;              // [b][8], zero between launches
  int* err;                  // set to 10 when a bounded wait expired
};

// byte offset of (row r, 16-byte chunk c) in a 128-byte-row tile written by TMA with 128-byte swizzle
__device__ __forceinline__ uint32_t swz128(int r, int c) { return (uint32_t)(r * 128 + ((c ^ (r & 7)) << 4)); }

__device__ __forceinline__ void st_row_range(const StreamArgs& a, int s, int& t_lo, int& L, int& p_first,
                                             int& n_pages) {
  L = a.lens[s];
  t_lo = max(a.t_min, a.window > 0 ? max(0, L - a.window) : 0);
  p_first = t_lo / PAGE;
  n_pages = L > t_lo ? (L - 1) / PAGE - p_first + 1 : 0;
}

// first page index of CTA c's share of `total` pages
__device__ __forceinline__ long long st_share(long long total, int c, int C) { return total * c / C; }
__device__ __forceinline__ int st_cta_of(long long u, long long total, int C) {
  int i = (int)(u * C / total);
  while (i + 1 < C && st_share(total, i + 1, C) <= u) ++i;
  while (i > 0 && st_share(total, i, C) > u) --i;
  return i;
}

template <typename T, int G>
__global__ void __launch_bounds__(ST_THREADS, 1)
    k_decode_stream(const __grid_constant__ CUtensorMap tm, const T* __restrict__ q, T* __restrict__ out,
                    StreamArgs a) {
  static_assert(G >= 1 && G <= 8, "query heads per kv head");
  constexpr int DH = ST_DH, KS = DH / 16, HKV = ST_HKV;
  const int Hq = HKV * G;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  int* row_start = reinterpret_cast<int*>(smem + ST_STAGES * ST_STAGE);      // [b + 1]
  uint16_t* pbuf = reinterpret_cast<uint16_t*>(row_start + ST_ROWS_MAX + 4);  // per warp: P hi [8][16], lo [8][16]
  uint64_t* full = reinterpret_cast<uint64_t*>(pbuf + HKV * 2 * 8 * PAGE);
  uint64_t* empty = full + ST_STAGES;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(empty + ST_STAGES);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t4 = lane & 3;

  if (threadIdx.x == 0) {
    for (int s = 0; s < ST_STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], HKV);
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  pdl_entry();  // lens, page tables, q and the prefix partials of the preceding launches are visible
  // row_start[s] = pages of rows 0 .. s-1 (block scan: each thread sums a run of consecutive rows)
  {
    const int per = (a.b + ST_THREADS - 1) / ST_THREADS;
    const int r0 = threadIdx.x * per, r1 = min(a.b, r0 + per);
    int sum = 0;
    for (int s = r0; s < r1; ++s) {
      int t_lo, L, pf, np;
      st_row_range(a, s, t_lo, L, pf, np);
      row_start[s] = np;  // own count for now
      sum += np;
    }
    // exclusive scan of the per-thread sums over the block (warp shuffles, then the warp totals)
    __shared__ int wsum[ST_THREADS / 32];
    int incl = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    int base = 0;
    for (int w = 0; w < warp; ++w) base += wsum[w];
    int run = base + incl - sum;
    for (int s = r0; s < r1; ++s) {
      const int np = row_start[s];
      row_start[s] = run;
      run += np;
    }
    if (threadIdx.x == ST_THREADS - 1) row_start[a.b] = run;
  }
  __syncthreads();
  const long long total = row_start[a.b];
  // shares over min(CTAs, pages) CTAs, so that every share holds a page (a row's segments are then
  // exactly the shares from the one holding its first page to the one holding its last)
  const int C = (int)min((long long)gridDim.x, total);
  if ((int)blockIdx.x >= C) return;
  const long long u0 = st_share(total, blockIdx.x, C), u1 = st_share(total, blockIdx.x + 1, C);
  // first row of the share: the last s with row_start[s] <= u0 (and a page)
  int s_first = 0;
  {
    int lo = 0, hi = a.b - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (row_start[mid] <= u0) lo = mid;
      else hi = mid - 1;
    }
    s_first = lo;
    while (row_start[s_first + 1] <= u0) ++s_first;  // skip rows without pages
  }
  const int n_units = (int)(u1 - u0);

  if (warp == HKV) {
    // ---------------- producer: K and V of every kv head for each page of the share ----------------
    // The 32 lanes look up the rows and page ids of the next 32 pages together (one round trip to memory per
    // 32 pages); lane 0 then waits for free stages and issues the copies.
    int stage = 0;
    uint32_t phase = 0;
    int armed[ST_STAGES];
    uint32_t armed_par[ST_STAGES];
    for (int i = 0; i < ST_STAGES; ++i) armed[i] = 0, armed_par[i] = 0;
    int ok = 1;
    int s_cur = s_first;  // row of the batch's first page
    for (long long ub = u0; ub < u1 && ok; ub += 32) {
      const long long u = ub + lane;
      int s = s_cur, page = 0;
      if (u < u1) {
        while (u >= row_start[s + 1]) ++s;
        int t_lo, L, pf, np;
        st_row_range(a, s, t_lo, L, pf, np);
        page = a.pt[(size_t)a.slot_ids[s] * a.pt_stride + pf + (int)(u - row_start[s])];
      }
      const int cnt = (int)min((long long)32, u1 - ub);
      s_cur = __shfl_sync(0xffffffffu, s, cnt - 1);
      for (int j = 0; j < cnt; ++j) {
        const int pg = __shfl_sync(0xffffffffu, page, j);
        if (lane == 0) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag)) {
            ok = 0;
          } else {
            mbar_expect_tx(&full[stage], ST_STAGE);
            uint8_t* dst = smem + stage * ST_STAGE;
            const int yk = pg * 2 * HKV * PAGE, yv = yk + HKV * PAGE;
            tma_load_2d(dst, &tm, &full[stage], 0, yk);
            tma_load_2d(dst + ST_TILE, &tm, &full[stage], 64, yk);
            tma_load_2d(dst + 2 * ST_TILE, &tm, &full[stage], 0, yv);
            tma_load_2d(dst + 3 * ST_TILE, &tm, &full[stage], 64, yv);
            armed[stage] = 1;
            armed_par[stage] = phase;
            if (++stage == ST_STAGES) stage = 0, phase ^= 1u;
          }
        }
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) break;
      }
    }
    if (lane == 0) {
      if (!ok) {
        if (a.err) atomicExch(a.err, 10);
        *abort_flag = 1;
      }
      for (int i = 0; i < ST_STAGES; ++i)  // every armed copy lands before the CTA exits
        if (armed[i]) mbar_wait(&full[i], armed_par[i], nullptr);
    }
    return;
  }

  // ---------------- consumer warp h: kv head h, query heads h G .. h G + G - 1 ----------------
  const int h = warp;
  uint16_t* sPh = pbuf + h * 2 * 8 * PAGE;
  uint16_t* sPl = sPh + 8 * PAGE;
  int stage = 0;
  uint32_t phase = 0;
  int s = s_first, t_lo = 0, L = 0, pf = 0, np = 0;
  st_row_range(a, s, t_lo, L, pf, np);
  uint32_t qb[KS][2];
  float m[2], l[2], o[KS][4];
  // the shared-prefix partial of this thread's (head column, dim) values, loaded when the row starts so that
  // its latency overlaps the row's pages
  float pre_o[KS][4], pre_m[2], pre_l[2];
  auto begin_row = [&]() {
    if (a.prefix_part) {
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const int hcol = min(2 * t4 + j, G - 1);
        const float* p0 = a.prefix_part + ((size_t)s * Hq + h * G + hcol) * a.max_splits * (DH + 2);
        pre_m[j] = p0[DH];
        pre_l[j] = p0[DH + 1];
#pragma unroll
        for (int mt = 0; mt < KS; ++mt) {
          pre_o[mt][j] = p0[mt * 16 + g];
          pre_o[mt][2 + j] = p0[mt * 16 + g + 8];
        }
      }
    }
    const T* qh = q + ((size_t)s * Hq + h * G + (g < G ? g : 0)) * DH;
#pragma unroll
    for (int k = 0; k < KS; ++k) {
      qb[k][0] = g < G ? *reinterpret_cast<const uint32_t*>(qh + k * 16 + 2 * t4) : 0u;
      qb[k][1] = g < G ? *reinterpret_cast<const uint32_t*>(qh + k * 16 + 8 + 2 * t4) : 0u;
    }
    m[0] = m[1] = -INFINITY;
    l[0] = l[1] = 0.f;
#pragma unroll
    for (int i = 0; i < KS; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  };
  begin_row();
  for (int i = 0; i < n_units; ++i) {
    const long long u = u0 + i;
    while (u >= row_start[s + 1]) {
      ++s;
      st_row_range(a, s, t_lo, L, pf, np);
      begin_row();
    }
    const int pl = (int)(u - row_start[s]);  // page of the row
    // every lane observes the stage's phase itself (the copies land through the async proxy)
    const bool ok = __all_sync(0xffffffffu, mbar_wait(&full[stage], phase, abort_flag));
    if (!ok) {
      if (lane == 0) {
        if (a.err) atomicExch(a.err, 10);
        *abort_flag = 1;
      }
      return;
    }
    const uint32_t st = smem_u32(smem + stage * ST_STAGE);
    // S^T = K Q^T: 16 positions x 8 head columns
    float sc[4] = {0.f, 0.f, 0.f, 0.f};
    {
      const int r = h * PAGE + (lane & 15);
#pragma unroll
      for (int k = 0; k < KS; ++k) {
        uint32_t a0, a1, a2, a3;
        ldm_x4(st + (k >> 2) * ST_TILE + swz128(r, (k & 3) * 2 + (lane >> 4)), a0, a1, a2, a3);
        mma16816<T>(sc, a0, a1, a2, a3, qb[k][0], qb[k][1]);
      }
    }
    const int tok0 = (pf + pl) * PAGE + g;
    const bool v0 = tok0 >= t_lo && tok0 < L, v1 = tok0 + 8 >= t_lo && tok0 + 8 < L;
    float corr[2];
#pragma unroll
    for (int j = 0; j < 2; ++j) {  // head columns 2 t4 + j
      const float x0 = v0 ? sc[j] * a.scale_log2 : -INFINITY;
      const float x1 = v1 ? sc[2 + j] * a.scale_log2 : -INFINITY;
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
    const uint32_t bh0 = *reinterpret_cast<const uint32_t*>(sPh + g * PAGE + 2 * t4);
    const uint32_t bh1 = *reinterpret_cast<const uint32_t*>(sPh + g * PAGE + 8 + 2 * t4);
    const uint32_t bl0 = *reinterpret_cast<const uint32_t*>(sPl + g * PAGE + 2 * t4);
    const uint32_t bl1 = *reinterpret_cast<const uint32_t*>(sPl + g * PAGE + 8 + 2 * t4);
    // O^T += V^T P^T: dims in m16 tiles, V rows (positions) read transposed
    {
      const int mi = lane >> 3, rr = h * PAGE + (lane & 7) + ((mi >> 1) << 3);
#pragma unroll
      for (int mt = 0; mt < KS; ++mt) {
        uint32_t a0, a1, a2, a3;
        ldm_x4_t(st + (2 + (mt >> 2)) * ST_TILE + swz128(rr, (mt & 3) * 2 + (mi & 1)), a0, a1, a2, a3);
        mma16816<T>(o[mt], a0, a1, a2, a3, bh0, bh1);
        if constexpr (std::is_same<T, bf16>::value) mma16816<T>(o[mt], a0, a1, a2, a3, bl0, bl1);
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[stage]);
    if (++stage == ST_STAGES) stage = 0, phase ^= 1u;
    if (pl != np - 1 && i != n_units - 1) continue;
    // ---------------- end of this CTA's segment of row s ----------------
    const long long rs = row_start[s], re = row_start[s + 1];
    const bool whole = rs >= u0 && re <= u1;
    const int which = rs > u0 ? 1 : 0;  // the row began inside the share: the share's last segment
    float* seg = a.seg_part + ((size_t)blockIdx.x * 2 + which) * Hq * (DH + 2);
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int hcol = 2 * t4 + j;
      if (hcol >= G) continue;
      const int hq = h * G + hcol;
      float M = m[j], Ls = l[j], fold = 1.f;
      float w0 = 0.f, m0 = -INFINITY, l0 = 0.f;
      const bool pre = whole && a.prefix_part;
      if (pre) {  // fold in the shared-prefix partial
        m0 = pre_m[j];
        l0 = pre_l[j];
        const float Mn = fmaxf(M, m0);
        w0 = (m0 == -INFINITY) ? 0.f : exp2f(m0 - Mn);
        fold = (M == -INFINITY) ? 0.f : exp2f(M - Mn);
        Ls = Ls * fold + l0 * w0;
      }
#pragma unroll
      for (int mt = 0; mt < KS; ++mt) {
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int d = mt * 16 + g + 8 * e;
          float O = o[mt][2 * e + j];
          if (whole) {
            if (pre) O = O * fold + pre_o[mt][2 * e + j] * w0;
            out[((size_t)s * Hq + hq) * DH + d] = f_to<T>(O / Ls);
          } else {
            seg[(size_t)hq * (DH + 2) + d] = O;
          }
        }
      }
      if (!whole && g == 0) {
        seg[(size_t)hq * (DH + 2) + DH] = M;
        seg[(size_t)hq * (DH + 2) + DH + 1] = Ls;
      }
    }
    if (whole) continue;
    // count this segment; the last of the row's segments (for this kv head) merges them
    __threadfence();
    __syncwarp();
    const int c0 = st_cta_of(rs, total, C), c1 = st_cta_of(re - 1, total, C);
    int last = 0;
    if (lane == 0) last = atomicAdd(&a.seg_cnt[(size_t)s * HKV + h], 1) == c1 - c0;
    last = __shfl_sync(0xffffffffu, last, 0);
    if (!last) continue;
    __threadfence();
    for (int hcol = 0; hcol < G; ++hcol) {
      const int hq = h * G + hcol;
      float M = -INFINITY, Ls = 0.f, O[DH / 32];
#pragma unroll
      for (int k = 0; k < DH / 32; ++k) O[k] = 0.f;
      auto merge = [&](const float* src) {
        const float ms = src[DH], ls = src[DH + 1];
        if (ms == -INFINITY) return;
        const float Mn = fmaxf(M, ms);
        const float wa = (M == -INFINITY) ? 0.f : exp2f(M - Mn), wb = exp2f(ms - Mn);
        Ls = Ls * wa + ls * wb;
#pragma unroll
        for (int k = 0; k < DH / 32; ++k) O[k] = O[k] * wa + src[lane + 32 * k] * wb;
        M = Mn;
      };
      if (a.prefix_part) merge(a.prefix_part + ((size_t)s * Hq + hq) * a.max_splits * (DH + 2));
      for (int c = c0; c <= c1; ++c) {
        const int wc = st_share(total, c, C) < rs ? 1 : 0;
        merge(a.seg_part + (((size_t)c * 2 + wc) * Hq + hq) * (DH + 2));
      }
#pragma unroll
      for (int k = 0; k < DH / 32; ++k) out[((size_t)s * Hq + hq) * DH + lane + 32 * k] = f_to<T>(O[k] / Ls);
    }
    if (lane == 0) a.seg_cnt[(size_t)s * HKV + h] = 0;
  }
}

// ------------------------------------------------------------------------------------------------
// Tensor-core shared-prefix pass (tcgen05; 16-bit KV, head_dim 128, 8 kv heads, prefix S <= 512 positions).
//
// The prompt's full pages are shared by every candidate, so the prefix part of decode attention is a dense
// attention of many queries against one key set: per kv head h, the b x G query rows (candidate s, query
// head h G + j) against the S prefix keys.  One CTA takes 128 query rows (128 / G candidates x G heads) of
// one kv head.  Warp 0 issues the TMA copies: the Q tile once (a 4D map over q [b][8][G][128]), then K and
// V of the kv head in blocks of 128 keys (16-row boxes out of the pool pages, 2 stages; keys past S read
// the zero fill of a box outside the pool).  Warp 1 issues tcgen05.mma: S = Q K^T (M 128, N 128, K 128)
// into one of two TMEM buffers, and O += P V (V read MN-major straight from the page rows) into a third.
// Warps 2-5 own one query row per thread (their TMEM lane quadrant): they read S, apply the scale and the
// per-row window, keep a reference maximum that is raised (and O rescaled in TMEM) only when a block's
// maximum exceeds it by more than 2^8, write P = exp2(s - m) as the K-major swizzled A operand, and at the
// end write (O, m, l) unnormalised as partial slot 0 in the decode kernels' log2-scaled convention.
constexpr int PX_KB = 128;                   // keys per block
constexpr int PX_HALF = 128 * 128;           // bytes of a 128-row x 64-column (128-byte) tile
constexpr int PX_STAGE = 4 * PX_HALF;        // K (two column halves) + V (two column halves)
constexpr int PX_STAGES = 2;
constexpr int PX_SMAX = 512;                 // longest prefix handled
constexpr size_t PX_SMEM = 1024 + 2 * PX_HALF + (size_t)PX_STAGES * PX_STAGE + 2 * PX_HALF + 256;
constexpr float PX_RAISE = 8.f;              // log2 units the block maximum may exceed the reference by

// instruction descriptor, kind::f16, fp32 D, M = 128, N = 128; b_mn: B is MN-major
__host__ __device__ constexpr uint32_t px_idesc(bool bf, bool b_mn) {
  return (1u << 4) | ((bf ? 1u : 0u) << 7) | ((bf ? 1u : 0u) << 10) | ((b_mn ? 1u : 0u) << 16) |
         ((uint32_t)(128 >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
}
// MN-major operand with 128-byte swizzle: rows of 64 MN elements (128 B), 8-row groups every 1024 B (SBO),
// the next 64 MN elements `lbo` bytes further (LBO)
__device__ __forceinline__ uint64_t sdesc_mn(uint32_t addr, uint32_t lbo) {
  return (uint64_t)((addr & 0x3FFFFu) >> 4) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
         ((uint64_t)(1024 >> 4) << 32) | ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

template <typename T, int G>
__global__ void __launch_bounds__(192, 1)
    k_prefix_tc(const __grid_constant__ CUtensorMap tmq, const __grid_constant__ CUtensorMap tmkv,
                const int* __restrict__ pt, int pt_stride, const int* __restrict__ slot_ids,
                const int* __restrict__ lens, int n,
                int S, int pool_rows, float scale_log2, int window, int max_splits, float* __restrict__ part,
                int* err) {
  static_assert(G == 1 || G == 2 || G == 4 || G == 8, "query heads per kv head");
  constexpr int HKV = 8, DH = 128, SPC = 128 / G;  // candidates per CTA
  constexpr bool BF = std::is_same<T, bf16>::value;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;                                  // 2 halves
  uint8_t* sKV = sQ + 2 * PX_HALF;                     // stages: K lo, K hi, V lo, V hi
  uint8_t* sP = sKV + PX_STAGES * PX_STAGE;            // 2 halves
  uint64_t* bars = reinterpret_cast<uint64_t*>(sP + 2 * PX_HALF);
  uint64_t* q_full = bars;
  uint64_t* full = bars + 1;                           // [2]
  uint64_t* empty = full + PX_STAGES;                  // [2]
  uint64_t* s_full = empty + PX_STAGES;                // [2]
  uint64_t* s_free = s_full + 2;                       // [2]
  uint64_t* p_full = s_free + 2;
  uint64_t* o_done = p_full + 1;
  uint64_t* mma_done = o_done + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.y, s0 = blockIdx.x * SPC;
  const int nkb = (S + PX_KB - 1) / PX_KB;
  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int i = 0; i < PX_STAGES; ++i) mbar_init(&full[i], 1), mbar_init(&empty[i], 1);
    for (int i = 0; i < 2; ++i) mbar_init(&s_full[i], 1), mbar_init(&s_free[i], 4);
    mbar_init(p_full, 4);
    mbar_init(o_done, 1);
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(512)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_entry();

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      bool ok = true;
      int armed[PX_STAGES] = {0, 0};
      uint32_t armed_par[PX_STAGES] = {0, 0};
      mbar_expect_tx(q_full, 2 * PX_HALF);
      for (int c = 0; c < 2; ++c) tma_load_4d(sQ + c * PX_HALF, &tmq, q_full, c * 64, 0, h, s0);
      const int* prow = pt + (size_t)slot_ids[0] * pt_stride;  // the prompt pages, the same in every row
      for (int kb = 0; kb < nkb && ok; ++kb) {
        const int st = kb % PX_STAGES;
        const uint32_t ph = (uint32_t)(kb / PX_STAGES) & 1u;
        if (!mbar_wait(&empty[st], ph ^ 1u, abort_flag)) {
          ok = false;
          break;
        }
        mbar_expect_tx(&full[st], PX_STAGE);
        uint8_t* dst = sKV + st * PX_STAGE;
        for (int pg = 0; pg < PX_KB / PAGE; ++pg) {
          const int key0 = kb * PX_KB + pg * PAGE;
          // a page past the prefix reads rows outside the pool: the zero fill
          const int yk = key0 < S ? prow[key0 / PAGE] * 2 * HKV * PAGE + h * PAGE : pool_rows;
          const int yv = key0 < S ? yk + HKV * PAGE : pool_rows;
          for (int c = 0; c < 2; ++c) {
            tma_load_2d(dst + c * PX_HALF + pg * PAGE * 128, &tmkv, &full[st], c * 64, yk);
            tma_load_2d(dst + (2 + c) * PX_HALF + pg * PAGE * 128, &tmkv, &full[st], c * 64, yv);
          }
        }
        armed[st] = 1;
        armed_par[st] = ph;
      }
      if (!ok) {
        if (err) atomicExch(err, 11);
        *abort_flag = 1;
      }
      mbar_wait(q_full, 0, nullptr);
      for (int i = 0; i < PX_STAGES; ++i)
        if (armed[i]) mbar_wait(&full[i], armed_par[i], nullptr);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      const uint32_t id_s = px_idesc(BF, false), id_o = px_idesc(BF, true);
      bool ok = mbar_wait(q_full, 0, abort_flag);
      tc_fence_after();
      auto issue_o = [&](int kb) -> bool {  // O += P V of block kb
        if (!mbar_wait(p_full, (uint32_t)kb & 1u, abort_flag)) return false;
        tc_fence_after();
        const uint32_t v = smem_u32(sKV + (kb % PX_STAGES) * PX_STAGE + 2 * PX_HALF);
#pragma unroll
        for (int k = 0; k < PX_KB / 16; ++k) {
          const uint64_t a = sdesc(smem_u32(sP + (k >> 2) * PX_HALF)) + (uint64_t)((k & 3) * 2);
          const uint64_t b = sdesc_mn(v + k * 16 * 128, PX_HALF);
          umma(tmem + 256, a, b, id_o, (kb > 0 || k > 0) ? 1u : 0u);
        }
        umma_commit(o_done);
        umma_commit(&empty[kb % PX_STAGES]);
        return true;
      };
      for (int kb = 0; kb < nkb && ok; ++kb) {
        const int st = kb % PX_STAGES, sb = kb & 1;
        if (!mbar_wait(&full[st], (uint32_t)(kb / PX_STAGES) & 1u, abort_flag) ||
            !mbar_wait(&s_free[sb], ((uint32_t)(kb >> 1) & 1u) ^ 1u, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t kbase = smem_u32(sKV + st * PX_STAGE);
#pragma unroll
        for (int k = 0; k < DH / 16; ++k) {
          const uint64_t a = sdesc(smem_u32(sQ + (k >> 2) * PX_HALF)) + (uint64_t)((k & 3) * 2);
          const uint64_t b = sdesc(kbase + (k >> 2) * PX_HALF) + (uint64_t)((k & 3) * 2);
          umma(tmem + sb * 128, a, b, id_s, k > 0 ? 1u : 0u);
        }
        umma_commit(&s_full[sb]);
        if (kb > 0 && !issue_o(kb - 1)) ok = false;
      }
      if (ok && !issue_o(nkb - 1)) ok = false;
      if (!ok) {
        if (err) atomicExch(err, 12);
        *abort_flag = 1;
      }
      umma_commit(mma_done);
      mbar_wait(mma_done, 0, nullptr);
    }
  } else {
    // ---------------- softmax: one query row per thread ----------------
    const int quad = warp & 3, r = quad * 32 + lane;
    const int s = s0 + r / G, j = r % G;
    const bool valid = s < n;
    const int qpos = valid ? lens[s] - 1 : 0;
    const uint32_t trow = tmem + ((uint32_t)(quad * 32) << 16);
    float m_ref = -INFINITY, l = 0.f;
    bool ok = true;
    for (int kb = 0; kb < nkb; ++kb) {
      const int sb = kb & 1;
      ok = __all_sync(0xffffffffu, mbar_wait(&s_full[sb], (uint32_t)(kb >> 1) & 1u, abort_flag));
      if (!ok) break;
      tc_fence_after();
      float x[PX_KB];
      tmem_ld64(trow + sb * 128, x);
      tmem_ld64(trow + sb * 128 + 64, x + 64);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_free[sb]);
      float bmax = -INFINITY;
#pragma unroll
      for (int c = 0; c < PX_KB; ++c) {
        const int t = kb * PX_KB + c;
        const bool in = t < S && (window <= 0 || t > qpos - window);
        x[c] = in ? x[c] * scale_log2 : -INFINITY;
        bmax = fmaxf(bmax, x[c]);
      }
      const bool raise = (m_ref == -INFINITY) ? (bmax > -INFINITY) : (bmax > m_ref + PX_RAISE);
      const float m_new = raise ? bmax : m_ref;
      const float corr = (raise && m_ref != -INFINITY) ? exp2f(m_ref - m_new) : 1.f;
      float psum = 0.f;
#pragma unroll
      for (int c = 0; c < PX_KB; ++c) {
        const float p = (x[c] == -INFINITY) ? 0.f : exp2f(x[c] - m_new);
        x[c] = p;
        psum += p;
      }
      l = l * corr + psum;
      m_ref = m_new;
      // the previous block's O MMA has read P and updated O before P is rewritten or O rescaled
      if (kb > 0) {
        ok = __all_sync(0xffffffffu, mbar_wait(o_done, (uint32_t)(kb - 1) & 1u, abort_flag));
        if (!ok) break;
        tc_fence_after();
      }
      // P row r as the K-major A operand (two 64-column halves, 128-byte swizzle)
#pragma unroll
      for (int ch = 0; ch < PX_KB / 8; ++ch) {
        uint32_t w[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const T a = f_to<T>(x[ch * 8 + 2 * e]), b = f_to<T>(x[ch * 8 + 2 * e + 1]);
          w[e] = (uint32_t)(*reinterpret_cast<const uint16_t*>(&a)) |
                 ((uint32_t)(*reinterpret_cast<const uint16_t*>(&b)) << 16);
        }
        uint8_t* dst = sP + (ch >> 3) * PX_HALF + r * 128 + (((ch & 7) ^ (r & 7)) << 4);
        *reinterpret_cast<uint4*>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
      }
      // a raised reference maximum rescales the O accumulated so far (rows whose maximum stayed multiply by 1)
      if (kb > 0 && __any_sync(0xffffffffu, corr != 1.f)) {
#pragma unroll 1
        for (int hh = 0; hh < 2; ++hh) {
          float o[64];
          tmem_ld64(trow + 256 + hh * 64, o);
#pragma unroll
          for (int c = 0; c < 64; ++c) o[c] *= corr;
          tmem_st64(trow + 256 + hh * 64, o);
        }
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // P is read by the tensor core
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full);
    }
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(o_done, (uint32_t)(nkb - 1) & 1u, abort_flag));
    if (ok) {
      tc_fence_after();
      float* pp = part + ((size_t)s * (HKV * G) + h * G + j) * max_splits * (DH + 2);
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        float o[64];
        tmem_ld64(trow + 256 + hh * 64, o);
        if (valid) {
          // a partial slot is DH + 2 = 130 floats (520 bytes): 8-byte aligned, so two floats per store
#pragma unroll
          for (int c = 0; c < 64; c += 2) *reinterpret_cast<float2*>(pp + hh * 64 + c) = make_float2(o[c], o[c + 1]);
        }
      }
      if (valid) pp[DH] = m_ref, pp[DH + 1] = l;
    } else if (lane == 0) {
      if (err) atomicExch(err, 13);
      *abort_flag = 1;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(512) : "memory");
  }
}

// ------------------------------------------------------------------------------------------------
// Tensor-core prefill attention (tcgen05; 16-bit, head_dim 128, 8 kv heads) for the reward model's scoring
// passes: packed sequences, each attending causally to the prompt prefix (contiguous [P][8][128] per layer),
// to its cached keys (reward-model cache pages, when the cache is on) and to its own new rows.
//
// One CTA takes 128 / G query positions (at most 64: a 64-position tile of the mma.sync kernel's tile list is
// split over 64 / min(128 / G, 64) CTAs) of one sequence for the G query heads of one kv head (128 rows, Q by a
// 4D map over q [rows][8][G][128]).  Keys come in blocks of 128 of one segment -- prefix rows and own rows by
// 3D maps ([rows][8][128], box of 128 positions of one kv head), cached keys by 16-row page boxes -- and
// blocks wholly outside the window or past the causal frontier are skipped; producer, MMA issuer and softmax
// warps derive the same block list.  The MMA / softmax scheme is the prefix pass's (S = Q K^T in one of two
// TMEM buffers, P written as the swizzled K-major operand, O += P V with V read MN-major, reference maximum
// raised by more than 2^8 only); the epilogue normalises O by l and stores the 16-bit output rows.
struct PrefillTcArgs {
  const int* seq_off;
  const int* tile_seq;
  const int* tile_q0;  // 64-position tiles of the mma.sync kernel: this kernel runs two 32-position halves
  int n_pre, pos0, window, rows_total, cache_rows;
  const int* cpt;       // cache page table (rows per candidate), or nullptr
  int cpt_stride;
  const int* seq_cand;
  const int* seq_cached;
  float scale_log2;
  int* err;
};

// key block kb of a CTA's list: segment (0 prefix, 1 cached, 2 own) and first key index within the segment
struct PxBlock {
  int seg, kbase, count, kpos0;
};

template <typename T, int G>
__global__ void __launch_bounds__(192, 1)
    k_prefill_tc(const __grid_constant__ CUtensorMap tmq, const __grid_constant__ CUtensorMap tmkp,
                 const __grid_constant__ CUtensorMap tmvp, const __grid_constant__ CUtensorMap tmk,
                 const __grid_constant__ CUtensorMap tmv, const __grid_constant__ CUtensorMap tmc, T* __restrict__ out,
                 PrefillTcArgs a) {
  static_assert(G == 1 || G == 2 || G == 4 || G == 8, "query heads per kv head");
  constexpr int HKV = 8, DH = 128, QP = 128 / G;  // query positions of the 128-row Q tile
  constexpr int PPC = QP < 64 ? QP : 64;           // positions a CTA answers for: a 64-position host tile
  constexpr int NSUB = 64 / PPC;                   // ... is split over NSUB CTAs
  constexpr bool BF = std::is_same<T, bf16>::value;
  const int tile = blockIdx.x / NSUB, h = blockIdx.y;
  const int j = a.tile_seq[tile];
  const int r0 = a.seq_off[j], nrows = a.seq_off[j + 1] - r0;
  const int q0 = a.tile_q0[tile] + (blockIdx.x % NSUB) * PPC;
  if (q0 >= nrows) return;  // a sub-tile past the end of a short tile
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;
  uint8_t* sKV = sQ + 2 * PX_HALF;
  uint8_t* sP = sKV + PX_STAGES * PX_STAGE;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sP + 2 * PX_HALF);
  uint64_t* q_full = bars;
  uint64_t* full = bars + 1;
  uint64_t* empty = full + PX_STAGES;
  uint64_t* s_full = empty + PX_STAGES;
  uint64_t* s_free = s_full + 2;
  uint64_t* p_full = s_free + 2;
  uint64_t* o_done = p_full + 1;
  uint64_t* mma_done = o_done + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  // the CTA's key blocks: prefix, cached, own (own keys up to the last query position of the CTA)
  const int ncache = a.cpt ? a.seq_cached[j] : 0;
  const int opos0 = a.pos0 + ncache;
  const int q_last = min(nrows, q0 + PPC) - 1;
  const int qpos_min = opos0 + q0, qpos_max = opos0 + q_last;
  const int n_own = q_last + 1;
  auto block_at = [&](int seg, int kbase) -> PxBlock {
    const int cnt = min(PX_KB, (seg == 0 ? a.n_pre : (seg == 1 ? ncache : n_own)) - kbase);
    const int kp0 = seg == 0 ? kbase : (seg == 1 ? a.pos0 + kbase : opos0 + kbase);
    return PxBlock{seg, kbase, cnt, kp0};
  };
  auto live = [&](const PxBlock& b) {  // some key of the block is visible to some query of the CTA
    if (a.window > 0 && b.kpos0 + b.count - 1 <= qpos_min - a.window) return false;
    return b.kpos0 <= qpos_max;
  };
  // blocks are enumerated by a running cursor (segment, key base) that skips dead blocks
  auto next_block = [&](int& seg, int& kbase, PxBlock& out_b) -> bool {
    while (seg < 3) {
      const int len = seg == 0 ? a.n_pre : (seg == 1 ? ncache : n_own);
      if (kbase >= len) {
        ++seg;
        kbase = 0;
        continue;
      }
      out_b = block_at(seg, kbase);
      kbase += PX_KB;
      if (live(out_b)) return true;
    }
    return false;
  };
  int nkb = 0;
  {
    int sg = 0, kb0 = 0;
    PxBlock b;
    while (next_block(sg, kb0, b)) ++nkb;
  }

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int i = 0; i < PX_STAGES; ++i) mbar_init(&full[i], 1), mbar_init(&empty[i], 1);
    for (int i = 0; i < 2; ++i) mbar_init(&s_full[i], 1), mbar_init(&s_free[i], 4);
    mbar_init(p_full, 4);
    mbar_init(o_done, 1);
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(512)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_entry();

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      bool ok = true;
      int armed[PX_STAGES] = {0, 0};
      uint32_t armed_par[PX_STAGES] = {0, 0};
      mbar_expect_tx(q_full, 2 * PX_HALF);
      for (int c = 0; c < 2; ++c) tma_load_4d(sQ + c * PX_HALF, &tmq, q_full, c * 64, 0, h, r0 + q0);
      const int* cpt = a.cpt ? a.cpt + (size_t)a.seq_cand[j] * a.cpt_stride : nullptr;
      int sg = 0, kbc = 0;
      PxBlock b;
      for (int kb = 0; kb < nkb && ok; ++kb) {
        next_block(sg, kbc, b);
        const int st = kb % PX_STAGES;
        const uint32_t ph = (uint32_t)(kb / PX_STAGES) & 1u;
        if (!mbar_wait(&empty[st], ph ^ 1u, abort_flag)) {
          ok = false;
          break;
        }
        mbar_expect_tx(&full[st], PX_STAGE);
        uint8_t* dst = sKV + st * PX_STAGE;
        if (b.seg == 1) {  // cached keys: 16-row page boxes (a page past the cached keys reads the zero fill)
          for (int pg = 0; pg < PX_KB / PAGE; ++pg) {
            const int key0 = b.kbase + pg * PAGE;
            const int yk = key0 < ncache ? cpt[key0 / PAGE] * 2 * HKV * PAGE + h * PAGE : a.cache_rows;
            const int yv = key0 < ncache ? yk + HKV * PAGE : a.cache_rows;
            for (int c = 0; c < 2; ++c) {
              tma_load_2d(dst + c * PX_HALF + pg * PAGE * 128, &tmc, &full[st], c * 64, yk);
              tma_load_2d(dst + (2 + c) * PX_HALF + pg * PAGE * 128, &tmc, &full[st], c * 64, yv);
            }
          }
        } else {  // prefix or own rows: one 128-position box of kv head h per column half
          const CUtensorMap* mk = b.seg == 0 ? &tmkp : &tmk;
          const CUtensorMap* mv = b.seg == 0 ? &tmvp : &tmv;
          const int row0 = b.seg == 0 ? b.kbase : r0 + b.kbase;
          for (int c = 0; c < 2; ++c) {
            tma_load_3d(dst + c * PX_HALF, mk, &full[st], c * 64, h, row0);
            tma_load_3d(dst + (2 + c) * PX_HALF, mv, &full[st], c * 64, h, row0);
          }
        }
        armed[st] = 1;
        armed_par[st] = ph;
      }
      if (!ok) {
        if (a.err) atomicExch(a.err, 14);
        *abort_flag = 1;
      }
      mbar_wait(q_full, 0, nullptr);
      for (int i = 0; i < PX_STAGES; ++i)
        if (armed[i]) mbar_wait(&full[i], armed_par[i], nullptr);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer (as in the prefix pass) ----------------
      const uint32_t id_s = px_idesc(BF, false), id_o = px_idesc(BF, true);
      bool ok = mbar_wait(q_full, 0, abort_flag);
      tc_fence_after();
      auto issue_o = [&](int kb) -> bool {
        if (!mbar_wait(p_full, (uint32_t)kb & 1u, abort_flag)) return false;
        tc_fence_after();
        const uint32_t v = smem_u32(sKV + (kb % PX_STAGES) * PX_STAGE + 2 * PX_HALF);
#pragma unroll
        for (int k = 0; k < PX_KB / 16; ++k) {
          const uint64_t ad = sdesc(smem_u32(sP + (k >> 2) * PX_HALF)) + (uint64_t)((k & 3) * 2);
          const uint64_t bd = sdesc_mn(v + k * 16 * 128, PX_HALF);
          umma(tmem + 256, ad, bd, id_o, (kb > 0 || k > 0) ? 1u : 0u);
        }
        umma_commit(o_done);
        umma_commit(&empty[kb % PX_STAGES]);
        return true;
      };
      for (int kb = 0; kb < nkb && ok; ++kb) {
        const int st = kb % PX_STAGES, sb = kb & 1;
        if (!mbar_wait(&full[st], (uint32_t)(kb / PX_STAGES) & 1u, abort_flag) ||
            !mbar_wait(&s_free[sb], ((uint32_t)(kb >> 1) & 1u) ^ 1u, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t kbase = smem_u32(sKV + st * PX_STAGE);
#pragma unroll
        for (int k = 0; k < DH / 16; ++k) {
          const uint64_t ad = sdesc(smem_u32(sQ + (k >> 2) * PX_HALF)) + (uint64_t)((k & 3) * 2);
          const uint64_t bd = sdesc(kbase + (k >> 2) * PX_HALF) + (uint64_t)((k & 3) * 2);
          umma(tmem + sb * 128, ad, bd, id_s, k > 0 ? 1u : 0u);
        }
        umma_commit(&s_full[sb]);
        if (kb > 0 && !issue_o(kb - 1)) ok = false;
      }
      if (ok && nkb > 0 && !issue_o(nkb - 1)) ok = false;
      if (!ok) {
        if (a.err) atomicExch(a.err, 15);
        *abort_flag = 1;
      }
      umma_commit(mma_done);
      mbar_wait(mma_done, 0, nullptr);
    }
  } else {
    // ---------------- softmax and epilogue: one query row per thread ----------------
    const int quad = warp & 3, r = quad * 32 + lane;
    const int qi = q0 + r / G, jh = r % G;
    const bool valid = qi < nrows && qi < q0 + PPC;
    const int qpos = opos0 + qi;
    const uint32_t trow = tmem + ((uint32_t)(quad * 32) << 16);
    float m_ref = -INFINITY, l = 0.f;
    bool ok = true;
    int sg = 0, kbc = 0;
    PxBlock b;
    for (int kb = 0; kb < nkb; ++kb) {
      next_block(sg, kbc, b);
      const int sb = kb & 1;
      ok = __all_sync(0xffffffffu, mbar_wait(&s_full[sb], (uint32_t)(kb >> 1) & 1u, abort_flag));
      if (!ok) break;
      tc_fence_after();
      float x[PX_KB];
      tmem_ld64(trow + sb * 128, x);
      tmem_ld64(trow + sb * 128 + 64, x + 64);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_free[sb]);
      float bmax = -INFINITY;
#pragma unroll
      for (int c = 0; c < PX_KB; ++c) {
        const int kpos = b.kpos0 + c;
        const bool in = c < b.count && kpos <= qpos && (a.window <= 0 || kpos > qpos - a.window);
        x[c] = in ? x[c] * a.scale_log2 : -INFINITY;
        bmax = fmaxf(bmax, x[c]);
      }
      const bool raise = (m_ref == -INFINITY) ? (bmax > -INFINITY) : (bmax > m_ref + PX_RAISE);
      const float m_new = raise ? bmax : m_ref;
      const float corr = (raise && m_ref != -INFINITY) ? exp2f(m_ref - m_new) : 1.f;
      float psum = 0.f;
#pragma unroll
      for (int c = 0; c < PX_KB; ++c) {
        const float p = (x[c] == -INFINITY) ? 0.f : exp2f(x[c] - m_new);
        x[c] = p;
        psum += p;
      }
      l = l * corr + psum;
      m_ref = m_new;
      if (kb > 0) {
        ok = __all_sync(0xffffffffu, mbar_wait(o_done, (uint32_t)(kb - 1) & 1u, abort_flag));
        if (!ok) break;
        tc_fence_after();
      }
#pragma unroll
      for (int ch = 0; ch < PX_KB / 8; ++ch) {
        uint32_t w[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const T lo = f_to<T>(x[ch * 8 + 2 * e]), hi = f_to<T>(x[ch * 8 + 2 * e + 1]);
          w[e] = (uint32_t)(*reinterpret_cast<const uint16_t*>(&lo)) |
                 ((uint32_t)(*reinterpret_cast<const uint16_t*>(&hi)) << 16);
        }
        uint8_t* dst = sP + (ch >> 3) * PX_HALF + r * 128 + (((ch & 7) ^ (r & 7)) << 4);
        *reinterpret_cast<uint4*>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
      }
      if (kb > 0 && __any_sync(0xffffffffu, corr != 1.f)) {
#pragma unroll 1
        for (int hh = 0; hh < 2; ++hh) {
          float o[64];
          tmem_ld64(trow + 256 + hh * 64, o);
#pragma unroll
          for (int c = 0; c < 64; ++c) o[c] *= corr;
          tmem_st64(trow + 256 + hh * 64, o);
        }
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full);
    }
    if (ok && nkb > 0) ok = __all_sync(0xffffffffu, mbar_wait(o_done, (uint32_t)(nkb - 1) & 1u, abort_flag));
    if (ok && nkb > 0) {
      tc_fence_after();
      const float inv = l > 0.f ? 1.f / l : 0.f;
      T* dst = out + ((size_t)(r0 + qi) * (HKV * G) + h * G + jh) * DH;
#pragma unroll 1
      for (int hh = 0; hh < 2; ++hh) {
        float o[64];
        tmem_ld64(trow + 256 + hh * 64, o);
        if (valid) {
#pragma unroll
          for (int c = 0; c < 64; c += 8) {
            uint32_t w[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const T lo = f_to<T>(o[c + 2 * e] * inv), hi = f_to<T>(o[c + 2 * e + 1] * inv);
              w[e] = (uint32_t)(*reinterpret_cast<const uint16_t*>(&lo)) |
                     ((uint32_t)(*reinterpret_cast<const uint16_t*>(&hi)) << 16);
            }
            *reinterpret_cast<uint4*>(dst + hh * 64 + c) = make_uint4(w[0], w[1], w[2], w[3]);
          }
        }
      }
    } else if (!ok && lane == 0) {
      if (a.err) atomicExch(a.err, 16);
      *abort_flag = 1;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(512) : "memory");
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

// fp16 with head_dim <= 128 fits 128 registers, so four CTAs share an SM (2 % faster than three on the scoring
// shapes); the bf16 (hi + lo P) and head_dim-256 forms need more registers and take no occupancy bound.
template <typename T, int DH, int DV>
__global__ void __launch_bounds__(128, (std::is_same<T, bf16>::value || DH > 128) ? 1 : 4) k_prefill_attn(const T* __restrict__ q, const T* __restrict__ k,
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

bool stream_enabled() {
  static const bool on = [] {
    const char* e = getenv("SR_ATTN_STREAM");
    return !(e && e[0] == '0');
  }();
  return on;
}

template <typename T, int G>
sr_status prefix_tc_t(const void* q, const void* pool, const int* pt, int pt_stride, const int* ids, const int* lens,
                      int b, int S, int window, float* part, int max_splits, const DecodeStreamWs& ws,
                      cudaStream_t st) {
  static bool attr = false;
  if (!attr) {
    SR_CUDA(cudaFuncSetAttribute(k_prefix_tc<T, G>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)PX_SMEM));
    attr = true;
  }
  constexpr bool BF = std::is_same<T, bf16>::value;
  const int pool_rows = ws.pool_pages * 2 * ST_HKV * PAGE;
  CUtensorMap tmkv, tmq;
  SR_TRY(encode_tma_2d(&tmkv, pool, BF, pool_rows, ST_DH, PAGE));
  const uint64_t dims[4] = {(uint64_t)ST_DH, (uint64_t)G, (uint64_t)ST_HKV, (uint64_t)b};
  const uint64_t strides[3] = {(uint64_t)ST_DH * 2, (uint64_t)G * ST_DH * 2, (uint64_t)ST_HKV * G * ST_DH * 2};
  const uint32_t box[4] = {64, (uint32_t)G, 1, (uint32_t)(128 / G)};
  SR_TRY(encode_tma_nd(&tmq, q, BF, 4, dims, strides, box));
  launch_k(k_prefix_tc<T, G>, dim3((b + 128 / G - 1) / (128 / G), ST_HKV), 192, PX_SMEM, st, tmq, tmkv, pt, pt_stride,
           ids, lens, b, S, pool_rows, 1.4426950408889634f / sqrtf((float)ST_DH), window, max_splits, part, ws.err);
  SR_LAUNCH();
  return SR_OK;
}

template <typename T, int G>
sr_status prefill_tc_t(const void* q, const void* k, const void* v, const void* kpre, const void* vpre, int npre,
                       const int* seq_off, const int* tile_seq, const int* tile_q0, int n_tiles, int pos0, int rows,
                       int window, void* out, const CachedKeys& ck, cudaStream_t st) {
  static bool attr = false;
  if (!attr) {
    SR_CUDA(cudaFuncSetAttribute(k_prefill_tc<T, G>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)PX_SMEM));
    attr = true;
  }
  constexpr bool BF = std::is_same<T, bf16>::value;
  constexpr int HKV = ST_HKV, DH = ST_DH;
  CUtensorMap tmq, tmk, tmv, tmkp, tmvp, tmc;
  {
    const uint64_t dims[4] = {(uint64_t)DH, (uint64_t)G, (uint64_t)HKV, (uint64_t)rows};
    const uint64_t strides[3] = {(uint64_t)DH * 2, (uint64_t)G * DH * 2, (uint64_t)HKV * G * DH * 2};
    const uint32_t box[4] = {64, (uint32_t)G, 1, (uint32_t)(128 / G)};
    SR_TRY(encode_tma_nd(&tmq, q, BF, 4, dims, strides, box));
  }
  auto kv3 = [&](CUtensorMap* m, const void* base, int n) -> sr_status {  // [n][8][128], 128-position boxes
    const uint64_t dims[3] = {(uint64_t)DH, (uint64_t)HKV, (uint64_t)n};
    const uint64_t strides[2] = {(uint64_t)DH * 2, (uint64_t)HKV * DH * 2};
    const uint32_t box[3] = {64, 1, (uint32_t)PX_KB};
    return encode_tma_nd(m, base, BF, 3, dims, strides, box);
  };
  SR_TRY(kv3(&tmk, k, rows));
  SR_TRY(kv3(&tmv, v, rows));
  if (npre > 0) {
    SR_TRY(kv3(&tmkp, kpre, npre));
    SR_TRY(kv3(&tmvp, vpre, npre));
  } else {
    tmkp = tmk, tmvp = tmv;  // no prefix segment: never read
  }
  const int cache_rows = ck.pool ? ck.pool_pages * 2 * HKV * PAGE : 0;
  if (ck.pool) SR_TRY(encode_tma_2d(&tmc, ck.pool, BF, cache_rows, DH, PAGE));
  else tmc = tmk;  // no cached segment: never read
  PrefillTcArgs a{seq_off, tile_seq, tile_q0, npre, pos0, window, rows, cache_rows,
                  ck.pool ? ck.page_table : nullptr, ck.pt_stride, ck.seq_cand, ck.seq_cached,
                  1.4426950408889634f / sqrtf((float)DH), tc_error_word()};
  constexpr int NSUB = 64 / ((128 / G) < 64 ? (128 / G) : 64);
  launch_k(k_prefill_tc<T, G>, dim3(n_tiles * NSUB, HKV), 192, PX_SMEM, st, tmq, tmkp, tmvp, tmk, tmv, tmc, (T*)out,
           a);
  SR_LAUNCH();
  return SR_OK;
}

// The tcgen05 prefill measured slower than the mma.sync kernel on the scoring shapes (1.03 against 0.66 ms for
// 37 sequences x 443 rows after a 288-position prefix: one CTA per SM, four softmax warps and a per-CTA TMEM
// allocation for a few key blocks each), so it runs only when SR_PREFILL_TC=1.
bool prefill_tc_enabled() {
  static const bool on = [] {
    const char* e = getenv("SR_PREFILL_TC");
    return e && e[0] == '1';
  }();
  return on;
}

// The tcgen05 prefix pass measured slower in the decode loop than the mma.sync one (one CTA and four softmax
// warps per SM against sixteen warps), so it runs only when SR_PREFIX_TC=1.
bool prefix_tc_enabled() {
  static const bool on = [] {
    const char* e = getenv("SR_PREFIX_TC");
    return e && e[0] == '1';
  }();
  return on;
}

template <typename T, int G>
sr_status decode_stream_t(const void* q, const void* pool, const int* pt, int pt_stride, const int* ids,
                          const int* lens, int b, int window, void* out, const float* prefix_part, int max_splits,
                          int shared_pos, const DecodeStreamWs& ws, cudaStream_t st) {
  static bool attr = false;
  if (!attr) {
    SR_CUDA(cudaFuncSetAttribute(k_decode_stream<T, G>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ST_SMEM));
    attr = true;
  }
  CUtensorMap tm;
  SR_TRY(encode_tma_2d(&tm, pool, std::is_same<T, bf16>::value, ws.pool_pages * 2 * ST_HKV * PAGE, ST_DH, 128));
  StreamArgs a{pt, pt_stride, ids, lens, b, window, shared_pos, max_splits,
               1.4426950408889634f / sqrtf((float)ST_DH), prefix_part, ws.seg_part, ws.seg_cnt, ws.err};
  launch_k(k_decode_stream<T, G>, ws.grid, ST_THREADS, ST_SMEM, st, tm, (const T*)q, (T*)out, a);
  SR_LAUNCH();
  return SR_OK;
}

template <typename T, int DH, int G>
sr_status decode_attn_tc_t(const void* q, const void* pool, const int* pt, int pt_stride, const int* ids,
                           const int* lens, int b, int Hkv, int window, void* out, float* part, int max_splits,
                           int shared_pos, int max_len, cudaStream_t st, int* err, const DecodeStreamWs* ws) {
  // with a shared prefix: slot 0 of the partials is the prefix pass, position splits follow
  const int sbase = shared_pos > 0 ? 1 : 0;
  const int t_min = shared_pos;
  bool prefix_done = false;
  if constexpr (DH == ST_DH) {
    if (sbase && part && ws && prefix_tc_enabled() && Hkv == ST_HKV && shared_pos <= PX_SMAX &&
        (G == 1 || G == 2 || G == 4 || G == 8)) {
      constexpr int GG = (G == 1 || G == 2 || G == 4 || G == 8) ? G : 1;
      const sr_status ps = prefix_tc_t<T, GG>(q, pool, pt, pt_stride, ids, lens, b, shared_pos, window, part,
                                              max_splits, *ws, st);
      if (ps != SR_OK) return ps;
      prefix_done = true;
    }
  }
  if (sbase && !prefix_done) {
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
  if constexpr (DH == ST_DH) {
    if (ws && stream_enabled() && Hkv == ST_HKV && b <= ST_ROWS_MAX)
      return decode_stream_t<T, G>(q, pool, pt, pt_stride, ids, lens, b, window, out, sbase ? part : nullptr,
                                   max_splits, shared_pos, *ws, st);
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
    // up to four CTAs per SM (see the launch bound): all of the SM's shared memory as carve-out
    SR_CUDA(cudaFuncSetAttribute(k_prefill_attn<T, DH, DV>, cudaFuncAttributePreferredSharedMemoryCarveout, 100));
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

size_t decode_stream_part_floats(int grid, int Hq) { return (size_t)grid * 2 * Hq * (ST_DH + 2); }
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
                                  int max_len, int* err, const DecodeStreamWs* ws) {
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
                                      shared_pos, max_len, st, err, ws);
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
                                   void* out, cudaStream_t st, CachedKeys ck, int rows) {
  (void)n_seq;
  if (n_tiles == 0) return SR_OK;
  if (Hq % Hkv) return set_err(SR_ERR_UNSUPPORTED, "prefill attention: n_heads %% n_kv_heads != 0");
  if (et != SR_DT_F16 && et != SR_DT_BF16) return set_err(SR_ERR_INVALID_ARG, "prefill attention: 16-bit types only");
  // head_dim 128 with 8 kv heads: the tensor-core kernel (every operand 16-byte aligned, as TMA needs)
  const int G = Hq / Hkv;
  const bool al = ((reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(k) | reinterpret_cast<uintptr_t>(v) |
                    reinterpret_cast<uintptr_t>(kpre) | reinterpret_cast<uintptr_t>(vpre) |
                    reinterpret_cast<uintptr_t>(ck.pool) | reinterpret_cast<uintptr_t>(out)) & 15) == 0;
  if (rows > 0 && prefill_tc_enabled() && dh == ST_DH && Hkv == ST_HKV && al &&
      (G == 1 || G == 2 || G == 4 || G == 8)) {
#define SR_PTC(TT, GG)                                                                                              \
  if (G == GG)                                                                                                      \
    return prefill_tc_t<TT, GG>(q, k, v, kpre, vpre, npre, seq_off, tile_seq, tile_q0, n_tiles, pos0, rows, window, \
                                out, ck, st);
    if (et == SR_DT_F16) {
      SR_PTC(f16, 1) SR_PTC(f16, 2) SR_PTC(f16, 4) SR_PTC(f16, 8)
    } else {
      SR_PTC(bf16, 1) SR_PTC(bf16, 2) SR_PTC(bf16, 4) SR_PTC(bf16, 8)
    }
#undef SR_PTC
  }
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
