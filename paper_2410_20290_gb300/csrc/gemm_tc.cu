// Dense layers on the 5th-generation tensor cores (tcgen05 + TMEM + TMA), C = A W^T, with A and W
// both fp16 or both bf16 (kind::f16) and fp32 accumulation.
//
// Every projection of the generator and reward model (QKV, O, gate/up, down, LM head) is one
// of these GEMMs (Section 4.2 generation and partial-reward scoring both run them; Section 3
// defines the models).  A [M][K] and W [N][K] are K-major 16-bit; the accumulator is fp32 in
// tensor memory.
//
// Design (persistent, warp-specialised, one CTA per SM):
//   warp 0      : TMA producer -- 128x64 A and BNx64 W tiles (BN = 256, 192, 128 or 64, chosen per
//                 shape by a waves x per-tile-cost model), 128-byte swizzle, STAGES-deep ring
//                 (up to 200 KB of shared memory in flight per SM)
//   warp 1      : allocates 2*BN TMEM columns; one elected lane issues tcgen05.mma (M=128, N=BN,
//                 K=16) and tcgen05.commit to release smem stages / publish accumulators
//   warps 2..5  : epilogue -- tcgen05.ld 32 lanes x 64 columns per warp and wait (the warp's TMEM
//                 lane quadrant is warp % 4), fused conversion / residual add / gated activation,
//                 direct global stores
// Two BN-column accumulators let the epilogue of tile i overlap the mainloop of tile i+1.
// Tiles are walked in groups of 16 M tiles, M fastest within a group, so that the CTAs running at the same
// time share W tiles and one band of A rows in L2.
// Two variants raise the MMA work per staged byte (the limit of the 128-row tiles on GB300):
// 256 x 256 tiles on one SM (two M = 128 MMAs per W tile, single-buffered accumulator), and
// 256 x 256 tiles on a CTA pair (cta_group::2, M = 256 MMAs, each SM staging half of A and W,
// double-buffered accumulators).  Decode batches of at most 512 rows can instead run the product
// transposed (C^T = W A^T) on a CTA pair, every activation row on the MMA's N side, with the K range
// split over the SMs and the fp32 partials summed in slice order.  The launcher picks per shape.
// Opt-in forms: stream-K shares of k-blocks on 128 x 256 tiles (SR_GEMM_STREAMK=1), and the LM head's
// sampling epilogue (EK = 1: Gumbel-max records instead of stored logits, sampling.cuh).
// Every mbarrier wait is bounded (about 2 s of %globaltimer); on expiry the CTA records an error,
// drains its own TMA copies and MMAs, frees TMEM and exits.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <map>
#include <mutex>
#include <type_traits>

#include "common.cuh"
#include "sampling.cuh"
#include "tma.cuh"

namespace sr {
namespace {

constexpr int BM = 128, BK = 64;  // BM: rows of one MMA (one TMEM lane block)
constexpr int BAR_BYTES = 256;

// TM = rows per CTA tile: 128 (one MMA per K step) or 256 (two MMAs sharing the W tile, which halves the
// staged bytes per flop; its 256 x 256 fp32 accumulator fills TMEM, so it is single-buffered and drained
// by eight epilogue warps instead of four).
template <int TM, int BN>
struct Cfg {
  static constexpr int MH = TM / BM;                          // 128-row halves per tile
  static constexpr int A_BYTES = TM * BK * 2;
  static constexpr int B_BYTES = BN * BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int STAGES = (200 * 1024) / STAGE_BYTES;  // 4 / 5 / 6 / 8 for BN 256 / 192 / 128 / 64; 3 for 256 x 256
  static constexpr int NACC = (MH * BN * 2 <= 512) ? 2 : 1;   // accumulator buffers in TMEM
  static constexpr int TMEM_USED = NACC * MH * BN;
  // tcgen05.alloc takes a power of two of at least 32 columns (384 for two BN = 192 accumulators -> 512)
  static constexpr int TMEM_COLS = TMEM_USED <= 32 ? 32 : TMEM_USED <= 64 ? 64 : TMEM_USED <= 128 ? 128
                                 : TMEM_USED <= 256 ? 256 : 512;
  static_assert(TMEM_USED <= 512, "accumulators exceed TMEM");
  static constexpr int EPI_WARPS = 4 * MH;
  static constexpr int THREADS = 64 + 32 * EPI_WARPS;
  static constexpr int SMEM_BYTES = 1024 /*alignment slack*/ + STAGES * STAGE_BYTES + BAR_BYTES;
};

// Instruction descriptor, kind::f16: D fp32 (bits 4-5 = 1), A and B format at bits 7-9 / 10-12
// (0 = fp16, 1 = bf16), both K-major (bits 15, 16 = 0), N >> 3 at bits 17-22, M >> 4 at bits 24-28.
__host__ __device__ constexpr uint32_t idesc_for(bool bf, int BN) {
  return (1u << 4) | ((bf ? 1u : 0u) << 7) | ((bf ? 1u : 0u) << 10) | ((uint32_t)(BN >> 3) << 17) |
         ((uint32_t)(BM >> 4) << 24);
}

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ float silu_f(float x) { return x / (1.f + __expf(-x)); }
__device__ __forceinline__ float gelu_f(float x) {
  const float c = 0.7978845608028654f;
  return 0.5f * x * (1.f + tanhf(c * (x + 0.044715f * x * x * x)));
}

// 32 consecutive outputs of one row as 16-bit values (bf16, or fp16 saturated at +-65504)
__device__ __forceinline__ void store16x32(void* dst, const float* v, bool bf) {
  uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    uint32_t w[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float a = v[q * 8 + 2 * j], b = v[q * 8 + 2 * j + 1];
      if (bf) {
        __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
        w[j] = *reinterpret_cast<uint32_t*>(&h);
      } else {
        __half2 h = __floats2half2_rn(fminf(fmaxf(a, -65504.f), 65504.f), fminf(fmaxf(b, -65504.f), 65504.f));
        w[j] = *reinterpret_cast<uint32_t*>(&h);
      }
    }
    d4[q] = make_uint4(w[0], w[1], w[2], w[3]);
  }
}

struct EpiArgs {
  void* out;
  int ldo;  // elements
  int kind;
  int bf;   // operands and 16-bit outputs are bf16 (1) or fp16 (0)
  // sampling epilogue (LM head): one SampleRec per row and 64 vocabulary ids, [rows][n_chunks]; each row's
  // candidate id and token count select its noise
  SampleRec* rec;
  int n_chunks;
  const int* ids;
  const int* lens;
  GumbelParams gp;
  int lp;  // also the log-sum-exp of the raw logits (self-likelihood reward)
};

// ---- CTA-pair (cta_group::2) forms ----
// Wait whose phase is completed by arrivals from the peer CTA: acquire at cluster scope.
__device__ __forceinline__ bool mbar_test_cl(uint32_t addr, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(addr), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __noinline__ bool mbar_wait_cl(uint64_t* bar, uint32_t parity, volatile int* abort_flag) {
  const uint32_t addr = smem_u32(bar);
  if (mbar_test_cl(addr, parity)) return true;
  const unsigned long long t0 = gtimer();
  while (true) {
#pragma unroll 1
    for (int i = 0; i < 32; ++i)
      if (mbar_test_cl(addr, parity)) return true;
    if (abort_flag && *abort_flag) return false;
    if (gtimer() - t0 > WAIT_NS) return false;
  }
}
// Address of the barrier at this smem offset in CTA `cta` of the cluster.
__device__ __forceinline__ uint32_t cluster_addr(const void* p, uint32_t cta) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(p)), "r"(cta));
  return remote;
}
// Arrive on the barrier at this smem offset in CTA `cta` of the cluster (release at cluster scope).
__device__ __forceinline__ void mbar_arrive_cta(uint64_t* bar, uint32_t cta) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr(bar, cta))
               : "memory");
}
// 2D TMA load into this CTA's shared memory whose completion (complete_tx) is counted on a barrier of
// either CTA of the pair (`bar_cluster`, a shared::cluster address).
__device__ __forceinline__ void tma_load_2d_pair(void* dst, const CUtensorMap* map, uint32_t bar_cluster, int x,
                                                 int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.cta_group::2 [%0], [%1, {%3, "
      "%4}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar_cluster), "r"(x), "r"(y)
      : "memory");
}
// One M = 256 MMA over the pair: A rows 0-127 and W rows 0 .. N/2-1 from the issuing CTA's shared
// memory, A rows 128-255 and W rows N/2 .. N-1 from the same offsets in the peer's; each CTA's TMEM
// receives its 128 rows x N columns.
__device__ __forceinline__ void umma_pair(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(
          d_tmem),
      "l"(a), "l"(b), "r"(idesc), "r"(accumulate));
}
__device__ __forceinline__ void umma_pair_commit_mc(uint64_t* bar, uint16_t mask) {
  asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
                   smem_u32(bar)),
               "h"(mask)
               : "memory");
}

// Epilogue of one accumulator row segment: this thread's row of BNC fp32 columns at TMEM address
// `tbase`, converted / activated / added and stored at (row, col0 ..).  Rows >= M and columns >= N are
// skipped (they hold the zero-filled tails of the TMA tiles).
// Epilogue of 64 accumulator values v (columns col .. col + 63 of `row`): conversion / residual add / gated or
// GELU activation and the store.  Rows >= M and columns >= N are skipped (the zero-filled tails of the tiles).
__device__ __forceinline__ void epi_chunk(const EpiArgs& ep, float* v, int row, int col, int M, int N) {
  if (ep.kind == EPI_SWIGLU || ep.kind == EPI_GEGLU) {
    // gate / up rows interleaved in blocks of 16: columns col..col+15 gate, col+16..col+31 up, then the next pair
    if (row < M && col < N) {
      float g[32];
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        const int gi = (j < 16) ? j : j + 16;
        g[j] = (ep.kind == EPI_SWIGLU ? silu_f(v[gi]) : gelu_f(v[gi])) * v[gi + 16];
      }
      uint16_t* dst = reinterpret_cast<uint16_t*>(ep.out) + (size_t)row * ep.ldo + col / 2;
      store16x32(dst, g, ep.bf != 0);
    }
    return;
  }
#pragma unroll
  for (int hh = 0; hh < 2; ++hh) {
    float* w = v + 32 * hh;
    const int cc = col + 32 * hh;
    if (row < M && cc < N) {
      if (ep.kind == EPI_F32 || ep.kind == EPI_ADD_F32) {
        float4* dst = reinterpret_cast<float4*>(reinterpret_cast<float*>(ep.out) + (size_t)row * ep.ldo + cc);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          float4 o = make_float4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
          if (ep.kind == EPI_ADD_F32) {
            const float4 r = dst[q];
            o.x += r.x, o.y += r.y, o.z += r.z, o.w += r.w;
          }
          dst[q] = o;
        }
      } else {
        if (ep.kind == EPI_GELU) {
#pragma unroll
          for (int j = 0; j < 32; ++j) w[j] = gelu_f(w[j]);
        }
        store16x32(reinterpret_cast<uint16_t*>(ep.out) + (size_t)row * ep.ldo + cc, w, ep.bf != 0);
      }
    }
  }
}

// Sampling epilogue of the LM head (fused next-token sampling): the logits of one row are never stored; the
// Gumbel-max scan of sampling.cuh runs over them in id order (Philox counters of 4 ids, the exact skip test) and
// the row's record for each 64-id chunk keeps the largest perturbed logit, its id and raw logit, and the chunk's
// log-sum-exp partial.  The values are the same fp32 accumulators the plain epilogue would store, so the sampled
// token equals k_sample's on stored logits.  TMEM is read 16 columns at a time in a loop that is not unrolled,
// which keeps the epilogue's code small next to the MMA and TMA warps it shares the SM with.
struct SampleState {
  float best, best_a, m, s;
  int best_v;
};

__device__ __forceinline__ void sample_reset(SampleState& q) {
  q.best = -__int_as_float(0x7f800000), q.best_a = 0.f, q.m = -__int_as_float(0x7f800000), q.s = 0.f;
  q.best_v = 0x7fffffff;
}

// ids col .. col+31 (col a multiple of 32), v their 32 logits.  The eight Philox calls are independent (eight
// dependency chains in flight: the epilogue has one warp per SMSP, so this is its only latency hiding); the
// skip tests run against `ref`, the row's best before these ids (never above the running best, so a skipped id
// still cannot win), and are independent too; the ids that pass are then scanned in order.
__device__ __forceinline__ void sample_piece(const EpiArgs& ep, const float* v, int col, int N, int id, int step,
                                             SampleState& q) {
  uint32_t words[32];
#pragma unroll
  for (int g4 = 0; g4 < 8; ++g4) {
    const uint4 w = philox4x32_10(make_uint4((uint32_t)((col >> 2) + g4), (uint32_t)id, (uint32_t)step, 0u),
                                  ep.gp.k0, ep.gp.k1);
    words[4 * g4] = w.x, words[4 * g4 + 1] = w.y, words[4 * g4 + 2] = w.z, words[4 * g4 + 3] = w.w;
  }
  const float ref = q.best;
  uint32_t pass = 0u;
#pragma unroll
  for (int j = 0; j < 32; ++j)
    if (col + j < N && !gumbel_skip(v[j], col + j, words[j], ep.gp, ref)) pass |= 1u << j;
  if (ep.lp) {
#pragma unroll
    for (int j = 0; j < 32; ++j)
      if (col + j < N) lse_step(v[j], q.m, q.s);
  }
#pragma unroll
  for (int j = 0; j < 32; ++j)
    if ((pass >> j) & 1u)
      if (gumbel_step(v[j], col + j, words[j], ep.gp, q.best, q.best_v)) q.best_a = v[j];
}

__device__ __forceinline__ void sample_record(const EpiArgs& ep, const SampleState& q, int row, int col, float a0) {
  float4* dst = reinterpret_cast<float4*>(ep.rec + (size_t)row * ep.n_chunks + col / 64);
  dst[0] = make_float4(q.best, __int_as_float(q.best_v), q.best_a, q.m);
  dst[1] = make_float4(q.s, a0, 0.f, 0.f);  // a0: id 0's raw logit in chunk 0 (the all -inf fallback)
}

// A 64-column chunk already in registers (the stream-K merge path).
__device__ __forceinline__ void sample_chunk(const EpiArgs& ep, const float* v, int row, int col, int M, int N) {
  if (row >= M || col >= N) return;
  const int id = ep.ids[row];
  const int step = ep.lens[id];
  SampleState q;
  sample_reset(q);
#pragma unroll
  for (int p = 0; p < 64; p += 32) sample_piece(ep, v + p, col + p, N, id, step, q);
  sample_record(ep, q, row, col, v[0]);
}

// The sampling epilogue of one accumulator row segment of BNC columns at TMEM address `tbase`.
template <int BNC>
__device__ __forceinline__ void sample_store(const EpiArgs& ep, uint32_t tbase, int row, int col0, int M, int N) {
  const bool live = row < M;
  const int id = live ? ep.ids[row] : 0;
  const int step = live ? ep.lens[id] : 0;
  // The scan of each chunk starts from the best of the tile's earlier chunks: an id not above it cannot win, and
  // a chunk whose record keeps that value carries no id (INT_MAX), which never wins the reduction's comparisons.
  float carry = -__int_as_float(0x7f800000);
#pragma unroll 1
  for (int c = 0; c < BNC; c += 64) {
    float w64[64];
    tmem_ld64(tbase + c, w64);  // warp-collective: every lane loads
    SampleState q;
    sample_reset(q);
    q.best = carry;
#pragma unroll 1
    for (int p = 0; p < 2; ++p) {
      float v[32];
      if (p == 0) {  // static register indices for the half
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = w64[j];
      } else {
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = w64[32 + j];
      }
      if (live && col0 + c + 32 * p < N) sample_piece(ep, v, col0 + c + 32 * p, N, id, step, q);
    }
    if (live && col0 + c < N) sample_record(ep, q, row, col0 + c, w64[0]);
    carry = q.best;
  }
}

// Epilogue of one accumulator row segment: this thread's row of BNC fp32 columns at TMEM address `tbase`,
// 64 columns per load and wait.  EK = 1: the sampling epilogue.
template <int BNC, int EK = 0>
__device__ __forceinline__ void epi_store(const EpiArgs& ep, uint32_t tbase, int row, int col0, int M, int N) {
  if constexpr (EK == 1) {
    sample_store<BNC>(ep, tbase, row, col0, M, N);
  } else {
#pragma unroll 1
    for (int c = 0; c < BNC; c += 64) {
      float v[64];
      tmem_ld64(tbase + c, v);
      epi_chunk(ep, v, row, col0 + c, M, N);
    }
  }
}

// Tile t -> (M tile, N tile): groups of up to RASTER_M consecutive M tiles, M fastest within a group and the
// group's N tiles in order, so the CTAs resident at one time share a band of A rows that stays in L2 while W
// streams past (a single group -- every shape up to RASTER_M M tiles -- is plain M-fastest order).
constexpr int RASTER_M = 16;
__device__ __forceinline__ void tile_mn(int t, int num_m, int num_n, int& mb, int& nb) {
  const int per_group = RASTER_M * num_n;
  const int g = t / per_group, r = t - g * per_group;
  const int m0 = g * RASTER_M, gm = min(RASTER_M, num_m - m0);
  mb = m0 + r % gm;
  nb = r / gm;
}

// Stream-K: the num_tiles x num_k k-block units of a launch, tile by tile, are cut into gridDim.x contiguous
// shares of (almost) equal size; a CTA's share is a run of segments (tile, k-blocks kb0..kb1).  A segment that
// is not a whole tile writes its fp32 accumulator rows to one of the CTA's two partial slots (the share's first
// or last segment) and each epilogue warp counts its 32 rows on the tile's counter for its lane quadrant; the
// last of a tile's segments for those rows sums the slots in CTA order -- k order, so the result does not
// depend on which CTA finishes last -- applies the epilogue and resets the counter.  No warp waits on another.
struct SkArgs {
  float* part = nullptr;  // [gridDim.x][2] slots of [BN / 4][TM] float4
  int* cnt = nullptr;     // [num_tiles][4] (tile, TMEM lane quadrant), zero between launches
  int on = 0;
};
struct Seg {
  int tile, kb0, kb1;
};
__device__ __forceinline__ long long sk_share(long long total, int c, int C) { return total * c / C; }
__device__ __forceinline__ int sk_cta_of(long long u, long long total, int C) {
  int i = (int)(u * C / total);
  while (i + 1 < C && sk_share(total, i + 1, C) <= u) ++i;
  while (i > 0 && sk_share(total, i, C) > u) --i;
  return i;
}
// The i-th segment of this CTA (false past the last): whole tiles t0 + i tstep without stream-K.
__device__ __forceinline__ bool sk_segment(bool on, int i, int num_tiles, int num_k, long long u0, long long u1,
                                           int t0, int tstep, long long& cursor, Seg& sg) {
  if (!on) {
    const int t = t0 + i * tstep;
    if (t >= num_tiles) return false;
    sg = Seg{t, 0, num_k};
    return true;
  }
  if (cursor >= u1) return false;
  const int t = (int)(cursor / num_k), kb0 = (int)(cursor % num_k);
  const int kb1 = (int)min((long long)num_k, kb0 + (u1 - cursor));
  sg = Seg{t, kb0, kb1};
  cursor += kb1 - kb0;
  return true;
}

template <int TM, int BN, int EK = 0>
__global__ void __launch_bounds__(Cfg<TM, BN>::THREADS, 1)
    k_gemm_tc(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, EpiArgs ep, int M,
              int N, int K, int* err, unsigned long long wait_ns, SkArgs sk) {
  using C = Cfg<TM, BN>;
  static_assert(TM == 128 || TM == 256, "tile height");
  constexpr int A_BYTES = C::A_BYTES, B_BYTES = C::B_BYTES, STAGE_BYTES = C::STAGE_BYTES, STAGES = C::STAGES;
  constexpr int TMEM_COLS = C::TMEM_COLS, MH = C::MH, NACC = C::NACC, EPI_WARPS = C::EPI_WARPS;
  constexpr int ACC_COLS = MH * BN;  // TMEM columns of one accumulator buffer
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + STAGES * A_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
  uint64_t* empty = full + STAGES;
  uint64_t* tfull = empty + STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* mma_done = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t idesc = idesc_for(ep.bf != 0, BN);
  const int num_m = (M + TM - 1) / TM, num_n = (N + BN - 1) / BN;
  const int num_k = (K + BK - 1) / BK;
  // tiles of this CTA: index t over (M tile, N tile), M fastest; with stream-K (TM = 128) a share of k-block units
  const int num_tiles = num_m * num_n;
  const int t0 = blockIdx.x, tstep = gridDim.x;
  const bool skon = TM == 128 && sk.on;
  const long long sk_total = (long long)num_tiles * num_k;
  const long long u0 = skon ? sk_share(sk_total, blockIdx.x, gridDim.x) : 0;
  const long long u1 = skon ? sk_share(sk_total, blockIdx.x + 1, gridDim.x) : 0;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], EPI_WARPS);
    }
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_entry();  // prologue done; the operands written by the previous kernel are visible from here

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      int stage = 0;
      uint32_t phase = 0;
      int armed[STAGES];
      uint32_t armed_par[STAGES];
      for (int s = 0; s < STAGES; ++s) armed[s] = 0, armed_par[s] = 0;
      bool ok = true;
      long long cur = u0;
      Seg sg;
      for (int i = 0; ok && sk_segment(skon, i, num_tiles, num_k, u0, u1, t0, tstep, cur, sg); ++i) {
        int mb, nb;
        tile_mn(sg.tile, num_m, num_n, mb, nb);
        for (int kb = sg.kb0; kb < sg.kb1; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, wait_ns)) {
            ok = false;
            break;
          }
          mbar_expect_tx(&full[stage], STAGE_BYTES);
          tma_load_2d(sA + stage * A_BYTES, &tmA, &full[stage], kb * BK, mb * TM);
          tma_load_2d(sB + stage * B_BYTES, &tmB, &full[stage], kb * BK, nb * BN);
          armed[stage] = 1;
          armed_par[stage] = phase;
          if (++stage == STAGES) stage = 0, phase ^= 1u;
        }
      }
      if (!ok) {
        atomicExch(err, 1);
        *abort_flag = 1;
      }
      // drain: every armed copy completes its stage's phase before the CTA exits (immediate after a normal run,
      // where the MMAs consumed them; needed when another role gave up while copies were in flight)
      for (int s = 0; s < STAGES; ++s)
        if (armed[s]) mbar_wait(&full[s], armed_par[s], nullptr);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      long long cur = u0;
      Seg sg;
      for (int i = 0; ok && sk_segment(skon, i, num_tiles, num_k, u0, u1, t0, tstep, cur, sg); ++i) {
        if (!mbar_wait(&tempty[acc], acc_phase ^ 1u, abort_flag, wait_ns)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * ACC_COLS);
        for (int kb = sg.kb0; kb < sg.kb1; ++kb) {
          if (!mbar_wait(&full[stage], phase, abort_flag, wait_ns)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t b0 = sdesc(smem_u32(sB + stage * B_BYTES));
#pragma unroll
          for (int h = 0; h < MH; ++h) {  // 128-row halves of the tile share the W tile
            const uint64_t a0 = sdesc(smem_u32(sA + stage * A_BYTES + h * (BM * BK * 2)));
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk)  // +32 bytes per K=16 step inside the swizzle atom
              umma(d_tmem + (uint32_t)(h * BN), a0 + (uint64_t)(kk * 2), b0 + (uint64_t)(kk * 2), idesc,
                   (kb != sg.kb0 || kk != 0) ? 1u : 0u);
          }
          umma_commit(&empty[stage]);
          if (++stage == STAGES) stage = 0, phase ^= 1u;
        }
        if (!ok) break;
        umma_commit(&tfull[acc]);
        if (++acc == NACC) acc = 0, acc_phase ^= 1u;
      }
      if (!ok) {
        atomicExch(err, 2);
        *abort_flag = 1;
      }
      // all MMAs issued by this thread are complete once mma_done flips
      umma_commit(mma_done);
      mbar_wait(mma_done, 0, nullptr);
    }
  } else {
    // ---------------- epilogue (warps 2 .. 2 + EPI_WARPS) ----------------
    // warp w reads TMEM lane quadrant w % 4 (the hardware's lane-access rule) of half (w - 2) / 4
    const int quad = warp & 3, half = (warp - 2) / 4;
    int acc = 0;
    uint32_t acc_phase = 0;
    long long cur = u0;
    Seg sg;
    for (int i = 0; sk_segment(skon, i, num_tiles, num_k, u0, u1, t0, tstep, cur, sg); ++i) {
      const int tile = sg.tile;
      int mb, nb;
      tile_mn(tile, num_m, num_n, mb, nb);
      // one lane waits and broadcasts, so the warp-collective tcgen05.ld below stays converged
      int ok = (lane == 0) ? (int)mbar_wait(&tfull[acc], acc_phase, abort_flag, wait_ns) : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) {
        if (lane == 0) {
          atomicExch(err, 3);
          *abort_flag = 1;
        }
        break;
      }
      tc_fence_after();
      const int row = mb * TM + half * BM + quad * 32 + lane;
      const uint32_t tbase = tmem_base + ((uint32_t)(quad * 32) << 16) + (uint32_t)(acc * ACC_COLS + half * BN);
      if (sg.kb0 == 0 && sg.kb1 == num_k) {
        epi_store<BN, EK>(ep, tbase, row, nb * BN, M, N);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&tempty[acc]);
        if (++acc == NACC) acc = 0, acc_phase ^= 1u;
        continue;
      }
      // ---- a part of the tile: fp32 rows to this CTA's slot, then the tile's counter ----
      const long long ts = (long long)tile * num_k;
      const int which = ts >= u0 ? 1 : 0;  // the tile began inside the share: the share's last segment
      // slot layout [column group of 4][row]: a warp's float4 accesses cover 512 contiguous bytes
      const int r = quad * 32 + lane;       // row within the tile (TM = 128)
      float4* slot = reinterpret_cast<float4*>(sk.part) + ((size_t)blockIdx.x * 2 + which) * (TM * BN / 4) + r;
#pragma unroll 1
      for (int c = 0; c < BN; c += 64) {
        float v[64];
        tmem_ld64(tbase + c, v);
#pragma unroll
        for (int q = 0; q < 16; ++q)
          __stcg(slot + (size_t)(c / 4 + q) * TM, make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]));
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[acc]);  // the accumulator is free for the next segment
      if (++acc == NACC) acc = 0, acc_phase ^= 1u;
      // each epilogue warp counts its own 32 rows (one counter per tile and lane quadrant), so no warp waits on
      // another; the last of the tile's segments for these rows merges them
      __threadfence();
      __syncwarp();
      const int c0 = sk_cta_of(ts, sk_total, gridDim.x), c1 = sk_cta_of(ts + num_k - 1, sk_total, gridDim.x);
      int last = 0;
      if (lane == 0) last = atomicAdd(&sk.cnt[(size_t)tile * 4 + quad], 1) == c1 - c0;
      last = __shfl_sync(0xffffffffu, last, 0);
      if (!last) continue;
      __threadfence();
#pragma unroll 1
      for (int c = 0; c < BN; c += 64) {
        float v[64];
#pragma unroll
        for (int e = 0; e < 64; ++e) v[e] = 0.f;
        for (int cc = c0; cc <= c1; ++cc) {  // k order
          // the writer's slot rule: slot 1 where the tile began inside the writer's share (only c0's can)
          const int wc = sk_share(sk_total, cc, gridDim.x) <= ts ? 1 : 0;
          const float4* src = reinterpret_cast<const float4*>(sk.part) + ((size_t)cc * 2 + wc) * (TM * BN / 4) + r;
#pragma unroll
          for (int q = 0; q < 16; ++q) {
            const float4 p = __ldcg(src + (size_t)(c / 4 + q) * TM);  // L2: written by other SMs
            v[4 * q] += p.x, v[4 * q + 1] += p.y, v[4 * q + 2] += p.z, v[4 * q + 3] += p.w;
          }
        }
        if constexpr (EK == 1)
          sample_chunk(ep, v, row, nb * BN + c, M, N);
        else
          epi_chunk(ep, v, row, nb * BN + c, M, N);
      }
      if (lane == 0) sk.cnt[(size_t)tile * 4 + quad] = 0;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(TMEM_COLS) : "memory");
  }
}

// ---------------------------------------------------------------------------------------------
// CTA-pair GEMM (cta_group::2): clusters of two CTAs on two SMs compute one 256 x BNP tile with
// M = 256 MMAs issued by the even CTA.  Each CTA stages only its own 128 rows of A and BNP/2 rows of
// W per K block (32 KB for BNP = 256: 128 flop per staged byte, against 85 for a 128 x 256 tile on
// one SM), so six stages fit, and each CTA's TMEM holds its 128 x BNP share of two accumulators,
// keeping the epilogue overlapped with the next tile's mainloop.
//   warp 0 (both CTAs) : TMA of the CTA's own A and W halves into its own shared memory; both CTAs'
//                        copies complete on the even CTA's full barrier, which expects both
//   warp 1, even CTA   : issues the MMAs, commits stage release and accumulator-ready to both CTAs
//   warps 2-5 (both)   : epilogue of the CTA's 128 rows; arrive on the even CTA's tempty barrier
// Every wait is bounded.  On abort the even CTA drains the stages it armed (their phases count both
// CTAs' copies); the odd CTA, whose copies complete on the other CTA's barriers, waits 1 ms for its
// own copies in flight before it leaves.
template <int BNP>
struct PairCfg {
  static constexpr int A_BYTES = BM * BK * 2;             // 16 KB
  static constexpr int B_BYTES = (BNP / 2) * BK * 2;      // 16 KB for BNP = 256
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int STAGES = (192 * 1024) / STAGE_BYTES;
  static constexpr int TMEM_COLS = 2 * BNP;
  static constexpr int THREADS = 192;
  static constexpr int GUARD = 32 * 1024;  // keeps any operand read of the last stage inside the allocation
  static constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + GUARD + BAR_BYTES;
};

__host__ __device__ constexpr uint32_t idesc_pair(bool bf, int N) {
  return (1u << 4) | ((bf ? 1u : 0u) << 7) | ((bf ? 1u : 0u) << 10) | ((uint32_t)(N >> 3) << 17) |
         ((uint32_t)(256 >> 4) << 24);
}

template <int BNP, int EK = 0>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(192, 1)
    k_gemm_pair(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, EpiArgs ep, int M,
                int N, int K, int* err) {
  using C = PairCfg<BNP>;
  constexpr int A_BYTES = C::A_BYTES, B_BYTES = C::B_BYTES, STAGE_BYTES = C::STAGE_BYTES, STAGES = C::STAGES;
  constexpr int TMEM_COLS = C::TMEM_COLS;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + STAGES * A_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES + C::GUARD);
  uint64_t* empty = full + STAGES;
  uint64_t* tfull = empty + STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* mma_done = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  const uint32_t idesc = idesc_pair(ep.bf != 0, BNP);
  const int num_m = (M + 255) / 256, num_n = (N + BNP - 1) / BNP;
  const int num_k = (K + BK - 1) / BK;
  const int num_tiles = num_m * num_n;
  const int t0 = blockIdx.x / 2, tstep = gridDim.x / 2;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 8);  // four epilogue warps in each CTA
    }
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // both CTAs' barriers are initialised (and TMEM allocated) before any cross-CTA signal
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_entry();

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer (own halves) ----------------
      int stage = 0;
      uint32_t phase = 0;
      int armed[STAGES];
      uint32_t armed_par[STAGES];
      for (int s = 0; s < STAGES; ++s) armed[s] = 0, armed_par[s] = 0;
      bool ok = true;
      for (int tile = t0; tile < num_tiles && ok; tile += tstep) {
        int mb, nb;
      tile_mn(tile, num_m, num_n, mb, nb);
        for (int kb = 0; kb < num_k; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag)) {
            ok = false;
            break;
          }
          // the even CTA's barrier counts both CTAs' bytes; the odd CTA's copies may land first (the
          // transaction count goes negative until the expect_tx, and the phase cannot complete before it)
          if (rank == 0) mbar_expect_tx(&full[stage], 2 * STAGE_BYTES);
          const uint32_t bar = cluster_addr(&full[stage], 0);
          tma_load_2d_pair(sA + stage * A_BYTES, &tmA, bar, kb * BK, mb * 256 + (int)rank * BM);
          tma_load_2d_pair(sB + stage * B_BYTES, &tmB, bar, kb * BK, nb * BNP + (int)rank * (BNP / 2));
          armed[stage] = 1;
          armed_par[stage] = phase;
          if (++stage == STAGES) stage = 0, phase ^= 1u;
        }
      }
      if (!ok) {
        atomicExch(err, 1);
        *abort_flag = 1;
        if (rank == 0) {
          for (int s = 0; s < STAGES; ++s)
            if (armed[s]) mbar_wait(&full[s], armed_par[s], nullptr);
        } else {
          const unsigned long long t = gtimer();
          while (gtimer() - t < 1000000ull) {
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {
      // ---------------- MMA issuer (even CTA) ----------------
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      for (int tile = t0; tile < num_tiles && ok; tile += tstep) {
        if (!mbar_wait_cl(&tempty[acc], acc_phase ^ 1u, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BNP);
        for (int kb = 0; kb < num_k; ++kb) {
          if (!mbar_wait(&full[stage], phase, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t a0 = sdesc(smem_u32(sA + stage * A_BYTES));
          const uint64_t b0 = sdesc(smem_u32(sB + stage * B_BYTES));
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk)
            umma_pair(d_tmem, a0 + (uint64_t)(kk * 2), b0 + (uint64_t)(kk * 2), idesc, (kb | kk) != 0);
          umma_pair_commit_mc(&empty[stage], 0x3);
          if (++stage == STAGES) stage = 0, phase ^= 1u;
        }
        if (!ok) break;
        umma_pair_commit_mc(&tfull[acc], 0x3);
        if (++acc == 2) acc = 0, acc_phase ^= 1u;
      }
      if (!ok) {
        atomicExch(err, 2);
        *abort_flag = 1;
      }
      umma_pair_commit_mc(mma_done, 0x1);
      mbar_wait(mma_done, 0, nullptr);
    }
  } else {
    // ---------------- epilogue (warps 2..5 of both CTAs) ----------------
    const int quad = warp & 3;
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int tile = t0; tile < num_tiles; tile += tstep) {
      int mb, nb;
      tile_mn(tile, num_m, num_n, mb, nb);
      int ok = (lane == 0) ? (int)mbar_wait(&tfull[acc], acc_phase, abort_flag) : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) {
        if (lane == 0) {
          atomicExch(err, 3);
          *abort_flag = 1;
        }
        break;
      }
      tc_fence_after();
      const int row = mb * 256 + (int)rank * BM + quad * 32 + lane;
      const uint32_t tbase = tmem_base + ((uint32_t)(quad * 32) << 16) + (uint32_t)(acc * BNP);
      epi_store<BNP, EK>(ep, tbase, row, nb * BNP, M, N);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cta(&tempty[acc], 0);
      if (++acc == 2) acc = 0, acc_phase ^= 1u;
    }
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // the even CTA's MMAs are complete and no CTA signals the other any more
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(TMEM_COLS) : "memory");
  }
}

// ---------------------------------------------------------------------------------------------
// Skinny GEMM (M <= 512 rows, the decode batch after rejection): the product is computed transposed,
// C^T = W A^T, on a CTA pair.  The M = 256 side of each cta_group::2 MMA is 256 rows of W (128 per SM)
// and the N side is every row of A (MP = Nb * Np rows, padded, Nb MMAs of N = Np), so each SM stages
// 128 rows of W and MP / 2 rows of A per K block: for 308 rows, 36 KB for 128 x 320 x 64 MACs (146 flop
// per staged byte, against 51 useful for 128 x 128 tiles of a 3-tile-high M).  Few W tiles exist
// (N / 256), so the K range is split into `s_split` slices to fill the SMs; with s_split > 1 every unit
// writes its fp32 partial C^T tile to `part` [s][M][N] and k_splitk_reduce adds the slices in slice
// order and applies the epilogue.  TMEM per SM: MP columns per accumulator (two when 2 MP <= 512).
struct SkinnyGeo {
  int Np, nb, MP, sub_bytes, stage_bytes, stages, nacc, tmem_cols, s_split, kps, n_tiles;
};

__device__ __forceinline__ void store_row_val(const EpiArgs& ep, int m, int n, float v) {
  if (ep.kind == EPI_F32) {
    reinterpret_cast<float*>(ep.out)[(size_t)m * ep.ldo + n] = v;
  } else if (ep.kind == EPI_ADD_F32) {
    reinterpret_cast<float*>(ep.out)[(size_t)m * ep.ldo + n] += v;
  } else {
    if (ep.kind == EPI_GELU) v = gelu_f(v);
    uint16_t h;
    if (ep.bf) {
      const __nv_bfloat16 b = __float2bfloat16_rn(v);
      h = *reinterpret_cast<const uint16_t*>(&b);
    } else {
      const __half b = __float2half_rn(fminf(fmaxf(v, -65504.f), 65504.f));
      h = *reinterpret_cast<const uint16_t*>(&b);
    }
    reinterpret_cast<uint16_t*>(ep.out)[(size_t)m * ep.ldo + n] = h;
  }
}

template <int NB>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(192, 1)
    k_gemm_skinny(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmA, EpiArgs ep,
                  float* __restrict__ part, SkinnyGeo geo, int M, int N, int K, int* err) {
  constexpr int MAXST = 8;
  const int STAGES = geo.stages, STAGE_BYTES = geo.stage_bytes, SUB = geo.sub_bytes, Np = geo.Np, MP = geo.MP;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES + PairCfg<256>::GUARD);
  uint64_t* empty = full + MAXST;
  uint64_t* tfull = empty + MAXST;
  uint64_t* tempty = tfull + 2;
  uint64_t* mma_done = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  const uint32_t idesc = idesc_pair(ep.bf != 0, Np);
  const int num_k = (K + BK - 1) / BK;
  const int units = geo.n_tiles * geo.s_split;
  const int t0 = blockIdx.x / 2, tstep = gridDim.x / 2;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 8);
    }
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(geo.tmem_cols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_entry();

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer: 128 W rows + this CTA's halves of the A blocks ----------------
      int stage = 0;
      uint32_t phase = 0;
      int armed[MAXST];
      uint32_t armed_par[MAXST];
      for (int s = 0; s < MAXST; ++s) armed[s] = 0, armed_par[s] = 0;
      bool ok = true;
      for (int u = t0; u < units && ok; u += tstep) {
        const int tile = u % geo.n_tiles, slice = u / geo.n_tiles;
        const int kb0 = slice * geo.kps, kb1 = min(num_k, kb0 + geo.kps);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag)) {
            ok = false;
            break;
          }
          if (rank == 0) mbar_expect_tx(&full[stage], 2 * STAGE_BYTES);
          const uint32_t bar = cluster_addr(&full[stage], 0);
          uint8_t* st = smem + stage * STAGE_BYTES;
          tma_load_2d_pair(st, &tmW, bar, kb * BK, tile * 256 + (int)rank * BM);
#pragma unroll
          for (int i = 0; i < NB; ++i)
            tma_load_2d_pair(st + 16384 + i * SUB, &tmA, bar, kb * BK, i * Np + (int)rank * (Np / 2));
          armed[stage] = 1;
          armed_par[stage] = phase;
          if (++stage == STAGES) stage = 0, phase ^= 1u;
        }
      }
      if (!ok) {
        atomicExch(err, 1);
        *abort_flag = 1;
        if (rank == 0) {
          for (int s = 0; s < STAGES; ++s)
            if (armed[s]) mbar_wait(&full[s], armed_par[s], nullptr);
        } else {
          const unsigned long long t = gtimer();
          while (gtimer() - t < 1000000ull) {
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {
      // ---------------- MMA issuer (even CTA) ----------------
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      for (int u = t0; u < units && ok; u += tstep) {
        const int slice = u / geo.n_tiles;
        const int kb0 = slice * geo.kps, kb1 = min(num_k, kb0 + geo.kps);
        if (!mbar_wait_cl(&tempty[acc], acc_phase ^ 1u, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * MP);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(&full[stage], phase, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t st = smem_u32(smem + stage * STAGE_BYTES);
          const uint64_t aw = sdesc(st);
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk) {
#pragma unroll
            for (int i = 0; i < NB; ++i)
              umma_pair(d_tmem + (uint32_t)(i * Np), aw + (uint64_t)(kk * 2),
                        sdesc(st + 16384 + i * SUB) + (uint64_t)(kk * 2), idesc, (kb > kb0 || kk > 0) ? 1u : 0u);
          }
          umma_pair_commit_mc(&empty[stage], 0x3);
          if (++stage == STAGES) stage = 0, phase ^= 1u;
        }
        if (!ok) break;
        umma_pair_commit_mc(&tfull[acc], 0x3);
        if (++acc == geo.nacc) acc = 0, acc_phase ^= 1u;
      }
      if (!ok) {
        atomicExch(err, 2);
        *abort_flag = 1;
      }
      umma_pair_commit_mc(mma_done, 0x1);
      mbar_wait(mma_done, 0, nullptr);
    }
  } else {
    // ---------------- epilogue: lane = one W row (output column n), TMEM column = output row m ----------
    const int quad = warp & 3;
    const bool gated = ep.kind == EPI_SWIGLU || ep.kind == EPI_GEGLU;
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int u = t0; u < units; u += tstep) {
      const int tile = u % geo.n_tiles, slice = u / geo.n_tiles;
      int ok = (lane == 0) ? (int)mbar_wait(&tfull[acc], acc_phase, abort_flag) : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) {
        if (lane == 0) {
          atomicExch(err, 3);
          *abort_flag = 1;
        }
        break;
      }
      tc_fence_after();
      const int nbase = tile * 256 + (int)rank * BM + quad * 32;  // first W row of this warp (multiple of 32)
      const int n = nbase + lane;
      const uint32_t tbase = tmem_base + ((uint32_t)(quad * 32) << 16) + (uint32_t)(acc * MP);
      // one output column n per lane; TMEM column c = output row m
      auto emit = [&](int c, const float* v, auto cnt_c) {
        constexpr int cnt = decltype(cnt_c)::value;
        if (geo.s_split > 1) {
          float* dst = part + ((size_t)slice * M) * N + n;
#pragma unroll
          for (int j = 0; j < cnt; ++j)
            if (c + j < M) dst[(size_t)(c + j) * N] = v[j];
        } else if (gated) {
          // W rows interleave gate / up in blocks of 16: lanes 0-15 gate, 16-31 up of features 16 (nbase/32) + lane
          const int f = 16 * (nbase / 32) + lane;
#pragma unroll
          for (int j = 0; j < cnt; ++j) {
            const float up = __shfl_xor_sync(0xffffffffu, v[j], 16);
            if (lane < 16 && c + j < M) {
              const float a = (ep.kind == EPI_SWIGLU ? silu_f(v[j]) : gelu_f(v[j])) * up;
              uint16_t* o = reinterpret_cast<uint16_t*>(ep.out) + (size_t)(c + j) * ep.ldo + f;
              if (ep.bf) {
                const __nv_bfloat16 b = __float2bfloat16_rn(a);
                *o = *reinterpret_cast<const uint16_t*>(&b);
              } else {
                const __half b = __float2half_rn(fminf(fmaxf(a, -65504.f), 65504.f));
                *o = *reinterpret_cast<const uint16_t*>(&b);
              }
            }
          }
        } else {
#pragma unroll
          for (int j = 0; j < cnt; ++j)
            if (c + j < M) store_row_val(ep, c + j, n, v[j]);
        }
      };
      int c = 0;
#pragma unroll 1
      for (; c + 64 <= MP; c += 64) {  // 64 columns per load / wait
        float v[64];
        tmem_ld64(tbase + c, v);
        if (c < M && nbase < N) emit(c, v, std::integral_constant<int, 64>{});
      }
#pragma unroll 1
      for (; c < MP; c += 16) {
        float v[16];
        tmem_ld16(tbase + c, v);
        if (c < M && nbase < N) emit(c, v, std::integral_constant<int, 16>{});
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cta(&tempty[acc], 0);
      if (++acc == geo.nacc) acc = 0, acc_phase ^= 1u;
    }
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(geo.tmem_cols)
                 : "memory");
  }
}

// Sums the s fp32 partials of a split-K skinny GEMM in slice order and applies the epilogue.
// Non-gated: one thread per 4 consecutive outputs of a row; gated: per 4 consecutive features.
__global__ void __launch_bounds__(256) k_splitk_reduce(const float* __restrict__ part, int s, int M, int N,
                                                       EpiArgs ep) {
  pdl_entry();
  const bool gated = ep.kind == EPI_SWIGLU || ep.kind == EPI_GEGLU;
  const int cols = gated ? N / 2 : N;
  const size_t total = (size_t)M * (cols / 4);
  for (size_t t = blockIdx.x * (size_t)blockDim.x + threadIdx.x; t < total; t += (size_t)gridDim.x * blockDim.x) {
    const int m = (int)(t / (cols / 4)), c = (int)(t % (cols / 4)) * 4;
    if (!gated) {
      float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int k = 0; k < s; ++k) {
        const float4 p = *reinterpret_cast<const float4*>(part + ((size_t)k * M + m) * N + c);
        a.x += p.x, a.y += p.y, a.z += p.z, a.w += p.w;
      }
      const float v[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
      for (int j = 0; j < 4; ++j) store_row_val(ep, m, c + j, v[j]);
    } else {
      const int ng = 32 * (c / 16) + c % 16;  // gate rows of features c..c+3; up rows 16 further
      float4 g = make_float4(0.f, 0.f, 0.f, 0.f), u = g;
      for (int k = 0; k < s; ++k) {
        const float* row = part + ((size_t)k * M + m) * N;
        const float4 pg = *reinterpret_cast<const float4*>(row + ng), pu = *reinterpret_cast<const float4*>(row + ng + 16);
        g.x += pg.x, g.y += pg.y, g.z += pg.z, g.w += pg.w;
        u.x += pu.x, u.y += pu.y, u.z += pu.z, u.w += pu.w;
      }
      const float gv[4] = {g.x, g.y, g.z, g.w}, uv[4] = {u.x, u.y, u.z, u.w};
      EpiArgs e2 = ep;
      e2.kind = EPI_STORE;
#pragma unroll
      for (int j = 0; j < 4; ++j)
        store_row_val(e2, m, c + j, (ep.kind == EPI_SWIGLU ? silu_f(gv[j]) : gelu_f(gv[j])) * uv[j]);
    }
  }
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;
int g_num_sms = 0;
int g_bn_override = 0;  // SR_GEMM_BN: force one N-tile width (tuning sweeps)
int g_tm_override = 0;  // SR_GEMM_TM: force the tile height (128 or 256)
int g_pair_override = -1;  // SR_GEMM_PAIR: 1 forces the CTA-pair kernel, 0 forbids it
int g_skinny_override = -1;  // SR_GEMM_SKINNY: 0 forbids the skinny kernel (else used for M <= 512)
// SR_GEMM_WAIT_NS: bound of the one-SM kernel's pipeline waits (tests make it expire; the drains of copies and
// MMAs already issued keep the 2 s bound, so an expired wait ends the kernel cleanly with the error word set)
unsigned long long g_wait_ns = WAIT_NS;
// SR_GEMM_STREAMK=1: stream-K shares of k-blocks on 128 x 256 tiles for every shape with a k-block per SM.  Off
// by default: on GB300 it measured slower than the launcher's tile choices on every decode shape (the merge of
// a tile's partial sums by its last contributor costs more than the idle SMs of the last wave).
int g_sk_override = 0;
std::mutex g_ws_mu;
// split-K partial workspace (floats) per (device, stream): launches on one stream run in order, so one
// buffer per stream keeps contexts on different streams from sharing it.  sr_destroy frees the buffers
// of the context's own and sr_set_stream streams; a stream passed only to sr_k_gemm or sr_generate_dev keeps
// its buffer until process exit.
std::map<std::pair<int, cudaStream_t>, std::pair<float*, size_t>> g_ws;
int* g_err = nullptr;

// Estimated relative time of a tile width: waves of persistent CTAs x per-tile cost.  The per-tile
// cost has a part proportional to BN * K (MMA work and W-tile bytes) and a fixed part (A-tile
// traffic, pipeline fill, epilogue) that a sweep of the decode and scoring shapes on GB300 puts
// at about the cost of 430 columns of a K = 4096 tile.
int pick_bn(int M, int N, int K) {
  if (g_bn_override == 64 || g_bn_override == 128 || g_bn_override == 192 || g_bn_override == 256) return g_bn_override;
  int best = 256;
  double best_cost = -1;
  for (int bn : {256, 192, 128, 64}) {
    const long long tiles = (long long)((M + BM - 1) / BM) * ((N + bn - 1) / bn);
    const long long waves = (tiles + g_num_sms - 1) / g_num_sms;
    const double cost = (double)waves * (bn * (K / 4096.0) + 430.0);
    if (best_cost < 0 || cost < best_cost) best_cost = cost, best = bn;
  }
  return best;
}

// Tall 256 x 256 tiles pay when they keep the SMs about as busy as the 128-row tiles: compare waves x
// per-tile cost, a 256 x 256 tile costing about 1.5 128 x 256 tiles (twice the MMA work at the higher
// tensor-pipe occupancy its halved staging allows).
bool pick_tall(int M, int N, int K) {
  (void)K;
  if (M < 2 * BM) return false;
  const int bn = pick_bn(M, N, K);
  const double t_small = std::ceil((double)((M + BM - 1) / BM) * ((N + bn - 1) / bn) / g_num_sms) *
                         (bn * (K / 4096.0) + 430.0);
  const double t_tall = std::ceil((double)((M + 255) / 256) * ((N + 255) / 256) / g_num_sms) * 1.5 *
                        (256 * (K / 4096.0) + 430.0);
  return t_tall < t_small;
}

// Stream-K workspace per (device, stream): partial slots and the per-(tile, quadrant) counters, zeroed when
// allocated (every launch leaves them zero).
struct SkWs {
  float* part = nullptr;
  size_t part_cap = 0;
  int* cnt = nullptr;
  size_t cnt_cap = 0;
};
std::map<std::pair<int, cudaStream_t>, SkWs> g_skws;

sr_status sk_workspace(size_t part_floats, size_t cnt_ints, cudaStream_t st, SkArgs* sk) {
  int dev;
  SR_CUDA(cudaGetDevice(&dev));
  std::lock_guard<std::mutex> lk(g_ws_mu);
  SkWs& w = g_skws[std::make_pair(dev, st)];
  if (w.part_cap < part_floats) {
    if (w.part) SR_CUDA(cudaFree(w.part));
    w.part = nullptr;
    w.part_cap = 0;
    SR_CUDA(cudaMalloc(&w.part, part_floats * sizeof(float)));
    w.part_cap = part_floats;
  }
  if (w.cnt_cap < cnt_ints) {
    if (w.cnt) SR_CUDA(cudaFree(w.cnt));
    w.cnt = nullptr;
    w.cnt_cap = 0;
    SR_CUDA(cudaMalloc(&w.cnt, cnt_ints * sizeof(int)));
    SR_CUDA(cudaMemsetAsync(w.cnt, 0, cnt_ints * sizeof(int), st));
    w.cnt_cap = cnt_ints;
  }
  sk->part = w.part;
  sk->cnt = w.cnt;
  sk->on = 1;
  return SR_OK;
}

template <int TM, int BN, int EK = 0>
sr_status launch_bn(const CUtensorMap& ta, const CUtensorMap& tb, const EpiArgs& ep, int M, int N, int K,
                    cudaStream_t st, bool streamk = false) {
  using C = Cfg<TM, BN>;
  static int max_ctas = 0;
  if (!max_ctas) {
    SR_CUDA(cudaFuncSetAttribute(k_gemm_tc<TM, BN, EK>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_BYTES));
    max_ctas = g_num_sms;
  }
  const int tiles = ((M + TM - 1) / TM) * ((N + BN - 1) / BN);
  SkArgs sk;
  int grid = std::min(tiles, max_ctas);
  // stream-K needs a unit for every CTA (an empty share would leave a split tile's count short)
  if (streamk && TM == 128 && (long long)tiles * ((K + BK - 1) / BK) >= max_ctas) {
    grid = max_ctas;
    SR_TRY(sk_workspace((size_t)grid * 2 * TM * BN, (size_t)tiles * 4, st, &sk));
  }
  launch_k(k_gemm_tc<TM, BN, EK>, grid, C::THREADS, C::SMEM_BYTES, st, ta, tb, ep, M, N, K, g_err, g_wait_ns, sk);
  SR_CUDA(cudaGetLastError());
  return SR_OK;
}

// Where the CTA-pair kernel measured faster on GB300 than the one-SM tiles: gated epilogues (its
// double-buffered accumulator hides them), LM-head widths, and down-projection shapes (N <= 4096,
// K >= 8192) below 8192 rows; at least two pair rows (M >= 512) so the 256-row tiles are not mostly padding.
bool pick_pair(int M, int N, int K, bool gated) {
  if (M < 512) return false;
  // gated shapes: only where padding M to 256-row pair tiles wastes no more rows than 128-row tiles (at 600 rows
  // the pair ran 161 us against 139 us on 128 x 256 tiles for 28672 x 4096)
  const double eff_pair = (double)M / (256.0 * ((M + 255) / 256)), eff_128 = (double)M / (128.0 * ((M + 127) / 128));
  if (gated && eff_pair + 0.02 < eff_128) return false;
  return gated || N >= 65536 || (N <= 4096 && K >= 8192 && M < 8192);
}

template <int BNP, int EK = 0>
sr_status launch_pair(const CUtensorMap& ta, const CUtensorMap& tb, const EpiArgs& ep, int M, int N, int K,
                      cudaStream_t st) {
  using C = PairCfg<BNP>;
  static int max_pairs = 0;
  if (!max_pairs) {
    SR_CUDA(cudaFuncSetAttribute(k_gemm_pair<BNP, EK>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_BYTES));
    max_pairs = g_num_sms / 2;
    cudaLaunchConfig_t qc = {};
    qc.gridDim = dim3(max_pairs * 2);
    qc.blockDim = dim3(C::THREADS);
    qc.dynamicSmemBytes = C::SMEM_BYTES;
    int clusters = 0;
    if (cudaOccupancyMaxActiveClusters(&clusters, k_gemm_pair<BNP, EK>, &qc) == cudaSuccess && clusters > 0)
      max_pairs = std::min(max_pairs, clusters);
    cudaGetLastError();
  }
  const int tiles = ((M + 255) / 256) * ((N + BNP - 1) / BNP);
  const int pairs = std::min(tiles, max_pairs);
  launch_k(k_gemm_pair<BNP, EK>, pairs * 2, C::THREADS, C::SMEM_BYTES, st, ta, tb, ep, M, N, K, g_err);
  SR_CUDA(cudaGetLastError());
  return SR_OK;
}

sr_status encode_kmajor(CUtensorMap* map, const void* base, bool bf, int rows, int K, int box_rows);

sr_status skinny_workspace(size_t floats, cudaStream_t st, float** out) {
  int dev;
  SR_CUDA(cudaGetDevice(&dev));
  std::lock_guard<std::mutex> lk(g_ws_mu);
  auto& w = g_ws[std::make_pair(dev, st)];
  if (w.second < floats) {
    if (w.first) SR_CUDA(cudaFree(w.first));
    w.first = nullptr;
    w.second = 0;
    SR_CUDA(cudaMalloc(&w.first, floats * sizeof(float)));
    w.second = floats;
  }
  *out = w.first;
  return SR_OK;
}

constexpr int SKINNY_SMEM_MAX = 1024 + 192 * 1024 + PairCfg<256>::GUARD + BAR_BYTES;

template <int NB>
int skinny_max_pairs() {
  static int max_pairs = 0;
  if (!max_pairs) {
    cudaFuncSetAttribute(k_gemm_skinny<NB>, cudaFuncAttributeMaxDynamicSharedMemorySize, SKINNY_SMEM_MAX);
    max_pairs = g_num_sms / 2;
    cudaLaunchConfig_t qc = {};
    qc.gridDim = dim3(max_pairs * 2);
    qc.blockDim = dim3(192);
    qc.dynamicSmemBytes = SKINNY_SMEM_MAX;
    int clusters = 0;
    if (cudaOccupancyMaxActiveClusters(&clusters, k_gemm_skinny<NB>, &qc) == cudaSuccess && clusters > 0)
      max_pairs = std::min(max_pairs, clusters);
    cudaGetLastError();
  }
  return max_pairs;
}

// Geometry and split of the skinny kernel for an M-row product (M <= 512).
SkinnyGeo skinny_geometry(int M, int N, int K, int max_pairs) {
  SkinnyGeo g{};
  const int mp32 = (M + 31) / 32 * 32;
  g.nb = mp32 > 256 ? 2 : 1;
  g.Np = (mp32 / g.nb + 15) / 16 * 16;
  g.MP = g.nb * g.Np;
  g.sub_bytes = (g.Np / 2) * 128;
  g.stage_bytes = 16384 + g.nb * g.sub_bytes;
  g.stages = std::min(8, (192 * 1024) / g.stage_bytes);
  g.nacc = 2 * g.MP <= 512 ? 2 : 1;
  int cols = 32;
  while (cols < g.nacc * g.MP) cols *= 2;
  g.tmem_cols = cols;
  g.n_tiles = (N + 255) / 256;
  const int num_k = (K + BK - 1) / BK;
  int s = g.n_tiles >= max_pairs ? 1 : std::max(1, max_pairs / g.n_tiles);
  s = std::max(1, std::min({s, 8, num_k / 4}));
  g.kps = (num_k + s - 1) / s;
  g.s_split = (num_k + g.kps - 1) / g.kps;
  return g;
}

// Where the skinny kernel measured faster on GB300 than the 128-row tiles: shapes with few W tiles,
// where split-K fills the SMs (N below 256 x the SM pairs), and among those the narrow outputs
// (N <= 4096: O and down projections), the large reductions (K >= 8192) and the small batches
// (M <= 256).  Wide single-slice shapes (gate/up, LM head) stay on the one-SM tiles.
bool pick_skinny(int M, int N, int K) {
  if (M > 512) return false;
  const int max_pairs = std::min(skinny_max_pairs<1>(), skinny_max_pairs<2>());
  const SkinnyGeo g = skinny_geometry(M, N, K, max_pairs);
  if (g.s_split < 2) return false;
  return M <= 256 || K >= 8192 || N <= 4096;
}

sr_status launch_skinny(const void* A, const void* W, bool bf, const EpiArgs& ep, int M, int N, int K,
                        cudaStream_t st) {
  const int max_pairs = std::min(skinny_max_pairs<1>(), skinny_max_pairs<2>());
  const SkinnyGeo g = skinny_geometry(M, N, K, max_pairs);
  CUtensorMap tw, ta;
  SR_TRY(encode_kmajor(&tw, W, bf, N, K, BM));
  SR_TRY(encode_kmajor(&ta, A, bf, M, K, g.Np / 2));
  float* part = nullptr;
  if (g.s_split > 1) SR_TRY(skinny_workspace((size_t)g.s_split * M * N, st, &part));
  const int units = g.n_tiles * g.s_split;
  const int pairs = std::min(units, max_pairs);
  const size_t smem = 1024 + (size_t)g.stages * g.stage_bytes + PairCfg<256>::GUARD + BAR_BYTES;
  if (g.nb == 1)
    launch_k(k_gemm_skinny<1>, pairs * 2, 192, smem, st, tw, ta, ep, part, g, M, N, K, g_err);
  else
    launch_k(k_gemm_skinny<2>, pairs * 2, 192, smem, st, tw, ta, ep, part, g, M, N, K, g_err);
  SR_CUDA(cudaGetLastError());
  if (g.s_split > 1) {
    const bool gated = ep.kind == EPI_SWIGLU || ep.kind == EPI_GEGLU;
    const size_t total = (size_t)M * ((gated ? N / 2 : N) / 4);
    const int blocks = (int)std::min<size_t>((total + 255) / 256, (size_t)g_num_sms * 8);
    launch_k(k_splitk_reduce, blocks, 256, 0, st, (const float*)part, g.s_split, M, N, ep);
    SR_CUDA(cudaGetLastError());
  }
  return SR_OK;
}

sr_status encode_kmajor(CUtensorMap* map, const void* base, bool bf, int rows, int K, int box_rows) {
  std::call_once(g_encode_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
  if (!g_encode) return set_err(SR_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
  cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)K * 2};
  cuuint32_t box[2] = {(cuuint32_t)BK, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(map, bf ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2,
                        const_cast<void*>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return set_err(SR_ERR_INVALID_ARG, "cuTensorMapEncodeTiled failed (%d)", (int)r);
  return SR_OK;
}

}  // namespace

// SM count, the error word and the tuning switches, on the first GEMM of the process.
sr_status gemm_init() {
  if (!g_num_sms) {
    int dev;
    SR_CUDA(cudaGetDevice(&dev));
    SR_CUDA(cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev));
    if (!tc_error_word()) return set_err(SR_ERR_OOM, "gemm: error word allocation failed");
    if (const char* e = getenv("SR_GEMM_BN")) g_bn_override = atoi(e);
    if (const char* e = getenv("SR_GEMM_TM")) g_tm_override = atoi(e);
    if (const char* e = getenv("SR_GEMM_PAIR")) g_pair_override = atoi(e);
    if (const char* e = getenv("SR_GEMM_SKINNY")) g_skinny_override = atoi(e);
    if (const char* e = getenv("SR_GEMM_WAIT_NS")) g_wait_ns = strtoull(e, nullptr, 10);
    if (const char* e = getenv("SR_GEMM_STREAMK")) g_sk_override = atoi(e);
  }
  return SR_OK;
}

sr_status gemm_tc(int et, const void* A, const void* W, void* C, int M, int N, int K, int epi, cudaStream_t st) {
  if (et != SR_DT_BF16 && et != SR_DT_F16) return set_err(SR_ERR_INVALID_ARG, "gemm: operands must be bf16 or fp16");
  const bool bf = et == SR_DT_BF16;
  if (M <= 0 || N <= 0 || K <= 0) return M == 0 ? SR_OK : set_err(SR_ERR_INVALID_ARG, "gemm: bad shape");
  if (K % 8 != 0 || N % 32 != 0 || ((epi == EPI_SWIGLU || epi == EPI_GEGLU) && N % 64 != 0))
    return set_err(SR_ERR_INVALID_ARG, "gemm: needs K %% 8 == 0 and N %% 32 == 0 (N %% 64 for gated)");
  if ((reinterpret_cast<uintptr_t>(A) | reinterpret_cast<uintptr_t>(W)) & 15)
    return set_err(SR_ERR_INVALID_ARG, "gemm: operands must be 16-byte aligned");
  SR_TRY(gemm_init());
  const bool gated = epi == EPI_SWIGLU || epi == EPI_GEGLU;
  CUtensorMap ta, tb;
  EpiArgs ep{C, gated ? N / 2 : N, epi, bf ? 1 : 0};
  const bool forced = g_pair_override == 1 || g_bn_override != 0 || g_tm_override != 0;
  if (g_sk_override == 1) {
    SR_TRY(encode_kmajor(&ta, A, bf, M, K, BM));
    SR_TRY(encode_kmajor(&tb, W, bf, N, K, 256));
    return launch_bn<128, 256>(ta, tb, ep, M, N, K, st, true);
  }
  if (M <= 512 && g_skinny_override != 0 && (g_skinny_override == 1 || (!forced && pick_skinny(M, N, K))))
    return launch_skinny(A, W, bf, ep, M, N, K, st);
  if (g_pair_override == 1 ||
      (g_pair_override == -1 && g_bn_override == 0 && g_tm_override == 0 && pick_pair(M, N, K, gated))) {
    SR_TRY(encode_kmajor(&ta, A, bf, M, K, BM));
    SR_TRY(encode_kmajor(&tb, W, bf, N, K, 128));
    return launch_pair<256>(ta, tb, ep, M, N, K, st);
  }
  int tm = 128, bn = pick_bn(M, N, K);
  // (gated epilogues are the longest, and the single-buffered tall tile cannot hide them: 128-row tiles there)
  if (g_tm_override == 256 || (g_tm_override == 0 && g_bn_override == 0 && !gated && pick_tall(M, N, K)))
    tm = 256, bn = 256;
  SR_TRY(encode_kmajor(&ta, A, bf, M, K, tm));
  SR_TRY(encode_kmajor(&tb, W, bf, N, K, bn));
  if (tm == 256) return launch_bn<256, 256>(ta, tb, ep, M, N, K, st);
  if (bn == 64) return launch_bn<128, 64>(ta, tb, ep, M, N, K, st);
  if (bn == 128) return launch_bn<128, 128>(ta, tb, ep, M, N, K, st);
  if (bn == 192) return launch_bn<128, 192>(ta, tb, ep, M, N, K, st);
  return launch_bn<128, 256>(ta, tb, ep, M, N, K, st);
}

// Fused LM head + sampling: 256 x 256 CTA-pair tiles from 512 rows (as the launcher picks for LM-head widths),
// 128 x 256 one-SM tiles below; the sampling epilogue replaces the logits store.
sr_status lm_head_sample(bool bf, const void* x, const void* W, int M, int V, int K, const int* ids, const int* lens,
                         uint64_t seed, float temperature, float eos_bias, int eos_id, int lp, SampleRec* rec,
                         cudaStream_t st) {
  if (M <= 0) return M == 0 ? SR_OK : set_err(SR_ERR_INVALID_ARG, "lm_head_sample: bad shape");
  if (V <= 0 || K <= 0 || K % 8 != 0 || V % 32 != 0)
    return set_err(SR_ERR_INVALID_ARG, "lm_head_sample: needs K %% 8 == 0 and V %% 32 == 0");
  if (!(temperature > 0.f)) return set_err(SR_ERR_INVALID_ARG, "temperature must be > 0");
  if ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(W) | reinterpret_cast<uintptr_t>(rec)) & 15)
    return set_err(SR_ERR_INVALID_ARG, "lm_head_sample: operands must be 16-byte aligned");
  SR_TRY(gemm_init());
  EpiArgs ep{};
  ep.kind = EPI_F32;  // unused by the sampling epilogue
  ep.bf = bf ? 1 : 0;
  ep.rec = rec;
  ep.n_chunks = (V + SAMPLE_CHUNK - 1) / SAMPLE_CHUNK;
  ep.ids = ids;
  ep.lens = lens;
  ep.gp = GumbelParams{(uint32_t)(seed & 0xFFFFFFFFu), (uint32_t)(seed >> 32), 1.0f / temperature, eos_bias, eos_id};
  ep.lp = lp;
  CUtensorMap ta, tb;
  SR_TRY(encode_kmajor(&ta, x, bf, M, K, BM));
  if (M >= 512) {
    SR_TRY(encode_kmajor(&tb, W, bf, V, K, 128));
    return launch_pair<256, 1>(ta, tb, ep, M, V, K, st);
  }
  SR_TRY(encode_kmajor(&tb, W, bf, V, K, 256));
  return launch_bn<128, 256, 1>(ta, tb, ep, M, V, K, st);
}

// The device error word shared by the kernels with bounded waits (allocated on first use; nullptr when
// the allocation failed, in which case waits still end but are not reported).
int* tc_error_word() {
  if (!g_err) {
    if (cudaMalloc(&g_err, sizeof(int)) != cudaSuccess) {
      g_err = nullptr;
      return nullptr;
    }
    cudaMemset(g_err, 0, sizeof(int));
  }
  return g_err;
}

sr_status encode_tma_2d(CUtensorMap* map, const void* base, bool bf, int rows, int cols, int box_rows) {
  return encode_kmajor(map, base, bf, rows, cols, box_rows);
}

sr_status encode_tma_nd(CUtensorMap* map, const void* base, bool bf, int rank, const uint64_t* dims,
                        const uint64_t* strides_bytes, const uint32_t* box) {
  CUtensorMap tmp;
  SR_TRY(encode_kmajor(&tmp, base, bf, 1, 64, 1));  // resolves the driver entry point once
  cuuint64_t d[5];
  cuuint64_t st[4];
  cuuint32_t bx[5], es[5];
  for (int i = 0; i < rank; ++i) d[i] = dims[i], bx[i] = box[i], es[i] = 1;
  for (int i = 0; i + 1 < rank; ++i) st[i] = strides_bytes[i];
  CUresult r = g_encode(map, bf ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16, (cuuint32_t)rank,
                        const_cast<void*>(base), d, st, bx, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return set_err(SR_ERR_INVALID_ARG, "cuTensorMapEncodeTiled (rank %d) failed (%d)", rank, (int)r);
  return SR_OK;
}

// Device error word of the tensor-core GEMM (nonzero after a bounded wait expired).
int* gemm_error_word() { return g_err; }

// Free the split-K workspace kept for `st` on the current device (called when a context that used the
// stream is destroyed; the stream must have no GEMM in flight).
void gemm_release_workspace(cudaStream_t st) {
  int dev;
  if (cudaGetDevice(&dev) != cudaSuccess) return;
  std::lock_guard<std::mutex> lk(g_ws_mu);
  auto it = g_ws.find(std::make_pair(dev, st));
  if (it != g_ws.end()) {
    if (it->second.first) cudaFree(it->second.first);
    g_ws.erase(it);
  }
  auto is = g_skws.find(std::make_pair(dev, st));
  if (is != g_skws.end()) {
    if (is->second.part) cudaFree(is->second.part);
    if (is->second.cnt) cudaFree(is->second.cnt);
    g_skws.erase(is);
  }
}

}  // namespace sr
