// Shared device helpers and host-side declarations of libsr.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "sr.h"

namespace sr {

typedef __nv_bfloat16 bf16;
typedef __half f16;
// Element types of device tensors use the SR_DT_* codes: SR_DT_F32, SR_DT_BF16, SR_DT_F16.  Models
// whose weights arrive in bf16 (or fp16) run with fp16 operands and KV cache: every bf16 value of
// magnitude >= 2^-17 is exact in fp16, and fp16's 11-bit significand makes the rounding of
// activations fed to the tensor cores 8x finer than bf16's, at the same tensor-core rate.
constexpr int PAGE = 16;            // positions per KV page
constexpr int MAX_BATCH = 4096;     // largest N handled by the single-CTA control kernels

// ---------------------------------------------------------------------------------------------
// error reporting (host)
// ---------------------------------------------------------------------------------------------
sr_status set_err(sr_status s, const char* fmt, ...);

#define SR_CUDA(call)                                                                                 \
  do {                                                                                                \
    cudaError_t e_ = (call);                                                                          \
    if (e_ != cudaSuccess)                                                                            \
      return ::sr::set_err(e_ == cudaErrorMemoryAllocation ? SR_ERR_OOM : SR_ERR_CUDA, "%s:%d %s: %s", \
                           __FILE__, __LINE__, #call, cudaGetErrorString(e_));                        \
  } while (0)
#define SR_LAUNCH() SR_CUDA(cudaGetLastError())

// Programmatic dependent launch: every kernel of the library starts with pdl_entry(), which waits until
// the preceding kernel of the stream has completed and its writes are visible (a no-op when the kernel
// was launched without the attribute) and then lets the next kernel's CTAs be scheduled, so launch
// latency and prologues overlap the previous kernel's tail.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_next() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_entry() {
  pdl_wait();
  pdl_launch_next();
}
bool pdl_enabled();  // SR_PDL=0 in the environment turns the launch attribute off

// Launch `k` on `st` with the programmatic-stream-serialisation attribute; errors surface through
// cudaGetLastError (SR_LAUNCH).
template <typename... KArgs, typename... Args>
inline void launch_k(void (*k)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = pdl_enabled() ? 1 : 0;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  (void)cudaLaunchKernelEx(&cfg, k, static_cast<KArgs>(args)...);
}
#define SR_TRY(expr)               \
  do {                             \
    sr_status s_ = (expr);         \
    if (s_ != SR_OK) return s_;    \
  } while (0)

// ---------------------------------------------------------------------------------------------
// device helpers
// ---------------------------------------------------------------------------------------------
__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(bf16 x) { return __bfloat162float(x); }
__device__ __forceinline__ float to_f(f16 x) { return __half2float(x); }
template <typename T>
__device__ __forceinline__ T f_to(float x);
template <>
__device__ __forceinline__ float f_to<float>(float x) { return x; }
template <>
__device__ __forceinline__ bf16 f_to<bf16>(float x) { return __float2bfloat16_rn(x); }
// fp16 conversions saturate at the largest finite value instead of overflowing to infinity
template <>
__device__ __forceinline__ f16 f_to<f16>(float x) { return __float2half_rn(fminf(fmaxf(x, -65504.f), 65504.f)); }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// block-wide sum for blockDim.x <= 1024; `red` holds >= 32 floats
__device__ __forceinline__ float block_sum(float v, float* red) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  v = warp_sum(v);
  __syncthreads();
  if (lane == 0) red[wid] = v;
  __syncthreads();
  float t = (threadIdx.x < nw) ? red[threadIdx.x] : 0.f;
  if (wid == 0) t = warp_sum(t);
  if (threadIdx.x == 0) red[0] = t;
  __syncthreads();
  return red[0];
}

// block-wide exclusive scan of ints for blockDim.x <= 1024; returns the total; `tmp` >= 33 ints
__device__ __forceinline__ int block_excl_scan(int v, int* tmp, int* total) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  __syncthreads();
  if (lane == 31) tmp[wid] = x;
  __syncthreads();
  if (wid == 0) {
    int s = (lane < nw) ? tmp[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int y = __shfl_up_sync(0xffffffffu, s, o);
      if (lane >= o) s += y;
    }
    tmp[lane] = s;  // inclusive scan of warp totals
  }
  __syncthreads();
  int base = (wid > 0) ? tmp[wid - 1] : 0;
  if (total) *total = tmp[nw - 1];
  return base + x - v;
}

// order-preserving map float -> uint32 (-0 folded onto +0, NaN ordered as -inf)
__device__ __forceinline__ uint32_t float_key(float r) {
  if (r != r) r = -__int_as_float(0x7f800000);
  if (r == 0.f) r = 0.f;
  uint32_t u = __float_as_uint(r);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float key_float(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

// Run `body` with T bound to the device element type of code `et` (SR_DT_*).
#define SR_DISPATCH_ET(et, T, body)                                                       \
  switch (et) {                                                                           \
    case SR_DT_F32: { typedef float T; body; } break;                                     \
    case SR_DT_BF16: { typedef ::sr::bf16 T; body; } break;                               \
    case SR_DT_F16: { typedef ::sr::f16 T; body; } break;                                 \
    default: return ::sr::set_err(SR_ERR_INVALID_ARG, "unknown element type %d", (int)(et)); \
  }

// ---------------------------------------------------------------------------------------------
// host launchers implemented in the kernel files
// ---------------------------------------------------------------------------------------------
enum Epi { EPI_F32 = 0, EPI_ADD_F32 = 1, EPI_STORE = 2, EPI_SWIGLU = 3, EPI_GEGLU = 4, EPI_GELU = 5 };

// gemm_tc.cu: tcgen05 GEMM, C = A W^T, A and W both bf16 or both fp16 (et = SR_DT_BF16 / SR_DT_F16).
sr_status gemm_tc(int et, const void* A, const void* W, void* C, int M, int N, int K, int epi, cudaStream_t st);

// One record of the LM head's sampling epilogue: row r, vocabulary ids 64 c .. 64 c + 63.  z = the largest
// perturbed logit (-inf if none was finite), id its vocabulary id (INT_MAX if none), a its raw logit, (m, s) the
// log-sum-exp partial of the raw logits (running max, sum of exp(logit - m)), a0 = id 0's raw logit (chunk 0).
struct SampleRec {
  float z;
  int id;
  float a, m, s, a0, pad0, pad1;
};
constexpr int SAMPLE_CHUNK = 64;
// gemm_tc.cu: logits = x W^T for M rows and V vocabulary ids (fp16 or, bf, bf16 operands, fp32 accumulators) reduced to
// SampleRec[M][ceil(V / 64)] in the GEMM's epilogue -- the logits are never stored.  Row r's noise is keyed on
// (seed, ids[r], lens[ids[r]]); lp != 0 adds the log-sum-exp partials.
sr_status lm_head_sample(bool bf, const void* x, const void* W, int M, int V, int K, const int* ids, const int* lens,
                         uint64_t seed, float temperature, float eos_bias, int eos_id, int lp, SampleRec* rec,
                         cudaStream_t st);
// gemm_f32.cu: fp32 SIMT GEMM (epilogues EPI_F32, EPI_ADD_F32, EPI_STORE).
sr_status gemm_f32(const float* A, const float* W, float* C, int M, int N, int K, int epi, cudaStream_t st);

// elementwise.cu
sr_status launch_embed(int dtype, const void* tok_emb, const void* pos_emb, const int* tokens, const int* positions,
                       int M, int d, float* x, cudaStream_t st);
sr_status launch_norm(int dtype, int norm, const float* x, const void* w, const void* b, float eps, int M, int d,
                      void* out, cudaStream_t st);
sr_status launch_rope_table(float2* tab, int max_pos, int head_dim, double theta, cudaStream_t st);
struct KvSink {        // where a layer's new K/V rows go besides the contiguous k/v outputs
  void* pool_layer;    // this layer's page 0 in the pool, or nullptr
  const int* page_table;
  int pt_stride;
  const int* row_seq;  // page-table row per input row (nullptr: row 0 for every input row; < 0: not stored)
  int pos_base = 0;    // the pool pages hold positions pos_base, pos_base + 1, ... (page index (pos - pos_base) / 16)
  const int* n_rows = nullptr;  // device count: rows >= *n_rows write nothing to the pool (nullptr: every row)
};
sr_status launch_rope_store(int dtype, const float* qkv, int M, const int* positions, const float2* rope, int Hq,
                            int Hkv, int dh, void* q_out, void* k_out, void* v_out, KvSink sink, cudaStream_t st);
sr_status launch_act(int dtype, int act, const float* in, int M, int F, void* out, cudaStream_t st);
sr_status launch_score_head(int dtype, int norm, const float* x, const int* rows, int n, const void* w,
                            const void* b, float eps, const void* head, int d, float* rewards, cudaStream_t st);
sr_status launch_copy_page(int dtype, void* pool, long long layer_stride_elems, int n_layers, int page_elems,
                           int src_page, const int* dst_pages, int n_dst, cudaStream_t st);

// sample.cu
sr_status launch_sample(const float* logits, long long ld, int b, int V, const int* orig_ids, const int* steps,
                        uint64_t seed, float temperature, float eos_bias, int eos_id, int* tokens_out,
                        int* tok_hist, int max_new, int* lens, int* status, cudaStream_t st,
                        double* lp_sum = nullptr,   // lp_sum: += ln p(token) per candidate id (Section 5.3 reward)
                        const int* n_rows = nullptr);  // device count: rows >= *n_rows are skipped
// The same decision from lm_head_sample's records (n_chunks per row), reduced in vocabulary order.
sr_status launch_sample_reduce(const SampleRec* rec, int n_chunks, int b, const int* orig_ids, int eos_id,
                               int* tokens_out, int* tok_hist, int max_new, int* lens, int* status, cudaStream_t st,
                               double* lp_sum = nullptr, const int* n_rows = nullptr);

// attention.cu
// Workspace of the streaming decode-attention kernel (16-bit KV, head_dim 128, 8 kv heads): one persistent
// CTA per SM (grid); segment partials [grid][2][n_heads][130] floats; per-(row, kv head) counters [b][8]
// that must be zero before the first launch (each launch leaves them zero); pool_pages = pages per layer of
// the pool; err: set to 10 when a bounded wait expired.  Without it (nullptr) the per-row kernels run.
struct DecodeStreamWs {
  float* seg_part = nullptr;
  int* seg_cnt = nullptr;
  int grid = 0;
  int pool_pages = 0;
  int* err = nullptr;
};
size_t decode_stream_part_floats(int grid, int Hq);
// gemm_tc.cu: device error word shared by the kernels with bounded waits (GEMMs 1-3, decode attention 10);
// allocated on first use, nullptr if that failed
int* tc_error_word();
// shared_pos > 0: positions [0, shared_pos) sit in pages shared by every row's page table (the prompt);
// a tensor-core prefix pass reads them once per 64 rows and `part` must hold
// decode_attention_slots(max_len, window, shared_pos) partial slots per (row, head).
sr_status launch_decode_attention(int dtype, const void* q, const void* pool_layer, const int* page_table,
                                  int pt_stride, const int* slot_ids, const int* lens, int b, int Hq, int Hkv, int dh,
                                  int window, void* out, float* part, int max_splits, cudaStream_t st,
                                  int shared_pos = 0, int max_len = 0,  // max_len > 0: longest lens[] (launch shape)
                                  int* err = nullptr,   // set to 1 when a row needs more splits than max_splits
                                  const DecodeStreamWs* ws = nullptr);  // workspace of the streaming kernel
int decode_attention_max_splits(int max_len);
int decode_attention_slots(int max_len, int window, int shared_pos);
size_t decode_attention_part_floats(int b, int Hq, int dh, int max_splits);
// Keys of a prefill sequence that sit between the shared prefix and the sequence's own rows: positions
// pos0 .. pos0 + seq_cached[j] - 1 of sequence j, kept in a paged pool ([page][2 (K, V)][Hkv][16][dh] per
// layer) under page-table row seq_cand[j]; the sequence's own rows then start at position pos0 + seq_cached[j].
// pool == nullptr: no such keys.
struct CachedKeys {
  const void* pool = nullptr;  // this layer's page 0
  const int* page_table = nullptr;
  int pt_stride = 0;
  const int* seq_cand = nullptr;
  const int* seq_cached = nullptr;
  int pool_pages = 0;          // pages per layer of the pool (bounds of its tensor map)
};
sr_status launch_prefill_attention_f32(const float* q, const float* k, const float* v, const float* k_pre,
                                       const float* v_pre, int n_pre, const int* seq_off, int n_seq, int rows,
                                       int pos0, int Hq, int Hkv, int dh, int window, float* out, cudaStream_t st,
                                       CachedKeys ck = CachedKeys(), int max_cached = 0);  // max_cached >= seq_cached[]
sr_status launch_prefill_attention(int et, const void* q, const void* k, const void* v, const void* k_pre,
                                   const void* v_pre, int n_pre, const int* seq_off, int n_seq, const int* tile_seq,
                                   const int* tile_q0, int n_tiles, int pos0, int Hq, int Hkv, int dh, int window,
                                   void* out, cudaStream_t st, CachedKeys ck = CachedKeys(),
                                   int rows = 0);  // rows > 0: q/k/v rows (the tensor-core kernel needs it)
// elementwise.cu: in-place bf16 -> fp16 conversion of n elements (weights at load)
sr_status launch_bf16_to_f16(void* p, size_t n, cudaStream_t st);

// select.cu -- device control words and candidate states
enum Ctrl { C_NLIVE = 0, C_TOP, C_NRSET, C_ERR, C_PEAK, C_K, C_KRAISED, C_NACC, C_BEST, C_NPOOL, C_N };
enum Status { ST_LIVE = 0, ST_PENDING = 1, ST_DONE = 2, ST_REJECTED = 3, ST_WAITING = 4 };
enum CtlErr { E_POOL_EMPTY = 1, E_STATE = 2 };
sr_status ctl_pool_init(int* free_stack, int n_pages, int* ctrl, cudaStream_t st);
sr_status ctl_prompt_pages(int* free_stack, int* ctrl, int n_sh, int has_tail, int template_page, int* prompt_row,
                           cudaStream_t st);
sr_status ctl_admit(int start, int count, int n_sh, int has_tail, const int* prompt_row, int* pt, int max_pages,
                    int* len, int* status, int* live, int* rset, const int* free_stack, int* ctrl, int* tail_dst,
                    cudaStream_t st);
sr_status ctl_step_begin(int P, const int* live, int* ctrl, const int* len, int* pt, int max_pages,
                         const int* free_stack, const int* tok, int max_new, int* tok_in, int* pos_in, int* kv_len,
                         cudaStream_t st);
sr_status ctl_step_end(int P, int n_sh, int* live, int* ctrl, const int* len, const int* status, const int* pt,
                       int max_pages, int* free_stack, cudaStream_t st);
sr_status ctl_round(int P, int n_sh, float alpha, int pool_need, const float* rewards, int* rset, int* live,
                    int* ctrl, float* ctrlf, int* status, const int* len, float* reward_final, const int* pt,
                    int max_pages, int* free_stack, uint8_t* mask_out, cudaStream_t st);
sr_status ctl_mark_done(const int* ids, const float* r, int n, int* status, float* reward_final, cudaStream_t st);
sr_status ctl_final(int N, const int* status, const float* reward_final, const int* tok, int max_new, const int* len,
                    int* out_tokens, int* out_len, float* out_score, int* ctrl, cudaStream_t st);
sr_status launch_rcut(const float* rewards, int b, float alpha, int k_override, float* r_cut_out, uint8_t* mask_out,
                      cudaStream_t st);

}  // namespace sr
