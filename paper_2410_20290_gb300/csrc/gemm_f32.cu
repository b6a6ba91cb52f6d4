// fp32 dense layers for float32 models, C = A W^T on the CUDA cores.
//
// Only models whose descriptor says float32 (the tiny parity workload) use this path; bf16
// models run the tcgen05 kernel.  64x64 output tile per 256-thread block, 4x4 outputs per
// thread, K staged through shared memory 16 at a time.
#include "common.cuh"

namespace sr {
namespace {

constexpr int TM = 64, TN = 64, TK = 16;

__global__ void __launch_bounds__(256) k_gemm_f32(const float* __restrict__ A, const float* __restrict__ W,
                                                  float* __restrict__ C, int M, int N, int K, int epi) {
  pdl_entry();
  __shared__ float sA[TK][TM + 4];
  __shared__ float sW[TK][TN + 4];
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  const int m0 = blockIdx.y * TM, n0 = blockIdx.x * TN;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += TK) {
    for (int i = threadIdx.x; i < TM * TK; i += 256) {
      const int r = i / TK, c = i % TK;
      const int gm = m0 + r, gn = n0 + r, gk = k0 + c;
      sA[c][r] = (gm < M && gk < K) ? A[(size_t)gm * K + gk] : 0.f;
      sW[c][r] = (gn < N && gk < K) ? W[(size_t)gn * K + gk] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < TK; ++kk) {
      float a[4], w[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = sA[kk][ty * 4 + i], w[i] = sW[kk][tx * 4 + i];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], w[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int gm = m0 + ty * 4 + i;
    if (gm >= M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int gn = n0 + tx * 4 + j;
      if (gn >= N) continue;
      float* c = C + (size_t)gm * N + gn;
      *c = (epi == EPI_ADD_F32) ? *c + acc[i][j] : acc[i][j];
    }
  }
}

}  // namespace

sr_status gemm_f32(const float* A, const float* W, float* C, int M, int N, int K, int epi, cudaStream_t st) {
  if (M == 0) return SR_OK;
  if (M < 0 || N <= 0 || K <= 0) return set_err(SR_ERR_INVALID_ARG, "gemm_f32: bad shape");
  if (epi != EPI_F32 && epi != EPI_ADD_F32 && epi != EPI_STORE)
    return set_err(SR_ERR_INVALID_ARG, "gemm_f32: epilogue %d not supported for fp32", epi);
  dim3 grid((N + TN - 1) / TN, (M + TM - 1) / TM);
  launch_k(k_gemm_f32, grid, 256, 0, st, A, W, C, M, N, K, epi);
  SR_LAUNCH();
  return SR_OK;
}

}  // namespace sr
