// fp32 GEMM on the CUDA cores (FFMA) for the fp32 workload, where TF32 or
// bf16 tensor-core inputs would exceed the 1e-4 tolerance:
//   C[M, N] = A[M, K] * W[N, K]^T  followed by the same fused epilogues as
// the tensor-core GEMM.  64 x 64 tiles, K in steps of 16, 128 threads, each
// thread 4 rows x 8 columns.
#include "common.cuh"
#include "epilogue.cuh"
#include "kernels.h"

namespace dc {

namespace {

constexpr int kTM = 64, kTN = 64, kTK = 16;

template <int MODE>
__global__ void __launch_bounds__(128)
    gemm_f32_kernel(const float* __restrict__ A, const float* __restrict__ W, int M, int N, int K,
                    EpiArgs ep, SlotMap map) {
  __shared__ float sA[kTK][kTM + 4];
  __shared__ float sW[kTK][kTN + 4];
  const int tid = threadIdx.x;
  const int tr = tid / 8;  // 16 row groups of 4
  const int tc = tid % 8;  // 8 column groups of 8
  const int m0 = blockIdx.y * kTM, n0 = blockIdx.x * kTN;
  float acc[4][8];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;
  for (int k0 = 0; k0 < K; k0 += kTK) {
    for (int i = tid; i < kTM * kTK; i += 128) {
      const int r = i / kTK, c = i % kTK;
      const int gr = m0 + r, gc = k0 + c;
      sA[c][r] = (gr < M && gc < K) ? A[(size_t)gr * K + gc] : 0.f;
      const int wr = n0 + r;
      sW[c][r] = (wr < N && gc < K) ? W[(size_t)wr * K + gc] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < kTK; ++kk) {
      float a[4], w[8];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = sA[kk][tr * 4 + i];
#pragma unroll
      for (int j = 0; j < 8; ++j) w[j] = sW[kk][tc * 8 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] += a[i] * w[j];
    }
    __syncthreads();
  }
  const int col = n0 + tc * 8;
  if (col >= N) return;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int row = m0 + tr * 4 + i;
    if (row < M) epilogue8<MODE, float>(ep, map, row, col, acc[i]);
  }
}

}  // namespace

cudaError_t launch_gemm_f32(int mode, const float* A, const float* W, int M, int N, int K,
                            const EpiArgs& ep, const SlotMap& map, cudaStream_t st) {
  if (M <= 0) return cudaSuccess;
  if (N % 8 != 0) return cudaErrorInvalidValue;
  dim3 grid((N + kTN - 1) / kTN, (M + kTM - 1) / kTM);
  switch (mode) {
    case kEpiQKV: gemm_f32_kernel<kEpiQKV><<<grid, 128, 0, st>>>(A, W, M, N, K, ep, map); break;
    case kEpiGELU: gemm_f32_kernel<kEpiGELU><<<grid, 128, 0, st>>>(A, W, M, N, K, ep, map); break;
    case kEpiResid: gemm_f32_kernel<kEpiResid><<<grid, 128, 0, st>>>(A, W, M, N, K, ep, map); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace dc
