// bf16 GEMM on the 5th-generation tensor cores (tcgen05), sm_103a.
//
//   C[M, N] = A[M, K] * W[N, K]^T   (A: activations, W: nn.Linear-style
//   weights, both K-major bf16), fp32 accumulation in TMEM, followed by one
//   of the fused DiT epilogues (QKV scatter, GELU, gated residual).
//
// Design: persistent CTAs (one per SM), 128 x 192 output tiles, K in steps
// of 64 (one 128-byte swizzle atom per row).  Warp 0 streams A/W tiles with
// TMA into a 4-stage shared-memory ring; warp 1 owns the TMEM allocation and
// one elected lane issues tcgen05.mma (M=128, N=192, K=16) into one of two
// TMEM accumulators; warps 2-9 drain the other accumulator with tcgen05.ld
// and run the epilogue, so the epilogue of tile i overlaps the MMAs of tile
// i+1.  N = 192 divides every projection width of the configured models
// (3d, d, 4d for d = 384, 1152, 3072).  Every mbarrier wait is bounded.
#include "common.cuh"
#include "epilogue.cuh"
#include "kernels.h"

namespace dc {

namespace {

constexpr int kBM = 128, kBN = 192, kBK = 64, kStages = 4;
constexpr int kABytes = kBM * kBK * 2;        // 16 KB
constexpr int kBBytes = kBN * kBK * 2;        // 24 KB
constexpr int kStageBytes = kABytes + kBBytes;
constexpr int kTmemCols = 512;                // two 192-column accumulators at 0 / 256
constexpr int kThreads = 320;                 // 10 warps
constexpr int kEpiWarps = 8;
constexpr uint32_t kIdesc = idesc_bf16_f32(kBM, kBN);
constexpr int kStgFloats = 32 * 33;           // per epilogue warp: 32 x 32 block, padded
constexpr size_t kSmemBytes =
    1024 + (size_t)kStages * kStageBytes + 256 + (size_t)kEpiWarps * kStgFloats * 4;

struct __align__(8) Barriers {
  uint64_t full[kStages];
  uint64_t empty[kStages];
  uint64_t tmem_full[2];
  uint64_t tmem_empty[2];
  uint64_t drain;
  uint32_t tmem_base;
};

template <int MODE>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_bf16_tc_kernel(const __grid_constant__ CUtensorMap tmA,
                        const __grid_constant__ CUtensorMap tmB, int M, int N, int K,
                        EpiArgs ep, SlotMap map, int* err) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t base = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + ((1024 - (base & 1023)) & 1023);
  uint8_t* sA = smem;
  uint8_t* sB = smem + (size_t)kStages * kABytes;
  Barriers* bar = reinterpret_cast<Barriers*>(smem + (size_t)kStages * kStageBytes);
  float* stg_all = reinterpret_cast<float*>(smem + (size_t)kStages * kStageBytes + 256);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int tiles_n = N / kBN;
  const int tiles_m = (M + kBM - 1) / kBM;
  const int n_tiles = tiles_m * tiles_n;
  const int KB = K / kBK;

  // a bounded wait of an earlier launch gave up: do nothing (the host
  // reports DC_ERR_DEVICE_TIMEOUT at its next check)
  if (*(volatile int*)err != 0) return;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&bar->full[s], 1);
      mbar_init(&bar->empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bar->tmem_full[b], 1);
      mbar_init(&bar->tmem_empty[b], kEpiWarps);
    }
    mbar_init(&bar->drain, 1);
    fence_barrier_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 1) {
    tmem_alloc(&bar->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = bar->tmem_base;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------ TMA producer
      int stage = 0;
      uint32_t phase = 0;
      int last_phase[kStages];
      for (int s = 0; s < kStages; ++s) last_phase[s] = -1;
      bool ok = true;
      for (int tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x) {
        const int m0 = (tile / tiles_n) * kBM;
        const int n0 = (tile % tiles_n) * kBN;
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(&bar->empty[stage], phase ^ 1, err, kDevTimeoutTma)) { ok = false; break; }
          mbar_arrive_expect_tx(&bar->full[stage], kStageBytes);
          tma_load_2d(sA + (size_t)stage * kABytes, &tmA, &bar->full[stage], kb * kBK, m0);
          tma_load_2d(sB + (size_t)stage * kBBytes, &tmB, &bar->full[stage], kb * kBK, n0);
          last_phase[stage] = (int)phase;
          if (++stage == kStages) { stage = 0; phase ^= 1; }
        }
      }
      // do not leave the CTA with copies still landing in shared memory
      for (int s = 0; s < kStages; ++s)
        if (last_phase[s] >= 0) mbar_wait(&bar->full[s], (uint32_t)last_phase[s], err, kDevTimeoutTma);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------ MMA issuer
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      int t = 0;
      for (int tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x, ++t) {
        const int b = t & 1;
        const uint32_t use = (uint32_t)(t >> 1);
        if (!mbar_wait(&bar->tmem_empty[b], (use & 1) ^ 1, err, kDevTimeoutMma)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(b * 256);
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(&bar->full[stage], phase, err, kDevTimeoutMma)) { ok = false; break; }
          tc_fence_after();
          const uint32_t a0 = smem_u32(sA + (size_t)stage * kABytes);
          const uint32_t b0 = smem_u32(sB + (size_t)stage * kBBytes);
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk) {
            tc_mma_f16(d_tmem, sw128_kmajor_desc(a0 + kk * 32), sw128_kmajor_desc(b0 + kk * 32),
                       kIdesc, (kb | kk) != 0 ? 1u : 0u);
          }
          tc_commit(&bar->empty[stage]);
          if (++stage == kStages) { stage = 0; phase ^= 1; }
        }
        if (ok) tc_commit(&bar->tmem_full[b]);
      }
      // every MMA this thread issued has completed once `drain` flips
      tc_commit(&bar->drain);
      mbar_wait(&bar->drain, 0, err, kDevTimeoutMma);
    }
  } else {
    // ---------------------------------------------------- epilogue warps
    const int q = warp & 3;             // TMEM lane quarter this warp may access
    const int half = (warp - 2) >> 2;   // which 96-column half of the tile
    int t = 0;
    for (int tile = blockIdx.x; tile < n_tiles; tile += gridDim.x, ++t) {
      const int b = t & 1;
      const uint32_t use = (uint32_t)(t >> 1);
      if (!mbar_wait(&bar->tmem_full[b], use & 1, err, kDevTimeoutEpi)) break;
      tc_fence_after();
      const int m0 = (tile / tiles_n) * kBM;
      const int n0 = (tile % tiles_n) * kBN;
      float acc[3][32];
#pragma unroll
      for (int c = 0; c < 3; ++c) {
        const uint32_t taddr =
            tmem_base + (uint32_t)(b * 256 + half * 96 + c * 32) + ((uint32_t)(q * 32) << 16);
        tmem_ld32(taddr, acc[c]);
      }
      tmem_ld_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bar->tmem_empty[b]);
      const int row0 = m0 + q * 32;
      if constexpr (MODE == kEpiResid) {
        // fp32 read-modify-write of the residual: transpose each 32 x 32
        // block through shared memory so that the warp reads and writes
        // whole 128-byte rows
        float* stg = stg_all + (warp - 2) * kStgFloats;
        if (row0 < M) {
#pragma unroll
          for (int c = 0; c < 3; ++c) {
#pragma unroll
            for (int i = 0; i < 32; ++i) stg[lane * 33 + i] = acc[c][i];
            __syncwarp();
            epilogue_block32<MODE>(ep, map, stg, row0, n0 + half * 96 + c * 32, lane);
            __syncwarp();
          }
        }
      } else {
        // bf16 outputs: each thread stores 16-byte pieces of its own row
        const int row = row0 + lane;
        if (row < M) {
#pragma unroll
          for (int c = 0; c < 3; ++c) {
#pragma unroll
            for (int g = 0; g < 4; ++g) {
              float v[8];
#pragma unroll
              for (int i = 0; i < 8; ++i) v[i] = acc[c][g * 8 + i];
              epilogue8<MODE, __nv_bfloat16>(ep, map, row, n0 + half * 96 + c * 32 + g * 8, v);
            }
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

}  // namespace

size_t gemm_tc_smem_bytes() { return kSmemBytes; }

template <int MODE>
static cudaError_t launch_mode(const CUtensorMap& tmA, const CUtensorMap& tmB, int M, int N, int K,
                               const EpiArgs& ep, const SlotMap& map, int* err, int n_sms,
                               cudaStream_t st) {
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(gemm_bf16_tc_kernel<MODE>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)kSmemBytes);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  const int tiles = ((M + kBM - 1) / kBM) * (N / kBN);
  const int grid = tiles < n_sms ? tiles : n_sms;
  gemm_bf16_tc_kernel<MODE><<<grid, kThreads, kSmemBytes, st>>>(tmA, tmB, M, N, K, ep, map, err);
  return cudaGetLastError();
}

cudaError_t launch_gemm_tc(int mode, const CUtensorMap& tmA, const CUtensorMap& tmB, int M, int N,
                           int K, const EpiArgs& ep, const SlotMap& map, int* err, int n_sms,
                           cudaStream_t st) {
  if (M <= 0) return cudaSuccess;
  if (N % kBN != 0 || K % kBK != 0) return cudaErrorInvalidValue;
  switch (mode) {
    case kEpiQKV: return launch_mode<kEpiQKV>(tmA, tmB, M, N, K, ep, map, err, n_sms, st);
    case kEpiGELU: return launch_mode<kEpiGELU>(tmA, tmB, M, N, K, ep, map, err, n_sms, st);
    case kEpiResid: return launch_mode<kEpiResid>(tmA, tmB, M, N, K, ep, map, err, n_sms, st);
  }
  return cudaErrorInvalidValue;
}

int gemm_tc_tile_n() { return kBN; }
int gemm_tc_tile_k() { return kBK; }
int gemm_tc_tile_m() { return kBM; }

}  // namespace dc
