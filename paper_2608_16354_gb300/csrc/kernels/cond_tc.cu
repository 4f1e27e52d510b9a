// adaLN modulation table of a call on the tensor cores (bf16 models):
//
//   mod[r][o] = sum_k silu(c_r)[k] W_ada[o][k] + b_ada[o],   r = (step, scene)
//
// for every step and scene of the call at once (K B rows) against the whole
// adaLN weight ((6 L + 2) d rows of d): a weight-streaming product whose
// bound is one read of W_ada (4.6 GB at d = 3072, L = 40).  The product is
// computed transposed, D[o][r] = W_ada[o][:] . X[r][:], so that the weight
// tile is the 128-row A operand streamed by TMA and the few activation rows
// are the B operand.  X = silu(c) is split into bf16 halves X = hi + lo
// (|lo| <= 2^-9 |X|), laid out per group of 64 rows as [64 hi rows; 64 lo
// rows], and one M = 128, N = 128 MMA per 16-deep step computes both
// products; the epilogue adds them (fp32 accuracy of the activations against
// the bf16 weights).
//
// Persistent CTAs, one per SM; work items (256 weight rows as two 128-row
// MMAs sharing each activation tile, 64-row group)
// ordered so that the groups of one weight tile run side by side (the tile
// is read from HBM once and from L2 by the other groups).  Warp 0 streams
// the tiles with TMA into a 4-stage ring, warp 1 issues the MMAs into one of
// two TMEM accumulators, warps 2-5 drain the other and write the table.
// Every mbarrier wait is bounded.
#include "common.cuh"
#include "kernels.h"

namespace dc {

namespace {

constexpr int kCM = 128, kCK = 64, kCRows = 64;  // weight rows, K step, activation rows per group
constexpr int kCTiles = 2;                       // weight tiles per item (sharing one activation tile)
constexpr int kCStages = 4;
constexpr int kCTileBytes = kCM * kCK * 2;       // 16 KB: a weight tile or a [hi; lo] tile
constexpr int kCStageBytes = (kCTiles + 1) * kCTileBytes;
constexpr int kCThreads = 192;
constexpr uint32_t kCIdesc = idesc_bf16_f32(kCM, 2 * kCRows);

struct __align__(8) CondBars {
  uint64_t full[kCStages];
  uint64_t empty[kCStages];
  uint64_t tmem_full[2];
  uint64_t tmem_empty[2];
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
};

constexpr int kCSmem = 1024 + kCStages * kCStageBytes + 256;

// silu(temb[k] + traj[s]) of row r = k B + s, split into bf16 hi / lo rows of
// its group: xs[(g * 128 + i) * d + e] = hi, xs[(g * 128 + 64 + i) * d + e] = lo
// (g = r / 64, i = r % 64)
__global__ void cond_split_kernel(const float* __restrict__ temb, const float* __restrict__ traj, int K,
                                  int B, int d, __nv_bfloat16* __restrict__ xs) {
  const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  const size_t total = (size_t)K * B * d;
  if (i >= total) return;
  const int e = (int)(i % d);
  const size_t r = i / d;
  const int s = (int)(r % B);
  const int k = (int)(r / B);
  const float v = silu(temb[(size_t)k * d + e] + traj[(size_t)s * d + e]);
  const __nv_bfloat16 hi = __float2bfloat16_rn(v);
  const size_t g = r / kCRows, w = r % kCRows;
  xs[(g * 2 * kCRows + w) * d + e] = hi;
  xs[(g * 2 * kCRows + kCRows + w) * d + e] = __float2bfloat16_rn(v - __bfloat162float(hi));
}

__global__ void __launch_bounds__(kCThreads, 1)
    cond_gemm_tc_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX,
                        int R, int O, int d, const float* __restrict__ bias, float* __restrict__ Y,
                        int* err) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t base = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + ((1024 - (base & 1023)) & 1023);
  uint8_t* sA = smem;                                // [stage][tile] weight tiles
  uint8_t* sB = smem + kCStages * kCTiles * kCTileBytes;  // [stage] activation tiles
  CondBars* bar = reinterpret_cast<CondBars*>(smem + kCStages * kCStageBytes);
  static_assert(sizeof(CondBars) <= 256, "barrier block exceeds its reserve");

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_rg = (R + kCRows - 1) / kCRows;
  const int n_items = ((O + kCTiles * kCM - 1) / (kCTiles * kCM)) * n_rg;
  const int KB = d / kCK;

  if (threadIdx.x == 0) {
    bar->abort = *(volatile int*)err;
    for (int s = 0; s < kCStages; ++s) {
      mbar_init(&bar->full[s], 1);
      mbar_init(&bar->empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bar->tmem_full[b], 1);
      mbar_init(&bar->tmem_empty[b], 4);  // one arrival per epilogue warp
    }
    mbar_init(&bar->drain, 1);
    fence_barrier_init();
    tma_prefetch_desc(&tmW);
    tma_prefetch_desc(&tmX);
  }
  if (warp == 1) {
    tmem_alloc(&bar->tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_trigger();
  pdl_wait();
  const uint32_t tmem_base = bar->tmem_base;
  const uint32_t wlim = work_wait_limit(err);

  if (bar->abort != 0) {
    // an earlier bounded wait gave up: do nothing, the host reports it
  } else if (warp == 0) {
    // ---------------------------------------------------------- TMA producer
    int stage = 0, issued = 0;
    uint32_t phase = 0;
    int last_phase[kCStages];
    for (int s = 0; s < kCStages; ++s) last_phase[s] = -1;
    bool ok = true;
    for (int it = blockIdx.x; it < n_items && ok; it += gridDim.x) {
      const int o0 = (it / n_rg) * kCTiles * kCM, rg = it % n_rg;
      for (int kb = 0; kb < KB; ++kb) {
        if (!mbar_wait_warp(&bar->empty[stage], phase ^ 1, err, kDevTimeoutTma, wlim)) { ok = false; break; }
        // copies issued by one thread complete one after another, so the three
        // boxes of a stage go out from three lanes that rotate over 0-7; a
        // weight tile past the last row is filled with zeros (its outputs are
        // not written)
        const int l0 = (3 * issued) & 7;
        if (lane == l0) mbar_arrive_expect_tx(&bar->full[stage], kCStageBytes);
        __syncwarp();
        for (int u = 0; u < kCTiles; ++u)
          if (lane == ((l0 + u) & 7))
            tma_load_2d(sA + (size_t)(stage * kCTiles + u) * kCTileBytes, &tmW, &bar->full[stage],
                        kb * kCK, o0 + u * kCM);
        if (lane == ((l0 + kCTiles) & 7))
          tma_load_2d(sB + (size_t)stage * kCTileBytes, &tmX, &bar->full[stage], kb * kCK,
                      rg * 2 * kCRows);
        __syncwarp();
        ++issued;
        last_phase[stage] = (int)phase;
        if (++stage == kCStages) { stage = 0; phase ^= 1; }
      }
    }
    // no copy may still be landing when the CTA leaves
    for (int s = 0; s < kCStages; ++s)
      if (last_phase[s] >= 0) mbar_wait_warp(&bar->full[s], (uint32_t)last_phase[s], err, kDevTimeoutTma);
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    int t = 0;
    const uint64_t dA = sw128_kmajor_desc(smem_u32(sA));
    const uint64_t dB = sw128_kmajor_desc(smem_u32(sB));
    for (int it = blockIdx.x; it < n_items && ok; it += gridDim.x, ++t) {
      const int b = t & 1;
      const uint32_t use = (uint32_t)(t >> 1);
      if (!mbar_wait_warp(&bar->tmem_empty[b], (use & 1) ^ 1, err, kDevTimeoutMma, wlim)) { ok = false; break; }
      tc_fence_after();
      const uint32_t d_tmem = tmem_base + (uint32_t)(b * kCTiles * 2 * kCRows);
      for (int kb = 0; kb < KB; ++kb) {
        if (!mbar_wait_warp(&bar->full[stage], phase, err, kDevTimeoutMma, wlim)) { ok = false; break; }
        tc_fence_after();
        if (elect_one()) {
#pragma unroll
          for (int kk = 0; kk < kCK / 16; ++kk)
#pragma unroll
            for (int u = 0; u < kCTiles; ++u)
              tc_mma_f16(d_tmem + (uint32_t)(u * 2 * kCRows),
                         dA + ((uint32_t)((stage * kCTiles + u) * kCTileBytes + kk * 32) >> 4),
                         dB + ((uint32_t)(stage * kCTileBytes + kk * 32) >> 4), kCIdesc,
                         (kb | kk) != 0 ? 1u : 0u);
          tc_commit(&bar->empty[stage]);
        }
        __syncwarp();
        if (++stage == kCStages) { stage = 0; phase ^= 1; }
      }
      if (ok) {
        if (elect_one()) tc_commit(&bar->tmem_full[b]);
        __syncwarp();
      }
    }
    // every MMA issued here has completed once `drain` flips
    if (elect_one()) tc_commit(&bar->drain);
    __syncwarp();
    mbar_wait_warp(&bar->drain, 0, err, kDevTimeoutMma);
  } else {
    // -------------------------------------------------------------- epilogue
    const int q = warp & 3;  // TMEM lane quarter: weight rows 32 q .. 32 q + 31
    int t = 0;
    for (int it = blockIdx.x; it < n_items; it += gridDim.x, ++t) {
      const int b = t & 1;
      const uint32_t use = (uint32_t)(t >> 1);
      if (!mbar_wait_warp(&bar->tmem_full[b], use & 1, err, kDevTimeoutEpi, wlim)) break;
      tc_fence_after();
      const int r0 = (it % n_rg) * kCRows;
#pragma unroll 1
      for (int u = 0; u < kCTiles; ++u) {
        const int o = (it / n_rg) * kCTiles * kCM + u * kCM + 32 * q + lane;
        const bool live = o < O;
        const float bo = live ? bias[o] : 0.f;
#pragma unroll 1
        for (int h = 0; h < 2; ++h) {
          float hv[32], lv[32];
          const uint32_t ta = tmem_base + (uint32_t)((b * kCTiles + u) * 2 * kCRows + 32 * h) +
                              ((uint32_t)(32 * q) << 16);
          tmem_ld32(ta, hv);
          tmem_ld32(ta + kCRows, lv);
          tmem_ld_wait();
          if (live) {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const int r = r0 + 32 * h + i;
              if (r < R) Y[(size_t)r * O + o] = (hv[i] + lv[i]) + bo;
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bar->tmem_empty[b]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, 512);
  }
}

}  // namespace

int cond_tc_group_rows() { return kCRows; }

cudaError_t launch_cond_split(const float* temb, const float* traj, int K, int B, int d,
                              __nv_bfloat16* xs, cudaStream_t st) {
  const size_t n = (size_t)K * B * d;
  if (n == 0) return cudaSuccess;
  cond_split_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(temb, traj, K, B, d, xs);
  return cudaGetLastError();
}

cudaError_t launch_cond_gemm_tc(const CUtensorMap& tmW, const CUtensorMap& tmX, int R, int O, int d,
                                const float* bias, float* Y, int* err, int n_sms, cudaStream_t st) {
  if (R <= 0) return cudaSuccess;
  if (O % kCM != 0 || d % kCK != 0) return cudaErrorInvalidValue;
  static std::atomic<unsigned long long> configured{0};
  const cudaError_t e = configure_once_per_device(configured, [] {
    return cudaFuncSetAttribute(cond_gemm_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kCSmem);
  });
  if (e != cudaSuccess) return e;
  const int n_items = ((O + kCTiles * kCM - 1) / (kCTiles * kCM)) * ((R + kCRows - 1) / kCRows);
  const int grid = n_items < n_sms ? n_items : n_sms;
  return launch_pdl(cond_gemm_tc_kernel, dim3(grid), dim3(kCThreads), kCSmem, st, tmW, tmX, R, O, d,
                    bias, Y, err);
}

}  // namespace dc
