// Reuse step of the bf16 path on tcgen05 (Eq. 1: the interface H_k on a
// reused cache row, and the Euler update).
//
// The cache row of a scene is c = h_L - x W_e^T (r + b_e + pos), so h = x_k
// W_e^T + c_j, and with W' = (1 + scale) W_f (see interface_tc.cu):
//   P_c     = (x G_s)_c + Q_c,   Q_c = sum_e c_e W'[c][e]
//   sum h   = x . w_sum + sum c
//   sum h^2 = x^T G x + 2 x . A + sum c^2,   A = W_e c
//   v_c     = rs (P_c - mu S'_c) + beta_c
// sum c and sum c^2 were stored beside the row when it was written, so the
// one contraction over d is [A | Q] = c [W_e^T | W'hi | W'lo]^T (N = 48): per
// CTA a 128-token tile of one scene is the A operand (M = 128), streamed in
// 64-column stages by TMA with the step's 48 B rows, one MMA per 16-deep
// step.  The fp32 accumulator (48 TMEM columns) stays in TMEM until the four
// epilogue warps (one token row per thread) read their row and finish the
// token, so each cache row is read once and no thread touches it.  A CTA
// finishes the first `rows` tokens of its tile (128, or fewer so that a
// scene's CTAs cover all SMs; the rest of the tile is the next CTA's).
//
//   warp 0      TMA: cache tile [128 rows][64] and B tile [48][64] per stage
//   warp 1      tcgen05.mma into TMEM; owns TMEM
//   warps 2-5   the per-token finish
// Every mbarrier wait is bounded.
#include "common.cuh"
#include "kernels.h"

namespace dc {

namespace {

constexpr int kRC = 16;                            // latent channels
constexpr int kRTab = 2 * kRC + kRC * kRC;         // S', beta, G_s per (step, scene)
constexpr int kRB = 3 * kRC;                       // B rows: W_e^T, W' hi, W' lo
constexpr int kRM = 128, kRK = 64;                 // tokens per CTA, columns per stage
constexpr int kRStages = 9;
constexpr int kRABytes = kRM * kRK * 2;            // 16 KB
constexpr int kRBBytes = kRB * kRK * 2;            // 6 KB
constexpr int kRStageBytes = kRABytes + kRBBytes;  // 22 KB (a multiple of 1024)
static_assert(kRStageBytes % 1024 == 0, "stages must keep the 1024-byte swizzle alignment");
constexpr int kRThreads = 192;
constexpr uint32_t kRIdesc = idesc_bf16_f32(kRM, kRB);     // [A | Q]: columns 0-47
constexpr int kRTmemCols = 64;

struct __align__(8) ReuseBars {
  uint64_t full[kRStages];
  uint64_t empty[kRStages];  // the stage's MMAs have read it
  uint64_t tmem_full;
  uint32_t tmem_base;
  int abort;
  uint32_t wlim;
};

constexpr int kRSmem = 1024 + kRStages * kRStageBytes + 256 +
                       (kRTab + kRC + kRC * kRC) * 4;  // + tables

__global__ void __launch_bounds__(kRThreads, 1)
    head_reuse_tc_kernel(const __grid_constant__ CUtensorMap tmC,
                         const __grid_constant__ CUtensorMap tmB, float* __restrict__ x,
                         const float2* __restrict__ cstat, SlotMap map, int N, int d, int rows,
                         int b_row0, const float* __restrict__ tab_k,
                         const float* __restrict__ wsum, const float* __restrict__ gram,
                         float dsig, float* __restrict__ vout, int* err) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t sbase = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + ((1024 - (sbase & 1023)) & 1023);
  ReuseBars* bar = reinterpret_cast<ReuseBars*>(smem + kRStages * kRStageBytes);
  float* stab = reinterpret_cast<float*>(smem + kRStages * kRStageBytes + 256);
  static_assert(sizeof(ReuseBars) <= 256, "barrier block exceeds its reserve");

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int slot = blockIdx.y, scene = map.scene[slot];
  const int tok0 = blockIdx.x * rows;  // this CTA finishes tokens tok0 .. tok0 + rows - 1
  const int KB = d / kRK;

  if (threadIdx.x == 0) {
    bar->abort = *(volatile int*)err;
    bar->wlim = work_wait_limit(err);
    for (int s = 0; s < kRStages; ++s) {
      mbar_init(&bar->full[s], 1);
      mbar_init(&bar->empty[s], 1);
    }
    mbar_init(&bar->tmem_full, 1);
    fence_barrier_init();
    tma_prefetch_desc(&tmC);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 1) {
    tmem_alloc(&bar->tmem_base, kRTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_trigger();
  pdl_wait();
  const uint32_t tmem = bar->tmem_base;
  const uint32_t wlim = bar->wlim;

  if (bar->abort != 0) {
    // an earlier bounded wait gave up: do nothing, the host reports it
  } else if (warp == 0) {
    // ------------------------------------------------------------ TMA
    // the box covers kRM rows from tok0: rows past `rows` (the next CTA's,
    // read by it at about the same time) and past the scene are not finished
    const int crow = scene * N + tok0;
    const int brow = b_row0 + scene * kRB;
    int stage = 0, issued = 0;
    uint32_t phase = 0;
    for (int kb = 0; kb < KB; ++kb) {
      if (!mbar_wait_warp(&bar->empty[stage], phase ^ 1, err, kDevTimeoutTma, wlim)) break;
      // two copies per stage, from two lanes (copies of one thread land one
      // after another), rotating over lanes 0-7
      const int l0 = (2 * kb) & 7;
      if (lane == l0) mbar_arrive_expect_tx(&bar->full[stage], kRStageBytes);
      __syncwarp();
      uint8_t* st = smem + (size_t)stage * kRStageBytes;
      if (lane == l0) tma_load_2d(st, &tmC, &bar->full[stage], kb * kRK, crow);
      if (lane == l0 + 1) tma_load_2d(st + kRABytes, &tmB, &bar->full[stage], kb * kRK, brow);
      __syncwarp();
      ++issued;
      if (++stage == kRStages) { stage = 0; phase ^= 1; }
    }
    // every copy in flight lands before the CTA can exit: stage s was last
    // filled by load s + kRStages ((issued - 1 - s) / kRStages), in that phase
    for (int s = 0; s < kRStages && s < issued; ++s)
      mbar_wait_warp(&bar->full[s], (uint32_t)(((issued - 1 - s) / kRStages) & 1), err, kDevTimeoutTma);
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA
    int stage = 0;
    uint32_t phase = 0;
    for (int kb = 0; kb < KB; ++kb) {
      if (!mbar_wait_warp(&bar->full[stage], phase, err, kDevTimeoutMma, wlim)) break;
      tc_fence_after();
      if (elect_one()) {
        const uint32_t sa = smem_u32(smem + (size_t)stage * kRStageBytes);
        const uint64_t da = sw128_kmajor_desc(sa), db = sw128_kmajor_desc(sa + kRABytes);
#pragma unroll
        for (int kk = 0; kk < kRK / 16; ++kk) {
          const uint32_t acc = (kb | kk) != 0 ? 1u : 0u;
          tc_mma_f16(tmem, da + (uint32_t)(kk * 2), db + (uint32_t)(kk * 2), kRIdesc, acc);
        }
        tc_commit(&bar->empty[stage]);
      }
      __syncwarp();
      if (++stage == kRStages) { stage = 0; phase ^= 1; }
    }
    // tmem_full flips once every MMA issued here has completed: it hands the
    // accumulator to the epilogue, and this warp waits for it too, so TMEM is
    // never freed under an MMA in flight (also when a wait gave up)
    if (elect_one()) tc_commit(&bar->tmem_full);
    __syncwarp();
    mbar_wait_warp(&bar->tmem_full, 0, err, kDevTimeoutMma);
  } else {
    // ------------------------------------------------------ token finish
    const int q = warp & 3;            // TMEM lane quarter
    const int r = q * 32 + lane;       // token row of the tile owned by this thread
    for (int i = threadIdx.x - 64; i < kRTab; i += 128) stab[i] = tab_k[(size_t)scene * kRTab + i];
    if (threadIdx.x - 64 < kRC) stab[kRTab + threadIdx.x - 64] = wsum[threadIdx.x - 64];
    for (int i = threadIdx.x - 64; i < kRC * kRC; i += 128) stab[kRTab + kRC + i] = gram[i];
    named_bar(1, 128);  // the tables are staged
    if (mbar_wait_warp(&bar->tmem_full, 0, err, kDevTimeoutEpi, wlim)) {
      tc_fence_after();
      float acc[64];  // columns 48-63 are not written by the MMA and not used
      {
        const uint32_t lanes = (uint32_t)(q * 32) << 16;
        tmem_ld32(tmem + lanes, *reinterpret_cast<float(*)[32]>(acc));
        tmem_ld32(tmem + 32 + lanes, *reinterpret_cast<float(*)[32]>(acc + 32));
        tmem_ld_wait();
      }
      const int tok = tok0 + r;
      if (r < rows && tok < N) {
        const float2 cs = cstat[(size_t)scene * N + tok];  // sum c, sum c^2
        float* xr = x + ((size_t)scene * N + tok) * kRC;
        float xv[kRC];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const float4 t4 = reinterpret_cast<const float4*>(xr)[k];
          xv[4 * k] = t4.x; xv[4 * k + 1] = t4.y; xv[4 * k + 2] = t4.z; xv[4 * k + 3] = t4.w;
        }
        const float *S = stab, *beta = stab + kRC, *Gs = stab + 2 * kRC, *ws = stab + kRTab,
                    *G = stab + kRTab + kRC;
        float sum1 = cs.x, xA = 0.f, xGx = 0.f;
#pragma unroll
        for (int a = 0; a < kRC; ++a) {
          xA = fmaf(xv[a], acc[a], xA);
          sum1 = fmaf(xv[a], ws[a], sum1);
          float t = 0.f;
#pragma unroll
          for (int b2 = 0; b2 < kRC; ++b2) t = fmaf(G[a * kRC + b2], xv[b2], t);
          xGx = fmaf(xv[a], t, xGx);
        }
        const float sq = xGx + 2.f * xA + cs.y;
        const float mu = sum1 / (float)d;
        const float var = fmaxf(sq / (float)d - mu * mu, 0.f);
        const float rs = rsqrtf(var + 1e-6f);
        float v[kRC];
#pragma unroll
        for (int c = 0; c < kRC; ++c) {
          float P = acc[kRC + c] + acc[2 * kRC + c];
#pragma unroll
          for (int a = 0; a < kRC; ++a) P = fmaf(xv[a], Gs[a * kRC + c], P);
          v[c] = fmaf(rs, P - mu * S[c], beta[c]);
        }
        float* out = vout ? vout + ((size_t)scene * N + tok) * kRC : xr;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          float4 o;
          if (vout) o = make_float4(v[4 * k], v[4 * k + 1], v[4 * k + 2], v[4 * k + 3]);
          else o = make_float4(fmaf(dsig, v[4 * k], xv[4 * k]), fmaf(dsig, v[4 * k + 1], xv[4 * k + 1]),
                               fmaf(dsig, v[4 * k + 2], xv[4 * k + 2]),
                               fmaf(dsig, v[4 * k + 3], xv[4 * k + 3]));
          reinterpret_cast<float4*>(out)[k] = o;
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kRTmemCols);
  }
}

}  // namespace

cudaError_t launch_head_reuse_tc(const CUtensorMap& tmC, const CUtensorMap& tmB, float* x,
                                 const float2* cstat, const SlotMap& map, int N, int d, int b_row0,
                                 const float* tab_k, const float* wsum, const float* gram, float dsig,
                                 int* err, int n_sms, cudaStream_t st, float* vout) {
  if (map.n <= 0) return cudaSuccess;
  if (d % kRK != 0) return cudaErrorInvalidValue;
  static std::atomic<unsigned long long> configured{0};
  const cudaError_t e = configure_once_per_device(configured, [] {
    return cudaFuncSetAttribute(head_reuse_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                kRSmem);
  });
  if (e != cudaSuccess) return e;
  // Tokens per CTA: kRM, or fewer when the scenes' 128-token tiles would
  // leave SMs idle (one CTA per SM): then every SM takes an equal share of a
  // scene (c5, 17550 tokens: 116 per CTA on 152 SMs instead of 128 on 138).
  int rows = kRM;
  const int tiles = (N + kRM - 1) / kRM;
  if (n_sms > 0 && (long long)tiles * map.n < n_sms) {
    const int per_scene = n_sms / map.n;  // >= tiles
    rows = max(16, (N + per_scene - 1) / per_scene);
  }
  const dim3 grid((unsigned)((N + rows - 1) / rows), (unsigned)map.n);
  return launch_pdl(head_reuse_tc_kernel, grid, dim3(kRThreads), kRSmem, st, tmC, tmB, x, cstat, map,
                    N, d, rows, b_row0, tab_k, wsum, gram, dsig, vout, err);
}

}  // namespace dc
