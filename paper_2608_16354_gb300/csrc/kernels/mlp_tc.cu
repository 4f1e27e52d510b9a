// Fused MLP of the DiT block on tcgen05 for d = 384, hidden 1536 (Eq. 1,
// the block stack F_k: h <- h + gate2 (GELU(a W1^T + b1) W2^T + b2)), bf16
// operands, fp32 accumulation, so that the [M][1536] hidden activation never
// goes to HBM.
//
// CTA pairs share M = 256 pair MMAs (tcgen05.mma.cta_group::2); each CTA
// keeps its 128 rows of a (all 384 columns) in shared memory for the whole
// tile.  Per pair tile and hidden chunk c (128 columns):
//   up(c):   D_up[256 x 128]   = a W1[c]^T              (TMEM columns 0-127)
//   epi(c):  G = bf16(GELU(D_up + b1[c])) -> shared memory (SW128, K-major),
//            both CTAs' halves handed to the MMA issuer with a cluster-scope
//            release / acquire
//   down(c): D_down[256 x 384] += G W2[:, c]^T         (TMEM columns 128-511,
//            two N = 192 MMAs)
// issued in the order up(0), up(1), down(0), up(2), down(1), ... so that the
// tensor core runs up(c+1) while the epilogue turns D_up(c) into G.  The
// weight chunks stream from L2 through a 3-stage ring in the MMA's order.
// After the last chunk the gated residual h = h_in + gate (D_down + b2) is
// formed in shared memory (the a tile's space) in two 192-column passes and
// stored with TMA.  The hidden dimension is accumulated in K steps of 16 in
// order, as the unfused MLP-down GEMM does, so the result equals MLP-up
// (GELU epilogue) followed by MLP-down (residual epilogue) bit for bit.
//
//   warp 0      TMA producer (a tile, weight ring, residual tiles)
//   warp 1      rank 0: MMA issuer; rank 1: waits for the pair's drain
//   warps 2-9   epilogue (GELU chunks, residual)
// Every wait is bounded.
#include "common.cuh"
#include "epilogue.cuh"
#include "kernels.h"

namespace dc {

namespace {

constexpr int kD = 384, kHid = 1536, kCh = 128, kNC = kHid / kCh;  // 12 chunks
constexpr int kBM = 128;                       // rows per CTA (256 per pair)
constexpr int kThreads = 320;                  // producer, MMA, 8 epilogue warps
constexpr int kEpiThreads = 256;
constexpr int kStages = 3;
constexpr int kStageBytes = 24576;             // W1: 3 atoms x 64 rows; W2: 2 atoms x 96 rows
constexpr int kOffA = 0;                       // 6 atoms x [128 rows][128 B]
constexpr int kOffG = kOffA + 6 * 16384;       // 2 atoms x [128 rows][128 B]
constexpr int kOffRing = kOffG + 2 * 16384;
constexpr int kOffB1 = kOffRing + kStages * kStageBytes;
constexpr int kOffVec = kOffB1 + kHid * 4;     // b2, gate_a, gate_b
constexpr int kOffBar = kOffVec + 3 * kD * 4;
constexpr int kSmem = 1024 + kOffBar + 256;
static_assert(kSmem <= 232448, "shared memory budget");
constexpr uint32_t kIdUp = idesc_bf16_f32(256, kCh);
constexpr uint32_t kIdDown = idesc_bf16_f32(256, 192);
constexpr int kTmemCols = 512;                 // D_up 0..127, D_down 128..511

struct __align__(8) Bars {
  uint64_t full[kStages], empty[kStages];
  uint64_t a_full, a_empty, up_full, up_empty, g_full, g_empty, down_full, down_empty;
  uint64_t hin_full, drain;
  uint32_t tmem_base;
  int abort;
};

__device__ __forceinline__ int sw128(int r, int c) { return r * 128 + ((c ^ (r & 7)) << 4); }

// release arrival on a barrier of either CTA of the pair: orders this
// thread's earlier shared-memory writes (and those ordered before them)
__device__ __forceinline__ void arrive_release_cluster(uint32_t bar_cluster) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar_cluster)
               : "memory");
}
__device__ __forceinline__ bool try_wait_acq_cluster(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n"
      " mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// bounded cluster-acquire wait, warp-uniform outcome
__device__ __forceinline__ bool wait_acq_cluster_warp(uint64_t* bar, uint32_t parity, int* err,
                                                      int code, uint32_t limit_ns) {
  bool ok = try_wait_acq_cluster(bar, parity);
  if (!ok) {
    const unsigned long long t0 = global_ns();
    while (true) {
      if (try_wait_acq_cluster(bar, parity)) { ok = true; break; }
      if (global_ns() - t0 > (unsigned long long)limit_ns) { atomicCAS(err, 0, code); break; }
    }
  }
  return __all_sync(0xffffffffu, ok);
}

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    mlp_tc_kernel(const __grid_constant__ CUtensorMap tmA,   // a  bf16 [M][384], box 64 x 128
                  const __grid_constant__ CUtensorMap tmW1,  // W1 bf16 [1536][384], box 64 x 64
                  const __grid_constant__ CUtensorMap tmW2,  // W2 bf16 [384][1536], box 64 x 96
                  const __grid_constant__ CUtensorMap tmH,   // h  fp32 [M][384], box 32 x 128
                  int M, const float* __restrict__ b1, const float* __restrict__ b2,
                  const float* __restrict__ mod, int mod_stride, int gate_off, int n_tok,
                  SlotMap map, int* err) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t base = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + ((1024 - (base & 1023)) & 1023);
  uint8_t* sA = smem + kOffA;
  uint8_t* sG = smem + kOffG;
  uint8_t* sRing = smem + kOffRing;
  float* b1s = reinterpret_cast<float*>(smem + kOffB1);
  float* vec = reinterpret_cast<float*>(smem + kOffVec);
  Bars* bar = reinterpret_cast<Bars*>(smem + kOffBar);
  static_assert(sizeof(Bars) <= 256, "barrier reserve");

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int rank = (int)cluster_rank();
  const int tiles_m = (M + kBM - 1) / kBM;
  const int n_pt = (tiles_m + 1) / 2;            // pair tiles
  const int pair = blockIdx.x >> 1, n_pairs = gridDim.x >> 1;
  auto m0_of = [&](int pt) { return (pt * 2 + rank) * kBM; };

  if (threadIdx.x == 0) {
    bar->abort = *(volatile int*)err;
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&bar->full[s], 2);
      mbar_init(&bar->empty[s], 1);
    }
    mbar_init(&bar->a_full, 2);
    mbar_init(&bar->a_empty, 1);
    mbar_init(&bar->up_full, 1);
    mbar_init(&bar->up_empty, 2 * 8);
    mbar_init(&bar->g_full, 2);
    mbar_init(&bar->g_empty, 1);
    mbar_init(&bar->down_full, 1);
    mbar_init(&bar->down_empty, 2 * 8);
    mbar_init(&bar->hin_full, 1);
    mbar_init(&bar->drain, 1);
    fence_barrier_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmW1);
    tma_prefetch_desc(&tmW2);
    tma_prefetch_desc(&tmH);
  }
  if (warp == 1) {
    tmem_alloc_pair(&bar->tmem_base, kTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync();
  tc_fence_after();
  pdl_trigger();
  pdl_wait();
  const uint32_t tmem_base = bar->tmem_base;
  const uint32_t wlim = work_wait_limit(err);  // waits on work in progress

  if (bar->abort != 0) {
  } else if (warp == 0) {
    // ------------------------------------------------------------ producer
    int stage = 0, box = 0;
    uint32_t phase = 0;
    int issued = 0;  // ring stages filled
    bool ok = true;
    const uint32_t a_full_c = cluster_addr(&bar->a_full, 0);
    // one ring stage: W1 chunk c, K half s (3 boxes of 64 rows), or W2 chunk c,
    // N half s (2 boxes of 96 rows); rank 1's copies complete on rank 0's barrier
    auto load_stage = [&](bool w1, int c, int s) -> bool {
      if (!mbar_wait_warp(&bar->empty[stage], phase ^ 1, err, kDevTimeoutTma, wlim)) return false;
      uint8_t* dst = sRing + stage * kStageBytes;
      const int nb = w1 ? 3 : 2;
      const int l0 = box & 31;
      if (rank == 0) {
        if (lane == l0) mbar_arrive_expect_tx(&bar->full[stage], kStageBytes);
      } else {
        if (lane == l0) mbar_arrive_expect_tx_cluster(cluster_addr(&bar->full[stage], 0), kStageBytes);
      }
      __syncwarp();
      for (int b = 0; b < nb; ++b) {
        const int l = (box + b) & 31;
        if (lane == l) {
          const int x = w1 ? 192 * s + 64 * b : kCh * c + 64 * b;
          const int y = w1 ? kCh * c + 64 * rank : 192 * s + 96 * rank;
          uint8_t* p = dst + b * (w1 ? 8192 : 12288);
          if (rank == 0) tma_load_2d(p, w1 ? &tmW1 : &tmW2, &bar->full[stage], x, y);
          else tma_load_2d_pair(p, w1 ? &tmW1 : &tmW2, cluster_addr(&bar->full[stage], 0), x, y);
        }
      }
      __syncwarp();
      box += nb;
      ++issued;
      if (++stage == kStages) { stage = 0; phase ^= 1; }
      return true;
    };
    int t = 0, a_issued = 0;
    for (int pt = pair; pt < n_pt && ok; pt += n_pairs, ++t) {
      const int m0 = m0_of(pt);
      if (t > 0 && !mbar_wait_warp(&bar->a_empty, (uint32_t)(t - 1) & 1, err, kDevTimeoutTma, wlim)) { ok = false; break; }
      ++a_issued;
      if (rank == 0) {
        if (lane == 0) mbar_arrive_expect_tx(&bar->a_full, 6 * 16384);
      } else {
        if (lane == 0) mbar_arrive_expect_tx_cluster(a_full_c, 6 * 16384);
      }
      __syncwarp();
      if (lane < 6) {
        if (rank == 0) tma_load_2d(sA + lane * 16384, &tmA, &bar->a_full, 64 * lane, m0);
        else tma_load_2d_pair(sA + lane * 16384, &tmA, a_full_c, 64 * lane, m0);
      }
      __syncwarp();
      // the MMA warp's order: up(0); then per chunk c: up(c+1), down(c)
      ok = load_stage(true, 0, 0) && load_stage(true, 0, 1);
      for (int c = 0; c < kNC && ok; ++c) {
        if (c + 1 < kNC) ok = load_stage(true, c + 1, 0) && load_stage(true, c + 1, 1);
        if (ok) ok = load_stage(false, c, 0) && load_stage(false, c, 1);
      }
    }
    if (rank == 0) {
      // stage s was last filled by load s + kStages ((issued - 1 - s) / kStages)
      for (int s = 0; s < kStages && s < issued; ++s)
        mbar_wait_warp(&bar->full[s], (uint32_t)(((issued - 1 - s) / kStages) & 1), err, kDevTimeoutTma);
      // the last A copies (both CTAs count on this barrier) have landed
      if (a_issued > 0) mbar_wait_warp(&bar->a_full, (uint32_t)(a_issued - 1) & 1, err, kDevTimeoutTma);
    }
  } else if (warp == 1 && rank != 0) {
    mbar_wait_warp(&bar->drain, 0, err, kDevTimeoutMma);
  } else if (warp == 1) {
    // ------------------------------------------------------- MMA issuer
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    const uint64_t dA = sw128_kmajor_desc(smem_u32(sA));
    const uint64_t dG = sw128_kmajor_desc(smem_u32(sG));
    const uint64_t dR = sw128_kmajor_desc(smem_u32(sRing));
    int u = 0;  // chunks issued so far (all tiles)
    auto up = [&](int uu) -> bool {
      if (uu > 0 && !mbar_wait_warp(&bar->up_empty, (uint32_t)(uu - 1) & 1, err, kDevTimeoutMma, wlim)) return false;
      tc_fence_after();
      for (int s = 0; s < 2; ++s) {
        if (!mbar_wait_warp(&bar->full[stage], phase, err, kDevTimeoutMma, wlim)) return false;
        tc_fence_after();
        if (elect_one()) {
#pragma unroll
          for (int kk = 0; kk < 12; ++kk) {
            const int atom = kk >> 2, k16 = kk & 3;
            tc_mma_f16_pair(tmem_base, dA + ((uint32_t)((3 * s + atom) * 16384 + k16 * 32) >> 4),
                            dR + ((uint32_t)(stage * kStageBytes + atom * 8192 + k16 * 32) >> 4), kIdUp,
                            (s | kk) != 0 ? 1u : 0u);
          }
          tc_commit_pair_mc(&bar->empty[stage], (uint16_t)0x3);
        }
        __syncwarp();
        if (++stage == kStages) { stage = 0; phase ^= 1; }
      }
      if (elect_one()) tc_commit_pair_mc(&bar->up_full, (uint16_t)0x3);
      __syncwarp();
      return true;
    };
    int t = 0;
    for (int pt = pair; pt < n_pt && ok; pt += n_pairs, ++t) {
      if (!mbar_wait_warp(&bar->a_full, (uint32_t)t & 1, err, kDevTimeoutMma, wlim)) { ok = false; break; }
      if (t > 0 && !mbar_wait_warp(&bar->down_empty, (uint32_t)(t - 1) & 1, err, kDevTimeoutMma, wlim)) { ok = false; break; }
      tc_fence_after();
      ok = up(u);
      for (int c = 0; c < kNC && ok; ++c) {
        if (c + 1 < kNC) ok = up(u + c + 1);
        if (!ok) break;
        // down(c): G from both CTAs' shared memory, written by their epilogues
        if (!wait_acq_cluster_warp(&bar->g_full, (uint32_t)(u + c) & 1, err, kDevTimeoutMma, wlim)) { ok = false; break; }
        tc_fence_after();
        for (int nh = 0; nh < 2 && ok; ++nh) {
          if (!mbar_wait_warp(&bar->full[stage], phase, err, kDevTimeoutMma, wlim)) { ok = false; break; }
          tc_fence_after();
          if (elect_one()) {
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
              const int atom = kk >> 2, k16 = kk & 3;
              tc_mma_f16_pair(tmem_base + 128 + 192 * nh,
                              dG + ((uint32_t)(atom * 16384 + k16 * 32) >> 4),
                              dR + ((uint32_t)(stage * kStageBytes + atom * 12288 + k16 * 32) >> 4),
                              kIdDown, (c | kk) != 0 ? 1u : 0u);
            }
            tc_commit_pair_mc(&bar->empty[stage], (uint16_t)0x3);
          }
          __syncwarp();
          if (++stage == kStages) { stage = 0; phase ^= 1; }
        }
        if (!ok) break;
        if (elect_one()) tc_commit_pair_mc(&bar->g_empty, (uint16_t)0x3);
        __syncwarp();
      }
      if (!ok) break;
      u += kNC;
      if (elect_one()) tc_commit_pair_mc(&bar->down_full, (uint16_t)0x3);
      __syncwarp();
    }
    if (elect_one()) tc_commit_pair_mc(&bar->drain, (uint16_t)0x3);
    __syncwarp();
    mbar_wait_warp(&bar->drain, 0, err, kDevTimeoutMma);
  } else {
    // ---------------------------------------------------- epilogue warps
    const int q = warp & 3;
    const int half = (warp - 2) >> 2;
    const int et = threadIdx.x - 64;
    const int r = q * 32 + lane;
    const bool copy_warp = warp == 2;
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    for (int i = et; i < kHid; i += kEpiThreads) b1s[i] = b1[i];
    named_bar(1, kEpiThreads);
    bool failed = false;
    int u = 0, t = 0, hp = 0;
    for (int pt = pair; pt < n_pt && !failed; pt += n_pairs, ++t) {
      const int m0 = m0_of(pt);
      const bool live = m0 < M;
      for (int c = 0; c < kNC; ++c, ++u) {
        bool ok = mbar_wait_warp(&bar->up_full, (uint32_t)u & 1, err, kDevTimeoutEpi, wlim);
        uint32_t w[32];  // 64 bf16 of this thread's row
        if (ok) {
          tc_fence_after();
          float acc[2][32];
          tmem_ld32(tmem_base + (uint32_t)(half * 64) + lane_off, acc[0]);
          tmem_ld32(tmem_base + (uint32_t)(half * 64 + 32) + lane_off, acc[1]);
          tmem_ld_wait();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_cluster_relaxed(cluster_addr(&bar->up_empty, 0));
          const float* bb = b1s + c * kCh + half * 64;
#pragma unroll
          for (int cc = 0; cc < 2; ++cc) {
#pragma unroll
            for (int i = 0; i < 32; i += 2) {
              const float2 x = f2_add(make_float2(acc[cc][i], acc[cc][i + 1]),
                                      make_float2(bb[cc * 32 + i], bb[cc * 32 + i + 1]));
              const float2 y = gelu_tanh_pair(x);
              __nv_bfloat162 p = __floats2bfloat162_rn(y.x, y.y);
              w[cc * 16 + i / 2] = *reinterpret_cast<uint32_t*>(&p);
            }
          }
        }
        // sG is free once down(u-1) has read it
        if (ok && u > 0) ok = mbar_wait_warp(&bar->g_empty, (uint32_t)(u - 1) & 1, err, kDevTimeoutEpi, wlim);
        if (ok) {
#pragma unroll
          for (int g = 0; g < 8; ++g)
            *reinterpret_cast<uint4*>(sG + half * 16384 + sw128(r, g)) =
                make_uint4(w[4 * g], w[4 * g + 1], w[4 * g + 2], w[4 * g + 3]);
        }
        fence_proxy_async();
        if (named_bar_or(1, kEpiThreads, !ok)) { failed = true; break; }
        if (et == 0) arrive_release_cluster(cluster_addr(&bar->g_full, 0));
      }
      if (failed) break;
      // ---- residual: h = h_in + gate (D_down + b2), two 192-column passes
      bool ok = mbar_wait_warp(&bar->down_full, (uint32_t)t & 1, err, kDevTimeoutEpi, wlim);
      const int last_row = live ? min(m0 + kBM, M) - 1 : m0;
      const int slot_a = m0 / n_tok, slot_b = last_row / n_tok;
      const int split = (slot_a + 1) * n_tok;
      const bool two_slots = slot_b - slot_a <= 1;
      for (int i = et; i < kD; i += kEpiThreads) {
        vec[i] = b2[i];
        if (live) {
          vec[kD + i] = mod[(size_t)map.scene[slot_a] * mod_stride + gate_off + i];
          vec[2 * kD + i] = mod[(size_t)map.scene[slot_b] * mod_stride + gate_off + i];
        }
      }
      if (named_bar_or(1, kEpiThreads, !ok)) { failed = true; break; }
      tc_fence_after();
      const int row = m0 + r;
      const float* gsel = vec + (row < split ? kD : 2 * kD);
      const float* grow = (!two_slots && row < M)
                              ? mod + (size_t)map.scene[row / n_tok] * mod_stride + gate_off
                              : nullptr;
      for (int p = 0; p < 2; ++p) {
        if (live && copy_warp) {
          if (lane == 0) mbar_arrive_expect_tx(&bar->hin_full, 6 * 16384);
          __syncwarp();
          if (lane < 6) tma_load_2d(sA + lane * 16384, &tmH, &bar->hin_full, 192 * p + 32 * lane, m0);
          __syncwarp();
        }
        float acc[3][32];
#pragma unroll
        for (int cc = 0; cc < 3; ++cc)
          tmem_ld32(tmem_base + (uint32_t)(128 + 192 * p + 96 * half + 32 * cc) + lane_off, acc[cc]);
        tmem_ld_wait();
        if (p == 1) {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_cluster_relaxed(cluster_addr(&bar->down_empty, 0));
        }
        bool hok = true;
        if (live) hok = mbar_wait_warp(&bar->hin_full, (uint32_t)(hp++) & 1, err, kDevTimeoutEpi, wlim);
        if (live && hok) {
#pragma unroll
          for (int cc = 0; cc < 3; ++cc) {
            uint8_t* bx = sA + (3 * half + cc) * 16384;
            const int col0 = 192 * p + 96 * half + 32 * cc;
#pragma unroll
            for (int ch = 0; ch < 8; ++ch) {
              float4* ptr = reinterpret_cast<float4*>(bx + sw128(r, ch));
              float4 h = *ptr;
              const int j = col0 + ch * 4;
              float g0, g1, g2, g3;
              if (two_slots) {
                g0 = gsel[j]; g1 = gsel[j + 1]; g2 = gsel[j + 2]; g3 = gsel[j + 3];
              } else if (grow) {
                g0 = grow[j]; g1 = grow[j + 1]; g2 = grow[j + 2]; g3 = grow[j + 3];
              } else {
                g0 = g1 = g2 = g3 = 0.f;
              }
              h.x += g0 * (acc[cc][ch * 4 + 0] + vec[j + 0]);
              h.y += g1 * (acc[cc][ch * 4 + 1] + vec[j + 1]);
              h.z += g2 * (acc[cc][ch * 4 + 2] + vec[j + 2]);
              h.w += g3 * (acc[cc][ch * 4 + 3] + vec[j + 3]);
              *ptr = h;
            }
          }
        }
        fence_proxy_async();
        if (named_bar_or(1, kEpiThreads, !hok)) { failed = true; break; }
        if (live && copy_warp) {
          if (lane < 6) {
            tma_store_2d(&tmH, sA + lane * 16384, 192 * p + 32 * lane, m0);
            bulk_commit();
            bulk_wait_read0();
          }
          __syncwarp();
        }
      }
      if (failed) break;
      // every store has read sA: the producer may load the next tile's A
      if (copy_warp && lane == 0) mbar_arrive(&bar->a_empty);
    }
    if (copy_warp && lane < 6) bulk_wait0();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, kTmemCols);
  }
  cluster_sync();
}

}  // namespace

bool mlp_tc_supported(int d, int md) { return d == kD && md == kHid; }

cudaError_t launch_mlp_tc(const CUtensorMap& tmA, const CUtensorMap& tmW1, const CUtensorMap& tmW2,
                          const CUtensorMap& tmH, int M, const float* b1, const float* b2,
                          const float* mod, int mod_stride, int gate_off, int n_tok,
                          const SlotMap& map, int* err, int n_sms, cudaStream_t st) {
  if (M <= 0) return cudaSuccess;
  static std::atomic<unsigned long long> configured{0};
  const cudaError_t e = configure_once_per_device(configured, [] {
    return cudaFuncSetAttribute(mlp_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
  });
  if (e != cudaSuccess) return e;
  // one CTA pair per pair tile, at most one pair per two SMs (persistent)
  const int n_pt = ((M + kBM - 1) / kBM + 1) / 2;
  const int grid = 2 * (n_pt < n_sms / 2 ? n_pt : n_sms / 2);
  return launch_pdl(mlp_tc_kernel, dim3(grid), dim3(kThreads), kSmem, st, tmA, tmW1, tmW2, tmH, M,
                    b1, b2, mod, mod_stride, gate_off, n_tok, map, err);
}

}  // namespace dc
