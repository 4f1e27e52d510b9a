// Full spatiotemporal attention on the 5th-generation tensor cores (sm_103a):
// o = softmax(q k^T / sqrt(dh)) v for head dims 64 and 128.
//
// One CTA per (slot, head, 128-query tile); keys stream in tiles of 128.
//   warp 0      TMA: Q once, K_j and V_j into a 2-stage ring
//   warp 1      owns TMEM (512 columns) and issues tcgen05.mma:
//                 S_j  = Q K_j^T      -> TMEM S[j % 2]   (M=128, N=128, K=dh)
//                 PV_j = P_j V_j      -> TMEM O[j % 2]   (M=128, N=64 per half, K=128)
//   warps 2-5   softmax, one query row per thread: read S_j with tcgen05.ld,
//               online max/sum in the log2 domain, write P_j = exp2(s - m) as
//               bf16 into shared memory in the 128-byte-swizzled K-major layout
//               the MMA reads, then fold PV_{j-1} into a register accumulator
//               with the running correction exp2(m_old - m_new).
// S, P and PV are double-buffered so that the MMAs of tile j+1 overlap the
// softmax of tile j.  V is consumed as an MN-major operand straight from its
// [keys][dh] layout.  Keys beyond N are masked; every mbarrier wait is bounded.
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace dc {

namespace {

constexpr int kAttThreads = 192;

template <int DHP>
struct AttCfg {
  static constexpr int kAtoms = DHP / 64;             // 64-element swizzle atoms along dh
  static constexpr int kTileBytes = kAtoms * 16384;   // 128 rows x DHP bf16
  static constexpr int kPBytes = 2 * 16384;           // 128 queries x 128 keys bf16
  static constexpr int kOffQ = 0;
  static constexpr int kOffK = kOffQ + kTileBytes;        // 2 stages
  static constexpr int kOffV = kOffK + 2 * kTileBytes;    // 2 stages
  static constexpr int kOffP = kOffV + 2 * kTileBytes;    // 2 buffers
  static constexpr int kOffBar = kOffP + 2 * kPBytes;
  static constexpr int kSmem = 1024 + kOffBar + 256;
};

struct __align__(8) AttBars {
  uint64_t q_full;
  uint64_t kv_full[2], kv_empty[2];
  uint64_t s_full[2], s_empty[2];
  uint64_t p_full[2], p_empty[2];
  uint64_t o_full[2], o_empty[2];
  uint64_t drain;
  uint32_t tmem_base;
};

// Descriptor of an MN-major operand tile written by TMA with 128-byte swizzle
// (rows = K index, 64 MN elements per 128-byte row).  One MN atom per MMA, so
// only the 8-row group stride along K (1024 bytes) is used; both offset
// fields carry it.
__device__ __forceinline__ uint64_t sw128_mnmajor_desc(uint32_t start) {
  uint64_t d = 0;
  d |= (uint64_t)((start & 0x3FFFF) >> 4);
  d |= (uint64_t)(1024 >> 4) << 16;
  d |= (uint64_t)(1024 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack2(float a, float b) {
  __nv_bfloat162 t = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&t);
}

template <int DHP>
__global__ void __launch_bounds__(kAttThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tm, int nslots, int heads, int N,
                   __nv_bfloat16* __restrict__ o, float scale_log2, int* err) {
  using Cfg = AttCfg<DHP>;
  constexpr uint32_t kIdS = idesc_bf16_f32(128, 128);
  constexpr uint32_t kIdPV = idesc_bf16_f32(128, 64) | (1u << 16);  // B (= V) MN-major
  extern __shared__ uint8_t smem_raw[];
  const uint32_t base = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + ((1024 - (base & 1023)) & 1023);
  AttBars* bar = reinterpret_cast<AttBars*>(smem + Cfg::kOffBar);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int bh = blockIdx.y;
  const int slot = bh / heads, head = bh - slot * heads;
  const int q0 = blockIdx.x * 128;
  const int n_kv = (N + 127) / 128;
  const int row_q = ((0 * nslots + slot) * heads + head) * N + q0;
  const int row_k = ((1 * nslots + slot) * heads + head) * N;
  const int row_v = ((2 * nslots + slot) * heads + head) * N;

  // a bounded wait of an earlier launch gave up: do nothing (the host
  // reports DC_ERR_DEVICE_TIMEOUT at its next check)
  if (*(volatile int*)err != 0) return;
  if (threadIdx.x == 0) {
    mbar_init(&bar->q_full, 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bar->kv_full[b], 1);
      mbar_init(&bar->kv_empty[b], 1);
      mbar_init(&bar->s_full[b], 1);
      mbar_init(&bar->s_empty[b], 4);
      mbar_init(&bar->p_full[b], 4);
      mbar_init(&bar->p_empty[b], 1);
      mbar_init(&bar->o_full[b], 1);
      mbar_init(&bar->o_empty[b], 4);
    }
    mbar_init(&bar->drain, 1);
    fence_barrier_init();
    tma_prefetch_desc(&tm);
  }
  if (warp == 1) {
    tmem_alloc(&bar->tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bar->tmem_base;
  // TMEM columns: S[0] 0..127, S[1] 128..255, O[0] 256.., O[1] 256 + DHP..

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ TMA
      bool ok = true;
      int last[2] = {-1, -1};
      mbar_arrive_expect_tx(&bar->q_full, Cfg::kTileBytes);
      for (int a = 0; a < Cfg::kAtoms; ++a)
        tma_load_2d(smem + Cfg::kOffQ + a * 16384, &tm, &bar->q_full, a * 64, row_q);
      for (int j = 0; j < n_kv && ok; ++j) {
        const int b = j & 1;
        const uint32_t u = (uint32_t)(j >> 1);
        if (!mbar_wait(&bar->kv_empty[b], (u & 1) ^ 1, err, kDevTimeoutTma)) { ok = false; break; }
        mbar_arrive_expect_tx(&bar->kv_full[b], 2 * Cfg::kTileBytes);
        for (int a = 0; a < Cfg::kAtoms; ++a) {
          tma_load_2d(smem + Cfg::kOffK + b * Cfg::kTileBytes + a * 16384, &tm, &bar->kv_full[b],
                      a * 64, row_k + j * 128);
          tma_load_2d(smem + Cfg::kOffV + b * Cfg::kTileBytes + a * 16384, &tm, &bar->kv_full[b],
                      a * 64, row_v + j * 128);
        }
        last[b] = (int)(u & 1);
      }
      mbar_wait(&bar->q_full, 0, err, kDevTimeoutTma);
      for (int b = 0; b < 2; ++b)
        if (last[b] >= 0) mbar_wait(&bar->kv_full[b], (uint32_t)last[b], err, kDevTimeoutTma);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------------------ MMA
      bool ok = mbar_wait(&bar->q_full, 0, err, kDevTimeoutMma);
      const uint32_t sQ = smem_u32(smem + Cfg::kOffQ);
      auto issue_pv = [&](int i) -> bool {
        const int b = i & 1;
        const uint32_t u = (uint32_t)(i >> 1);
        if (!mbar_wait(&bar->p_full[b], u & 1, err, kDevTimeoutMma)) return false;
        if (!mbar_wait(&bar->o_empty[b], (u & 1) ^ 1, err, kDevTimeoutMma)) return false;
        tc_fence_after();
        const uint32_t sP = smem_u32(smem + Cfg::kOffP + b * Cfg::kPBytes);
        const uint32_t sV = smem_u32(smem + Cfg::kOffV + b * Cfg::kTileBytes);
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint64_t ad = sw128_kmajor_desc(sP + (kk >> 2) * 16384 + (kk & 3) * 32);
#pragma unroll
          for (int a = 0; a < Cfg::kAtoms; ++a)
            tc_mma_f16(tmem + 256 + b * DHP + a * 64, ad,
                       sw128_mnmajor_desc(sV + a * 16384 + kk * 2048), kIdPV, kk > 0 ? 1u : 0u);
        }
        tc_commit(&bar->o_full[b]);
        tc_commit(&bar->p_empty[b]);
        tc_commit(&bar->kv_empty[b]);
        return true;
      };
      for (int j = 0; j < n_kv && ok; ++j) {
        const int b = j & 1;
        const uint32_t u = (uint32_t)(j >> 1);
        if (!mbar_wait(&bar->kv_full[b], u & 1, err, kDevTimeoutMma)) { ok = false; break; }
        if (!mbar_wait(&bar->s_empty[b], (u & 1) ^ 1, err, kDevTimeoutMma)) { ok = false; break; }
        tc_fence_after();
        const uint32_t sK = smem_u32(smem + Cfg::kOffK + b * Cfg::kTileBytes);
#pragma unroll
        for (int kk = 0; kk < DHP / 16; ++kk) {
          const uint32_t off = (kk >> 2) * 16384 + (kk & 3) * 32;
          tc_mma_f16(tmem + b * 128, sw128_kmajor_desc(sQ + off), sw128_kmajor_desc(sK + off), kIdS,
                     kk > 0 ? 1u : 0u);
        }
        tc_commit(&bar->s_full[b]);
        if (j >= 1 && !issue_pv(j - 1)) { ok = false; break; }
      }
      if (ok) issue_pv(n_kv - 1);
      tc_commit(&bar->drain);
      mbar_wait(&bar->drain, 0, err, kDevTimeoutMma);
    }
  } else {
    // ------------------------------------------------------------ softmax
    const int q = warp & 3;
    const int row = q * 32 + lane;
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    float O[DHP];
#pragma unroll
    for (int i = 0; i < DHP; ++i) O[i] = 0.f;
    float m = -INFINITY, l = 0.f, corr_prev = 1.f;
    bool ok = true;
    auto accumulate = [&](int i, float c) -> bool {
      const int b = i & 1;
      const uint32_t u = (uint32_t)(i >> 1);
      if (!mbar_wait(&bar->o_full[b], u & 1, err, kDevTimeoutEpi)) return false;
      tc_fence_after();
#pragma unroll
      for (int ch = 0; ch < DHP / 32; ++ch) {
        float v[32];
        tmem_ld32(tmem + 256 + b * DHP + ch * 32 + lane_off, v);
        tmem_ld_wait();
#pragma unroll
        for (int t = 0; t < 32; ++t) O[ch * 32 + t] = O[ch * 32 + t] * c + v[t];
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bar->o_empty[b]);
      return true;
    };
    for (int j = 0; j < n_kv && ok; ++j) {
      const int b = j & 1;
      const uint32_t u = (uint32_t)(j >> 1);
      if (!mbar_wait(&bar->s_full[b], u & 1, err, kDevTimeoutEpi)) { ok = false; break; }
      tc_fence_after();
      const uint32_t tS = tmem + b * 128 + lane_off;
      const int kbase = j * 128;
      float mx = -INFINITY;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        float v[32];
        tmem_ld32(tS + c * 32, v);
        tmem_ld_wait();
#pragma unroll
        for (int t = 0; t < 32; ++t)
          if (kbase + c * 32 + t < N) mx = fmaxf(mx, v[t]);
      }
      const float m_new = fmaxf(m, mx * scale_log2);
      const float corr = ex2(m - m_new);
      m = m_new;
      if (!mbar_wait(&bar->p_empty[b], (u & 1) ^ 1, err, kDevTimeoutEpi)) { ok = false; break; }
      uint8_t* Pb = smem + Cfg::kOffP + b * Cfg::kPBytes;
      float rs = 0.f;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        float v[32];
        tmem_ld32(tS + c * 32, v);
        tmem_ld_wait();
#pragma unroll
        for (int t = 0; t < 32; ++t) {
          const float p = kbase + c * 32 + t < N ? ex2(v[t] * scale_log2 - m) : 0.f;
          v[t] = p;
          rs += p;
        }
#pragma unroll
        for (int g = 0; g < 4; ++g) {
          const int ch = c * 4 + g;  // 16-byte chunk of the row (8 keys)
          uint4 w;
          w.x = pack2(v[g * 8 + 0], v[g * 8 + 1]);
          w.y = pack2(v[g * 8 + 2], v[g * 8 + 3]);
          w.z = pack2(v[g * 8 + 4], v[g * 8 + 5]);
          w.w = pack2(v[g * 8 + 6], v[g * 8 + 7]);
          *reinterpret_cast<uint4*>(Pb + (ch >> 3) * 16384 + row * 128 +
                                    (((ch & 7) ^ (row & 7)) << 4)) = w;
        }
      }
      tc_fence_before();
      fence_proxy_async();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&bar->s_empty[b]);
        mbar_arrive(&bar->p_full[b]);
      }
      l = l * corr + rs;
      if (j >= 1 && !accumulate(j - 1, corr_prev)) { ok = false; break; }
      corr_prev = corr;
    }
    if (ok) ok = accumulate(n_kv - 1, corr_prev);
    if (ok && q0 + row < N) {
      const float inv = 1.f / l;
      __nv_bfloat16* dst = o + ((size_t)slot * N + q0 + row) * ((size_t)heads * DHP) + head * DHP;
#pragma unroll
      for (int e = 0; e < DHP; e += 8) {
        uint4 w;
        w.x = pack2(O[e] * inv, O[e + 1] * inv);
        w.y = pack2(O[e + 2] * inv, O[e + 3] * inv);
        w.z = pack2(O[e + 4] * inv, O[e + 5] * inv);
        w.w = pack2(O[e + 6] * inv, O[e + 7] * inv);
        *reinterpret_cast<uint4*>(dst + e) = w;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

template <int DHP>
cudaError_t launch_tc(const CUtensorMap& tm, int nslots, int heads, int N, __nv_bfloat16* o,
                      int* err, cudaStream_t st) {
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(attn_tc_kernel<DHP>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         AttCfg<DHP>::kSmem);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  dim3 grid((N + 127) / 128, nslots * heads);
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)DHP);
  attn_tc_kernel<DHP><<<grid, kAttThreads, AttCfg<DHP>::kSmem, st>>>(tm, nslots, heads, N, o,
                                                                      scale_log2, err);
  return cudaGetLastError();
}

}  // namespace

bool attention_tc_supported(int dh) { return dh == 64 || dh == 128; }

cudaError_t launch_attention_tc(const CUtensorMap& tm, int nslots, int heads, int N, int dh,
                                __nv_bfloat16* o, int* err, cudaStream_t st) {
  if (nslots <= 0) return cudaSuccess;
  if (dh == 64) return launch_tc<64>(tm, nslots, heads, N, o, err, st);
  if (dh == 128) return launch_tc<128>(tm, nslots, heads, N, o, err, st);
  return cudaErrorInvalidValue;
}

}  // namespace dc
