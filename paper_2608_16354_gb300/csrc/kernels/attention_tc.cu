// Full spatiotemporal attention on the 5th-generation tensor cores (sm_103a):
// o = softmax(q k^T / sqrt(dh)) v for head dims 64 and 128.
//
// One CTA per (slot, head, NQ x 128 queries); keys stream in tiles of 128.
//   warp 0        TMA: the NQ query tiles once, K_j and V_j into a 2-stage ring
//   warp 1        owns TMEM and issues tcgen05.mma for every query tile t:
//                   S_{t,j}  = Q_t K_j^T  -> TMEM buffer (t, j % 2)  (M=128, N=128, K=dh)
//                   PV_{t,j} = P_{t,j} V_j -> the same buffer once S_{t,j} has been
//                                             read (M=128, N=64 per MMA, K=128)
//   warps 2..     one softmax warpgroup per query tile, one query row per
//                 thread.
// Softmax of tile j (per row): P = exp2(s * scale - ref) against a reference
// max `ref` that only moves when the row's max exceeds it by more than 8
// (log2 units), so one pass over S suffices; P is written as bf16 into shared
// memory (double-buffered) in the 128-byte-swizzled K-major layout the MMA
// reads.  Halfway through the pass the thread folds PV_{j-1} into its
// register accumulator (O = (O + PV) * c, c = exp2(ref_old - ref_new)) and
// frees that TMEM buffer, so S_{j+1} is computed during the second half and
// PV_j during the first half of the next tile.  Both softmax warpgroups share
// the tensor core.  A quarter of the exponentials run on the FMA pipe
// (Cody-Waite split into integer and fraction, degree-3 minimax polynomial
// for 2^r on [0, 1], max relative error 8.6e-5) to relieve the MUFU unit.
// V is consumed as an MN-major operand straight from its [keys][dh] layout.
// Keys beyond N are masked (last tile only).  Every mbarrier wait is bounded.
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace dc {

namespace {

constexpr float kRefSlack = 8.0f;    // move the reference max only beyond this (log2 units)
constexpr float kRedoExcess = 64.0f; // larger jumps redo the tile against the new max

template <int DHP, int NQ>
struct AttCfg {
  static constexpr int kAtoms = DHP / 64;             // 64-element swizzle atoms along dh
  static constexpr int kTileBytes = kAtoms * 16384;   // 128 rows x DHP bf16
  static constexpr int kPBytes = 2 * 16384;           // 128 queries x 128 keys bf16
  static constexpr int kOffQ = 0;                           // NQ tiles
  static constexpr int kOffK = kOffQ + NQ * kTileBytes;     // 2 stages
  static constexpr int kOffV = kOffK + 2 * kTileBytes;      // 2 stages
  static constexpr int kOffP = kOffV + 2 * kTileBytes;      // NQ x 2 buffers
  static constexpr int kOffBar = kOffP + NQ * 2 * kPBytes;
  static constexpr int kSmem = 1024 + kOffBar + 256;
  static constexpr int kThreads = 64 + NQ * 128;
  static constexpr int kTmemCols = NQ * 256;  // two 128-column buffers per query tile
};

template <int NQ>
struct __align__(8) AttBars {
  uint64_t q_full;
  uint64_t k_full[2], k_empty[2];   // key ring: loader <-> S MMAs
  uint64_t v_full[2], v_empty[2];   // value ring: loader <-> PV MMAs
  uint64_t s_full[NQ][2];    // MMA -> softmax: S ready in buffer
  uint64_t p_full[NQ][2];    // softmax -> MMA: P written, S consumed
  uint64_t o_full[NQ][2];    // MMA -> softmax: PV ready in buffer (P buffer free again)
  uint64_t buf_free[NQ][2];  // softmax -> MMA: PV folded, buffer free
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

// 2^x on the MUFU unit
__device__ __forceinline__ float ex2_mufu(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Packed fp32x2 arithmetic (one instruction for two lanes of work).
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) {
  float2 r;
  asm("{\n .reg .b64 a, b, c, d;\n mov.b64 a, {%2, %3};\n mov.b64 b, {%4, %5};\n"
      " mov.b64 c, {%6, %7};\n fma.rn.f32x2 d, a, b, c;\n mov.b64 {%0, %1}, d;\n}\n"
      : "=f"(r.x), "=f"(r.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  return r;
}
__device__ __forceinline__ float2 fadd2(float2 a, float2 b) {
  float2 r;
  asm("{\n .reg .b64 a, b, d;\n mov.b64 a, {%2, %3};\n mov.b64 b, {%4, %5};\n"
      " add.rn.f32x2 d, a, b;\n mov.b64 {%0, %1}, d;\n}\n"
      : "=f"(r.x), "=f"(r.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return r;
}
__device__ __forceinline__ float2 fmul2(float2 a, float2 b) {
  float2 r;
  asm("{\n .reg .b64 a, b, d;\n mov.b64 a, {%2, %3};\n mov.b64 b, {%4, %5};\n"
      " mul.rn.f32x2 d, a, b;\n mov.b64 {%0, %1}, d;\n}\n"
      : "=f"(r.x), "=f"(r.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return r;
}

// 2^x for a pair, on the FMA/ALU pipes, given y = x - 1/2 (x <= kRedoExcess):
// n = round(y) = floor(x) from the rounding against 1.5 * 2^23, r' = y - n in
// [-1/2, 1/2], 2^(r' + 1/2) by a degree-3 minimax polynomial (the [0, 1]
// minimax for 2^r re-expanded around 1/2), and n (clamped at -126 so tiny
// values stay tiny) added to the exponent bits.
__device__ __forceinline__ float2 ex2_poly2(float2 y) {
  const float magic = 12582912.0f;  // 1.5 * 2^23
  const float2 t = fadd2(y, make_float2(magic, magic));
  const float2 n = fadd2(t, make_float2(-magic, -magic));
  const float2 r = fadd2(y, make_float2(-n.x, -n.y));
  float2 q = ffma2(make_float2(7.706703991e-02f, 7.706703991e-02f), r,
                   make_float2(3.432455659e-01f, 3.432455659e-01f));
  q = ffma2(q, r, make_float2(9.805620313e-01f, 9.805620313e-01f));
  q = ffma2(q, r, make_float2(1.414103031e+00f, 1.414103031e+00f));
  const int n0 = max(__float_as_int(t.x) - 0x4B400000, -126);
  const int n1 = max(__float_as_int(t.y) - 0x4B400000, -126);
  return make_float2(__int_as_float(__float_as_int(q.x) + (n0 << 23)),
                     __int_as_float(__float_as_int(q.y) + (n1 << 23)));
}

__device__ __forceinline__ uint32_t pack2(float a, float b) {
  __nv_bfloat162 t = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&t);
}

// One 32-column chunk of the softmax pass: p = 2^(s * scale - ref) (chunk 3
// on the FMA pipe), masked beyond `valid`, raw max and row sum updated on
// four independent chains, P chunk written to shared memory.
template <bool MASKED>
__device__ __forceinline__ void softmax_chunk(const uint32_t (&raw)[32], int c, int valid,
                                              float scale_log2, float neg_ref, float (&tmax)[4],
                                              float2 (&rs)[2], uint8_t* P, int row) {
  const float2 sc = make_float2(scale_log2, scale_log2);
  float v[32];
  if (c == 3) {
    const float2 nr = make_float2(neg_ref - 0.5f, neg_ref - 0.5f);
#pragma unroll
    for (int e = 0; e < 32; e += 2) {
      const float2 y = ffma2(make_float2(__uint_as_float(raw[e]), __uint_as_float(raw[e + 1])), sc, nr);
      const float2 p = ex2_poly2(y);
      v[e] = p.x;
      v[e + 1] = p.y;
    }
  } else {
    const float2 nr = make_float2(neg_ref, neg_ref);
#pragma unroll
    for (int e = 0; e < 32; e += 2) {
      const float2 x = ffma2(make_float2(__uint_as_float(raw[e]), __uint_as_float(raw[e + 1])), sc, nr);
      v[e] = ex2_mufu(x.x);
      v[e + 1] = ex2_mufu(x.y);
    }
  }
#pragma unroll
  for (int e = 0; e < 32; ++e) {
    if (!MASKED || c * 32 + e < valid) {
      tmax[e & 3] = fmaxf(tmax[e & 3], __uint_as_float(raw[e]));
    } else {
      v[e] = 0.f;
    }
  }
#pragma unroll
  for (int e = 0; e < 32; e += 4) {
    rs[0] = fadd2(rs[0], make_float2(v[e], v[e + 1]));
    rs[1] = fadd2(rs[1], make_float2(v[e + 2], v[e + 3]));
  }
#pragma unroll
  for (int g = 0; g < 4; ++g) {
    const int ch = c * 4 + g;  // 16-byte chunk of the row (8 keys)
    uint4 w;
    w.x = pack2(v[g * 8 + 0], v[g * 8 + 1]);
    w.y = pack2(v[g * 8 + 2], v[g * 8 + 3]);
    w.z = pack2(v[g * 8 + 4], v[g * 8 + 5]);
    w.w = pack2(v[g * 8 + 6], v[g * 8 + 7]);
    *reinterpret_cast<uint4*>(P + (ch >> 3) * 16384 + row * 128 + (((ch & 7) ^ (row & 7)) << 4)) = w;
  }
}

template <int DHP, int NQ>
__global__ void __launch_bounds__(AttCfg<DHP, NQ>::kThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tm, int nslots, int heads, int N,
                   __nv_bfloat16* __restrict__ o, float scale_log2, int* err) {
  using Cfg = AttCfg<DHP, NQ>;
  constexpr uint32_t kIdS = idesc_bf16_f32(128, 128);
  constexpr uint32_t kIdPV = idesc_bf16_f32(128, 64) | (1u << 16);  // B (= V) MN-major
  extern __shared__ uint8_t smem_raw[];
  const uint32_t base = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + ((1024 - (base & 1023)) & 1023);
  AttBars<NQ>* bar = reinterpret_cast<AttBars<NQ>*>(smem + Cfg::kOffBar);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int bh = blockIdx.y;
  const int slot = bh / heads, head = bh - slot * heads;
  const int q0 = blockIdx.x * (128 * NQ);
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
      mbar_init(&bar->k_full[b], 1);
      mbar_init(&bar->k_empty[b], 1);
      mbar_init(&bar->v_full[b], 1);
      mbar_init(&bar->v_empty[b], 1);
      for (int t = 0; t < NQ; ++t) {
        mbar_init(&bar->s_full[t][b], 1);
        mbar_init(&bar->p_full[t][b], 4);
        mbar_init(&bar->o_full[t][b], 1);
        mbar_init(&bar->buf_free[t][b], 4);
      }
    }
    mbar_init(&bar->drain, 1);
    fence_barrier_init();
    tma_prefetch_desc(&tm);
  }
  if (warp == 1) {
    tmem_alloc(&bar->tmem_base, Cfg::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bar->tmem_base;
  // TMEM buffer (t, b) = columns (2 t + b) * 128 .. + 127

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ TMA
      // K and V have rings of their own: K_j is released as soon as every
      // S_{t,j} is issued, so the next key tile streams in while the PV
      // products on V_j are still pending.
      bool ok = true;
      int last_k[2] = {-1, -1}, last_v[2] = {-1, -1};
      mbar_arrive_expect_tx(&bar->q_full, NQ * Cfg::kTileBytes);
      for (int t = 0; t < NQ; ++t)
        for (int a = 0; a < Cfg::kAtoms; ++a)
          tma_load_2d(smem + Cfg::kOffQ + t * Cfg::kTileBytes + a * 16384, &tm, &bar->q_full,
                      a * 64, row_q + t * 128);
      int nk = 0, nv = 0;
      unsigned long long t_idle = global_ns();
      while (ok && nv < n_kv) {
        bool progressed = false;
        if (nk < n_kv) {
          const int b = nk & 1;
          const uint32_t u = (uint32_t)(nk >> 1);
          if (mbar_test(&bar->k_empty[b], (u & 1) ^ 1)) {
            mbar_arrive_expect_tx(&bar->k_full[b], Cfg::kTileBytes);
            for (int a = 0; a < Cfg::kAtoms; ++a)
              tma_load_2d(smem + Cfg::kOffK + b * Cfg::kTileBytes + a * 16384, &tm,
                          &bar->k_full[b], a * 64, row_k + nk * 128);
            last_k[b] = (int)(u & 1);
            ++nk;
            progressed = true;
          }
        }
        if (nv < nk) {
          const int b = nv & 1;
          const uint32_t u = (uint32_t)(nv >> 1);
          if (mbar_test(&bar->v_empty[b], (u & 1) ^ 1)) {
            mbar_arrive_expect_tx(&bar->v_full[b], Cfg::kTileBytes);
            for (int a = 0; a < Cfg::kAtoms; ++a)
              tma_load_2d(smem + Cfg::kOffV + b * Cfg::kTileBytes + a * 16384, &tm,
                          &bar->v_full[b], a * 64, row_v + nv * 128);
            last_v[b] = (int)(u & 1);
            ++nv;
            progressed = true;
          }
        }
        if (progressed) {
          t_idle = global_ns();
        } else if (*(volatile int*)err != 0) {
          ok = false;
        } else if (global_ns() - t_idle > kWaitLimitNs) {
          atomicCAS(err, 0, kDevTimeoutTma);
          ok = false;
        }
      }
      // every copy in flight lands before the CTA can exit
      mbar_wait(&bar->q_full, 0, err, kDevTimeoutTma);
      for (int b = 0; b < 2; ++b) {
        if (last_k[b] >= 0) mbar_wait(&bar->k_full[b], (uint32_t)last_k[b], err, kDevTimeoutTma);
        if (last_v[b] >= 0) mbar_wait(&bar->v_full[b], (uint32_t)last_v[b], err, kDevTimeoutTma);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------------------ MMA
      // Issue whichever operation is ready (non-blocking tests), so that a
      // lagging softmax warpgroup never holds up the other one:
      //   S_{t,j}  needs K_j loaded and buffer (t, j % 2) freed (PV_{t,j-2} folded)
      //   PV_{t,j} needs P_{t,j} written (S_{t,j} consumed) and V_j loaded
      bool ok = mbar_wait(&bar->q_full, 0, err, kDevTimeoutMma);
      int next_s[NQ], next_pv[NQ];
      for (int t = 0; t < NQ; ++t) next_s[t] = next_pv[t] = 0;
      int released = 0, k_released = 0;  // stages handed back to the loader (V, K)
      unsigned long long t_idle = global_ns();
      while (ok) {
        bool progressed = false, done = true;
        for (int t = 0; t < NQ; ++t) {
          const int js = next_s[t];
          if (js < n_kv) {
            done = false;
            const int b = js & 1;
            const uint32_t u = (uint32_t)(js >> 1);
            if (mbar_test(&bar->k_full[b], u & 1) && mbar_test(&bar->buf_free[t][b], (u & 1) ^ 1)) {
              tc_fence_after();
              const uint32_t sK = smem_u32(smem + Cfg::kOffK + b * Cfg::kTileBytes);
              const uint32_t sQ = smem_u32(smem + Cfg::kOffQ + t * Cfg::kTileBytes);
#pragma unroll
              for (int kk = 0; kk < DHP / 16; ++kk) {
                const uint32_t off = (kk >> 2) * 16384 + (kk & 3) * 32;
                tc_mma_f16(tmem + (2 * t + b) * 128, sw128_kmajor_desc(sQ + off),
                           sw128_kmajor_desc(sK + off), kIdS, kk > 0 ? 1u : 0u);
              }
              tc_commit(&bar->s_full[t][b]);
              next_s[t] = js + 1;
              progressed = true;
            }
          }
          const int jp = next_pv[t];
          if (jp < n_kv) {
            done = false;
            const int b = jp & 1;
            const uint32_t u = (uint32_t)(jp >> 1);
            if (jp < next_s[t] && mbar_test(&bar->p_full[t][b], u & 1) &&
                mbar_test(&bar->v_full[b], u & 1)) {
              tc_fence_after();
              const uint32_t sV = smem_u32(smem + Cfg::kOffV + b * Cfg::kTileBytes);
              const uint32_t sP = smem_u32(smem + Cfg::kOffP + (2 * t + b) * Cfg::kPBytes);
#pragma unroll
              for (int kk = 0; kk < 8; ++kk) {
                const uint64_t ad = sw128_kmajor_desc(sP + (kk >> 2) * 16384 + (kk & 3) * 32);
#pragma unroll
                for (int a = 0; a < Cfg::kAtoms; ++a)
                  tc_mma_f16(tmem + (2 * t + b) * 128 + a * 64, ad,
                             sw128_mnmajor_desc(sV + a * 16384 + kk * 2048), kIdPV,
                             kk > 0 ? 1u : 0u);
              }
              tc_commit(&bar->o_full[t][b]);
              next_pv[t] = jp + 1;
              progressed = true;
            }
          }
        }
        // a K stage goes back to the loader once every tile's S on it is
        // issued, a V stage once every tile's PV on it is
        int min_s = n_kv, min_pv = n_kv;
        for (int t = 0; t < NQ; ++t) {
          min_s = min(min_s, next_s[t]);
          min_pv = min(min_pv, next_pv[t]);
        }
        while (k_released < min_s) {
          tc_commit(&bar->k_empty[k_released & 1]);
          ++k_released;
        }
        while (released < min_pv) {
          tc_commit(&bar->v_empty[released & 1]);
          ++released;
        }
        if (done) break;
        if (progressed) {
          t_idle = global_ns();
        } else if (global_ns() - t_idle > kWaitLimitNs) {
          atomicCAS(err, 0, kDevTimeoutMma);
          ok = false;
        }
      }
      tc_commit(&bar->drain);
      mbar_wait(&bar->drain, 0, err, kDevTimeoutMma);
    }
  } else {
    // ------------------------------------------------------------ softmax
    const int t = (warp - 2) >> 2;  // query tile of this warpgroup
    const int q = warp & 3;         // TMEM lane quarter
    const int row = q * 32 + lane;
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    float O[DHP];
#pragma unroll
    for (int i = 0; i < DHP; ++i) O[i] = 0.f;
    float ref = -INFINITY, l = 0.f, c_prev = 1.f;
    bool ok = true;
    // fold PV_{t,i} (relative to the reference of tile i) and free its buffer
    auto fold = [&](int i, float c) -> bool {
      const int b = i & 1;
      if (!mbar_wait_warp(&bar->o_full[t][b], (uint32_t)(i >> 1) & 1, err, kDevTimeoutEpi)) return false;
      tc_fence_after();
      const uint32_t tb = tmem + (2 * t + b) * 128 + lane_off;
      const bool scale = __any_sync(0xffffffffu, c != 1.f);
      const float2 c2 = make_float2(c, c);
#pragma unroll
      for (int ch = 0; ch < DHP / 32; ++ch) {
        uint32_t r[32];
        tmem_ld32_async(tb + ch * 32, r);
        tmem_ld_wait_regs(r);
#pragma unroll
        for (int e = 0; e < 32; e += 2) {
          float2 acc = fadd2(make_float2(O[ch * 32 + e], O[ch * 32 + e + 1]),
                             make_float2(__uint_as_float(r[e]), __uint_as_float(r[e + 1])));
          if (scale) acc = fmul2(acc, c2);
          O[ch * 32 + e] = acc.x;
          O[ch * 32 + e + 1] = acc.y;
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bar->buf_free[t][b]);
      return true;
    };
    for (int j = 0; j < n_kv && ok; ++j) {
      const int b = j & 1;
      if (!mbar_wait_warp(&bar->s_full[t][b], (uint32_t)(j >> 1) & 1, err, kDevTimeoutEpi)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t tS = tmem + (2 * t + b) * 128 + lane_off;
      uint8_t* Pb = smem + Cfg::kOffP + (2 * t + b) * Cfg::kPBytes;
      const int valid = min(128, N - j * 128);
      if (j == 0) {
        // the first tile sets the reference max
        float mx = -INFINITY;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          uint32_t r[32];
          tmem_ld32_async(tS + c * 32, r);
          tmem_ld_wait_regs(r);
#pragma unroll
          for (int e = 0; e < 32; ++e)
            if (c * 32 + e < valid) mx = fmaxf(mx, __uint_as_float(r[e]));
        }
        ref = mx * scale_log2;
      }
      float tmax4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
      float2 rs2[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
      const float neg_ref = -ref;
      uint32_t ra[32], rb[32];
      // first half: chunks 0 and 1
      tmem_ld32_async(tS + 0, ra);
      tmem_ld_wait_regs(ra);
      tmem_ld32_async(tS + 32, rb);
      if (valid == 128) softmax_chunk<false>(ra, 0, valid, scale_log2, neg_ref, tmax4, rs2, Pb, row);
      else softmax_chunk<true>(ra, 0, valid, scale_log2, neg_ref, tmax4, rs2, Pb, row);
      tmem_ld_wait_regs(rb);
      if (valid == 128) softmax_chunk<false>(rb, 1, valid, scale_log2, neg_ref, tmax4, rs2, Pb, row);
      else softmax_chunk<true>(rb, 1, valid, scale_log2, neg_ref, tmax4, rs2, Pb, row);
      // fold PV_{j-1} (issued at the end of the previous tile)
      if (j >= 1 && !fold(j - 1, c_prev)) { ok = false; break; }
      // second half: chunks 2 and 3
      tmem_ld32_async(tS + 64, ra);
      tmem_ld_wait_regs(ra);
      tmem_ld32_async(tS + 96, rb);
      if (valid == 128) softmax_chunk<false>(ra, 2, valid, scale_log2, neg_ref, tmax4, rs2, Pb, row);
      else softmax_chunk<true>(ra, 2, valid, scale_log2, neg_ref, tmax4, rs2, Pb, row);
      tmem_ld_wait_regs(rb);
      if (valid == 128) softmax_chunk<false>(rb, 3, valid, scale_log2, neg_ref, tmax4, rs2, Pb, row);
      else softmax_chunk<true>(rb, 3, valid, scale_log2, neg_ref, tmax4, rs2, Pb, row);
      const float tmax = fmaxf(fmaxf(tmax4[0], tmax4[1]), fmaxf(tmax4[2], tmax4[3]));
      float rs = (rs2[0].x + rs2[0].y) + (rs2[1].x + rs2[1].y);
      const float tm = tmax * scale_log2;
      if (__any_sync(0xffffffffu, tm - ref > kRedoExcess)) {
        // rare: a row's max jumped far above its reference; rescale what is
        // accumulated to the new max and redo this tile against it
        if (tm > ref) {
          const float c = ex2_mufu(ref - tm);
#pragma unroll
          for (int i = 0; i < DHP; ++i) O[i] *= c;
          l *= c;
          ref = tm;
        }
        float dummy[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
        float2 rr[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          tmem_ld32_async(tS + c * 32, ra);
          tmem_ld_wait_regs(ra);
          softmax_chunk<true>(ra, c, valid, scale_log2, -ref, dummy, rr, Pb, row);
        }
        l += (rr[0].x + rr[0].y) + (rr[1].x + rr[1].y);
        c_prev = 1.f;
      } else {
        float c = 1.f;
        if (tm > ref + kRefSlack) {
          c = ex2_mufu(ref - tm);
          ref = tm;
        }
        l = (l + rs) * c;
        c_prev = c;
      }
      // S consumed, P written: hand the buffer to the PV MMA
      tc_fence_before();
      fence_proxy_async();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bar->p_full[t][b]);
    }
    if (ok) ok = fold(n_kv - 1, c_prev);
    const int qrow = q0 + t * 128 + row;
    if (ok && qrow < N) {
      const float inv = 1.f / l;
      __nv_bfloat16* dst = o + ((size_t)slot * N + qrow) * ((size_t)heads * DHP) + head * DHP;
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
    tmem_dealloc(tmem, Cfg::kTmemCols);
  }
}

template <int DHP, int NQ>
cudaError_t launch_tc(const CUtensorMap& tm, int nslots, int heads, int N, __nv_bfloat16* o,
                      int* err, cudaStream_t st) {
  using Cfg = AttCfg<DHP, NQ>;
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(attn_tc_kernel<DHP, NQ>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmem);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  dim3 grid((N + 128 * NQ - 1) / (128 * NQ), nslots * heads);
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)DHP);
  attn_tc_kernel<DHP, NQ><<<grid, Cfg::kThreads, Cfg::kSmem, st>>>(tm, nslots, heads, N, o,
                                                                   scale_log2, err);
  return cudaGetLastError();
}

}  // namespace

bool attention_tc_supported(int dh) { return dh == 64 || dh == 128; }

cudaError_t launch_attention_tc(const CUtensorMap& tm, int nslots, int heads, int N, int dh,
                                __nv_bfloat16* o, int* err, cudaStream_t st) {
  if (nslots <= 0) return cudaSuccess;
  if (dh == 64) return launch_tc<64, 2>(tm, nslots, heads, N, o, err, st);
  if (dh == 128) return launch_tc<128, 1>(tm, nslots, heads, N, o, err, st);
  return cudaErrorInvalidValue;
}

}  // namespace dc
