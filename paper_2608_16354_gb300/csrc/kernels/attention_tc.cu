// Full spatiotemporal attention on the 5th-generation tensor cores (sm_103a):
// o = softmax(q k^T / sqrt(dh)) v for head dims 64, 72 and 128 (72 runs in
// the 128-column layout: S over 5 K steps of 16, O over 80 columns).
//
// One CTA per (slot, head, NQ x 128 queries); keys stream in tiles of 128.
//   warp 0        TMA: the NQ query tiles once; K_j and V_j into two rings of
//                 their own (kKStages and kVStages stages)
//   warps 1..NQ   one MMA-issuing warp per query tile t (warp 1 also owns
//                 TMEM); for key tile j it issues
//                   S_{t,j}    = Q_t K_j^T   (M=128, N=128, K=dh; Q, K from shared memory)
//                   O_t       += P_{t,j-1} V_{j-1}  (M=128, N=64 per MMA, K=128;
//                                P from TMEM, V from shared memory)
//   other warps of the control warpgroup are idle
//   warps 4..     one softmax warpgroup per query tile, one query row per
//                 thread.
// TMEM per query tile t: O_t (dh columns), S_t (128), P_t (64: 128 bf16 keys).
// Keeping P in TMEM means the PV products read only V from shared memory,
// which halves the shared-memory traffic per key tile (the MMA operand path
// shares shared-memory bandwidth with TMA writes and the mbarriers).
// Softmax of tile j (per row): the whole 128-column S row is loaded into
// registers and S_t handed straight back, so S_{t,j+1} is computed while this
// tile's exponentials run.  P = exp2(s * scale - ref) against a reference max
// `ref` that only moves when the row's max exceeds it by more than 8 (log2
// units); when it moves, the row of O_t (and the row sum) is rescaled by
// exp2(ref_old - ref_new) once PV_{t,j-1} has landed and before P_{t,j} is
// released.  On a full key tile the exponentials run against the current
// reference while the row max is taken alongside (ALU and MUFU in parallel);
// the rare row whose max moves the reference recomputes its P.  Every
// exponential runs on MUFU (ex2.approx): moving a share of them to a
// polynomial on the FMA pipe measured slower here (MUFU is about half busy;
// the loop is bound by the latency of the S -> softmax -> P -> PV chain, not
// by one unit).  V is consumed as an MN-major operand straight from its
// [keys][dh] layout.  Keys beyond N are masked (last tile only).  Every
// mbarrier wait is bounded.
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace dc {

namespace {

constexpr float kRefSlack = 8.0f;  // move the reference max only beyond this (log2 units)

template <int DHP, int NQ>
struct AttCfg {
  static constexpr int kAtoms = DHP / 64;             // 64-element swizzle atoms along dh
  // Two 128-column query tiles (dh in the 128-column layout): O 2 x 128 and
  // S 2 x 128 fill TMEM, so P_t is written over the first 64 columns of S_t
  // once S_t is in registers, and S_{t,j+1} is issued after PV_{t,j} (the
  // MMAs of one thread run in issue order).
  static constexpr bool kAliasP = DHP == 128 && NQ == 2;
  // ring depths (key, value): deeper rings measured no faster at dh 64
  static constexpr int kKStages = kAliasP ? 2 : 3;
  static constexpr int kVStages = kAliasP ? 2 : 3;
  static constexpr int kTileBytes = kAtoms * 16384;   // 128 rows x DHP bf16
  static constexpr int kOffQ = 0;                              // NQ tiles
  static constexpr int kOffK = kOffQ + NQ * kTileBytes;        // kKStages stages
  static constexpr int kOffV = kOffK + kKStages * kTileBytes;  // kVStages stages
  static constexpr int kOffBar = kOffV + kVStages * kTileBytes;
  static constexpr int kSmem = 1024 + kOffBar + 512;
  static constexpr int kThreads = 128 + NQ * 128;   // control warpgroup + softmax
  // two query tiles: the control warpgroup gives registers to the softmax
  // warpgroups (128 x 72 + 256 x 216 = 384 x 168, the launch allocation)
  static constexpr bool kSplitRegs = NQ == 2;
  static constexpr int kRegsLaunch = 168, kRegsCtl = 72, kRegsSoftmax = 216;
  static_assert(!kSplitRegs || 128 * kRegsCtl + NQ * 128 * kRegsSoftmax <= kThreads * kRegsLaunch,
                "register split exceeds the launch allocation");
  // TMEM columns
  static constexpr int kColO = 0;                     // O_t at t * DHP
  static constexpr int kColS = NQ * DHP;              // S_t at kColS + t * 128
  static constexpr int kColP = kAliasP ? kColS : kColS + NQ * 128;  // P_t at kColP + t * kPStride
  static constexpr int kPStride = kAliasP ? 128 : 64;
  static constexpr int kTmemCols = 512;
  static_assert(kColS + NQ * 128 <= kTmemCols && kColP + (NQ - 1) * kPStride + 64 <= kTmemCols,
                "TMEM budget");
  static_assert(kSmem <= 232448, "shared memory budget");
};

template <int NQ, int kKStages, int kVStages>
struct __align__(8) AttBars {
  uint64_t q_full;
  uint64_t k_full[kKStages], k_empty[kKStages];  // key ring: loader <-> S MMAs
  uint64_t v_full[kVStages], v_empty[kVStages];  // value ring: loader <-> PV MMAs
  uint64_t s_full[NQ];    // MMA -> softmax: S_{t,j} ready
  uint64_t s_free[NQ];    // softmax -> MMA: S_{t,j} read into registers
  uint64_t p_full[NQ];    // softmax -> MMA: P_{t,j} in TMEM (and O_t rescaled)
  uint64_t p_free[NQ];    // MMA -> softmax: PV_{t,j} done (P_t free, O_t current)
  uint64_t drain;
  uint32_t tmem_base;
  int abort;              // the error word was set before this CTA started
  uint32_t wlim;          // limit of the waits on work in progress (ns)
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
__device__ __forceinline__ uint32_t pack2(float a, float b) {
  __nv_bfloat162 t = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&t);
}


// max of three (one instruction on sm_100 and later)
__device__ __forceinline__ float fmax3f(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// One 32-column chunk: p = 2^(s * scale - ref), masked beyond `valid`, row
// sum on two packed chains, and the chunk packed into 16 bf16 pairs (even
// key in the low half) for P in TMEM.
template <bool MASKED>
__device__ __forceinline__ void p_chunk(const uint32_t (&v)[32], int c, int valid,
                                        float scale_log2, float neg_ref, float2 (&rs)[2],
                                        uint32_t* pk) {
  const float2 sc = make_float2(scale_log2, scale_log2);
  const float2 nr = make_float2(neg_ref, neg_ref);
#pragma unroll
  for (int e = 0; e < 32; e += 2) {
    const float2 s2 = make_float2(__uint_as_float(v[e]), __uint_as_float(v[e + 1]));
    const float2 x = ffma2(s2, sc, nr);
    float2 p = make_float2(ex2_mufu(x.x), ex2_mufu(x.y));
    if (MASKED) {
      if (c * 32 + e >= valid) p.x = 0.f;
      if (c * 32 + e + 1 >= valid) p.y = 0.f;
    }
    rs[(e >> 1) & 1] = fadd2(rs[(e >> 1) & 1], p);
    pk[e >> 1] = pack2(p.x, p.y);
  }
}

// Raw max of a 32-column chunk (columns at or beyond `valid` ignored).
template <bool MASKED>
__device__ __forceinline__ float chunk_max(const uint32_t (&raw)[32], int c, int valid, float m) {
  float m0 = m, m1 = -INFINITY;
#pragma unroll
  for (int e = 0; e < 32; e += 4) {
    float a = __uint_as_float(raw[e]), b = __uint_as_float(raw[e + 1]);
    float x = __uint_as_float(raw[e + 2]), y = __uint_as_float(raw[e + 3]);
    if (MASKED) {
      if (c * 32 + e >= valid) a = -INFINITY;
      if (c * 32 + e + 1 >= valid) b = -INFINITY;
      if (c * 32 + e + 2 >= valid) x = -INFINITY;
      if (c * 32 + e + 3 >= valid) y = -INFINITY;
    }
    m0 = fmax3f(m0, a, b);
    m1 = fmax3f(m1, x, y);
  }
  return fmaxf(m0, m1);
}

// One unmasked 32-column chunk against the current reference, as p_chunk,
// with the raw chunk max folded in on the ALU pipe (four chains) while MUFU
// runs the exponentials.
__device__ __forceinline__ void p_chunk_max(const uint32_t (&v)[32], float scale_log2,
                                            float neg_ref, float2 (&rs)[2], uint32_t* pk,
                                            float (&m)[4]) {
  const float2 sc = make_float2(scale_log2, scale_log2);
  const float2 nr = make_float2(neg_ref, neg_ref);
#pragma unroll
  for (int e = 0; e < 32; e += 2) {
    const float a = __uint_as_float(v[e]), b = __uint_as_float(v[e + 1]);
    const float2 x = ffma2(make_float2(a, b), sc, nr);
    const float2 p = make_float2(ex2_mufu(x.x), ex2_mufu(x.y));
    m[(e >> 1) & 3] = fmax3f(m[(e >> 1) & 3], a, b);
    rs[(e >> 1) & 1] = fadd2(rs[(e >> 1) & 1], p);
    pk[e >> 1] = pack2(p.x, p.y);
  }
}

// DH: the head dimension; DHP: its storage in shared memory and TMEM (64 or
// 128 columns, 64-element swizzle atoms).  DH < DHP (72 in 128) computes S
// over ceil(DH / 16) K steps of 16 and O over DH rounded up to 16 columns;
// the query/key/value rows hold round16(DH) elements, the rest of each
// 64-element atom is the zero fill of the TMA loads.
template <int DHP, int NQ, int DH = DHP>
__global__ void __launch_bounds__(AttCfg<DHP, NQ>::kThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tm, int nslots, int heads, int N,
                   __nv_bfloat16* __restrict__ o, float scale_log2, int* err) {
  using Cfg = AttCfg<DHP, NQ>;
  constexpr uint32_t kIdS = idesc_bf16_f32(128, 128);
  constexpr uint32_t kIdPV = idesc_bf16_f32(128, 64) | (1u << 16);  // B (= V) MN-major
  static_assert(DH % 8 == 0 && DH <= DHP && DH > DHP - 64, "head dim within the last atom");
  constexpr int kDHR = (DH + 15) / 16 * 16;         // O columns computed
  constexpr int kKSteps = kDHR / 16;                // K steps of the S products
  constexpr int kLastN = kDHR - 64 * (Cfg::kAtoms - 1);  // N of the last atom's PV product
  constexpr uint32_t kIdPVLast = idesc_bf16_f32(128, kLastN) | (1u << 16);
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  constexpr int kKStages = Cfg::kKStages, kVStages = Cfg::kVStages;
  using Bars = AttBars<NQ, kKStages, kVStages>;
  Bars* bar = reinterpret_cast<Bars*>(smem + Cfg::kOffBar);
  static_assert(sizeof(Bars) <= 512, "barrier block exceeds its reserve");

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int bh = blockIdx.y;
  const int slot = bh / heads, head = bh - slot * heads;
  const int q0 = blockIdx.x * (128 * NQ);
  const int n_kv = (N + 127) / 128;
  const int row_q = ((0 * nslots + slot) * heads + head) * N + q0;
  const int row_k = ((1 * nslots + slot) * heads + head) * N;
  const int row_v = ((2 * nslots + slot) * heads + head) * N;

  if (threadIdx.x == 0) {
    // read once, so that the whole CTA takes the same decision below
    bar->abort = *(volatile int*)err;
    bar->wlim = work_wait_limit(err);
    mbar_init(&bar->q_full, 1);
    for (int b = 0; b < kKStages; ++b) {
      mbar_init(&bar->k_full[b], 1);
      mbar_init(&bar->k_empty[b], NQ);  // every query tile's MMA warp releases it
    }
    for (int b = 0; b < kVStages; ++b) {
      mbar_init(&bar->v_full[b], 1);
      mbar_init(&bar->v_empty[b], NQ);
    }
    for (int t = 0; t < NQ; ++t) {
      mbar_init(&bar->s_full[t], 1);
      mbar_init(&bar->s_free[t], 4);
      mbar_init(&bar->p_full[t], 4);
      mbar_init(&bar->p_free[t], 1);
    }
    mbar_init(&bar->drain, NQ);
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
  // the prologue above overlaps the previous kernel; q/k/v are read below
  pdl_trigger();
  pdl_wait();
  const uint32_t tmem = bar->tmem_base;
  const uint32_t wlim = bar->wlim;
  if (bar->abort != 0) {
    // a bounded wait of an earlier launch gave up: do nothing (the host
    // reports DC_ERR_DEVICE_TIMEOUT at its next check)
    if (warp == 1) tmem_dealloc(tmem, Cfg::kTmemCols);
    return;
  }

  // Each register region runs to its own end: the control warpgroup and the
  // softmax warpgroups meet only at the named barrier before TMEM is freed.
  if (warp < 4) {
    if constexpr (Cfg::kSplitRegs)
      asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(Cfg::kRegsCtl));
    if (warp == 0) {
      // ------------------------------------------------------------ TMA
      // The whole warp runs the loop (warp-uniform decisions, taken by lane
      // 0 and broadcast).  Copies issued by one thread complete one after
      // another, so K_j and V_j go out from lanes that rotate over 0-7.  K and V have
      // rings of their own: K_j is released as soon as every S_{t,j} is
      // issued, so later key tiles stream in while the PV products on V_j
      // are still pending.
      bool ok = true;
      int last_k[kKStages], last_v[kVStages];
      for (int b = 0; b < kKStages; ++b) last_k[b] = -1;
      for (int b = 0; b < kVStages; ++b) last_v[b] = -1;
      if (elect_one()) {
        mbar_arrive_expect_tx(&bar->q_full, NQ * Cfg::kTileBytes);
        for (int t = 0; t < NQ; ++t)
          for (int a = 0; a < Cfg::kAtoms; ++a)
            tma_load_2d(smem + Cfg::kOffQ + t * Cfg::kTileBytes + a * 16384, &tm, &bar->q_full,
                        a * 64, row_q + t * 128);
      }
      __syncwarp();
      int nk = 0, nv = 0;
      long long t_idle = clock64();
      while (ok && nv < n_kv) {
        bool progressed = false;
        if (nk < n_kv) {
          const int b = nk % kKStages;
          const uint32_t u = (uint32_t)(nk / kKStages);
          int ready = 0;
          if (lane == 0) ready = mbar_test(&bar->k_empty[b], (u & 1) ^ 1);
          if (__shfl_sync(0xffffffffu, ready, 0)) {
            if (lane == ((2 * nk) & 7)) {
              mbar_arrive_expect_tx(&bar->k_full[b], Cfg::kTileBytes);
              for (int a = 0; a < Cfg::kAtoms; ++a)
                tma_load_2d(smem + Cfg::kOffK + b * Cfg::kTileBytes + a * 16384, &tm,
                            &bar->k_full[b], a * 64, row_k + nk * 128);
            }
            __syncwarp();
            last_k[b] = (int)(u & 1);
            ++nk;
            progressed = true;
          }
        }
        if (nv < nk) {
          const int b = nv % kVStages;
          const uint32_t u = (uint32_t)(nv / kVStages);
          int ready = 0;
          if (lane == 0) ready = mbar_test(&bar->v_empty[b], (u & 1) ^ 1);
          if (__shfl_sync(0xffffffffu, ready, 0)) {
            if (lane == ((2 * nv + 1) & 7)) {
              mbar_arrive_expect_tx(&bar->v_full[b], Cfg::kTileBytes);
              for (int a = 0; a < Cfg::kAtoms; ++a)
                tma_load_2d(smem + Cfg::kOffV + b * Cfg::kTileBytes + a * 16384, &tm,
                            &bar->v_full[b], a * 64, row_v + nv * 128);
            }
            __syncwarp();
            last_v[b] = (int)(u & 1);
            ++nv;
            progressed = true;
          }
        }
        if (progressed) {
          t_idle = clock64();
        } else {
          int stop = 0;
          if (lane == 0) {
            if (*(volatile int*)err != 0) {
              stop = 1;
            } else if (clock64() - t_idle > kWaitLimitCycles) {
              atomicCAS(err, 0, kDevTimeoutTma);
              stop = 1;
            }
          }
          if (__shfl_sync(0xffffffffu, stop, 0)) ok = false;
        }
      }
      // every copy in flight lands before the CTA can exit
      mbar_wait_warp(&bar->q_full, 0, err, kDevTimeoutTma);
      for (int b = 0; b < kKStages; ++b)
        if (last_k[b] >= 0) mbar_wait_warp(&bar->k_full[b], (uint32_t)last_k[b], err, kDevTimeoutTma);
      for (int b = 0; b < kVStages; ++b)
        if (last_v[b] >= 0) mbar_wait_warp(&bar->v_full[b], (uint32_t)last_v[b], err, kDevTimeoutTma);
    } else if (warp >= 1 && warp <= NQ) {
      // ------------------------------------------------------------ MMA
      // One warp per query tile t, fixed order with blocking waits.  Round j
      // issues S_{t,j} (needs K_j and S_{t,j-1} read by the softmax, which
      // happens at the start of that softmax tile), then PV_{t,j-1} (needs
      // P_{t,j-1} and V_{j-1}).  Nothing waited for depends on a later issue
      // of this warp or on the other tile's warp, so the order cannot
      // deadlock.  The whole warp runs the loop with uniform descriptors; one
      // elected lane (the same one throughout, as tcgen05.commit tracks the
      // issuing thread) issues.
      const int t = warp - 1;
      bool ok = mbar_wait_warp(&bar->q_full, 0, err, kDevTimeoutMma, wlim);
      // descriptor + (byte offset >> 4) moves the start address (no carry:
      // shared-memory addresses are below 256 KB)
      const uint64_t dQ = sw128_kmajor_desc(smem_u32(smem + Cfg::kOffQ + t * Cfg::kTileBytes));
      const uint64_t dK = sw128_kmajor_desc(smem_u32(smem + Cfg::kOffK));
      const uint64_t dV = sw128_mnmajor_desc(smem_u32(smem + Cfg::kOffV));
      // S_{t,j} = Q_t K_j^T: needs K_j, and S_t no longer needed (read by the
      // softmax; with P aliased onto S_t, PV_{t,j-1} issued before it)
      auto issue_s = [&](int j) -> bool {
        const int kb = j % kKStages;
        bool good = mbar_wait_warp(&bar->k_full[kb], (uint32_t)(j / kKStages) & 1, err, kDevTimeoutMma, wlim);
        if (!Cfg::kAliasP)
          good = good && mbar_wait_warp(&bar->s_free[t], ((uint32_t)j & 1) ^ 1, err, kDevTimeoutMma, wlim);
        if (!good) return false;
        tc_fence_after();
        if (elect_one()) {
#pragma unroll
          for (int kk = 0; kk < kKSteps; ++kk) {
            const uint32_t off = (kk >> 2) * 16384 + (kk & 3) * 32;
            tc_mma_f16(tmem + Cfg::kColS + t * 128, dQ + (off >> 4),
                       dK + ((uint32_t)(kb * Cfg::kTileBytes + off) >> 4), kIdS, kk > 0 ? 1u : 0u);
          }
          tc_commit(&bar->s_full[t]);
          tc_commit(&bar->k_empty[kb]);
        }
        __syncwarp();
        return true;
      };
      // O_t += P_{t,jp} V_jp: needs V_jp and P_{t,jp} in TMEM
      auto issue_pv = [&](int jp) -> bool {
        const int vb = jp % kVStages;
        const bool good =
            mbar_wait_warp(&bar->v_full[vb], (uint32_t)(jp / kVStages) & 1, err, kDevTimeoutMma, wlim) &&
            mbar_wait_warp(&bar->p_full[t], (uint32_t)jp & 1, err, kDevTimeoutMma, wlim);
        if (!good) return false;
        tc_fence_after();
        if (elect_one()) {
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
#pragma unroll
            for (int a = 0; a < Cfg::kAtoms; ++a)
              tc_mma_f16_ta(tmem + Cfg::kColO + t * DHP + a * 64,
                            tmem + Cfg::kColP + t * Cfg::kPStride + kk * 8,
                            dV + ((uint32_t)(vb * Cfg::kTileBytes + a * 16384 + kk * 2048) >> 4),
                            a == Cfg::kAtoms - 1 ? kIdPVLast : kIdPV, (jp > 0 || kk > 0) ? 1u : 0u);
          }
          tc_commit(&bar->p_free[t]);
          tc_commit(&bar->v_empty[vb]);
        }
        __syncwarp();
        return true;
      };
      for (int j = 0; j <= n_kv && ok; ++j) {
        if (Cfg::kAliasP) {
          if (j >= 1) ok = issue_pv(j - 1);
          if (ok && j < n_kv) ok = issue_s(j);
        } else {
          if (j < n_kv) ok = issue_s(j);
          if (ok && j >= 1) ok = issue_pv(j - 1);
        }
      }
      if (elect_one()) tc_commit(&bar->drain);
      __syncwarp();
      mbar_wait_warp(&bar->drain, 0, err, kDevTimeoutMma);
    }
    tc_fence_before();
    named_bar(1, Cfg::kThreads);
    if (warp == 1) {
      tc_fence_after();
      tmem_dealloc(tmem, Cfg::kTmemCols);
    }
  } else {
    if constexpr (Cfg::kSplitRegs)
      asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(Cfg::kRegsSoftmax));
    // ------------------------------------------------------------ softmax
    const int t = (warp - 4) >> 2;  // query tile of this warpgroup
    const int q = warp & 3;         // TMEM lane quarter
    const int row = q * 32 + lane;
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    const uint32_t tO = tmem + Cfg::kColO + t * DHP + lane_off;
    const uint32_t tS = tmem + Cfg::kColS + t * 128 + lane_off;
    const uint32_t tP = tmem + Cfg::kColP + t * Cfg::kPStride + lane_off;
    float ref = -INFINITY, l = 0.f;
    bool ok = true;
    // (Making the two query tiles take turns on MUFU through named barriers
    // measured slower: the tiles' own S -> P -> PV chains set the pace.)
    for (int j = 0; j < n_kv; ++j) {
      ok = ok && mbar_wait_warp_sl(&bar->s_full[t], (uint32_t)j & 1, err, kDevTimeoutEpi, &bar->wlim);
      if (!ok) break;
      float c = 1.f;
      uint32_t pk[64];
      {
        uint32_t s0[32], s1[32], s2[32], s3[32];
        const int valid = min(128, N - j * 128);
        float2 rs2[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
        // With P aliased onto S_t nothing waits for S_t to be in registers,
        // so on a full key tile after the first the four 32-column loads are
        // chained with the exponentials: each chunk's load is in flight
        // while the previous chunk is exponentiated.
        const bool chained = Cfg::kAliasP && j > 0 && valid == 128;
        tc_fence_after();
        if (chained) {
          tmem_ld32_async(tS + 0, s0);
          tmem_ld_wait_regs(s0);
        } else {
          tmem_ld32_async(tS + 0, s0);
          tmem_ld32_async(tS + 32, s1);
          tmem_ld32_async(tS + 64, s2);
          tmem_ld32_async(tS + 96, s3);
          tmem_ld_wait_regs(s0);
          tmem_ld_wait_regs(s1);
          tmem_ld_wait_regs(s2);
          tmem_ld_wait_regs(s3);
        }
        // S is in registers: hand S_t back to the MMA warp (with P aliased
        // onto S_t, the hand-back is p_full below)
        if (!Cfg::kAliasP) {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&bar->s_free[t]);
        }
        if (chained) {
          float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
          tmem_ld32_async(tS + 32, s1);
          p_chunk_max(s0, scale_log2, -ref, rs2, pk + 0, m4);
          tmem_ld_wait_regs(s1);
          tmem_ld32_async(tS + 64, s2);
          p_chunk_max(s1, scale_log2, -ref, rs2, pk + 16, m4);
          tmem_ld_wait_regs(s2);
          tmem_ld32_async(tS + 96, s3);
          p_chunk_max(s2, scale_log2, -ref, rs2, pk + 32, m4);
          tmem_ld_wait_regs(s3);
          p_chunk_max(s3, scale_log2, -ref, rs2, pk + 48, m4);
          const float tm = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3])) * scale_log2;
          if (tm > ref + kRefSlack) {  // as below: move the reference, recompute P
            c = ex2_mufu(ref - tm);
            ref = tm;
            rs2[0] = make_float2(0.f, 0.f);
            rs2[1] = make_float2(0.f, 0.f);
            p_chunk<false>(s0, 0, 128, scale_log2, -ref, rs2, pk + 0);
            p_chunk<false>(s1, 1, 128, scale_log2, -ref, rs2, pk + 16);
            p_chunk<false>(s2, 2, 128, scale_log2, -ref, rs2, pk + 32);
            p_chunk<false>(s3, 3, 128, scale_log2, -ref, rs2, pk + 48);
          }
        } else if (j > 0 && valid == 128) {
          // Speculate that the reference stays: exponentials against the
          // current reference with the row max computed alongside, so the max
          // is off the critical path.  A row whose max exceeds the reference by
          // more than the slack (rare once the first tiles are in) moves it and
          // recomputes its P and row sum from the S values still in registers;
          // every row ends with exactly the values of the max-first order.
          float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
          p_chunk_max(s0, scale_log2, -ref, rs2, pk + 0, m4);
          p_chunk_max(s1, scale_log2, -ref, rs2, pk + 16, m4);
          p_chunk_max(s2, scale_log2, -ref, rs2, pk + 32, m4);
          p_chunk_max(s3, scale_log2, -ref, rs2, pk + 48, m4);
          const float tm = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3])) * scale_log2;
          if (tm > ref + kRefSlack) {
            c = ex2_mufu(ref - tm);
            ref = tm;
            rs2[0] = make_float2(0.f, 0.f);
            rs2[1] = make_float2(0.f, 0.f);
            p_chunk<false>(s0, 0, 128, scale_log2, -ref, rs2, pk + 0);
            p_chunk<false>(s1, 1, 128, scale_log2, -ref, rs2, pk + 16);
            p_chunk<false>(s2, 2, 128, scale_log2, -ref, rs2, pk + 32);
            p_chunk<false>(s3, 3, 128, scale_log2, -ref, rs2, pk + 48);
          }
        } else {
          float mx;
          if (valid == 128) {
            mx = chunk_max<false>(s0, 0, valid, -INFINITY);
            mx = chunk_max<false>(s1, 1, valid, mx);
            mx = chunk_max<false>(s2, 2, valid, mx);
            mx = chunk_max<false>(s3, 3, valid, mx);
          } else {
            mx = chunk_max<true>(s0, 0, valid, -INFINITY);
            mx = chunk_max<true>(s1, 1, valid, mx);
            mx = chunk_max<true>(s2, 2, valid, mx);
            mx = chunk_max<true>(s3, 3, valid, mx);
          }
          const float tm = mx * scale_log2;
          if (j == 0) {
            ref = tm;
          } else if (tm > ref + kRefSlack) {
            c = ex2_mufu(ref - tm);
            ref = tm;
          }
          const float neg_ref = -ref;
          if (valid == 128) {
            p_chunk<false>(s0, 0, valid, scale_log2, neg_ref, rs2, pk + 0);
            p_chunk<false>(s1, 1, valid, scale_log2, neg_ref, rs2, pk + 16);
            p_chunk<false>(s2, 2, valid, scale_log2, neg_ref, rs2, pk + 32);
            p_chunk<false>(s3, 3, valid, scale_log2, neg_ref, rs2, pk + 48);
          } else {
            p_chunk<true>(s0, 0, valid, scale_log2, neg_ref, rs2, pk + 0);
            p_chunk<true>(s1, 1, valid, scale_log2, neg_ref, rs2, pk + 16);
            p_chunk<true>(s2, 2, valid, scale_log2, neg_ref, rs2, pk + 32);
            p_chunk<true>(s3, 3, valid, scale_log2, neg_ref, rs2, pk + 48);
          }
        }
        l = l * c + ((rs2[0].x + rs2[0].y) + (rs2[1].x + rs2[1].y));
      }
      // P_t and O_t are free once PV_{t,j-1} has landed
      ok = mbar_wait_warp_sl(&bar->p_free[t], ((uint32_t)j & 1) ^ 1, err, kDevTimeoutEpi, &bar->wlim);
      if (!ok) break;
      tc_fence_after();
      if (__any_sync(0xffffffffu, c != 1.f)) {
        // the reference moved for some row of this warp: rescale the warp's
        // 32 rows of O_t (c = 1 elsewhere) before PV_{t,j} accumulates
#pragma unroll
        for (int ch = 0; ch < (kDHR + 31) / 32; ++ch) {
          uint32_t r[32];
          tmem_ld32_async(tO + ch * 32, r);
          tmem_ld_wait_regs(r);
#pragma unroll
          for (int e = 0; e < 32; ++e) r[e] = __float_as_uint(__uint_as_float(r[e]) * c);
          tmem_st32(tO + ch * 32, r);
        }
      }
      tmem_st32(tP + 0, *reinterpret_cast<const uint32_t(*)[32]>(pk));
      tmem_st32(tP + 32, *reinterpret_cast<const uint32_t(*)[32]>(pk + 32));
      tmem_st_wait();
      // P in TMEM (and O rescaled): hand both to the PV MMA
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bar->p_full[t]);
    }
    // the last PV product of this query tile completes O_t
    if (ok) ok = mbar_wait_warp_sl(&bar->p_free[t], (uint32_t)(n_kv - 1) & 1, err, kDevTimeoutEpi, &bar->wlim);
    const int qrow = q0 + t * 128 + row;
    if (ok) {
      tc_fence_after();
      const float inv = 1.f / l;
      __nv_bfloat16* dst = o + ((size_t)slot * N + qrow) * ((size_t)heads * DH) + head * DH;
#pragma unroll
      for (int ch = 0; ch < (DH + 31) / 32; ++ch) {
        uint32_t r[32];
        tmem_ld32_async(tO + ch * 32, r);
        tmem_ld_wait_regs(r);
        if (qrow < N) {
#pragma unroll
          for (int e = 0; e < 32 && ch * 32 + e < DH; e += 8) {
            uint4 w;
            w.x = pack2(__uint_as_float(r[e]) * inv, __uint_as_float(r[e + 1]) * inv);
            w.y = pack2(__uint_as_float(r[e + 2]) * inv, __uint_as_float(r[e + 3]) * inv);
            w.z = pack2(__uint_as_float(r[e + 4]) * inv, __uint_as_float(r[e + 5]) * inv);
            w.w = pack2(__uint_as_float(r[e + 6]) * inv, __uint_as_float(r[e + 7]) * inv);
            *reinterpret_cast<uint4*>(dst + ch * 32 + e) = w;
          }
        }
      }
    }
    tc_fence_before();
    named_bar(1, Cfg::kThreads);
  }
}

template <int DHP, int NQ, int DH = DHP>
cudaError_t launch_tc(const CUtensorMap& tm, int nslots, int heads, int N, __nv_bfloat16* o,
                      int* err, cudaStream_t st) {
  using Cfg = AttCfg<DHP, NQ>;
  static std::atomic<unsigned long long> configured{0};
  const cudaError_t e = configure_once_per_device(configured, [] {
    cudaError_t r = cudaFuncSetAttribute(attn_tc_kernel<DHP, NQ, DH>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmem);
    if (r != cudaSuccess) return r;
    // setmaxnreg.inc waits until the CTA's launch allocation can serve it:
    // never launch a build whose allocation is not the one the split assumes
    cudaFuncAttributes fa;
    r = cudaFuncGetAttributes(&fa, attn_tc_kernel<DHP, NQ, DH>);
    if (r != cudaSuccess) return r;
    if (Cfg::kSplitRegs && fa.numRegs != Cfg::kRegsLaunch) return cudaErrorInvalidConfiguration;
    return cudaSuccess;
  });
  if (e != cudaSuccess) return e;
  dim3 grid((N + 128 * NQ - 1) / (128 * NQ), nslots * heads);
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)DH);
  return launch_pdl(attn_tc_kernel<DHP, NQ, DH>, grid, dim3(Cfg::kThreads), Cfg::kSmem, st, tm,
                    nslots, heads, N, o, scale_log2, err);
}

}  // namespace

bool attention_tc_supported(int dh) { return dh == 64 || dh == 72 || dh == 128; }

cudaError_t launch_attention_tc(const CUtensorMap& tm, int nslots, int heads, int N, int dh,
                                __nv_bfloat16* o, int* err, cudaStream_t st) {
  if (nslots <= 0) return cudaSuccess;
  if (dh == 64) return launch_tc<64, 2>(tm, nslots, heads, N, o, err, st);
  if (dh == 128) return launch_tc<128, 2>(tm, nslots, heads, N, o, err, st);
  if (dh == 72) return launch_tc<128, 2, 72>(tm, nslots, heads, N, o, err, st);
  return cudaErrorInvalidValue;
}

}  // namespace dc
