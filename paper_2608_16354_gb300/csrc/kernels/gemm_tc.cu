// bf16 GEMM on the 5th-generation tensor cores (tcgen05), sm_103a.
//
//   C[M, N] = A[M, K] * W[N, K]^T   (A: activations, W: nn.Linear-style
//   weights, both K-major bf16), fp32 accumulation in TMEM, followed by one
//   of the fused DiT epilogues (QKV scatter, GELU, gated residual).
//
// Design: persistent CTAs (one per SM) in clusters of two that share one
// M = 256 pair MMA (tcgen05.mma.cta_group::2): the pair owns a 256 x 192
// output tile, each CTA holds its 128 rows of A and half of the W tile (96
// rows) in its own shared memory at the same offsets, rank 0 issues the MMAs
// and each CTA receives its 128 rows of the accumulator in its own TMEM.  A
// CTA so pulls 28 KB per 64-deep K step instead of 40 KB, which buys six
// ring stages (four for the residual kernels) within shared memory -- the
// loads, whose latency reaches several thousand cycles under full load, not
// the tensor core bound these GEMMs.  Rank 1's copies complete on rank 0's
// full barriers; the MMA commits release the stages and hand the
// accumulators to the epilogues of both CTAs (multicast), and both CTAs'
// epilogue warps free an accumulator on rank 0.  Warp 0 streams the tiles
// with TMA; warp 1 of rank 0 issues the MMAs into one of two TMEM
// accumulators (warp 1 of each CTA takes part in the pair TMEM allocation);
// warps 2-9 drain the other accumulator with tcgen05.ld and run the
// epilogue, so the epilogue of tile i overlaps the MMAs of tile i+1.
// N = 192 divides every projection width of the configured models (3d, d,
// 4d for d = 384, 1152, 3072).
//
// Epilogues (bias and gate vectors of the tile are staged in shared memory):
//   QKV      y = acc + b, 16-byte stores into head-major q / k / v
//   GELU     y = gelu(acc + b) in bf16, written to a swizzled shared tile and
//            stored with TMA
//   residual the fp32 residual tile is prefetched with TMA into shared memory
//            while the MMAs run, h = h_in + gate (acc + b) is formed in place
//            and the tile goes back with TMA stores, so the epilogue moves
//            whole tiles at DRAM speed instead of single rows
// Every mbarrier wait is bounded.
#include "common.cuh"
#include "epilogue.cuh"
#include "kernels.h"

namespace dc {

namespace {

constexpr int kBM = 128, kBN = 192, kBK = 64;
constexpr int kABytes = kBM * kBK * 2;        // 16 KB
constexpr int kBBytes = kBN * kBK * 2;        // 24 KB: the pair's W tile
constexpr int kBHalf = kBBytes / 2;            // 12 KB: this CTA's half (96 rows)
constexpr int kStageBytes = kABytes + kBHalf;  // 28 KB per CTA and K step
constexpr int kTmemCols = 512;                // two 192-column accumulators at 0 / 256
constexpr int kThreads = 320;                 // 10 warps
constexpr int kEpiWarps = 8;
constexpr int kEpiThreads = kEpiWarps * 32;
constexpr uint32_t kIdesc = idesc_bf16_f32(2 * kBM, kBN);  // one M = 256 MMA over the pair

// HALF (residual mode, long K): the fp32 residual tile is staged and
// written in two 96-column halves, which frees 48 KB of shared memory for two
// more ring stages.
template <int MODE, bool HALF = false>
struct GemmCfg {
  static constexpr int kStages = MODE == kEpiResid && !HALF ? 4 : 6;
  // epilogue staging tile: residual 6 boxes of [128 rows][32 fp32], GELU and
  // QKV 3 boxes of [128 rows][64 bf16]; 16 KB per box, 128-byte swizzle
  static constexpr int kOutBytes = MODE == kEpiResid && !HALF ? 6 * 16384 : 3 * 16384;
  static constexpr int kOffA = 0;
  static constexpr int kOffB = kOffA + kStages * kABytes;
  static constexpr int kOffOut = kOffB + kStages * kBHalf;
  static constexpr int kOffVec = kOffOut + kOutBytes;            // bias + two gate rows
  static constexpr int kOffBar = kOffVec + 3 * kBN * 4;
  static constexpr int kSmem = 1024 + kOffBar + 256;
  static_assert(kStages <= 6, "barrier arrays hold six stages");
  static_assert(kSmem <= 232448, "shared memory budget");
};

struct __align__(8) Barriers {
  uint64_t full[6];   // rank 0: both CTAs' loads of a stage landed
  uint64_t empty[6];  // each CTA: the pair MMAs have read its stage
  uint64_t tmem_full[2];
  uint64_t tmem_empty[2];
  uint64_t hin_full;
  uint64_t drain;
  uint32_t tmem_base;
  int abort;  // the error word was set before this CTA started
};

// byte offset of 16-byte chunk `c` of row `r` in a [rows][128 B] box written
// with 128-byte swizzle (the layout TMA produces and consumes)
__device__ __forceinline__ int sw128_off(int r, int c) { return r * 128 + ((c ^ (r & 7)) << 4); }

template <int MODE, bool HALF = false>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    gemm_bf16_tc_kernel(const __grid_constant__ CUtensorMap tmA,
                        const __grid_constant__ CUtensorMap tmB,
                        const __grid_constant__ CUtensorMap tmCin,
                        const __grid_constant__ CUtensorMap tmCout, int M, int N, int K,
                        EpiArgs ep, SlotMap map, int* err) {
  using Cfg = GemmCfg<MODE, HALF>;
  constexpr int kStages = Cfg::kStages;
  constexpr int kHinBoxes = HALF ? 3 : 6;  // residual boxes staged at a time
  extern __shared__ uint8_t smem_raw[];
  const uint32_t base = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + ((1024 - (base & 1023)) & 1023);
  uint8_t* sA = smem + Cfg::kOffA;
  uint8_t* sB = smem + Cfg::kOffB;
  uint8_t* sOut = smem + Cfg::kOffOut;
  float* vec = reinterpret_cast<float*>(smem + Cfg::kOffVec);
  Barriers* bar = reinterpret_cast<Barriers*>(smem + Cfg::kOffBar);
  static_assert(sizeof(Barriers) <= 256, "barrier block exceeds its reserve");

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int tiles_n = N / kBN;
  const int tiles_m = (M + kBM - 1) / kBM;
  const int KB = K / kBK;
  // pair tiles: (pair of m tiles, n tile); this CTA takes m tile 2 p + rank
  const int rank = (int)cluster_rank();
  const int n_pt = ((tiles_m + 1) / 2) * tiles_n;
  const int pair = blockIdx.x >> 1, n_pairs = gridDim.x >> 1;
  auto m0_of = [&](int pt) { return ((pt / tiles_n) * 2 + rank) * kBM; };
  auto n0_of = [&](int pt) { return (pt % tiles_n) * kBN; };

  if (threadIdx.x == 0) {
    // read once, so that the whole CTA takes the same decision below
    bar->abort = *(volatile int*)err;
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&bar->full[s], 2);   // one expect_tx arrival from each CTA's producer
      mbar_init(&bar->empty[s], 1);  // the pair MMAs' commit, multicast to both CTAs
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bar->tmem_full[b], 1);
      mbar_init(&bar->tmem_empty[b], 2 * kEpiWarps);  // used on rank 0: both CTAs' epilogues
    }
    mbar_init(&bar->hin_full, 1);
    mbar_init(&bar->drain, 1);
    fence_barrier_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    if (MODE != kEpiQKV) tma_prefetch_desc(&tmCout);
    if (MODE == kEpiResid) tma_prefetch_desc(&tmCin);
  }
  if (warp == 1) {
    tmem_alloc_pair(&bar->tmem_base, kTmemCols);
    tmem_relinquish_pair();
  }
  // the peer's barriers are initialised before any multicast or remote arrive
  tc_fence_before();
  cluster_sync();
  tc_fence_after();
  // the prologue above overlaps the previous kernel; its outputs are read below
  pdl_trigger();
  pdl_wait();
  const uint32_t tmem_base = bar->tmem_base;
  const uint32_t wlim = work_wait_limit(err);
  // a bounded wait of an earlier launch gave up: do nothing (the host reports
  // DC_ERR_DEVICE_TIMEOUT at its next check), but still meet the peer at the
  // final cluster barrier
  if (bar->abort != 0) {
  } else if (warp == 0) {
    // -------------------------------------------------- TMA producer
    // The whole warp runs the loop (uniform waits).  Copies issued by one
    // thread complete one after another (about one box per 300-400 cycles
    // whatever its size), so the boxes of successive stages rotate over
    // lanes 0-7: A from an even lane, the W half from the next odd one.
    int stage = 0, issued = 0;
    uint32_t phase = 0;
    int last_phase[kStages];
    for (int s = 0; s < kStages; ++s) last_phase[s] = -1;
    bool ok = true;
    for (int pt = pair; pt < n_pt && ok; pt += n_pairs) {
      const int m0 = m0_of(pt);
      const int n0 = n0_of(pt);
      for (int kb = 0; kb < KB; ++kb) {
        // the stage is free once the pair MMAs have read it; both CTAs'
        // copies are counted on rank 0's full barrier
        if (!mbar_wait_warp(&bar->empty[stage], phase ^ 1, err, kDevTimeoutTma, wlim)) { ok = false; break; }
        const int la = (2 * issued) & 7;
        if (rank == 0) {
          if (lane == la) mbar_arrive_expect_tx(&bar->full[stage], kStageBytes);
          __syncwarp();
          if (lane == la) tma_load_2d(sA + (size_t)stage * kABytes, &tmA, &bar->full[stage], kb * kBK, m0);
          if (lane == la + 1)
            tma_load_2d(sB + (size_t)stage * kBHalf, &tmB, &bar->full[stage], kb * kBK, n0);
        } else {
          const uint32_t fb = cluster_addr(&bar->full[stage], 0);
          if (lane == la) mbar_arrive_expect_tx_cluster(fb, kStageBytes);
          __syncwarp();
          if (lane == la) tma_load_2d_pair(sA + (size_t)stage * kABytes, &tmA, fb, kb * kBK, m0);
          if (lane == la + 1)
            tma_load_2d_pair(sB + (size_t)stage * kBHalf, &tmB, fb, kb * kBK, n0 + kBN / 2);
        }
        __syncwarp();
        ++issued;
        last_phase[stage] = (int)phase;
        if (++stage == kStages) { stage = 0; phase ^= 1; }
      }
    }
    // do not leave the pair with copies still landing in shared memory: rank
    // 0's full barriers count both CTAs' copies, and rank 1 stays until rank
    // 0 has passed here (final cluster barrier)
    if (rank == 0)
      for (int s = 0; s < kStages; ++s)
        if (last_phase[s] >= 0) mbar_wait_warp(&bar->full[s], (uint32_t)last_phase[s], err, kDevTimeoutTma);
  } else if (warp == 1 && rank != 0) {
    // rank 1 issues nothing; its shared memory and TMEM are in use by rank
    // 0's pair MMAs until they drain
    mbar_wait_warp(&bar->drain, 0, err, kDevTimeoutMma);
  } else if (warp == 1) {
    // -------------------------------------------------- MMA issuer (rank 0)
    // The whole warp runs the loop with uniform descriptors; one elected lane
    // (the same one throughout: tcgen05.commit tracks the issuing thread)
    // issues the pair MMAs (M = 256: rows of A and half of the W columns from
    // each CTA's shared memory at the same offsets, 128 rows of D in each
    // CTA's TMEM) and commits.
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    int t = 0;
    // descriptor + (byte offset >> 4) moves the start address (no carry:
    // shared-memory addresses are below 256 KB)
    const uint64_t dA = sw128_kmajor_desc(smem_u32(sA));
    const uint64_t dB = sw128_kmajor_desc(smem_u32(sB));
    for (int pt = pair; pt < n_pt && ok; pt += n_pairs, ++t) {
      const int b = t & 1;
      const uint32_t use = (uint32_t)(t >> 1);
      if (!mbar_wait_warp(&bar->tmem_empty[b], (use & 1) ^ 1, err, kDevTimeoutMma, wlim)) { ok = false; break; }
      tc_fence_after();
      const uint32_t d_tmem = tmem_base + (uint32_t)(b * 256);
      for (int kb = 0; kb < KB; ++kb) {
        if (!mbar_wait_warp(&bar->full[stage], phase, err, kDevTimeoutMma, wlim)) { ok = false; break; }
        tc_fence_after();
        if (elect_one()) {
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk) {
            tc_mma_f16_pair(d_tmem, dA + ((uint32_t)(stage * kABytes + kk * 32) >> 4),
                            dB + ((uint32_t)(stage * kBHalf + kk * 32) >> 4), kIdesc,
                            (kb | kk) != 0 ? 1u : 0u);
          }
          tc_commit_pair_mc(&bar->empty[stage], (uint16_t)0x3);  // release it in both CTAs
        }
        __syncwarp();
        if (++stage == kStages) { stage = 0; phase ^= 1; }
      }
      if (ok) {
        if (elect_one()) tc_commit_pair_mc(&bar->tmem_full[b], (uint16_t)0x3);
        __syncwarp();
      }
    }
    // every pair MMA this warp issued has completed once `drain` flips (in
    // both CTAs)
    if (elect_one()) tc_commit_pair_mc(&bar->drain, (uint16_t)0x3);
    __syncwarp();
    mbar_wait_warp(&bar->drain, 0, err, kDevTimeoutMma);
  } else {
    // ---------------------------------------------------- epilogue warps
    const int q = warp & 3;             // TMEM lane quarter this warp may access
    const int half = (warp - 2) >> 2;   // which 96-column half of the tile
    const int et = threadIdx.x - 64;    // epilogue thread 0..255
    const bool copy_warp = warp == 2;   // issues the tile's bulk copies, one box per lane
    const int r = q * 32 + lane;        // row of the tile owned by this thread
    int hin_loads = 0, hin_used = 0;    // residual stagings requested / consumed
    if (MODE == kEpiResid && copy_warp && pair < n_pt) {
      if (lane == 0) mbar_arrive_expect_tx(&bar->hin_full, Cfg::kOutBytes);
      __syncwarp();
      if (lane < kHinBoxes)
        tma_load_2d(sOut + lane * 16384, &tmCin, &bar->hin_full, n0_of(pair) + 32 * lane, m0_of(pair));
      hin_loads = 1;
    }
    // bias (and gate rows) of the next tile are loaded into registers while
    // the current tile is processed, and staged to shared memory at its start
    float nb = 0.f, nga = 0.f, ngb = 0.f;
    auto fetch_vec = [&](int pt) {
      if (pt < n_pt && et < kBN && m0_of(pt) < M) {
        const int fm0 = m0_of(pt), fn0 = n0_of(pt);
        nb = ep.bias[fn0 + et];
        if (MODE == kEpiResid) {
          const int sa = fm0 / ep.n_tok, sb = (min(fm0 + kBM, M) - 1) / ep.n_tok;
          nga = ep.mod[(size_t)map.scene[sa] * ep.mod_stride + ep.gate_off + fn0 + et];
          ngb = ep.mod[(size_t)map.scene[sb] * ep.mod_stride + ep.gate_off + fn0 + et];
        }
      }
    };
    fetch_vec(pair);
    int t = 0;
    bool ok = true;
    for (int pt = pair; pt < n_pt && ok; pt += n_pairs, ++t) {
      const int b = t & 1;
      const uint32_t use = (uint32_t)(t >> 1);
      // every wait outcome is made uniform (warp, then the 8 epilogue warps at
      // the named barrier) so that an abort is taken by all of them together
      const bool acc_ok = mbar_wait_warp(&bar->tmem_full[b], use & 1, err, kDevTimeoutEpi, wlim);
      const int m0 = m0_of(pt);
      const int n0 = n0_of(pt);
      // the second tile of the last pair may lie below M: it runs (its A rows
      // are zero) but writes nothing
      const bool live = m0 < M;
      float acc[3][32];
      if (acc_ok) {
        tc_fence_after();
#pragma unroll
        for (int c = 0; c < 3; ++c) {
          const uint32_t taddr =
              tmem_base + (uint32_t)(b * 256 + half * 96 + c * 32) + ((uint32_t)(q * 32) << 16);
          tmem_ld32(taddr, acc[c]);
        }
        tmem_ld_wait();
        tc_fence_before();
        __syncwarp();
        // the accumulator is in registers (wait::ld): rank 0 may reuse it
        if (lane == 0) mbar_arrive_cluster_relaxed(cluster_addr(&bar->tmem_empty[b], 0));
      }

      // stage bias (and gate rows) of this tile once the previous tile is done
      if (named_bar_or(1, kEpiThreads, !acc_ok)) { ok = false; break; }
      const int last_row = live ? min(m0 + kBM, M) - 1 : m0;
      const int slot_a = m0 / ep.n_tok, slot_b = last_row / ep.n_tok;
      const int split = (slot_a + 1) * ep.n_tok;  // first row that belongs to slot_b
      if (et < kBN) {
        vec[et] = nb;
        if (MODE == kEpiResid) {
          vec[kBN + et] = nga;
          vec[2 * kBN + et] = ngb;
        }
      }
      fetch_vec(pt + n_pairs);
      if (MODE != kEpiResid && copy_warp && lane < 3) bulk_wait_read0();  // previous stores read sOut
      named_bar(1, kEpiThreads);

      if constexpr (MODE == kEpiResid) {
        // rows spanning more than two slots (tokens per scene < 128) take the
        // gate from global memory per row
        const bool two_slots = slot_b - slot_a <= 1;
        const int row = m0 + r;
        const float* gsel = vec + (row < split ? kBN : 2 * kBN);
        const float* grow = nullptr;
        if (!two_slots && row < M)
          grow = ep.mod + (size_t)map.scene[row / ep.n_tok] * ep.mod_stride + ep.gate_off + n0;
        // h = h_in + gate (acc + b) on this thread's 96 columns, in the staged
        // boxes whose first column is `base`
        auto apply = [&](int base) {
#pragma unroll
          for (int c = 0; c < 3; ++c) {
            const int col0 = half * 96 + c * 32;  // tile column of this 32-column chunk
            uint8_t* box = sOut + ((col0 - base) >> 5) * 16384;
#pragma unroll
            for (int ch = 0; ch < 8; ++ch) {
              float4* p = reinterpret_cast<float4*>(box + sw128_off(r, ch));
              float4 h = *p;
              const int j = col0 + ch * 4;
              float g0, g1, g2, g3;
              if (two_slots) {
                g0 = gsel[j]; g1 = gsel[j + 1]; g2 = gsel[j + 2]; g3 = gsel[j + 3];
              } else if (grow) {
                g0 = grow[j]; g1 = grow[j + 1]; g2 = grow[j + 2]; g3 = grow[j + 3];
              } else {
                g0 = g1 = g2 = g3 = 0.f;
              }
              h.x += g0 * (acc[c][ch * 4 + 0] + vec[j + 0]);
              h.y += g1 * (acc[c][ch * 4 + 1] + vec[j + 1]);
              h.z += g2 * (acc[c][ch * 4 + 2] + vec[j + 2]);
              h.w += g3 * (acc[c][ch * 4 + 3] + vec[j + 3]);
              *p = h;
            }
          }
        };
        const int next = pt + n_pairs;
        bool failed = false;  // the same for all epilogue threads (named_bar_or)
#pragma unroll 1
        for (int pass = 0; pass < (HALF ? 2 : 1); ++pass) {
          // pass p stages columns 96 p .. (all 192 without HALF)
          const bool hin_ok = mbar_wait_warp(&bar->hin_full, HALF ? (uint32_t)pass : (uint32_t)t & 1,
                                             err, kDevTimeoutEpi, wlim);
          if (hin_ok) ++hin_used;
          if (hin_ok && (!HALF || half == pass)) apply(HALF ? 96 * pass : 0);
          fence_proxy_async();
          failed = named_bar_or(1, kEpiThreads, !hin_ok);
          if (failed) break;
          if (copy_warp) {
            const int c0 = HALF ? 96 * pass : 0;
            if (live && lane < kHinBoxes) {
              tma_store_2d(&tmCout, sOut + lane * 16384, n0 + c0 + 32 * lane, m0);
              bulk_commit();
              bulk_wait_read0();
            }
            __syncwarp();  // every box has been read out before the next staging lands
            // next staging: the second half of this tile, else the next tile
            const bool second = HALF && pass == 0;
            if (second || next < n_pt) {
              if (lane == 0) mbar_arrive_expect_tx(&bar->hin_full, Cfg::kOutBytes);
              __syncwarp();
              if (lane < kHinBoxes)
                tma_load_2d(sOut + lane * 16384, &tmCin, &bar->hin_full,
                            (second ? n0 + 96 : n0_of(next)) + 32 * lane, second ? m0 : m0_of(next));
              ++hin_loads;
            }
          }
        }
        if (failed) { ok = false; break; }
      } else if constexpr (MODE == kEpiGELU) {
#pragma unroll
        for (int c = 0; c < 3; ++c) {
#pragma unroll
          for (int g = 0; g < 4; ++g) {
            const int j = half * 96 + c * 32 + g * 8;  // tile column of this 8-column group
            uint4 w;
            float v[8];
#pragma unroll
            for (int i = 0; i < 8; i += 2) {
              const float2 x = f2_add(make_float2(acc[c][g * 8 + i], acc[c][g * 8 + i + 1]),
                                      make_float2(vec[j + i], vec[j + i + 1]));
              const float2 y = gelu_tanh_pair(x);
              v[i] = y.x;
              v[i + 1] = y.y;
            }
            __nv_bfloat162 p0 = __floats2bfloat162_rn(v[0], v[1]);
            __nv_bfloat162 p1 = __floats2bfloat162_rn(v[2], v[3]);
            __nv_bfloat162 p2 = __floats2bfloat162_rn(v[4], v[5]);
            __nv_bfloat162 p3 = __floats2bfloat162_rn(v[6], v[7]);
            w.x = *reinterpret_cast<uint32_t*>(&p0);
            w.y = *reinterpret_cast<uint32_t*>(&p1);
            w.z = *reinterpret_cast<uint32_t*>(&p2);
            w.w = *reinterpret_cast<uint32_t*>(&p3);
            *reinterpret_cast<uint4*>(sOut + (j >> 6) * 16384 + sw128_off(r, (j & 63) >> 3)) = w;
          }
        }
        fence_proxy_async();
        named_bar(1, kEpiThreads);
        if (copy_warp && live && lane < 3) {
          tma_store_2d(&tmCout, sOut + lane * 16384, n0 + 64 * lane, m0);
          bulk_commit();
        }
      } else if (ep.qkv_tma && (!live || (m0 + kBM <= M && (m0 + kBM - 1) / ep.n_tok == slot_a))) {
        // QKV, tile inside one slot: each 64-column group is one head's
        // [128 tokens][64] block of q, k or v, contiguous in the head-major
        // layout; stage the bf16 tile swizzled and store it with TMA
#pragma unroll
        for (int c = 0; c < 3; ++c) {
#pragma unroll
          for (int g = 0; g < 4; ++g) {
            const int j = half * 96 + c * 32 + g * 8;  // tile column of this 8-column group
            float v[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) v[i] = acc[c][g * 8 + i] + vec[j + i];
            Pack8<__nv_bfloat16>::store(
                reinterpret_cast<__nv_bfloat16*>(sOut + (j >> 6) * 16384 + sw128_off(r, (j & 63) >> 3)), v);
          }
        }
        fence_proxy_async();
        named_bar(1, kEpiThreads);
        if (copy_warp && live && lane < 3) {
          const int tok0 = m0 - slot_a * ep.n_tok;
          const int col = n0 + 64 * lane;
          const int which = col / ep.d;
          const int within = col - which * ep.d;
          const int head = within / ep.dh;
          const int e = within - head * ep.dh;
          tma_store_2d(&tmCout, sOut + lane * 16384, e,
                       ((which * ep.nslots + slot_a) * ep.heads + head) * ep.n_tok + tok0);
          bulk_commit();
        }
      } else {
        // QKV: each thread stores 16-byte pieces of its own row
        const int row = m0 + r;
        if (row < M) {
          const int slot = row / ep.n_tok;
          const int tok = row - slot * ep.n_tok;
#pragma unroll
          for (int c = 0; c < 3; ++c) {
#pragma unroll
            for (int g = 0; g < 4; ++g) {
              const int j = half * 96 + c * 32 + g * 8;
              const int col = n0 + j;
              const int which = col / ep.d;
              const int within = col - which * ep.d;
              const int head = within / ep.dh;
              const int e = within - head * ep.dh;
              float v[8];
#pragma unroll
              for (int i = 0; i < 8; ++i) v[i] = acc[c][g * 8 + i] + vec[j + i];
              __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(ep.out) +
                                   ((((size_t)which * ep.nslots + slot) * ep.heads + head) * ep.n_tok + tok) *
                                       ep.dhp + e;
              Pack8<__nv_bfloat16>::store(dst, v);
            }
          }
        }
      }
    }
    if (copy_warp) {
      if (lane < 6) bulk_wait0();
      // a residual prefetch that was never consumed (aborted run) must land first
      if (MODE == kEpiResid && lane == 0 && !ok && hin_loads > hin_used)
        mbar_wait(&bar->hin_full, (uint32_t)(hin_loads - 1) & 1, err, kDevTimeoutEpi);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, kTmemCols);
  }
  // no CTA leaves while its peer may still multicast into it or arrive on
  // its barriers
  cluster_sync();
}

template <int MODE, bool HALF = false>
cudaError_t launch_mode(const CUtensorMap& tmA, const CUtensorMap& tmB, const CUtensorMap& tmCin,
                        const CUtensorMap& tmCout, int M, int N, int K, const EpiArgs& ep,
                        const SlotMap& map, int* err, int n_sms, cudaStream_t st) {
  using Cfg = GemmCfg<MODE, HALF>;
  static std::atomic<unsigned long long> configured{0};
  const cudaError_t e = configure_once_per_device(configured, [] {
    return cudaFuncSetAttribute(gemm_bf16_tc_kernel<MODE, HALF>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmem);
  });
  if (e != cudaSuccess) return e;
  // clusters of two CTAs over pairs of m tiles (the grid is even)
  const int pair_tiles = ((M + kBM - 1) / kBM + 1) / 2 * (N / kBN);
  const int grid = 2 * (pair_tiles < n_sms / 2 ? pair_tiles : n_sms / 2);
  return launch_pdl(gemm_bf16_tc_kernel<MODE, HALF>, dim3(grid), dim3(kThreads), Cfg::kSmem, st, tmA,
                    tmB, tmCin, tmCout, M, N, K, ep, map, err);
}

}  // namespace

cudaError_t launch_gemm_tc(int mode, const CUtensorMap& tmA, const CUtensorMap& tmB,
                           const CUtensorMap& tmCin, const CUtensorMap& tmCout, int M, int N,
                           int K, const EpiArgs& ep, const SlotMap& map, int* err, int n_sms,
                           cudaStream_t st) {
  if (M <= 0) return cudaSuccess;
  if (N % kBN != 0 || K % kBK != 0) return cudaErrorInvalidValue;
  switch (mode) {
    case kEpiQKV:
      return launch_mode<kEpiQKV>(tmA, tmB, tmCin, tmCout, M, N, K, ep, map, err, n_sms, st);
    case kEpiGELU:
      return launch_mode<kEpiGELU>(tmA, tmB, tmCin, tmCout, M, N, K, ep, map, err, n_sms, st);
    case kEpiResid:
      // long K: more ring stages, residual tile in two halves
      if (K >= 1024)
        return launch_mode<kEpiResid, true>(tmA, tmB, tmCin, tmCout, M, N, K, ep, map, err, n_sms, st);
      return launch_mode<kEpiResid>(tmA, tmB, tmCin, tmCout, M, N, K, ep, map, err, n_sms, st);
  }
  return cudaErrorInvalidValue;
}

int gemm_tc_tile_n() { return kBN; }
int gemm_tc_w_box_rows() { return kBN / 2; }
int gemm_tc_tile_k() { return kBK; }
int gemm_tc_tile_m() { return kBM; }

}  // namespace dc
