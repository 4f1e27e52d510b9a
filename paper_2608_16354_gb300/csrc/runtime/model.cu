// Sampler runtime of the DriveCache hot path: model construction (weights to
// HBM, TMA descriptors), and the K-step Euler sampler with the causal cache
// controller (Eq. 1, Eq. 12, Sec. 3.2).
//
// Per step: scenes whose plan says REUSE are checked first (drift sums on
// the device, one readback, fp64 decision on the host); refused reuses turn
// into full evaluations and the scene's suffix is replanned.  Scenes that
// compute are packed into slots 0..n-1 of the activation workspace and run
// the block stack together; reusing scenes run the fused reuse kernel.
// Everything is enqueued on the caller's stream.

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "drivecache.h"
#include "kernels/kernels.h"
#include "plan/planner.h"
#include "runtime/snapshot.h"

using dc::SlotMap;

struct BlockW {
  void *w_qkv, *w_o, *w_1, *w_2;
  float *b_qkv, *b_o, *b_1, *b_2;
  CUtensorMap tm_qkv, tm_o, tm_1, tm_2;
  CUtensorMap tm_1f;  // W1 in 64-row boxes (the fused MLP)
};

struct dc_model {
  dc_model_desc desc{};
  int device = 0, n_sms = 0;
  bool bf16 = false;
  int N = 0, C = 0, d = 0, L = 0, heads = 0, dh = 0, dhp = 0, md = 0, P = 0, Bmax = 0, Kmax = 0;
  int mod_stride = 0;
  size_t elt = 4;
  // weights
  void* wbuf = nullptr;
  float *w_e = nullptr, *b_e = nullptr, *w_t1 = nullptr, *b_t1 = nullptr, *w_t2 = nullptr,
        *b_t2 = nullptr, *w_traj = nullptr, *b_traj = nullptr, *b_ada = nullptr, *w_f = nullptr,
        *b_f = nullptr;
  void *pos = nullptr, *w_ada = nullptr;
  std::vector<BlockW> blk;
  // workspace
  void* ws = nullptr;
  float *u = nullptr, *h = nullptr, *xj = nullptr, *mod = nullptr, *silu_c = nullptr,
        *temb_f = nullptr, *temb_h = nullptr, *temb = nullptr, *pose_f = nullptr, *traj = nullptr,
        *drift_part = nullptr, *drift_out = nullptr, *lat_stage = nullptr,
        *cfg_x = nullptr, *cfg_v = nullptr;  // guidance: latents and velocities of both branches
  void *a = nullptr, *qkv = nullptr, *o = nullptr, *m = nullptr, *r = nullptr;
  double *poses_d = nullptr, *sig_d = nullptr;
  int* err_d = nullptr;
  float* drift_host = nullptr;  // pinned
  // derived tables: W_e^T [C][d] and the Gram tables of the drift sums
  float *w_eT = nullptr, *gram = nullptr, *gp = nullptr, *gs = nullptr;
  // tensor-core interface (bf16 models, C = 16): W_e^T in bf16, its row
  // sums, and per (step, scene) head tables of the call
  bool head_tc = false;
  bool mlp_tc = false;  // fused MLP kernel (bf16, d 384, hidden 1536)
  __nv_bfloat16 *head_wp = nullptr, *cond_xs = nullptr, *we_frag = nullptr;
  CUtensorMap tm_ada, tm_xs;  // adaLN weight and the split activations (bf16 models)
  CUtensorMap tm_cache, tm_headb;  // the cache rows and the head tables' B rows (reuse steps)
  float *wsum = nullptr, *head_tab = nullptr;
  float2* cstat = nullptr;  // per cache row: sum c, sum c^2 of its bf16 values
  CUtensorMap tm_a, tm_oact, tm_m, tm_qkv, tm_u32, tm_h32;
  long long launches = 0;
  // per-kernel profiling (dc_profile)
  struct ProfRec { int cat; cudaEvent_t a, b; double flops, bytes; };
  bool prof_on = false;
  std::vector<cudaEvent_t> ev_pool;
  std::vector<ProfRec> prof_pending;
  double prof_ms[DC_PROF_N] = {}, prof_flops[DC_PROF_N] = {}, prof_bytes[DC_PROF_N] = {};
  long long prof_cnt[DC_PROF_N] = {};
};

namespace {

#define DC_CK(expr)                                                                \
  do {                                                                             \
    cudaError_t e_ = (expr);                                                       \
    if (e_ != cudaSuccess) {                                                       \
      dc::set_error(std::string(#expr) + ": " + cudaGetErrorString(e_));           \
      return DC_ERR_CUDA;                                                          \
    }                                                                              \
  } while (0)

#define DC_TRY(expr)                    \
  do {                                  \
    dc_status s_ = (expr);              \
    if (s_ != DC_OK) return s_;         \
  } while (0)

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

// row groups of the split activations of the tensor-core adaLN product
size_t cond_groups(size_t rows) {
  const size_t g = (size_t)dc::cond_tc_group_rows();
  return (rows + g - 1) / g;
}

cudaEvent_t take_event(dc_model* m) {
  if (!m->ev_pool.empty()) {
    cudaEvent_t e = m->ev_pool.back();
    m->ev_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}

dc_status prof_start(dc_model* m, cudaStream_t st, cudaEvent_t* ev) {
  *ev = nullptr;
  if (!m->prof_on) return DC_OK;
  *ev = take_event(m);
  if (!*ev) { dc::set_error("cudaEventCreate failed"); return DC_ERR_CUDA; }
  DC_CK(cudaEventRecord(*ev, st));
  return DC_OK;
}

dc_status prof_stop(dc_model* m, int cat, cudaStream_t st, cudaEvent_t a, double flops,
                    double bytes) {
  if (!m->prof_on || !a) return DC_OK;
  cudaEvent_t b = take_event(m);
  if (!b) { dc::set_error("cudaEventCreate failed"); return DC_ERR_CUDA; }
  DC_CK(cudaEventRecord(b, st));
  m->prof_pending.push_back({cat, a, b, flops, bytes});
  return DC_OK;
}

// after the stream has been synchronised: fold pending timings into totals
void prof_flush(dc_model* m) {
  for (auto& r : m->prof_pending) {
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, r.a, r.b) == cudaSuccess) {
      m->prof_ms[r.cat] += ms;
      m->prof_flops[r.cat] += r.flops;
      m->prof_bytes[r.cat] += r.bytes;
      m->prof_cnt[r.cat] += 1;
    }
    m->ev_pool.push_back(r.a);
    m->ev_pool.push_back(r.b);
  }
  m->prof_pending.clear();
}

// Launch one kernel (or a fixed pair) with optional per-category timing.
#define DC_LAUNCH(cat, flops, bytes, expr)                           \
  do {                                                               \
    cudaEvent_t ev_ = nullptr;                                       \
    DC_TRY(prof_start(m, st, &ev_));                                 \
    DC_CK(expr);                                                     \
    DC_TRY(prof_stop(m, (cat), st, ev_, (double)(flops), (double)(bytes))); \
  } while (0)

PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    cudaDriverEntryPointQueryResult q;
    void* p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// 2-D row-major tensor [rows][inner] with 128-byte rows per box (64 bf16 or
// 32 fp32 elements), box_rows rows, 128-byte swizzle.
dc_status make_map(CUtensorMap* map, const void* ptr, uint64_t inner, uint64_t rows,
                   uint32_t box_rows, bool fp32 = false) {
  auto enc = get_encode();
  if (!enc) {
    dc::set_error("cuTensorMapEncodeTiled is unavailable");
    return DC_ERR_CUDA;
  }
  const uint32_t esize = fp32 ? 4 : 2;
  cuuint64_t dims[2] = {inner, rows};
  cuuint64_t strides[1] = {inner * esize};
  cuuint32_t box[2] = {128 / esize, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(map, fp32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                   const_cast<void*>(ptr), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                   CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    dc::set_error("cuTensorMapEncodeTiled failed with CUresult " + std::to_string((int)r));
    return DC_ERR_CUDA;
  }
  return DC_OK;
}

uint16_t f2bf_host(float f) {
  uint32_t u;
  std::memcpy(&u, &f, 4);
  if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x7FFFFFu)) return (uint16_t)((u >> 16) | 0x40);
  const uint32_t lsb = (u >> 16) & 1u;
  u += 0x7FFFu + lsb;
  return (uint16_t)(u >> 16);
}

dc_status check_desc(const dc_model_desc* d) {
  if (!d) { dc::set_error("desc is NULL"); return DC_ERR_INVALID_ARG; }
  if (d->dtype != DC_DTYPE_F32 && d->dtype != DC_DTYPE_BF16) {
    dc::set_error("dtype must be DC_DTYPE_F32 or DC_DTYPE_BF16");
    return DC_ERR_INVALID_ARG;
  }
  if (d->n_blocks < 1 || d->d_model < 8 || d->n_heads < 1 || d->mlp_ratio < 1 ||
      d->channels < 1 || d->n_tokens < 1 || d->n_poses < 1 || d->max_batch < 1 ||
      d->max_steps < 1 || d->d_model % d->n_heads != 0) {
    dc::set_error("model shape fields must be positive and d_model divisible by n_heads");
    return DC_ERR_INVALID_ARG;
  }
  // index bounds: every row index (max_batch * n_tokens rows, 32 threads a
  // row in the row kernels) and step index stays far inside int
  if (d->n_blocks > 4096 || d->mlp_ratio > 16 || d->n_tokens > (1 << 22) ||
      (long long)d->max_batch * d->n_tokens > (1LL << 25) || d->n_poses > 65536 ||
      d->max_steps > 100000) {
    dc::set_error("model shape beyond the index bounds (n_blocks <= 4096, mlp_ratio <= 16, "
                  "n_tokens <= 2^22, max_batch * n_tokens <= 2^25, n_poses <= 65536, "
                  "max_steps <= 100000)");
    return DC_ERR_UNSUPPORTED;
  }
  if (d->max_batch > dc::kMaxBatch) {
    dc::set_error("max_batch above " + std::to_string(dc::kMaxBatch));
    return DC_ERR_UNSUPPORTED;
  }
  if (d->channels != 4 && d->channels != 16) {
    dc::set_error("channels must be 4 or 16");
    return DC_ERR_UNSUPPORTED;
  }
  const int dh = d->d_model / d->n_heads;
  if (d->d_model % 4 != 0 || d->d_model > 3072) {
    dc::set_error("d_model must be a multiple of 4 and <= 3072");
    return DC_ERR_UNSUPPORTED;
  }
  if (d->dtype == DC_DTYPE_BF16) {
    if (d->d_model % 192 != 0 || (d->mlp_ratio * d->d_model) % 192 != 0 ||
        !(dh == 64 || dh == 72 || dh == 128)) {
      dc::set_error("bf16 kernels need d_model % 192 == 0 and head_dim in {64, 72, 128}");
      return DC_ERR_UNSUPPORTED;
    }
  } else {
    if (d->d_model % 8 != 0 || !(dh == 8 || dh == 16 || dh == 32 || dh == 64)) {
      dc::set_error("fp32 kernels need d_model % 8 == 0 and head_dim in {8, 16, 32, 64}");
      return DC_ERR_UNSUPPORTED;
    }
  }
  return DC_OK;
}

struct WeightLayout {
  struct T { const char* name; size_t n; bool big; };
  std::vector<T> t;
  size_t total = 0;
};

void weight_layout(const dc_model_desc& d, WeightLayout* w) {
  const size_t D = d.d_model, Cc = d.channels, L = d.n_blocks, N = d.n_tokens,
               M = (size_t)d.mlp_ratio * D, P = d.n_poses;
  auto add = [&](const char* n, size_t cnt, bool big) { w->t.push_back({n, cnt, big}); w->total += cnt; };
  add("w_embed", D * Cc, false); add("b_embed", D, false); add("pos", N * D, true);
  add("w_t1", D * 256, false); add("b_t1", D, false);
  add("w_t2", D * D, false); add("b_t2", D, false);
  add("w_traj", D * 3 * P, false); add("b_traj", D, false);
  add("w_ada", (6 * L + 2) * D * D, true); add("b_ada", (6 * L + 2) * D, false);
  for (size_t l = 0; l < L; ++l) {
    add("w_qkv", 3 * D * D, true); add("b_qkv", 3 * D, false);
    add("w_o", D * D, true); add("b_o", D, false);
    add("w_1", M * D, true); add("b_1", M, false);
    add("w_2", D * M, true); add("b_2", D, false);
  }
  add("w_final", Cc * D, false); add("b_final", Cc, false);
}

template <typename T>
dc_status enqueue_conditioning(dc_model* m, int B, int K, cudaStream_t st) {
  const int d = m->d;
  cudaEvent_t ev = nullptr;
  DC_TRY(prof_start(m, st, &ev));
  DC_CK(dc::launch_temb_features(m->sig_d, K, m->temb_f, st));
  DC_CK(dc::launch_rows_linear<float>(m->temb_f, K, 256, m->w_t1, m->b_t1, d, m->temb_h, 0, st));
  DC_CK(dc::launch_rows_linear<float>(m->temb_h, K, d, m->w_t2, m->b_t2, d, m->temb, 1, st));
  DC_CK(dc::launch_pose_features(m->poses_d, B, m->P, m->pose_f, st));
  DC_CK(dc::launch_rows_linear<float>(m->pose_f, B, 3 * m->P, m->w_traj, m->b_traj, d, m->traj, 0,
                                      st));
  // algorithmic work: the small MLPs' weights read once
  DC_TRY(prof_stop(m, DC_PROF_COND_MLP, st, ev,
                   2.0 * K * (256.0 * d + (double)d * d) + 2.0 * B * 3.0 * m->P * d,
                   4.0 * (256.0 * d + (double)d * d + 3.0 * m->P * d)));
  DC_TRY(prof_start(m, st, &ev));
  if (m->bf16) {
    // the adaLN weight streamed once through the tensor cores
    DC_CK(dc::launch_cond_split(m->temb, m->traj, K, B, d, m->cond_xs, st));
    DC_CK(dc::launch_cond_gemm_tc(m->tm_ada, m->tm_xs, K * B, m->mod_stride, d, m->b_ada, m->mod,
                                  m->err_d, m->n_sms, st));
  } else {
    DC_CK(dc::launch_cond_combine(m->temb, m->traj, K, B, d, m->silu_c, st));
    DC_CK(dc::launch_rows_linear<T>(m->silu_c, K * B, d, static_cast<const T*>(m->w_ada), m->b_ada,
                                    m->mod_stride, m->mod, 0, st));
  }
  // algorithmic bytes: the adaLN weight table read once + the table written
  DC_TRY(prof_stop(m, DC_PROF_CONDITION, st, ev, 2.0 * K * B * d * m->mod_stride,
                   (double)m->mod_stride * d * m->elt + 4.0 * K * B * m->mod_stride));
  m->launches += 7;
  if (m->head_tc) {
    DC_LAUNCH(DC_PROF_COND_MLP, 2.0 * K * B * 18.0 * 16.0 * d, 4.0 * K * B * 64.0 * d,
              dc::launch_head_tables(m->mod, K * B, m->mod_stride, 6 * m->L * d, d, m->w_f, m->b_f,
                                     m->w_eT, m->head_wp, m->head_tab, st));
    m->launches += 1;
  }
  return DC_OK;
}

// This step's head tables (tensor-core interface): items (k - 1) * Bi + scene.
const __nv_bfloat16* head_wp_k(const dc_model* m, int k, int Bi) {
  return m->head_wp + (size_t)(k - 1) * Bi * dc::head_b_rows() * m->d;
}
const float* head_tab_k(const dc_model* m, int k, int Bi) {
  return m->head_tab + (size_t)(k - 1) * Bi * dc::head_table_floats();
}

template <typename T>
dc_status enqueue_compute(dc_model* m, float* lat, const float* mod_k, const SlotMap& map,
                          float dsig, int k, int Bi, cudaStream_t st, float* vout = nullptr) {
  const int N = m->N, d = m->d, nc = map.n, M = nc * N;
  if (nc == 0) return DC_OK;
  T* a = static_cast<T*>(m->a);
  T* qkv = static_cast<T*>(m->qkv);
  T* o = static_cast<T*>(m->o);
  T* mm = static_cast<T*>(m->m);
  const double Md = (double)M * d, E = (double)m->elt;
  DC_LAUNCH(DC_PROF_EMBED, 2.0 * M * d * m->C, 4.0 * M * m->C + 4.0 * Md + (double)N * d * E,
            dc::launch_embed<T>(lat, m->w_eT, m->b_e, static_cast<const T*>(m->pos), map, N, m->C,
                                d, m->u, st));
  m->launches += 1;
  const double ln_bytes = 4.0 * Md + E * Md;
  const double attn_flops = 4.0 * nc * (double)N * N * d;
  const double attn_bytes = E * (3.0 * Md + Md);
  dc::EpiArgs ep{};
  ep.M = M;
  ep.n_tok = N;
  ep.mod = mod_k;
  ep.mod_stride = m->mod_stride;
  ep.d = d;
  ep.heads = m->heads;
  ep.dh = m->dh;
  ep.dhp = m->dhp;
  ep.nslots = nc;
  for (int l = 0; l < m->L; ++l) {
    const BlockW& w = m->blk[l];
    const int base = l * 6 * d;
    // block 0 reads the block-stack input u directly (h = u is never copied)
    const float* h_in = l == 0 ? m->u : m->h;
    DC_LAUNCH(DC_PROF_LN, 0.0, ln_bytes,
              dc::launch_ln_mod<T>(h_in, M, N, d, mod_k, m->mod_stride, base + 0 * d, base + 1 * d,
                                   map, a, st));
    dc::EpiArgs e1 = ep;
    e1.N = 3 * d; e1.bias = w.b_qkv; e1.out = qkv;
    // q/k/v tiles go out by TMA through the attention's map when dh = 64 or 128
    // head blocks of whole 64-column swizzle atoms go out by TMA
    e1.qkv_tma = dc::attention_tc_supported(m->dh) && m->dh % 64 == 0 ? 1 : 0;
    dc::EpiArgs e2 = ep;
    e2.N = d; e2.bias = w.b_o; e2.h = m->h; e2.h_in = h_in; e2.gate_off = base + 2 * d;
    dc::EpiArgs e3 = ep;
    e3.N = m->md; e3.bias = w.b_1; e3.out = mm;
    dc::EpiArgs e4 = ep;
    e4.N = d; e4.bias = w.b_2; e4.h = m->h; e4.h_in = m->h; e4.gate_off = base + 5 * d;
    const double f_qkv = 2.0 * M * 3.0 * d * d, f_o = 2.0 * M * (double)d * d,
                 f_mlp = 2.0 * M * (double)m->md * d;
    const double b_qkv = E * (Md + 3.0 * d * d + 3.0 * Md), b_o = E * (Md + (double)d * d) + 8.0 * Md,
                 b_1 = E * (Md + (double)m->md * d + (double)M * m->md),
                 b_2 = E * ((double)M * m->md + (double)m->md * d) + 8.0 * Md;
    if constexpr (sizeof(T) == 2) {
      DC_LAUNCH(DC_PROF_GEMM_QKV, f_qkv, b_qkv,
                dc::launch_gemm_tc(dc::kEpiQKV, m->tm_a, w.tm_qkv, m->tm_a, m->tm_qkv, M, 3 * d, d,
                                   e1, map, m->err_d, m->n_sms, st));
      if (dc::attention_tc_supported(m->dh)) {
        DC_LAUNCH(DC_PROF_ATTENTION, attn_flops, attn_bytes,
                  dc::launch_attention_tc(m->tm_qkv, nc, m->heads, N, m->dh,
                                          reinterpret_cast<__nv_bfloat16*>(o), m->err_d, st));
      } else {
        DC_LAUNCH(DC_PROF_ATTENTION, attn_flops, attn_bytes,
                  dc::launch_attention_bf16(reinterpret_cast<const __nv_bfloat16*>(qkv), nc,
                                            m->heads, N, m->dh, m->dhp,
                                            reinterpret_cast<__nv_bfloat16*>(o), st));
      }
      DC_LAUNCH(DC_PROF_GEMM_OUT, f_o, b_o,
                dc::launch_gemm_tc(dc::kEpiResid, m->tm_oact, w.tm_o, l == 0 ? m->tm_u32 : m->tm_h32,
                                   m->tm_h32, M, d, d, e2, map, m->err_d, m->n_sms, st));
      DC_LAUNCH(DC_PROF_LN, 0.0, ln_bytes,
                dc::launch_ln_mod<T>(m->h, M, N, d, mod_k, m->mod_stride, base + 3 * d,
                                     base + 4 * d, map, a, st));
      if (m->mlp_tc) {
        // both projections in one kernel (the hidden activation stays on
        // chip): counted under MLP-up with the flops of both
        DC_LAUNCH(DC_PROF_GEMM_MLP1, 2.0 * f_mlp,
                  E * (Md + 2.0 * m->md * d) + 8.0 * Md,
                  dc::launch_mlp_tc(m->tm_a, w.tm_1f, w.tm_2, m->tm_h32, M, w.b_1, w.b_2, mod_k,
                                    m->mod_stride, base + 5 * d, N, map, m->err_d, m->n_sms, st));
        m->launches -= 1;  // one launch where the block counts two
      } else {
        DC_LAUNCH(DC_PROF_GEMM_MLP1, f_mlp, b_1,
                  dc::launch_gemm_tc(dc::kEpiGELU, m->tm_a, w.tm_1, m->tm_m, m->tm_m, M, m->md, d,
                                     e3, map, m->err_d, m->n_sms, st));
        DC_LAUNCH(DC_PROF_GEMM_MLP2, f_mlp, b_2,
                  dc::launch_gemm_tc(dc::kEpiResid, m->tm_m, w.tm_2, m->tm_h32, m->tm_h32, M, d,
                                     m->md, e4, map, m->err_d, m->n_sms, st));
      }
    } else {
      DC_LAUNCH(DC_PROF_GEMM_QKV, f_qkv, b_qkv,
                dc::launch_gemm_f32(dc::kEpiQKV, reinterpret_cast<const float*>(a),
                                    static_cast<const float*>(w.w_qkv), M, 3 * d, d, e1, map, st));
      DC_LAUNCH(DC_PROF_ATTENTION, attn_flops, attn_bytes,
                dc::launch_attention_f32(reinterpret_cast<const float*>(qkv), nc, m->heads, N,
                                         m->dh, m->dhp, reinterpret_cast<float*>(o), st));
      DC_LAUNCH(DC_PROF_GEMM_OUT, f_o, b_o,
                dc::launch_gemm_f32(dc::kEpiResid, reinterpret_cast<const float*>(o),
                                    static_cast<const float*>(w.w_o), M, d, d, e2, map, st));
      DC_LAUNCH(DC_PROF_LN, 0.0, ln_bytes,
                dc::launch_ln_mod<T>(m->h, M, N, d, mod_k, m->mod_stride, base + 3 * d,
                                     base + 4 * d, map, a, st));
      DC_LAUNCH(DC_PROF_GEMM_MLP1, f_mlp, b_1,
                dc::launch_gemm_f32(dc::kEpiGELU, reinterpret_cast<const float*>(a),
                                    static_cast<const float*>(w.w_1), M, m->md, d, e3, map, st));
      DC_LAUNCH(DC_PROF_GEMM_MLP2, f_mlp, b_2,
                dc::launch_gemm_f32(dc::kEpiResid, reinterpret_cast<const float*>(mm),
                                    static_cast<const float*>(w.w_2), M, d, m->md, e4, map, st));
    }
    m->launches += 7;
  }
  // algorithmic bytes: h_L read, the cache row written (with its two sums on
  // the tensor-core path), x read, x and x_j written
  if (m->head_tc && sizeof(T) == 2) {
    DC_LAUNCH(DC_PROF_FINAL, 4.0 * M * d * m->C, 4.0 * Md + E * Md + 12.0 * M * m->C + 8.0 * M,
              dc::launch_head_compute(m->h, lat, m->xj, reinterpret_cast<__nv_bfloat16*>(m->r),
                                      m->cstat, map, N, d, m->we_frag, head_wp_k(m, k, Bi),
                                      head_tab_k(m, k, Bi), dsig, st, vout));
  } else {
    DC_LAUNCH(DC_PROF_FINAL, 4.0 * M * d * m->C, 4.0 * Md + E * Md + 12.0 * M * m->C,
              dc::launch_final_compute<T>(m->h, m->w_eT, lat, m->xj, static_cast<T*>(m->r), map, N,
                                          m->C, d, mod_k, m->mod_stride, 6 * m->L * d, m->w_f,
                                          m->b_f, dsig, st, vout));
  }
  m->launches += 1;
  return DC_OK;
}

template <typename T>
dc_status enqueue_reuse(dc_model* m, float* lat, const float* mod_k, const SlotMap& map, float dsig,
                        int k, int Bi, cudaStream_t st, float* vout = nullptr) {
  if (map.n == 0) return DC_OK;
  const double M = (double)map.n * m->N;
  // algorithmic bytes of a reuse scene-step: the cached row (N d elements) +
  // x_k read, x_{k+1} written and x_j read by the drift check (3 N C fp32),
  // and on the tensor-core path the row's two stored sums
  if (m->head_tc && sizeof(T) == 2) {
    DC_LAUNCH(DC_PROF_REUSE, 2.0 * M * m->d * 3 * m->C,
              M * ((double)m->d * m->elt + 12.0 * m->C + 8.0),
              dc::launch_head_reuse_tc(m->tm_cache, m->tm_headb, lat, m->cstat, map, m->N, m->d,
                                       (k - 1) * Bi * dc::head_b_rows(), head_tab_k(m, k, Bi),
                                       m->wsum, m->gram, dsig, m->err_d, m->n_sms, st, vout));
  } else {
    DC_LAUNCH(DC_PROF_REUSE, 4.0 * M * m->d * m->C, M * ((double)m->d * m->elt + 12.0 * m->C),
              dc::launch_final_reuse<T>(lat, static_cast<const T*>(m->r), m->w_eT, map, m->N, m->C,
                                        m->d, mod_k, m->mod_stride, 6 * m->L * m->d, m->w_f, m->b_f,
                                        dsig, st, vout));
  }
  m->launches += 1;
  return DC_OK;
}

template <typename T>
dc_status enqueue_drift(dc_model* m, const dc::DriftItems& it, float* out, cudaStream_t st) {
  // algorithmic bytes: x_now and x_ref of every item (2 N C fp32)
  DC_LAUNCH(DC_PROF_DRIFT, 4.0 * it.n * m->N * m->C * m->C, 8.0 * it.n * m->N * m->C,
            dc::launch_drift(it, m->gram, m->gp, m->gs, m->N, m->C, m->drift_part, out, st));
  m->launches += 2;
  return DC_OK;
}

dc_status check_device_error(dc_model* m, cudaStream_t st) {
  int err = 0;
  DC_CK(cudaMemcpyAsync(&err, m->err_d, sizeof(int), cudaMemcpyDeviceToHost, st));
  DC_CK(cudaStreamSynchronize(st));
  prof_flush(m);
  if (err != 0) {
    dc::set_error("a bounded device wait gave up (code " + std::to_string(err) + ")");
    cudaMemsetAsync(m->err_d, 0, sizeof(int), st);
    return DC_ERR_DEVICE_TIMEOUT;
  }
  return DC_OK;
}

struct SceneState {
  double C = 0.0;
  int j = 0, age = 0;
};

// The call's record, always kept (the caller's dc_run_stats and snapshots
// are filled from it).
struct Record {
  std::vector<unsigned char> planned, executed, checked;  // [B][K+1]
  std::vector<double> d_obs, d_bar;                       // [B][K+1]
  std::vector<int> n_compute, n_reuse, n_veto, n_replan, supported;
  std::vector<double> D;
  long long backbone_calls = 0;
  void init(int B, size_t W) {
    planned.assign((size_t)B * W, 0);
    executed.assign((size_t)B * W, 0);
    checked.assign((size_t)B * W, 0);
    d_obs.assign((size_t)B * W, NAN);
    d_bar.assign((size_t)B * W, NAN);
    n_compute.assign(B, 0); n_reuse.assign(B, 0); n_veto.assign(B, 0); n_replan.assign(B, 0);
    supported.assign(B, 0);
    D.assign(B, 0.0);
  }
};

// Snapshot requests of one call: run steps k0+1 .. k_stop, resuming from
// `in` (validated, digest checked) when non-null, saving into `out`.
struct SnapIO {
  int k_stop = 0;
  const uint8_t* in = nullptr;
  uint8_t* out = nullptr;
  uint64_t digest = 0;
};

// The sampler.  trace (optional, device [K][B][N][C]) receives x_k before
// step k; r_trace (optional, device [K][N][d] of the cache type) receives
// scene 0's cached r after step k.
template <typename T>
dc_status run_sampler(dc_model* m, float* lat, const dc_cond* cond, const dc_sched* sc,
                      cudaStream_t st, dc_run_stats* stats, float* trace,
                      void* r_trace = nullptr, const SnapIO* io = nullptr) {
  const int B = cond->B, K = sc->K, N = m->N, C = m->C;
  // guidance: every scene s runs two branches -- internal scene s with its
  // trajectory and internal scene B + s with the null trajectory -- each with
  // its own cache; the plan and the drift check stay per scene
  const bool cfg = sc->cfg_scale != 0.0;
  const int Bi = cfg ? 2 * B : B;
  const dc_anchor_responses* anc = sc->anchors;
  const double eps = anc ? anc->eps : 1e-6;
  const int W = K + 1;
  const int k_stop = io ? io->k_stop : K;
  const dc::SnapLayout lay = dc::snap_layout(B, K, cfg ? 1 : 0, N, m->d, C, m->elt);
  std::vector<unsigned char> acts((size_t)B * W, dc::kCompute);
  std::vector<dc::SceneTables> tabs(B);
  std::vector<SceneState> state(B);
  Record rec;
  rec.init(B, W);
  const bool forced = sc->forced != nullptr;
  for (int s = 0; s < B; ++s) {
    unsigned char* a = &acts[(size_t)s * W];
    a[0] = 0;
    if (forced) {
      for (int k = 1; k <= K; ++k) a[k] = sc->forced[(size_t)s * W + k];
      a[1] = dc::kCompute;
      continue;
    }
    // the shuffled-trajectory ablation plans scene s from scene s+1's poses
    const dc_trajectory& pt = cond->traj[anc->variant == DC_VAR_SHUFFLED ? (s + 1) % B : s];
    double L, Th, D, cost;
    int n_reuse;
    dc::motion_stats(pt.poses, pt.n_poses, &L, &Th);
    rec.supported[s] = dc::plan_scene(L, Th, *anc, sc->tau, a, &n_reuse, &cost, &D, &tabs[s]);
    rec.D[s] = D;
  }
  rec.planned = acts;
  // the fixed-interval baseline runs its pattern with no charge and no checks
  const bool unchecked = !forced && anc->variant == DC_VAR_FIXED_INTERVAL;

  int k0 = 0;
  if (io && io->in) {
    // resume: the controller state and the record come from the snapshot
    // (the scene tables above are a pure function of the same inputs)
    const uint8_t* in = io->in;
    dc::SnapHeader h;
    std::memcpy(&h, in, sizeof(h));
    k0 = h.k_done;
    rec.backbone_calls = h.backbone_calls;
    for (int s = 0; s < B; ++s) {
      dc::SnapScene r;
      std::memcpy(&r, in + lay.scene + (size_t)s * sizeof(r), sizeof(r));
      state[s].C = r.charge;
      state[s].j = r.j;
      state[s].age = r.age;
      rec.D[s] = r.D;
      rec.supported[s] = r.supported;
      rec.n_compute[s] = r.n_compute;
      rec.n_reuse[s] = r.n_reuse;
      rec.n_veto[s] = r.n_veto;
      rec.n_replan[s] = r.n_replan;
    }
    const size_t bw = (size_t)B * W;
    std::memcpy(rec.planned.data(), in + lay.planned, bw);
    std::memcpy(acts.data(), in + lay.plan, bw);
    std::memcpy(rec.executed.data(), in + lay.executed, bw);
    std::memcpy(rec.checked.data(), in + lay.checked, bw);
    std::memcpy(rec.d_obs.data(), in + lay.d_obs, bw * sizeof(double));
    std::memcpy(rec.d_bar.data(), in + lay.d_bar, bw * sizeof(double));
    const size_t xb = (size_t)B * N * C * sizeof(float);
    DC_CK(cudaMemcpyAsync(lat, in + lay.lat, xb, cudaMemcpyHostToDevice, st));
    DC_CK(cudaMemcpyAsync(m->xj, in + lay.xj, xb, cudaMemcpyHostToDevice, st));
    DC_CK(cudaMemcpyAsync(m->r, in + lay.r, (size_t)Bi * N * m->d * m->elt,
                          cudaMemcpyHostToDevice, st));
    if (lay.cs_bytes)
      DC_CK(cudaMemcpyAsync(m->cstat, in + lay.cs, lay.cs_bytes, cudaMemcpyHostToDevice, st));
  }
  const long long launches0 = m->launches;

  // inputs of the conditioning: poses (the null trajectory of the second
  // branch is all zeros, so its pose features vanish) and sigmas
  std::vector<double> poses((size_t)Bi * m->P * 3, 0.0);
  for (int s = 0; s < B; ++s)
    for (int t = 0; t < m->P; ++t) {
      const dc_pose& p = cond->traj[s].poses[t];
      double* q = &poses[((size_t)s * m->P + t) * 3];
      q[0] = p.x; q[1] = p.y; q[2] = p.psi;
    }
  DC_CK(cudaMemcpyAsync(m->poses_d, poses.data(), poses.size() * sizeof(double),
                        cudaMemcpyHostToDevice, st));
  DC_CK(cudaMemcpyAsync(m->sig_d, sc->sigmas, (size_t)(K + 1) * sizeof(double),
                        cudaMemcpyHostToDevice, st));
  DC_TRY(enqueue_conditioning<T>(m, Bi, K, st));

  std::vector<unsigned char> reuse_now(B);
  for (int k = k0 + 1; k <= k_stop; ++k) {
    const float dsig = (float)(sc->sigmas[k] - sc->sigmas[k - 1]);
    const float* mod_k = m->mod + (size_t)(k - 1) * Bi * m->mod_stride;
    if (trace) {
      DC_CK(cudaMemcpyAsync(trace + (size_t)(k - 1) * B * N * C, lat, (size_t)B * N * C * 4,
                            cudaMemcpyDeviceToDevice, st));
    }
    std::vector<int> chk;
    for (int s = 0; s < B; ++s) {
      reuse_now[s] = 0;
      if (k == 1 || acts[(size_t)s * W + k] != dc::kReuse) continue;
      if (forced || !sc->veto || unchecked) {
        reuse_now[s] = 1;
        if (!forced && !unchecked) state[s].C = state[s].C + tabs[s].at_c(state[s].j, state[s].age + 1);
      } else {
        chk.push_back(s);
      }
    }
    if (!chk.empty()) {
      dc::DriftItems it{};
      it.n = (int)chk.size();
      for (int i = 0; i < it.n; ++i) {
        it.now[i] = lat + (size_t)chk[i] * N * C;
        it.ref[i] = m->xj + (size_t)chk[i] * N * C;
      }
      DC_TRY(enqueue_drift<T>(m, it, m->drift_out, st));
      DC_CK(cudaMemcpyAsync(m->drift_host, m->drift_out, (size_t)2 * it.n * sizeof(float),
                            cudaMemcpyDeviceToHost, st));
      DC_TRY(check_device_error(m, st));  // synchronises the stream
      for (int i = 0; i < it.n; ++i) {
        const int s = chk[i];
        const double Sd = m->drift_host[2 * i], Su = m->drift_host[2 * i + 1];
        if (!std::isfinite(Sd) || !std::isfinite(Su)) {
          dc::set_error("non-finite drift statistic for scene " + std::to_string(s) + " at step " +
                        std::to_string(k));
          return DC_ERR_NONFINITE;
        }
        SceneState& S = state[s];
        const int h = S.age + 1, j = S.j;
        const double d_obs = std::sqrt(Sd) / (std::sqrt(Su) + eps);
        const double dbar = tabs[s].at_d(j, h);
        const double c = tabs[s].at_c(j, h);
        const bool ok = d_obs <= dbar + eps && S.C + c <= sc->tau;
        rec.d_obs[(size_t)s * W + k] = d_obs;
        rec.d_bar[(size_t)s * W + k] = dbar;
        rec.checked[(size_t)s * W + k] = ok ? 1 : 2;
        if (ok) {
          reuse_now[s] = 1;
          S.C = S.C + c;
        } else {
          rec.n_veto[s]++;
          if (anc->variant != DC_VAR_FIXED_PLACEMENT) {  // the fixed pattern is kept
            rec.n_replan[s]++;
            double cost;
            dc::plan_suffix(tabs[s], anc->legal, k, sc->tau - S.C, &acts[(size_t)s * W], &cost);
          }
        }
      }
    }
    SlotMap cm{}, rm{};
    for (int s = 0; s < B; ++s) {
      SlotMap& mp = reuse_now[s] ? rm : cm;
      mp.scene[mp.n++] = s;
      if (cfg) mp.scene[mp.n++] = B + s;
    }
    if (cfg) {
      // both branches see x_k; their velocities are combined into x_{k+1}
      const size_t xb = (size_t)B * N * C * 4;
      DC_CK(cudaMemcpyAsync(m->cfg_x, lat, xb, cudaMemcpyDeviceToDevice, st));
      DC_CK(cudaMemcpyAsync(m->cfg_x + (size_t)B * N * C, lat, xb, cudaMemcpyDeviceToDevice, st));
      DC_TRY(enqueue_compute<T>(m, m->cfg_x, mod_k, cm, dsig, k, Bi, st, m->cfg_v));
      DC_TRY(enqueue_reuse<T>(m, m->cfg_x, mod_k, rm, dsig, k, Bi, st, m->cfg_v));
      DC_CK(dc::launch_cfg_combine(lat, m->cfg_v, B, (size_t)N * C, (float)sc->cfg_scale, dsig,
                                   st));
      m->launches += 1;
    } else {
      DC_TRY(enqueue_compute<T>(m, lat, mod_k, cm, dsig, k, Bi, st));
      DC_TRY(enqueue_reuse<T>(m, lat, mod_k, rm, dsig, k, Bi, st));
    }
    if (r_trace) {
      const size_t rb = (size_t)N * m->d * m->elt;
      DC_CK(cudaMemcpyAsync(static_cast<uint8_t*>(r_trace) + (size_t)(k - 1) * rb, m->r, rb,
                            cudaMemcpyDeviceToDevice, st));
    }
    for (int s = 0; s < B; ++s) {
      if (reuse_now[s]) {
        state[s].age += 1;
      } else {
        state[s].j = k;
        state[s].age = 0;
      }
      rec.executed[(size_t)s * W + k] = reuse_now[s] ? dc::kReuse : dc::kCompute;
      if (reuse_now[s]) rec.n_reuse[s]++;
      else rec.n_compute[s]++;
    }
    rec.backbone_calls += cm.n;
  }
  if (io && io->out) {
    // save: host state now, device payload after the stream drains
    uint8_t* out = io->out;
    dc::SnapHeader h{};
    std::memcpy(h.magic, dc::kSnapMagic, sizeof(h.magic));
    h.version = dc::kSnapVersion;
    h.B = B; h.K = K; h.cfg = cfg ? 1 : 0; h.k_done = k_stop;
    h.dtype = m->bf16 ? DC_DTYPE_BF16 : DC_DTYPE_F32;
    h.N = N; h.d = m->d; h.C = C; h.elt = (uint32_t)m->elt;
    h.digest = io->digest;
    h.bytes = lay.total;
    h.backbone_calls = rec.backbone_calls;
    std::memset(out, 0, lay.lat);
    std::memcpy(out, &h, sizeof(h));
    for (int s = 0; s < B; ++s) {
      dc::SnapScene r{};
      r.charge = state[s].C; r.D = rec.D[s];
      r.j = state[s].j; r.age = state[s].age; r.supported = rec.supported[s];
      r.n_compute = rec.n_compute[s]; r.n_reuse = rec.n_reuse[s];
      r.n_veto = rec.n_veto[s]; r.n_replan = rec.n_replan[s];
      std::memcpy(out + lay.scene + (size_t)s * sizeof(r), &r, sizeof(r));
    }
    const size_t bw = (size_t)B * W;
    std::memcpy(out + lay.planned, rec.planned.data(), bw);
    std::memcpy(out + lay.plan, acts.data(), bw);
    std::memcpy(out + lay.executed, rec.executed.data(), bw);
    std::memcpy(out + lay.checked, rec.checked.data(), bw);
    std::memcpy(out + lay.d_obs, rec.d_obs.data(), bw * sizeof(double));
    std::memcpy(out + lay.d_bar, rec.d_bar.data(), bw * sizeof(double));
    const size_t xb = (size_t)B * N * C * sizeof(float);
    std::memset(out + lay.lat + 2 * xb, 0, lay.r - (lay.lat + 2 * xb));
    DC_CK(cudaMemcpyAsync(out + lay.lat, lat, xb, cudaMemcpyDeviceToHost, st));
    DC_CK(cudaMemcpyAsync(out + lay.xj, m->xj, xb, cudaMemcpyDeviceToHost, st));
    DC_CK(cudaMemcpyAsync(out + lay.r, m->r, (size_t)Bi * N * m->d * m->elt,
                          cudaMemcpyDeviceToHost, st));
    if (lay.cs_bytes) {
      const size_t r_end = lay.r + (size_t)Bi * N * m->d * m->elt;
      std::memset(out + r_end, 0, lay.cs - r_end);
      DC_CK(cudaMemcpyAsync(out + lay.cs, m->cstat, lay.cs_bytes, cudaMemcpyDeviceToHost, st));
    }
  }
  DC_TRY(check_device_error(m, st));  // synchronises the stream
  if (stats) {
    const size_t bw = (size_t)B * W;
    if (stats->planned) std::memcpy(stats->planned, rec.planned.data(), bw);
    if (stats->executed) std::memcpy(stats->executed, rec.executed.data(), bw);
    if (stats->checked) std::memcpy(stats->checked, rec.checked.data(), bw);
    if (stats->d_obs) std::memcpy(stats->d_obs, rec.d_obs.data(), bw * sizeof(double));
    if (stats->d_bar) std::memcpy(stats->d_bar, rec.d_bar.data(), bw * sizeof(double));
    for (int s = 0; s < B; ++s) {
      if (stats->n_compute) stats->n_compute[s] = rec.n_compute[s];
      if (stats->n_reuse) stats->n_reuse[s] = rec.n_reuse[s];
      if (stats->n_veto) stats->n_veto[s] = rec.n_veto[s];
      if (stats->n_replan) stats->n_replan[s] = rec.n_replan[s];
      if (stats->supported) stats->supported[s] = rec.supported[s];
      if (stats->D) stats->D[s] = rec.D[s];
      if (stats->charge) stats->charge[s] = state[s].C;
    }
    stats->backbone_calls = rec.backbone_calls;
    stats->launches = m->launches - launches0;
  }
  return DC_OK;
}

dc_status check_call(dc_model* m, const dc_cond* cond, const dc_sched* sc) {
  if (!m || !cond || !sc) { dc::set_error("NULL model/cond/sched"); return DC_ERR_INVALID_ARG; }
  if (cond->B < 1 || cond->B > m->Bmax || !cond->traj) {
    dc::set_error("cond->B must be in [1, max_batch] with non-NULL trajectories");
    return DC_ERR_INVALID_ARG;
  }
  if (sc->K < 1 || sc->K > m->Kmax || !sc->sigmas) {
    dc::set_error("sched->K must be in [1, max_steps] with non-NULL sigmas");
    return DC_ERR_INVALID_ARG;
  }
  if (!std::isfinite(sc->cfg_scale) || (sc->cfg_scale != 0.0 && 2 * cond->B > m->Bmax)) {
    dc::set_error("cfg_scale must be finite, and guidance needs 2 B <= max_batch");
    return DC_ERR_INVALID_ARG;
  }
  for (int k = 0; k <= sc->K; ++k)
    if (!std::isfinite(sc->sigmas[k])) {
      dc::set_error("non-finite sigma");
      return DC_ERR_INVALID_ARG;
    }
  for (int s = 0; s < cond->B; ++s) {
    const dc_trajectory& t = cond->traj[s];
    if (!t.poses || t.n_poses != m->P) {
      dc::set_error("trajectory " + std::to_string(s) + " must have n_poses = " + std::to_string(m->P));
      return DC_ERR_INVALID_ARG;
    }
    for (int i = 0; i < t.n_poses; ++i)
      if (!std::isfinite(t.poses[i].x) || !std::isfinite(t.poses[i].y) ||
          !std::isfinite(t.poses[i].psi)) {
        dc::set_error("non-finite pose");
        return DC_ERR_INVALID_ARG;
      }
  }
  if (sc->forced) {
    for (int s = 0; s < cond->B; ++s)
      for (int k = 1; k <= sc->K; ++k) {
        const unsigned char a = sc->forced[(size_t)s * (sc->K + 1) + k];
        if (a != dc::kCompute && a != dc::kReuse) {
          dc::set_error("forced actions must be DC_ACT_COMPUTE or DC_ACT_REUSE");
          return DC_ERR_INVALID_ARG;
        }
      }
  } else {
    dc_status s = dc::check_anchors(sc->anchors);
    if (s != DC_OK) return s;
    if (sc->anchors->K != sc->K || std::isnan(sc->tau)) {
      dc::set_error("anchors->K must equal sched->K and tau must not be NaN");
      return DC_ERR_INVALID_ARG;
    }
    if ((s = dc::check_reuse_count(*sc->anchors, sc->tau)) != DC_OK) return s;
  }
  return DC_OK;
}

// ------------------------------------------- joint run responses (Eq. 6-7)

// Device buffers of one dc_anchor_response call, freed on every exit.
struct DevBufs {
  std::vector<void*> p;
  ~DevBufs() {
    for (void* q : p) cudaFree(q);
  }
  template <typename X>
  bool get(X** out, size_t bytes) {
    void* q = nullptr;
    if (cudaMalloc(&q, bytes ? bytes : 16) != cudaSuccess) return false;
    p.push_back(q);
    *out = static_cast<X*>(q);
    return true;
  }
};

template <typename T>
struct ResponseWork {
  int N, C, d, L, md, heads, dh;
  // trace and interface outputs
  float *xs, *vbar, *e, *vtmp;
  T* rs;
  // primal activations at one trace point
  float *hin, *qkv, *h1, *z, *hcur, *hL, *abuf, *obuf, *mbuf;
  // tangents
  float *th, *ta, *tqkv, *tout, *tm, *tv;
};

// v = H_t(x, r): u(x) + r through the step's final modulated LayerNorm and
// head (the reuse interface of Eq. 1).
template <typename T>
dc_status interface_f32(dc_model* m, ResponseWork<T>& w, const float* x, const T* r,
                        const float* mod, float* v, cudaStream_t st) {
  const size_t Nd = (size_t)w.N * w.d;
  const float* fsh = mod + (size_t)6 * w.L * w.d;
  // the cache row c = r + b_e + pos: u + r = x W_e^T + c
  DC_LAUNCH(DC_PROF_JVP_OTHER, 0.0, 0.0,
              dc::launch_embed_f32<T>(x, m->w_eT, nullptr, static_cast<const T*>(nullptr), w.N, w.N,
                                      w.C, w.d, w.hcur, st));
  DC_LAUNCH(DC_PROF_JVP_OTHER, 0.0, 0.0,
              dc::launch_add_cache<T>(w.hcur, r, w.hcur, Nd, st));
  DC_LAUNCH(DC_PROF_JVP_OTHER, 0.0, 0.0,
              dc::launch_ln_mod_f32(w.hcur, w.N, w.d, fsh, fsh + w.d, w.abuf, st));
  dc::JEpi ep{};
  ep.mode = dc::kJStore; ep.bias = m->b_f; ep.out = v;
  DC_LAUNCH(DC_PROF_JVP_GEMM, 2.0 * (w.N) * (w.C) * (w.d), 0.0,
              dc::launch_gemm_f32w<float>(w.abuf, m->w_f, w.N, w.C, w.d, ep, st));
  return DC_OK;
}

// Full evaluation at one trace point, keeping what the tangents need.
template <typename T>
dc_status primal_f32(dc_model* m, ResponseWork<T>& w, const float* x, const float* mod,
                     cudaStream_t st) {
  const int N = w.N, d = w.d, md = w.md;
  const size_t Nd = (size_t)N * d;
  DC_LAUNCH(DC_PROF_JVP_OTHER, 0.0, 0.0,
            dc::launch_embed_f32<T>(x, m->w_eT, m->b_e, static_cast<const T*>(m->pos), N, N, w.C,
                                    d, w.hcur, st));
  for (int l = 0; l < w.L; ++l) {
    const BlockW& b = m->blk[l];
    const float* mb = mod + (size_t)l * 6 * d;
    float* qkv = w.qkv + (size_t)l * N * 3 * d;
    DC_CK(cudaMemcpyAsync(w.hin + l * Nd, w.hcur, Nd * 4, cudaMemcpyDeviceToDevice, st));
    DC_LAUNCH(DC_PROF_JVP_OTHER, 0.0, 0.0,
              dc::launch_ln_mod_f32(w.hcur, N, d, mb, mb + d, w.abuf, st));
    dc::JEpi e1{};
    e1.mode = dc::kJStore; e1.bias = b.b_qkv; e1.out = qkv;
    DC_LAUNCH(DC_PROF_JVP_GEMM, 2.0 * (N) * (3 * d) * (d), 0.0,
              dc::launch_gemm_f32w<T>(w.abuf, static_cast<const T*>(b.w_qkv), N, 3 * d, d, e1, st));
    // primal attention: 4 N^2 dh flops per head (scores and weighted sum)
    DC_LAUNCH(DC_PROF_JVP_ATTENTION, 4.0 * w.heads * (double)N * N * w.dh, 0.0,
              dc::launch_attention_f32_jvp(qkv, nullptr, N, d, w.heads, w.dh, 1, w.obuf, nullptr,
                                           st));
    dc::JEpi e2{};
    e2.mode = dc::kJGatedAdd; e2.bias = b.b_o; e2.gate = mb + 2 * d; e2.base = w.hcur; e2.out = w.hcur;
    DC_LAUNCH(DC_PROF_JVP_GEMM, 2.0 * (N) * (d) * (d), 0.0,
              dc::launch_gemm_f32w<T>(w.obuf, static_cast<const T*>(b.w_o), N, d, d, e2, st));
    DC_CK(cudaMemcpyAsync(w.h1 + l * Nd, w.hcur, Nd * 4, cudaMemcpyDeviceToDevice, st));
    DC_LAUNCH(DC_PROF_JVP_OTHER, 0.0, 0.0,
              dc::launch_ln_mod_f32(w.hcur, N, d, mb + 3 * d, mb + 4 * d, w.abuf, st));
    dc::JEpi e3{};
    e3.mode = dc::kJGeluPrimal; e3.bias = b.b_1; e3.out = w.z + (size_t)l * N * md; e3.out2 = w.mbuf;
    DC_LAUNCH(DC_PROF_JVP_GEMM, 2.0 * (N) * (md) * (d), 0.0,
              dc::launch_gemm_f32w<T>(w.abuf, static_cast<const T*>(b.w_1), N, md, d, e3, st));
    dc::JEpi e4{};
    e4.mode = dc::kJGatedAdd; e4.bias = b.b_2; e4.gate = mb + 5 * d; e4.base = w.hcur; e4.out = w.hcur;
    DC_LAUNCH(DC_PROF_JVP_GEMM, 2.0 * (N) * (d) * (md), 0.0,
              dc::launch_gemm_f32w<T>(w.mbuf, static_cast<const T*>(b.w_2), N, d, md, e4, st));
  }
  DC_CK(cudaMemcpyAsync(w.hL, w.hcur, Nd * 4, cudaMemcpyDeviceToDevice, st));
  return DC_OK;
}

// dv = J dx for T perturbations dx [T][N][C] of the last primal point.
template <typename T>
dc_status tangent_f32(dc_model* m, ResponseWork<T>& w, const float* dx, int Tn, const float* mod,
                      float* dv, cudaStream_t st) {
  const int N = w.N, d = w.d, md = w.md, R = Tn * N;
  const size_t Nd = (size_t)N * d;
  DC_LAUNCH(DC_PROF_JVP_OTHER, 0.0, 0.0,
            dc::launch_embed_f32<T>(dx, m->w_eT, nullptr, static_cast<const T*>(nullptr), R, N,
                                    w.C, d, w.th, st));
  for (int l = 0; l < w.L; ++l) {
    const BlockW& b = m->blk[l];
    const float* mb = mod + (size_t)l * 6 * d;
    DC_LAUNCH(DC_PROF_JVP_OTHER, 0.0, 0.0,
              dc::launch_ln_jvp_f32(w.hin + l * Nd, w.th, N, Tn, d, mb + d, w.ta, st));
    dc::JEpi e1{};
    e1.mode = dc::kJStore; e1.out = w.tqkv;
    DC_LAUNCH(DC_PROF_JVP_GEMM, 2.0 * (R) * (3 * d) * (d), 0.0,
              dc::launch_gemm_f32w<T>(w.ta, static_cast<const T*>(b.w_qkv), R, 3 * d, d, e1, st));
    // tangent: scores, their tangent and the three weighted sums, 12 N^2 dh
    DC_LAUNCH(DC_PROF_JVP_ATTENTION, 12.0 * Tn * w.heads * (double)N * N * w.dh, 0.0,
              dc::launch_attention_f32_jvp(w.qkv + (size_t)l * N * 3 * d, w.tqkv, N, d, w.heads,
                                           w.dh, Tn, nullptr, w.tout, st));
    dc::JEpi e2{};
    e2.mode = dc::kJGatedAdd; e2.gate = mb + 2 * d; e2.base = w.th; e2.out = w.th;
    DC_LAUNCH(DC_PROF_JVP_GEMM, 2.0 * (R) * (d) * (d), 0.0,
              dc::launch_gemm_f32w<T>(w.tout, static_cast<const T*>(b.w_o), R, d, d, e2, st));
    DC_LAUNCH(DC_PROF_JVP_OTHER, 0.0, 0.0,
              dc::launch_ln_jvp_f32(w.h1 + l * Nd, w.th, N, Tn, d, mb + 4 * d, w.ta, st));
    dc::JEpi e3{};
    e3.mode = dc::kJGeluGrad; e3.out = w.tm; e3.z = w.z + (size_t)l * N * md; e3.zrows = N;
    DC_LAUNCH(DC_PROF_JVP_GEMM, 2.0 * (R) * (md) * (d), 0.0,
              dc::launch_gemm_f32w<T>(w.ta, static_cast<const T*>(b.w_1), R, md, d, e3, st));
    dc::JEpi e4{};
    e4.mode = dc::kJGatedAdd; e4.gate = mb + 5 * d; e4.base = w.th; e4.out = w.th;
    DC_LAUNCH(DC_PROF_JVP_GEMM, 2.0 * (R) * (d) * (md), 0.0,
              dc::launch_gemm_f32w<T>(w.tm, static_cast<const T*>(b.w_2), R, d, md, e4, st));
  }
  const float* fsh = mod + (size_t)6 * w.L * d;
  DC_LAUNCH(DC_PROF_JVP_OTHER, 0.0, 0.0,
              dc::launch_ln_jvp_f32(w.hL, w.th, N, Tn, d, fsh + d, w.ta, st));
  dc::JEpi ef{};
  ef.mode = dc::kJStore; ef.out = dv;
  DC_LAUNCH(DC_PROF_JVP_GEMM, 2.0 * (R) * (w.C) * (d), 0.0,
              dc::launch_gemm_f32w<float>(w.ta, m->w_f, R, w.C, d, ef, st));
  return DC_OK;
}

template <typename T>
dc_status anchor_response_impl(dc_model* m, const float* noise, const dc_trajectory* traj, int K,
                               const double* sig, int H, double eps, double* q_out,
                               cudaStream_t st) {
  ResponseWork<T> w{};
  w.N = m->N; w.C = m->C; w.d = m->d; w.L = m->L; w.md = m->md; w.heads = m->heads; w.dh = m->dh;
  const int N = w.N, C = w.C, d = w.d, md = w.md;
  const size_t NC = (size_t)N * C, Nd = (size_t)N * d;
  // perturbation chains (j, l), injected after step t = j + l, ordered by t
  std::vector<std::pair<int, int>> chains;
  std::vector<int> first_at(K + 2, 0);
  for (int t = 2; t <= K; ++t) {
    first_at[t] = (int)chains.size();
    for (int l = 1; l <= std::min(H, t - 1); ++l) chains.push_back({t - l, l});
  }
  first_at[K + 1] = (int)chains.size();
  const int nch = (int)chains.size();
  // tangent batch: at most 64, within about 8 GB of tangent workspace
  const size_t per_tan = (size_t)N * (6 * (size_t)d + md + 2 * (size_t)C) * 4;
  const int Tmax = (int)std::max<size_t>(1, std::min<size_t>(64, (size_t)8e9 / per_tan));
  DevBufs buf;
  const bool ok =
      buf.get(&w.xs, (size_t)(K + 1) * NC * 4) && buf.get(&w.rs, (size_t)K * Nd * sizeof(T)) &&
      buf.get(&w.vbar, (size_t)K * NC * 4) && buf.get(&w.e, NC * 4) && buf.get(&w.vtmp, NC * 4) &&
      buf.get(&w.hin, (size_t)w.L * Nd * 4) && buf.get(&w.qkv, (size_t)w.L * Nd * 3 * 4) &&
      buf.get(&w.h1, (size_t)w.L * Nd * 4) && buf.get(&w.z, (size_t)w.L * N * md * 4) &&
      buf.get(&w.hcur, Nd * 4) && buf.get(&w.hL, Nd * 4) && buf.get(&w.abuf, Nd * 4) &&
      buf.get(&w.obuf, Nd * 4) && buf.get(&w.mbuf, (size_t)N * md * 4) &&
      buf.get(&w.th, (size_t)Tmax * Nd * 4) && buf.get(&w.ta, (size_t)Tmax * Nd * 4) &&
      buf.get(&w.tqkv, (size_t)Tmax * Nd * 3 * 4) && buf.get(&w.tout, (size_t)Tmax * Nd * 4) &&
      buf.get(&w.tm, (size_t)Tmax * N * md * 4) && buf.get(&w.tv, (size_t)Tmax * NC * 4);
  float* dxs = nullptr;
  if (!ok || !buf.get(&dxs, (size_t)std::max(nch, 1) * NC * 4)) {
    dc::set_error("dc_anchor_response: device allocation failed");
    return DC_ERR_NOMEM;
  }
  // the frozen full trace: x_1..x_K, the cached r_1..r_K, then x_{K+1}
  std::vector<unsigned char> forced((size_t)K + 1, dc::kCompute);
  dc_sched sc{};
  sc.K = K; sc.sigmas = sig; sc.anchors = nullptr; sc.tau = 0.0; sc.veto = 0;
  sc.forced = forced.data();
  dc_cond cond{1, traj};
  DC_TRY(check_call(m, &cond, &sc));
  float* lat = w.xs + (size_t)K * NC;
  DC_CK(cudaMemcpyAsync(lat, noise, NC * 4, cudaMemcpyDeviceToDevice, st));
  DC_TRY(run_sampler<T>(m, lat, &cond, &sc, st, nullptr, w.xs, w.rs));
  auto x_at = [&](int k) { return w.xs + (size_t)(k - 1) * NC; };      // x_k, k = 1..K+1
  auto r_at = [&](int k) { return w.rs + (size_t)(k - 1) * Nd; };      // r_k, k = 1..K
  auto mod_at = [&](int k) { return m->mod + (size_t)(k - 1) * m->mod_stride; };
  // H_t(x_t, r_t) of every step (the second term of Eq. 6)
  for (int t = 1; t <= K; ++t)
    DC_TRY(interface_f32<T>(m, w, x_at(t), r_at(t), mod_at(t), w.vbar + (size_t)(t - 1) * NC, st));
  for (int step = 2; step <= K + 1; ++step) {
    // chains injected after step t = step - 1: dx_{t+1} = dsig_t e_{j,l} (Eq. 6)
    const int t = step - 1;
    const float dsig_t = (float)(sig[t] - sig[t - 1]);
    for (int c = first_at[t]; c < first_at[t + 1]; ++c) {
      DC_TRY(interface_f32<T>(m, w, x_at(t), r_at(chains[c].first), mod_at(t), w.vtmp, st));
      DC_LAUNCH(DC_PROF_JVP_OTHER, 0.0, 0.0,
                dc::launch_scaled_diff(w.vtmp, w.vbar + (size_t)(t - 1) * NC, dsig_t, dxs + c * NC,
                                       NC, st));
    }
    if (step > K) break;
    // carry every live chain through step `step`: dx += dsig J dx
    const int live = first_at[step];
    if (live == 0) continue;
    DC_TRY(primal_f32<T>(m, w, x_at(step), mod_at(step), st));
    const float dsig = (float)(sig[step] - sig[step - 1]);
    for (int g0 = 0; g0 < live; g0 += Tmax) {
      const int Tn = std::min(Tmax, live - g0);
      DC_TRY(tangent_f32<T>(m, w, dxs + (size_t)g0 * NC, Tn, mod_at(step), w.tv, st));
      DC_LAUNCH(DC_PROF_JVP_OTHER, 0.0, 0.0,
                dc::launch_axpy_f32(dxs + (size_t)g0 * NC, w.tv, dsig, (size_t)Tn * NC, st));
    }
  }
  // Eq. 7 on the host in fp64: G_{j,h} = sum_{l<=h} P_{j+l} e_{j,l}
  std::vector<float> Y((size_t)nch * NC), xK(NC);
  if (nch) DC_CK(cudaMemcpyAsync(Y.data(), dxs, Y.size() * 4, cudaMemcpyDeviceToHost, st));
  DC_CK(cudaMemcpyAsync(xK.data(), x_at(K + 1), NC * 4, cudaMemcpyDeviceToHost, st));
  DC_TRY(check_device_error(m, st));
  double nx = 0.0;
  for (float v : xK) nx += (double)v * v;
  const double den = std::sqrt(nx) + eps;
  for (size_t i = 0; i < (size_t)K * (H + 1); ++i) q_out[i] = 0.0;
  std::vector<int> idx((size_t)(K + 1) * (H + 1), -1);
  for (int c = 0; c < nch; ++c) idx[(size_t)chains[c].first * (H + 1) + chains[c].second] = c;
  std::vector<double> G(NC);
  for (int j = 1; j < K; ++j) {
    std::fill(G.begin(), G.end(), 0.0);
    for (int l = 1; l <= std::min(H, K - j); ++l) {
      const float* y = Y.data() + (size_t)idx[(size_t)j * (H + 1) + l] * NC;
      double g2 = 0.0;
      for (size_t i = 0; i < NC; ++i) {
        G[i] += y[i];
        g2 += G[i] * G[i];
      }
      if (!std::isfinite(g2)) {
        dc::set_error("dc_anchor_response: non-finite response");
        return DC_ERR_NONFINITE;
      }
      q_out[(size_t)j * (H + 1) + l] = std::sqrt(g2) / den;
    }
  }
  return DC_OK;
}

}  // namespace

extern "C" {

size_t dc_model_weight_count(const dc_model_desc* desc) {
  if (check_desc(desc) != DC_OK) return 0;
  WeightLayout w;
  weight_layout(*desc, &w);
  return w.total;
}

dc_status dc_model_create(const dc_model_desc* desc, const float* host_weights, size_t n_floats,
                          int device, dc_model** out) {
  DC_TRY(check_desc(desc));
  if (!host_weights || !out) { dc::set_error("NULL weights/out"); return DC_ERR_INVALID_ARG; }
  WeightLayout lay;
  weight_layout(*desc, &lay);
  if (n_floats != lay.total) {
    dc::set_error("weight blob has " + std::to_string(n_floats) + " floats, expected " +
                  std::to_string(lay.total));
    return DC_ERR_INVALID_ARG;
  }
  if (device >= 0) DC_CK(cudaSetDevice(device));
  int dev = 0;
  DC_CK(cudaGetDevice(&dev));
  int major = 0, minor = 0;
  DC_CK(cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev));
  DC_CK(cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev));
  if (major != 10 || minor != 3) {
    dc::set_error("this library is built for sm_103a only (device is sm_" + std::to_string(major) +
                  std::to_string(minor) + ")");
    return DC_ERR_UNSUPPORTED;
  }
  dc_model* m = new dc_model();
  m->desc = *desc;
  m->device = dev;
  DC_CK(cudaDeviceGetAttribute(&m->n_sms, cudaDevAttrMultiProcessorCount, dev));
  m->bf16 = desc->dtype == DC_DTYPE_BF16;
  m->elt = m->bf16 ? 2 : 4;
  m->N = desc->n_tokens; m->C = desc->channels; m->d = desc->d_model; m->L = desc->n_blocks;
  m->heads = desc->n_heads; m->dh = m->d / m->heads;
  m->dhp = m->bf16 ? ((m->dh + 15) / 16) * 16 : m->dh;
  m->md = desc->mlp_ratio * m->d; m->P = desc->n_poses; m->Bmax = desc->max_batch;
  m->Kmax = desc->max_steps;
  m->mod_stride = (6 * m->L + 2) * m->d;

  // ---- weights
  std::vector<size_t> off(lay.t.size());
  size_t bytes = 0;
  for (size_t i = 0; i < lay.t.size(); ++i) {
    off[i] = bytes;
    bytes += align256(lay.t[i].n * (lay.t[i].big ? m->elt : 4));
  }
  std::vector<uint8_t> host(bytes, 0);
  {
    const float* src = host_weights;
    for (size_t i = 0; i < lay.t.size(); ++i) {
      const size_t n = lay.t[i].n;
      if (lay.t[i].big && m->bf16) {
        uint16_t* dst = reinterpret_cast<uint16_t*>(host.data() + off[i]);
        for (size_t k = 0; k < n; ++k) dst[k] = f2bf_host(src[k]);
      } else {
        std::memcpy(host.data() + off[i], src, n * 4);
      }
      src += n;
    }
  }
  auto fail = [&](dc_status s) { dc_model_destroy(m); return s; };
  if (cudaMalloc(&m->wbuf, bytes) != cudaSuccess) {
    dc::set_error("cudaMalloc of " + std::to_string(bytes) + " weight bytes failed");
    return fail(DC_ERR_NOMEM);
  }
  if (cudaMemcpy(m->wbuf, host.data(), bytes, cudaMemcpyHostToDevice) != cudaSuccess) {
    dc::set_error("weight upload failed");
    return fail(DC_ERR_CUDA);
  }
  {
    uint8_t* b = static_cast<uint8_t*>(m->wbuf);
    size_t i = 0;
    auto nxt = [&]() { return b + off[i++]; };
    m->w_e = (float*)nxt(); m->b_e = (float*)nxt(); m->pos = nxt();
    m->w_t1 = (float*)nxt(); m->b_t1 = (float*)nxt();
    m->w_t2 = (float*)nxt(); m->b_t2 = (float*)nxt();
    m->w_traj = (float*)nxt(); m->b_traj = (float*)nxt();
    m->w_ada = nxt(); m->b_ada = (float*)nxt();
    m->blk.resize(m->L);
    for (int l = 0; l < m->L; ++l) {
      BlockW& w = m->blk[l];
      w.w_qkv = nxt(); w.b_qkv = (float*)nxt();
      w.w_o = nxt(); w.b_o = (float*)nxt();
      w.w_1 = nxt(); w.b_1 = (float*)nxt();
      w.w_2 = nxt(); w.b_2 = (float*)nxt();
    }
    m->w_f = (float*)nxt(); m->b_f = (float*)nxt();
  }

  // ---- workspace
  m->head_tc = m->bf16 && m->C == 16;
  m->mlp_tc = m->bf16 && dc::mlp_tc_supported(m->d, m->md);
  const size_t B = m->Bmax, N = m->N, d = m->d, K = m->Kmax;
  struct Buf { void** p; size_t bytes; };
  std::vector<Buf> bufs = {
      {(void**)&m->u, B * N * d * 4}, {(void**)&m->h, B * N * d * 4},
      {&m->a, B * N * d * m->elt}, {&m->qkv, 3 * B * m->heads * N * m->dhp * m->elt},
      {&m->o, B * N * d * m->elt}, {&m->m, B * N * m->md * m->elt},
      {&m->r, B * N * d * m->elt}, {(void**)&m->xj, B * N * m->C * 4},
      {(void**)&m->lat_stage, B * N * m->C * 4},
      {(void**)&m->cfg_x, B * N * m->C * 4}, {(void**)&m->cfg_v, B * N * m->C * 4},
      {(void**)&m->mod, K * B * m->mod_stride * 4}, {(void**)&m->silu_c, K * B * d * 4},
      {(void**)&m->temb_f, K * 256 * 4}, {(void**)&m->temb_h, K * d * 4},
      {(void**)&m->temb, K * d * 4}, {(void**)&m->pose_f, B * 3 * m->P * 4},
      {(void**)&m->traj, B * d * 4},
      {(void**)&m->drift_part, (size_t)dc::kMaxBatch * dc::kDriftParts * 2 * 4},
      {(void**)&m->drift_out, (size_t)dc::kMaxBatch * 2 * 4},
      {(void**)&m->poses_d, B * m->P * 3 * 8}, {(void**)&m->sig_d, (K + 1) * 8},
      {(void**)&m->err_d, 256}, {(void**)&m->w_eT, (size_t)m->C * d * 4},
      {(void**)&m->gram, (size_t)m->C * m->C * 4}, {(void**)&m->gp, N * m->C * 4},
      {(void**)&m->gs, N * 4},
      {(void**)&m->wsum, (size_t)m->C * 4}, {(void**)&m->we_frag, (size_t)m->C * d * 2},
      {(void**)&m->head_wp, m->head_tc ? K * B * (size_t)dc::head_b_rows() * d * 2 : 0},
      {(void**)&m->head_tab, m->head_tc ? K * B * (size_t)dc::head_table_floats() * 4 : 0},
      {(void**)&m->cstat, m->head_tc ? B * N * sizeof(float2) : 0},
      {(void**)&m->cond_xs, m->bf16 ? cond_groups(K * B) * 2 * dc::cond_tc_group_rows() * d * 2 : 0}};
  size_t wsb = 0;
  for (auto& b : bufs) wsb += align256(b.bytes);
  if (cudaMalloc(&m->ws, wsb) != cudaSuccess) {
    dc::set_error("cudaMalloc of " + std::to_string(wsb) + " workspace bytes failed");
    return fail(DC_ERR_NOMEM);
  }
  {
    uint8_t* p = static_cast<uint8_t*>(m->ws);
    for (auto& b : bufs) { *b.p = p; p += align256(b.bytes); }
  }
  // zero everything once: the head-dim pad columns of q/k/v stay zero
  if (cudaMemset(m->ws, 0, wsb) != cudaSuccess) return fail(DC_ERR_CUDA);
  {
    // W_e^T and the Gram tables of the drift sums (fp64 on the host, from the
    // values the device uses: pos rounded to bf16 for bf16 models)
    const int C = m->C, D = (int)d;
    const float* we = host_weights;                 // w_embed [d][C]
    const float* be = host_weights + (size_t)D * C;  // b_embed [d]
    const float* ps = be + D;                        // pos [N][d]
    std::vector<float> weT((size_t)C * D), gram((size_t)C * C), gp(N * C), gs(N), wsum(C);
    for (int e = 0; e < D; ++e)
      for (int c = 0; c < C; ++c) {
        weT[(size_t)c * D + e] = we[(size_t)e * C + c];
      }
    for (int c = 0; c < C; ++c) {
      double acc = 0.0;
      for (int e = 0; e < D; ++e) acc += (double)we[(size_t)e * C + c];
      wsum[c] = (float)acc;
    }
    std::vector<uint16_t> we_frag(m->head_tc ? (size_t)C * D : 0);
    if (m->head_tc) dc::head_we_fragments(weT.data(), D, we_frag.data());
    for (int a = 0; a < C; ++a)
      for (int b = 0; b < C; ++b) {
        double acc = 0.0;
        for (int e = 0; e < D; ++e) acc += (double)we[(size_t)e * C + a] * we[(size_t)e * C + b];
        gram[(size_t)a * C + b] = (float)acc;
      }
    std::vector<double> g(D);
    for (size_t t = 0; t < N; ++t) {
      double sq = 0.0;
      for (int e = 0; e < D; ++e) {
        float pv = ps[t * D + e];
        if (m->bf16) {
          const uint32_t bits = (uint32_t)f2bf_host(pv) << 16;
          std::memcpy(&pv, &bits, 4);
        }
        g[e] = (double)be[e] + (double)pv;
        sq += g[e] * g[e];
      }
      gs[t] = (float)sq;
      for (int c = 0; c < C; ++c) {
        double acc = 0.0;
        for (int e = 0; e < D; ++e) acc += (double)we[(size_t)e * C + c] * g[e];
        gp[t * C + c] = (float)acc;
      }
    }
    if (cudaMemcpy(m->w_eT, weT.data(), weT.size() * 4, cudaMemcpyHostToDevice) != cudaSuccess ||
        cudaMemcpy(m->gram, gram.data(), gram.size() * 4, cudaMemcpyHostToDevice) != cudaSuccess ||
        cudaMemcpy(m->gp, gp.data(), gp.size() * 4, cudaMemcpyHostToDevice) != cudaSuccess ||
        cudaMemcpy(m->gs, gs.data(), gs.size() * 4, cudaMemcpyHostToDevice) != cudaSuccess ||
        cudaMemcpy(m->wsum, wsum.data(), wsum.size() * 4, cudaMemcpyHostToDevice) != cudaSuccess ||
        (m->head_tc && cudaMemcpy(m->we_frag, we_frag.data(), we_frag.size() * 2,
                                  cudaMemcpyHostToDevice) != cudaSuccess)) {
      dc::set_error("upload of the derived tables failed");
      return fail(DC_ERR_CUDA);
    }
  }
  if (cudaMallocHost(&m->drift_host, (size_t)dc::kMaxBatch * 2 * 4) != cudaSuccess) {
    dc::set_error("cudaMallocHost failed");
    return fail(DC_ERR_NOMEM);
  }
  if (m->bf16) {
    const uint32_t bn = (uint32_t)dc::gemm_tc_w_box_rows(), bm = (uint32_t)dc::gemm_tc_tile_m();
    dc_status s;
    if ((s = make_map(&m->tm_a, m->a, d, B * N, bm)) != DC_OK) return fail(s);
    if ((s = make_map(&m->tm_oact, m->o, d, B * N, bm)) != DC_OK) return fail(s);
    if ((s = make_map(&m->tm_m, m->m, m->md, B * N, bm)) != DC_OK) return fail(s);
    if ((s = make_map(&m->tm_u32, m->u, d, B * N, bm, true)) != DC_OK) return fail(s);
    if ((s = make_map(&m->tm_h32, m->h, d, B * N, bm, true)) != DC_OK) return fail(s);
    if ((s = make_map(&m->tm_ada, m->w_ada, d, m->mod_stride, 128)) != DC_OK) return fail(s);
    if (m->head_tc) {
      if ((s = make_map(&m->tm_cache, m->r, d, B * N, 128)) != DC_OK) return fail(s);
      if ((s = make_map(&m->tm_headb, m->head_wp, d, K * B * dc::head_b_rows(), dc::head_b_rows())) !=
          DC_OK)
        return fail(s);
    }
    if ((s = make_map(&m->tm_xs, m->cond_xs, d, cond_groups(K * B) * 2 * dc::cond_tc_group_rows(),
                      128)) != DC_OK)
      return fail(s);
    if (dc::attention_tc_supported(m->dh) &&
        (s = make_map(&m->tm_qkv, m->qkv, m->dhp, 3 * B * m->heads * N, 128)) != DC_OK)
      return fail(s);
    for (int l = 0; l < m->L; ++l) {
      BlockW& w = m->blk[l];
      if ((s = make_map(&w.tm_qkv, w.w_qkv, d, 3 * d, bn)) != DC_OK) return fail(s);
      if ((s = make_map(&w.tm_o, w.w_o, d, d, bn)) != DC_OK) return fail(s);
      if ((s = make_map(&w.tm_1, w.w_1, d, m->md, bn)) != DC_OK) return fail(s);
      if ((s = make_map(&w.tm_2, w.w_2, m->md, d, bn)) != DC_OK) return fail(s);
      if (m->mlp_tc && (s = make_map(&w.tm_1f, w.w_1, d, m->md, 64)) != DC_OK) return fail(s);
    }
  }
  if (cudaDeviceSynchronize() != cudaSuccess) return fail(DC_ERR_CUDA);
  *out = m;
  return DC_OK;
}

void dc_model_destroy(dc_model* m) {
  if (!m) return;
  if (m->wbuf) cudaFree(m->wbuf);
  if (m->ws) cudaFree(m->ws);
  if (m->drift_host) cudaFreeHost(m->drift_host);
  for (auto& r : m->prof_pending) { cudaEventDestroy(r.a); cudaEventDestroy(r.b); }
  for (auto e : m->ev_pool) cudaEventDestroy(e);
  delete m;
}

dc_status dc_denoise(dc_model* m, float* latents, const dc_cond* cond, const dc_sched* sched,
                     void* stream, dc_run_stats* stats) {
  DC_TRY(check_call(m, cond, sched));
  if (!latents) { dc::set_error("latents is NULL"); return DC_ERR_INVALID_ARG; }
  DC_CK(cudaSetDevice(m->device));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (m->bf16) return run_sampler<__nv_bfloat16>(m, latents, cond, sched, st, stats, nullptr);
  return run_sampler<float>(m, latents, cond, sched, st, stats, nullptr);
}

dc_status dc_denoise_steps(dc_model* m, float* latents, const dc_cond* cond, const dc_sched* sched,
                           int k_stop, const void* resume, size_t resume_bytes, void* save,
                           size_t save_bytes, void* stream, dc_run_stats* stats) {
  DC_TRY(check_call(m, cond, sched));
  if (!latents) { dc::set_error("latents is NULL"); return DC_ERR_INVALID_ARG; }
  const int cfg = sched->cfg_scale != 0.0 ? 1 : 0;
  const dc::SnapLayout lay = dc::snap_layout(cond->B, sched->K, cfg, m->N, m->d, m->C, m->elt);
  SnapIO io;
  io.k_stop = k_stop;
  io.digest = dc::call_digest(cond, sched);
  int k0 = 0;
  if (resume) {
    dc::SnapHeader h;
    DC_TRY(dc::read_header(resume, resume_bytes, &h));
    const int dtype = m->bf16 ? DC_DTYPE_BF16 : DC_DTYPE_F32;
    if (h.B != cond->B || h.K != sched->K || h.cfg != cfg || h.dtype != dtype || h.N != m->N ||
        h.d != m->d || h.C != m->C) {
      dc::set_error("snapshot shape (B, K, guidance, dtype, N, d, C) does not match this call");
      return DC_ERR_INVALID_ARG;
    }
    if (h.digest != io.digest) {
      dc::set_error("snapshot was taken from a call with other inputs (digest mismatch)");
      return DC_ERR_INVALID_ARG;
    }
    k0 = h.k_done;
    io.in = static_cast<const uint8_t*>(resume);
  }
  if (k_stop <= k0 || k_stop > sched->K) {
    dc::set_error("k_stop must satisfy k_done < k_stop <= K (k_done = " + std::to_string(k0) + ")");
    return DC_ERR_INVALID_ARG;
  }
  if (save) {
    if (save_bytes != lay.total) {
      dc::set_error("save buffer must be dc_snapshot_bytes(...) = " + std::to_string(lay.total) +
                    " bytes");
      return DC_ERR_INVALID_ARG;
    }
    if (resume && static_cast<const uint8_t*>(save) < static_cast<const uint8_t*>(resume) + resume_bytes &&
        static_cast<const uint8_t*>(resume) < static_cast<const uint8_t*>(save) + save_bytes) {
      dc::set_error("save and resume buffers overlap");
      return DC_ERR_INVALID_ARG;
    }
    io.out = static_cast<uint8_t*>(save);
  }
  DC_CK(cudaSetDevice(m->device));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (m->bf16) return run_sampler<__nv_bfloat16>(m, latents, cond, sched, st, stats, nullptr, nullptr, &io);
  return run_sampler<float>(m, latents, cond, sched, st, stats, nullptr, nullptr, &io);
}

dc_status dc_denoise_host(dc_model* m, float* host_latents, const dc_cond* cond,
                          const dc_sched* sched, void* stream, dc_run_stats* stats) {
  DC_TRY(check_call(m, cond, sched));
  if (!host_latents) { dc::set_error("host_latents is NULL"); return DC_ERR_INVALID_ARG; }
  DC_CK(cudaSetDevice(m->device));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const size_t bytes = (size_t)cond->B * m->N * m->C * sizeof(float);
  DC_CK(cudaMemcpyAsync(m->lat_stage, host_latents, bytes, cudaMemcpyHostToDevice, st));
  dc_status s = m->bf16 ? run_sampler<__nv_bfloat16>(m, m->lat_stage, cond, sched, st, stats, nullptr)
                        : run_sampler<float>(m, m->lat_stage, cond, sched, st, stats, nullptr);
  if (s != DC_OK) return s;
  DC_CK(cudaMemcpyAsync(host_latents, m->lat_stage, bytes, cudaMemcpyDeviceToHost, st));
  DC_CK(cudaStreamSynchronize(st));
  return DC_OK;
}

dc_status dc_anchor_drift(dc_model* m, const float* noise, const dc_trajectory* traj, int K,
                          const double* sigmas, int H_max, double eps, double* d_out,
                          void* stream) {
  if (!m || !noise || !traj || !sigmas || !d_out || K < 1 || K > m->Kmax || H_max < 1 ||
      H_max > 4096 || !(eps > 0.0)) {
    dc::set_error("dc_anchor_drift: NULL argument, K outside [1, max_steps], H_max outside "
                  "[1, 4096] or eps <= 0");
    return DC_ERR_INVALID_ARG;
  }
  DC_CK(cudaSetDevice(m->device));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const size_t NC = (size_t)m->N * m->C;
  float* trace = nullptr;
  float* x = nullptr;
  if (cudaMalloc(&trace, (size_t)K * NC * 4) != cudaSuccess ||
      cudaMalloc(&x, NC * 4) != cudaSuccess) {
    if (trace) cudaFree(trace);
    dc::set_error("dc_anchor_drift: trace allocation failed");
    return DC_ERR_NOMEM;
  }
  std::vector<unsigned char> forced((size_t)K + 1, dc::kCompute);
  dc_sched sc{};
  sc.K = K; sc.sigmas = sigmas; sc.anchors = nullptr; sc.tau = 0.0; sc.veto = 0;
  sc.forced = forced.data();
  dc_cond cond{1, traj};
  dc_status s = check_call(m, &cond, &sc);
  if (s == DC_OK && cudaMemcpyAsync(x, noise, NC * 4, cudaMemcpyDeviceToDevice, st) != cudaSuccess) {
    dc::set_error("dc_anchor_drift: copy failed");
    s = DC_ERR_CUDA;
  }
  if (s == DC_OK)
    s = m->bf16 ? run_sampler<__nv_bfloat16>(m, x, &cond, &sc, st, nullptr, trace)
                : run_sampler<float>(m, x, &cond, &sc, st, nullptr, trace);
  for (int j = 0; j < K; ++j)
    for (int h = 0; h <= H_max; ++h) d_out[(size_t)j * (H_max + 1) + h] = 0.0;
  // pairs (j + h, j) for j = 1..K-1, h = 1..min(H_max, K - j); trace[k-1] = x_k
  std::vector<std::pair<int, int>> pairs;
  for (int j = 1; j < K; ++j)
    for (int h = 1; h <= H_max && j + h <= K; ++h) pairs.push_back({j, h});
  for (size_t p0 = 0; s == DC_OK && p0 < pairs.size(); p0 += dc::kMaxBatch) {
    dc::DriftItems it{};
    it.n = (int)std::min(pairs.size() - p0, (size_t)dc::kMaxBatch);
    for (int i = 0; i < it.n; ++i) {
      const auto& pr = pairs[p0 + i];
      it.now[i] = trace + (size_t)(pr.first + pr.second - 1) * NC;
      it.ref[i] = trace + (size_t)(pr.first - 1) * NC;
    }
    s = m->bf16 ? enqueue_drift<__nv_bfloat16>(m, it, m->drift_out, st)
                : enqueue_drift<float>(m, it, m->drift_out, st);
    if (s != DC_OK) break;
    if (cudaMemcpyAsync(m->drift_host, m->drift_out, (size_t)2 * it.n * 4, cudaMemcpyDeviceToHost,
                        st) != cudaSuccess ||
        cudaStreamSynchronize(st) != cudaSuccess) {
      dc::set_error("dc_anchor_drift: readback failed");
      s = DC_ERR_CUDA;
      break;
    }
    for (int i = 0; i < it.n; ++i) {
      const auto& pr = pairs[p0 + i];
      const double Sd = m->drift_host[2 * i], Su = m->drift_host[2 * i + 1];
      if (!std::isfinite(Sd) || !std::isfinite(Su)) {
        dc::set_error("non-finite drift along the anchor trace");
        s = DC_ERR_NONFINITE;
        break;
      }
      d_out[(size_t)pr.first * (H_max + 1) + pr.second] = std::sqrt(Sd) / (std::sqrt(Su) + eps);
    }
  }
  cudaStreamSynchronize(st);
  cudaFree(trace);
  cudaFree(x);
  return s;
}

dc_status dc_anchor_response(dc_model* m, const float* noise, const dc_trajectory* traj, int K,
                             const double* sigmas, int H_max, double eps, double* q_out,
                             void* stream) {
  if (!m || !noise || !traj || !sigmas || !q_out || K < 1 || K > m->Kmax || H_max < 1 ||
      H_max > 4096 || !(eps > 0.0)) {
    dc::set_error("dc_anchor_response: NULL argument, K outside [1, max_steps], H_max outside "
                  "[1, 4096] or eps <= 0");
    return DC_ERR_INVALID_ARG;
  }
  if (!dc::attention_f32_jvp_supported(m->dh)) {
    dc::set_error("dc_anchor_response: head_dim must be 8, 16, 32, 64, 72 or 128");
    return DC_ERR_UNSUPPORTED;
  }
  DC_CK(cudaSetDevice(m->device));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  dc_status s = m->bf16 ? anchor_response_impl<__nv_bfloat16>(m, noise, traj, K, sigmas, H_max, eps,
                                                               q_out, st)
                        : anchor_response_impl<float>(m, noise, traj, K, sigmas, H_max, eps, q_out,
                                                      st);
  cudaStreamSynchronize(st);
  return s;
}

dc_status dc_drift_sums(dc_model* m, const float* x_now, const float* x_ref, int B, float* out,
                        void* stream) {
  if (!m || !x_now || !x_ref || !out || B < 1 || B > m->Bmax) {
    dc::set_error("dc_drift_sums: NULL pointer or B outside [1, max_batch]");
    return DC_ERR_INVALID_ARG;
  }
  DC_CK(cudaSetDevice(m->device));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  dc::DriftItems it{};
  it.n = B;
  const size_t NC = (size_t)m->N * m->C;
  for (int i = 0; i < B; ++i) {
    it.now[i] = x_now + i * NC;
    it.ref[i] = x_ref + i * NC;
  }
  return m->bf16 ? enqueue_drift<__nv_bfloat16>(m, it, out, st) : enqueue_drift<float>(m, it, out, st);
}

dc_status dc_set_wait_limit(dc_model* m, unsigned int ns) {
  if (!m) { dc::set_error("model is NULL"); return DC_ERR_INVALID_ARG; }
  DC_CK(cudaSetDevice(m->device));
  DC_CK(cudaDeviceSynchronize());  // no launch of this model is in flight
  DC_CK(cudaMemcpy(m->err_d + 1, &ns, sizeof(ns), cudaMemcpyHostToDevice));
  return DC_OK;
}

dc_status dc_profile(dc_model* m, int enable) {
  if (!m) { dc::set_error("model is NULL"); return DC_ERR_INVALID_ARG; }
  if (enable) {
    for (int i = 0; i < DC_PROF_N; ++i) {
      m->prof_ms[i] = m->prof_flops[i] = m->prof_bytes[i] = 0.0;
      m->prof_cnt[i] = 0;
    }
  }
  m->prof_on = enable != 0;
  return DC_OK;
}

dc_status dc_profile_read(dc_model* m, double* ms, long long* launches, double* flops,
                          double* bytes) {
  if (!m) { dc::set_error("model is NULL"); return DC_ERR_INVALID_ARG; }
  for (int i = 0; i < DC_PROF_N; ++i) {
    if (ms) ms[i] = m->prof_ms[i];
    if (launches) launches[i] = m->prof_cnt[i];
    if (flops) flops[i] = m->prof_flops[i];
    if (bytes) bytes[i] = m->prof_bytes[i];
  }
  return DC_OK;
}

dc_status dc_cache_copy(dc_model* m, int scene, void* dst, size_t bytes, void* stream) {
  if (!m || !dst || scene < 0 || scene >= m->Bmax ||
      bytes != (size_t)m->N * m->d * m->elt) {
    dc::set_error("dc_cache_copy: NULL pointer, scene outside [0, max_batch) or wrong size");
    return DC_ERR_INVALID_ARG;
  }
  DC_CK(cudaSetDevice(m->device));
  // the cache row is c = r + b_e + pos: return r
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const size_t off = (size_t)scene * m->N * m->d;
  if (m->bf16) {
    DC_CK(dc::launch_cache_to_residual(static_cast<const __nv_bfloat16*>(m->r) + off, m->b_e,
                                       static_cast<const __nv_bfloat16*>(m->pos), m->N, m->d,
                                       static_cast<__nv_bfloat16*>(dst), st));
  } else {
    DC_CK(dc::launch_cache_to_residual(static_cast<const float*>(m->r) + off, m->b_e,
                                       static_cast<const float*>(m->pos), m->N, m->d,
                                       static_cast<float*>(dst), st));
  }
  return DC_OK;
}

dc_status dc_attention(int dtype, const void* qkv, int slots, int heads, int n_tokens,
                       int head_dim, void* out, void* stream) {
  if (!qkv || !out || slots < 1 || heads < 1 || n_tokens < 1 || head_dim < 1) {
    dc::set_error("dc_attention: NULL pointer or non-positive size");
    return DC_ERR_INVALID_ARG;
  }
  // keeps the work-item count (slot, head, 128-query tile) inside int
  if ((long long)slots * heads > (1 << 15) || n_tokens > (1 << 22)) {
    dc::set_error("dc_attention: slots * heads above 2^15 or n_tokens above 2^22");
    return DC_ERR_UNSUPPORTED;
  }
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (dtype == DC_DTYPE_BF16) {
    if (!(head_dim == 16 || head_dim == 64 || head_dim == 72 || head_dim == 128)) {
      dc::set_error("dc_attention: bf16 head_dim must be 16, 64, 72 or 128");
      return DC_ERR_UNSUPPORTED;
    }
    const int dhp = ((head_dim + 15) / 16) * 16;
    if (dc::attention_tc_supported(head_dim)) {
      // the tensor-core kernel: a TMA map over the caller's buffer and an
      // error word of this call's own (stream-ordered allocation, so calls
      // from several threads, streams or devices never share one); the call
      // waits for the kernel to report
      CUtensorMap tm;
      DC_TRY(make_map(&tm, qkv, dhp, (uint64_t)3 * slots * heads * n_tokens, 128));
      int* err_d = nullptr;
      DC_CK(cudaMallocAsync(reinterpret_cast<void**>(&err_d), 2 * sizeof(int), st));
      cudaError_t e = cudaMemsetAsync(err_d, 0, 2 * sizeof(int), st);  // code, wait limit
      if (e == cudaSuccess)
        e = dc::launch_attention_tc(tm, slots, heads, n_tokens, head_dim,
                                    static_cast<__nv_bfloat16*>(out), err_d, st);
      int err = 0;
      if (e == cudaSuccess)
        e = cudaMemcpyAsync(&err, err_d, sizeof(int), cudaMemcpyDeviceToHost, st);
      const cudaError_t ef = cudaFreeAsync(err_d, st);
      if (e == cudaSuccess) e = ef;
      if (e == cudaSuccess) e = cudaStreamSynchronize(st);
      if (e != cudaSuccess) {
        dc::set_error(std::string("dc_attention: ") + cudaGetErrorString(e));
        return DC_ERR_CUDA;
      }
      if (err) {
        dc::set_error("dc_attention: a bounded device wait gave up");
        return DC_ERR_DEVICE_TIMEOUT;
      }
      return DC_OK;
    }
    DC_CK(dc::launch_attention_bf16(static_cast<const __nv_bfloat16*>(qkv), slots, heads, n_tokens,
                                    head_dim, dhp, static_cast<__nv_bfloat16*>(out), st));
    return DC_OK;
  }
  if (dtype == DC_DTYPE_F32) {
    if (!(head_dim == 8 || head_dim == 16 || head_dim == 32 || head_dim == 64)) {
      dc::set_error("dc_attention: fp32 head_dim must be 8, 16, 32 or 64");
      return DC_ERR_UNSUPPORTED;
    }
    DC_CK(dc::launch_attention_f32(static_cast<const float*>(qkv), slots, heads, n_tokens, head_dim,
                                   head_dim, static_cast<float*>(out), st));
    return DC_OK;
  }
  dc::set_error("dc_attention: unknown dtype");
  return DC_ERR_INVALID_ARG;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Drift sums without allocation.
//
// Some callers cannot allocate device memory once they are running: a planner
// loop with a memory budget fixed at start-up, or a host process where a
// cudaMalloc (which may synchronise the device and can fail under
// fragmentation) is not allowed after initialisation.  For them the
// reduction scratch of the drift sums lives in a fixed array in device
// memory that every GPU loading this library holds until the process exits.
// ---------------------------------------------------------------------------

namespace {

// Up to this many scenes per call: kNoAllocMaxScenes x kDriftParts x 2 fp32
// partial sums = 32 KiB of device memory per GPU.
constexpr int kNoAllocMaxScenes = dc::kMaxBatch;
static __device__ __align__(256) float g_drift_scratch[kNoAllocMaxScenes * dc::kDriftParts * 2];

std::mutex g_scratch_mu;
constexpr int kScratchDevices = 64;
float* g_scratch_addr[kScratchDevices] = {};

// Device address of the scratch array on `dev` (which must be current).  The
// array's name is only a host-side stand-in; the address is looked up once
// per device and cached for the life of the process.  A cudaDeviceReset
// unloads the module and so invalidates the cached address -- and, with it,
// every model on that device, whose weights it frees as well: models must be
// destroyed before a reset and created again after it, and no call may use
// this entry point across a reset.
dc_status scratch_address(int dev, float** out) {
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (dev < 0 || dev >= kScratchDevices) {
    dc::set_error("dc_drift_sums_noalloc: device ordinal out of range");
    return DC_ERR_UNSUPPORTED;
  }
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_drift_scratch);
    if (e != cudaSuccess || !p) {
      dc::set_error(std::string("cudaGetSymbolAddress(drift scratch) failed: ") +
                    cudaGetErrorString(e));
      return DC_ERR_CUDA;
    }
    g_scratch_addr[dev] = static_cast<float*>(p);
  }
  *out = g_scratch_addr[dev];
  return DC_OK;
}

}  // namespace

extern "C" dc_status dc_drift_sums_noalloc(dc_model* m, const float* x_now, const float* x_ref,
                                           int B, float* out, void* stream) {
  if (!m || !x_now || !x_ref || !out) {
    dc::set_error("dc_drift_sums_noalloc: NULL pointer");
    return DC_ERR_INVALID_ARG;
  }
  if (B < 1 || B > m->Bmax || B > kNoAllocMaxScenes) {
    dc::set_error("dc_drift_sums_noalloc: B = " + std::to_string(B) + " outside [1, " +
                  std::to_string(std::min(m->Bmax, kNoAllocMaxScenes)) +
                  "] (fixed scratch holds " + std::to_string(kNoAllocMaxScenes) + " scenes)");
    return DC_ERR_INVALID_ARG;
  }
  DC_CK(cudaSetDevice(m->device));
  float* scratch = nullptr;
  DC_TRY(scratch_address(m->device, &scratch));
  dc::DriftItems it{};
  it.n = B;
  const size_t NC = (size_t)m->N * m->C;
  for (int i = 0; i < B; ++i) {
    it.now[i] = x_now + i * NC;
    it.ref[i] = x_ref + i * NC;
  }
  // every partial the final pass reads is written by the first pass of the
  // same call, so nothing in the scratch needs clearing; the two launches are
  // counted (and timed under dc_profile) like those of dc_drift_sums
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  DC_LAUNCH(DC_PROF_DRIFT, 4.0 * it.n * m->N * m->C * m->C, 8.0 * it.n * m->N * m->C,
            dc::launch_drift(it, m->gram, m->gp, m->gs, m->N, m->C, scratch, out, st));
  m->launches += 2;
  return DC_OK;
}
