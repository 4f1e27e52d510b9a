// Launchers of the device kernels (host-callable, all asynchronous on `st`).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "common.cuh"
#include "epilogue.cuh"

namespace dc {

// ---- conditioning (once per dc_denoise call) -------------------------
// pose features (dx/10, dy/10, wrap(dpsi)) of B trajectories [B][P][3] fp64
cudaError_t launch_pose_features(const double* poses, int B, int P, float* out, cudaStream_t st);
// sinusoidal features of t = 1000 sigma for K sigmas -> [K][256]
cudaError_t launch_temb_features(const double* sigmas, int K, float* out, cudaStream_t st);
// Y[r][o] = sum_i act(X[r][i]) W[o][i] + b[o]  (act = silu if in_silu), W fp32 or bf16
template <typename TW>
cudaError_t launch_rows_linear(const float* X, int R, int I, const TW* W, const float* b, int O,
                               float* Y, int in_silu, cudaStream_t st);
// adaLN table on the tensor cores (bf16 models, cond_tc.cu): xs = silu(temb[k]
// + traj[s]) split into bf16 hi / lo rows per group of cond_tc_group_rows()
// rows ([groups][2 x 64][d]), then Y[r][o] = xs_r . W[o] + b[o] for R = K B
// rows against W [O][d] bf16 (tmW: box 64 x 128, tmX over xs: box 64 x 128)
int cond_tc_group_rows();
cudaError_t launch_cond_split(const float* temb, const float* traj, int K, int B, int d,
                              __nv_bfloat16* xs, cudaStream_t st);
cudaError_t launch_cond_gemm_tc(const CUtensorMap& tmW, const CUtensorMap& tmX, int R, int O, int d,
                                const float* bias, float* Y, int* err, int n_sms, cudaStream_t st);
// c[k][s] = temb[k] + traj[s]; out = silu(c)   ([K][B][d])
cudaError_t launch_cond_combine(const float* temb, const float* traj, int K, int B, int d,
                                float* silu_c, cudaStream_t st);

// ---- per-step kernels --------------------------------------------------
// u = x W_e^T + b_e + pos (fp32) for each compute slot; w_eT = W_e^T [C][d]
template <typename T>
cudaError_t launch_embed(const float* x, const float* w_eT, const float* b_e, const T* pos,
                         const SlotMap& map, int N, int C, int d, float* u, cudaStream_t st);
// a = LN(h) * (1 + scale) + shift  (per-slot modulation)  -> T
template <typename T>
cudaError_t launch_ln_mod(const float* h, int rows, int N, int d, const float* mod, int mod_stride,
                          int shift_off, int scale_off, const SlotMap& map, T* a, cudaStream_t st);
// GEMMs
// tmCin / tmCout: epilogue maps (residual: fp32 [rows][N] box 32 x 128 for
// h_in and h; GELU: bf16 [rows][N] box 64 x 128 for the output; QKV: unused)
cudaError_t launch_gemm_tc(int mode, const CUtensorMap& tmA, const CUtensorMap& tmB,
                           const CUtensorMap& tmCin, const CUtensorMap& tmCout, int M, int N,
                           int K, const EpiArgs& ep, const SlotMap& map, int* err, int n_sms,
                           cudaStream_t st);
cudaError_t launch_gemm_f32(int mode, const float* A, const float* W, int M, int N, int K,
                            const EpiArgs& ep, const SlotMap& map, cudaStream_t st);
size_t gemm_tc_smem_bytes();
int gemm_tc_tile_n();
int gemm_tc_w_box_rows();  // rows of the W box: each CTA of a cluster loads half the tile
int gemm_tc_tile_k();
int gemm_tc_tile_m();
// attention: q/k/v [3][slots][heads][N][dhp] -> o [slots][N][heads*dh]
cudaError_t launch_attention_bf16(const __nv_bfloat16* qkv, int slots, int heads, int N, int dh,
                                  int dhp, __nv_bfloat16* o, cudaStream_t st);
cudaError_t launch_attention_f32(const float* qkv, int slots, int heads, int N, int dh, int dhp,
                                 float* o, cudaStream_t st);
// tcgen05 attention (dh 64, 72 or 128; dhp = dh rounded up to 16, pad
// columns zero): tm is a 2-D bf16 map over the q/k/v buffer viewed as
// [3 * slots * heads * N][dhp], box 64 x 128, 128-byte swizzle; o is
// [slots][N][heads * dh]; err receives a code if a bounded wait gives up
bool attention_tc_supported(int dh);
cudaError_t launch_attention_tc(const CUtensorMap& tm, int nslots, int heads, int N, int dh,
                                __nv_bfloat16* o, int* err, cudaStream_t st);
// The cache row of a scene is c = h_L - x W_e^T of its last full evaluation
// (the block-stack residual r = h_L - u plus b_e + pos), so a reuse step
// forms u_k + r_j = x_k W_e^T + c_j.
// SIMT interface (fp32 models and C = 4): compute step v = head(h_L),
// x_j <- x, x += dsig v, c <- h_L - x W_e^T; reuse step h = x W_e^T + c_j,
// v = head(h), x += dsig v  (w_eT = W_e^T [C][d] fp32)
template <typename T>
cudaError_t launch_final_compute(const float* hL, const float* w_eT, float* x, float* xj, T* r,
                                 const SlotMap& map, int N, int C, int d, const float* mod,
                                 int mod_stride, int fin_off, const float* w_f, const float* b_f,
                                 float dsig, cudaStream_t st, float* vout = nullptr);
template <typename T>
cudaError_t launch_final_reuse(float* x, const T* r, const float* w_eT, const SlotMap& map, int N,
                               int C, int d, const float* mod, int mod_stride, int fin_off,
                               const float* w_f, const float* b_f, float dsig, cudaStream_t st,
                               float* vout = nullptr);
// r_j = c_j - b_e - pos (inspection of a cache row), out [N][d]
template <typename T>
cudaError_t launch_cache_to_residual(const T* c, const float* b_e, const T* pos, int N, int d, T* out,
                                     cudaStream_t st);
// Fused MLP of the block stack for d = 384, hidden 1536 (mlp_tc.cu):
// h <- h + gate2 (GELU(a W1^T + b1) W2^T + b2) in one launch, equal bit for
// bit to the MLP-up (GELU) and MLP-down (residual) GEMMs.  tmA: a [M][384]
// bf16 (box 64 x 128); tmW1: W1 [1536][384] bf16 (box 64 x 64); tmW2: W2
// [384][1536] bf16 (box 64 x 96); tmH: h [M][384] fp32 (box 32 x 128), read
// and written; gate row gate_off of each slot's modulation row.
bool mlp_tc_supported(int d, int md);
cudaError_t launch_mlp_tc(const CUtensorMap& tmA, const CUtensorMap& tmW1, const CUtensorMap& tmW2,
                          const CUtensorMap& tmH, int M, const float* b1, const float* b2,
                          const float* mod, int mod_stride, int gate_off, int n_tok,
                          const SlotMap& map, int* err, int n_sms, cudaStream_t st);
// Tensor-core interface of bf16 models with C = 16 (interface_tc.cu).  Per
// (step, scene) item of the call's modulation table: head_b_rows() = 48 bf16
// rows of d (W_e^T, then W' = (1 + scale) W_f as hi and lo halves), and S',
// beta, G_s (head_table_floats() fp32).  Beside the cache rows [B_max][N][d]
// the compute step keeps cstat [B_max][N] = (sum c, sum c^2) of each row's
// bf16 values, which the reuse step reads instead of the row's moments.
int head_table_floats();
int head_b_rows();
cudaError_t launch_head_tables(const float* mod, int n_items, int mod_stride, int fin_off, int d,
                               const float* w_f, const float* b_f, const float* w_eT,
                               __nv_bfloat16* wp, float* tab, cudaStream_t st);
// reuse step on tcgen05 (reuse_tc.cu): tmC over the cache [B_max N][d] bf16
// (box 64 x 128), tmB over the head tables' B rows [K B_max 48][d] (box 64 x
// 48); b_row0: first B row of this step; tab_k: the step's fp32 tables; wsum:
// row sums of W_e^T; gram: W_e^T W_e [16][16]; err: the model's error word;
// n_sms: the device's SM count (the CTA size follows it)
cudaError_t launch_head_reuse_tc(const CUtensorMap& tmC, const CUtensorMap& tmB, float* x,
                                 const float2* cstat, const SlotMap& map, int N, int d, int b_row0,
                                 const float* tab_k, const float* wsum, const float* gram, float dsig,
                                 int* err, int n_sms, cudaStream_t st, float* vout = nullptr);
// compute step: writes the cache rows and their cstat, x_j <- x, x += dsig v;
// we_frag: W_e^T (16 x d, bf16) in the fragment order head_we_fragments
// builds (host)
cudaError_t launch_head_compute(const float* hL, float* x, float* xj, __nv_bfloat16* cache,
                                float2* cstat, const SlotMap& map, int N, int d,
                                const __nv_bfloat16* we_frag, const __nv_bfloat16* wp_k, const float* tab_k, float dsig,
                                cudaStream_t st, float* vout = nullptr);
void head_we_fragments(const float* w_eT, int d, uint16_t* out /* 16 d values */);
// vout != NULL (both): write the velocity v[scene][tok][c] instead of the
// Euler update (x is left as it is; the compute step still sets x_j = x).
// guidance: x_s += dsig (v_u + g (v_c - v_u)), v_c = v[s], v_u = v[B + s]
cudaError_t launch_cfg_combine(float* x, const float* v, int B, size_t per_scene, float g,
                               float dsig, cudaStream_t st);

// drift sums over items: out[2i] = sum ||(now_i - ref_i) W_e^T||^2,
// out[2i+1] = sum ||now_i W_e^T + b_e + pos||^2   (deterministic order),
// evaluated with the Gram tables gram = W_e^T W_e [C][C],
// gp[t] = W_e^T (b_e + pos_t) [N][C] and gs[t] = ||b_e + pos_t||^2 [N]
struct DriftItems {
  int n;
  const float* now[kMaxBatch];
  const float* ref[kMaxBatch];
};
constexpr int kDriftParts = 64;
cudaError_t launch_drift(const DriftItems& items, const float* gram, const float* gp,
                         const float* gs, int N, int C, float* partials /* [n][kDriftParts][2] */,
                         float* out /* [2n] */, cudaStream_t st);

// ---- fp32 forward-mode kernels for the joint run responses (Eq. 6-7) ----
// C[M][N] = A[M][K] W[N][K]^T + epilogue (W fp32 or bf16, fp32 accumulate):
enum { kJStore = 0, kJGatedAdd = 1, kJGeluPrimal = 2, kJGeluGrad = 3 };
struct JEpi {
  int mode;
  const float* bias;   // optional [N], added to the product first
  const float* gate;   // kJGatedAdd: out = base + gate (acc + bias)
  const float* base;   // kJGatedAdd: [M][N], may equal out
  float* out;          // [M][N]
  float* out2;         // kJGeluPrimal: out = z = acc + bias, out2 = gelu(z)
  const float* z;      // kJGeluGrad: out = gelu'(z[row % zrows]) acc
  int zrows;
};
template <typename TW>
cudaError_t launch_gemm_f32w(const float* A, const TW* W, int M, int N, int K, const JEpi& ep,
                             cudaStream_t st);
// out = LN(h) (1 + scale) + shift per row of d
cudaError_t launch_ln_mod_f32(const float* h, int R, int d, const float* shift, const float* scale,
                              float* out, cudaStream_t st);
// tangent of the modulated LayerNorm at primal rows h [N][d] for dh [T][N][d]
cudaError_t launch_ln_jvp_f32(const float* h, const float* dh, int N, int T, int d,
                              const float* scale, float* out, cudaStream_t st);
// u = x W_e^T (+ b_e + pos when b_e != NULL), x [R][C], rows r use pos[r % N]
template <typename TP>
cudaError_t launch_embed_f32(const float* x, const float* w_eT, const float* b_e, const TP* pos,
                             int R, int N, int C, int d, float* out, cudaStream_t st);
// attention of one scene (qkv [N][3d] fp32 rows) -> o [N][d]; with dqkv
// [T][N][3d] (non-NULL) the tangent -> dout [T][N][d] instead
bool attention_f32_jvp_supported(int dh);
cudaError_t launch_attention_f32_jvp(const float* qkv, const float* dqkv, int N, int d, int heads,
                                     int dh, int T, float* o, float* dout, cudaStream_t st);
cudaError_t launch_axpy_f32(float* y, const float* x, float a, size_t n, cudaStream_t st);
template <typename T>
cudaError_t launch_add_cache(const float* a, const T* r, float* out, size_t n, cudaStream_t st);
cudaError_t launch_scaled_diff(const float* a, const float* b, float s, float* out, size_t n,
                               cudaStream_t st);

}  // namespace dc
