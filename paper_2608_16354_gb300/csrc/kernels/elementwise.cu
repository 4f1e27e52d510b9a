// HBM-bound kernels of the hot path: conditioning (timestep + trajectory
// features, small MLPs, adaLN modulation table), patch embedding, adaLN
// LayerNorm, the interface + Euler update on compute and on reuse steps, and
// the deterministic drift reduction of Eq. 12.
//
// Row-wise kernels use one warp per token row with float4 accesses; each
// lane holds NV float4 of the row in registers (NV = ceil(d / 128)).
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace dc {

namespace {

constexpr double kPiD = 3.141592653589793238462643383279502884;

// ------------------------------------------------------------ conditioning

__global__ void pose_features_kernel(const double* __restrict__ poses, int B, int P,
                                     float* __restrict__ out) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= B * P) return;
  const int s = i / P, t = i - s * P;
  const double* p0 = poses + (size_t)s * P * 3;
  const double* pt = p0 + (size_t)t * 3;
  double dpsi = remainder(pt[2] - p0[2], 2.0 * kPiD);
  if (dpsi == -kPiD) dpsi = kPiD;
  float* o = out + (size_t)s * 3 * P + 3 * t;
  o[0] = (float)((pt[0] - p0[0]) / 10.0);
  o[1] = (float)((pt[1] - p0[1]) / 10.0);
  o[2] = (float)dpsi;
}

__global__ void temb_features_kernel(const double* __restrict__ sig, int K, float* __restrict__ out) {
  const int k = blockIdx.x, i = threadIdx.x;  // 128 threads
  if (k >= K) return;
  const double t = 1000.0 * sig[k];
  const double f = exp(-log(10000.0) * (double)i / 128.0);
  out[(size_t)k * 256 + i] = (float)cos(t * f);
  out[(size_t)k * 256 + 128 + i] = (float)sin(t * f);
}

// Y[R][O] = act(X)[R][I] W[O][I]^T + b, fp32 accumulation.  A CTA computes a
// 64-row x 128-output tile: 32-deep slices of X and W are staged k-major in
// shared memory and each thread accumulates 8 rows x 4 outputs (outputs
// lane + 32 c, so that stores are coalesced), summing over i in order.
constexpr int kRlRows = 64, kRlCols = 128, kRlK = 32;

template <typename TW>
__global__ void __launch_bounds__(256) rows_linear_kernel(const float* __restrict__ X, int R, int I,
                                                          const TW* __restrict__ W,
                                                          const float* __restrict__ b, int O,
                                                          float* __restrict__ Y, int in_silu) {
  // row strides: 68 keeps the float4 reads aligned, 129 spreads the
  // transposing stores over the banks
  __shared__ __align__(16) float xs[kRlK][kRlRows + 4];
  __shared__ float ws[kRlK][kRlCols + 1];
  const int tid = threadIdx.x, lane = tid & 31, ty = tid >> 5;
  const int o0 = blockIdx.x * kRlCols, r0 = blockIdx.y * kRlRows;
  float acc[8][4];
#pragma unroll
  for (int j = 0; j < 8; ++j)
#pragma unroll
    for (int c = 0; c < 4; ++c) acc[j][c] = 0.f;
  for (int k0 = 0; k0 < I; k0 += kRlK) {
    const int kk = tid & (kRlK - 1), k = k0 + kk;
#pragma unroll
    for (int e = 0; e < kRlRows * kRlK / 256; ++e) {
      const int row = (tid >> 5) + 8 * e, r = r0 + row;
      float v = r < R && k < I ? X[(size_t)r * I + k] : 0.f;
      if (in_silu && r < R && k < I) v = silu(v);
      xs[kk][row] = v;
    }
#pragma unroll
    for (int e = 0; e < kRlCols * kRlK / 256; ++e) {
      const int col = (tid >> 5) + 8 * e, o = o0 + col;
      ws[kk][col] = o < O && k < I ? to_f(W[(size_t)o * I + k]) : 0.f;
    }
    __syncthreads();
#pragma unroll 4
    for (int q = 0; q < kRlK; ++q) {
      const float4 xa = *reinterpret_cast<const float4*>(&xs[q][ty * 8]);
      const float4 xb = *reinterpret_cast<const float4*>(&xs[q][ty * 8 + 4]);
      const float xv[8] = {xa.x, xa.y, xa.z, xa.w, xb.x, xb.y, xb.z, xb.w};
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const float wv = ws[q][lane + 32 * c];
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[j][c] = fmaf(xv[j], wv, acc[j][c]);
      }
    }
    __syncthreads();
  }
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const int r = r0 + ty * 8 + j;
    if (r >= R) break;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int o = o0 + lane + 32 * c;
      if (o < O) Y[(size_t)r * O + o] = acc[j][c] + b[o];
    }
  }
}

__global__ void cond_combine_kernel(const float* __restrict__ temb, const float* __restrict__ traj,
                                    int K, int B, int d, float* __restrict__ out) {
  const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  const size_t total = (size_t)K * B * d;
  if (i >= total) return;
  const int e = (int)(i % d);
  const int s = (int)((i / d) % B);
  const int k = (int)(i / ((size_t)d * B));
  out[i] = silu(temb[(size_t)k * d + e] + traj[(size_t)s * d + e]);
}

// ------------------------------------------------------------- embedding

template <typename T>
__device__ __forceinline__ float4 load4(const T* src);

// u = x W_e^T + b_e + pos: a thread computes 4 consecutive outputs of
// kEmbedRows consecutive tokens, so that its W_e columns (read transposed,
// [C][d], contiguous float4 across the warp) are loaded once for all of them:
// 16 rows keep those W_e reads (C float4 per thread, from L2) below the
// row bytes the thread moves.
constexpr int kEmbedRows = 16;

template <typename T, int C>
__global__ void embed_kernel(const float* __restrict__ x, const float* __restrict__ w_eT,
                             const float* __restrict__ b_e, const T* __restrict__ pos, SlotMap map,
                             int N, int d, float* __restrict__ u) {
  pdl_trigger();
  pdl_wait();
  const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int d4 = d >> 2;
  const size_t rows = (size_t)map.n * N;
  const size_t groups = (rows + kEmbedRows - 1) / kEmbedRows;
  if (i >= groups * d4) return;
  const int e4 = (int)(i % d4);
  const size_t g = i / d4;
  float4 w[C];
#pragma unroll
  for (int c = 0; c < C; ++c) w[c] = __ldg(reinterpret_cast<const float4*>(w_eT + (size_t)c * d) + e4);
  const float4 bv = __ldg(reinterpret_cast<const float4*>(b_e) + e4);
  const int nrow = (int)min((size_t)kEmbedRows, rows - g * kEmbedRows);
#pragma unroll 4
  for (int t = 0; t < nrow; ++t) {
    const size_t row = g * kEmbedRows + t;  // slot * N + tok
    const int slot = (int)(row / N), tok = (int)(row - (size_t)slot * N);
    const float4* xr = reinterpret_cast<const float4*>(x + ((size_t)map.scene[slot] * N + tok) * C);
    float xv[C];
#pragma unroll
    for (int c = 0; c < C / 4; ++c) {
      const float4 v = __ldg(xr + c);
      xv[4 * c] = v.x; xv[4 * c + 1] = v.y; xv[4 * c + 2] = v.z; xv[4 * c + 3] = v.w;
    }
    const float4 pv = load4<T>(pos + (size_t)tok * d + 4 * e4);
    float4 acc = make_float4(bv.x + pv.x, bv.y + pv.y, bv.z + pv.z, bv.w + pv.w);
#pragma unroll
    for (int c = 0; c < C; ++c) {
      acc.x += w[c].x * xv[c]; acc.y += w[c].y * xv[c];
      acc.z += w[c].z * xv[c]; acc.w += w[c].w * xv[c];
    }
    reinterpret_cast<float4*>(u)[row * d4 + e4] = acc;
  }
}

// --------------------------------------------------------------- LN + mod

template <int NV>
__device__ __forceinline__ void load_row(const float* __restrict__ src, int d4, int lane,
                                         float4 (&v)[NV]) {
#pragma unroll
  for (int j = 0; j < NV; ++j) {
    const int i = lane + 32 * j;
    v[j] = i < d4 ? reinterpret_cast<const float4*>(src)[i] : make_float4(0.f, 0.f, 0.f, 0.f);
  }
}

// mean and rstd of the row held in registers (two-pass)
template <int NV>
__device__ __forceinline__ void row_stats(const float4 (&v)[NV], int d, int d4, int lane,
                                          float* mean, float* rstd) {
  float s = 0.f;
#pragma unroll
  for (int j = 0; j < NV; ++j) s += (v[j].x + v[j].y) + (v[j].z + v[j].w);
  const float mu = warp_sum(s) / (float)d;
  float q = 0.f;
#pragma unroll
  for (int j = 0; j < NV; ++j) {
    if (lane + 32 * j < d4) {
      const float a = v[j].x - mu, b = v[j].y - mu, c = v[j].z - mu, e = v[j].w - mu;
      q += (a * a + b * b) + (c * c + e * e);
    }
  }
  const float var = warp_sum(q) / (float)d;
  *mean = mu;
  *rstd = rsqrtf(var + 1e-6f);
}

template <typename T>
__device__ __forceinline__ void store4(T* dst, float a, float b, float c, float d_);
template <>
__device__ __forceinline__ void store4<float>(float* dst, float a, float b, float c, float d_) {
  *reinterpret_cast<float4*>(dst) = make_float4(a, b, c, d_);
}
template <>
__device__ __forceinline__ void store4<__nv_bfloat16>(__nv_bfloat16* dst, float a, float b, float c,
                                                      float d_) {
  __align__(8) __nv_bfloat162 t[2] = {__floats2bfloat162_rn(a, b), __floats2bfloat162_rn(c, d_)};
  *reinterpret_cast<uint2*>(dst) = *reinterpret_cast<const uint2*>(t);
}

template <typename T>
__device__ __forceinline__ float4 load4(const T* src);
template <>
__device__ __forceinline__ float4 load4<float>(const float* src) {
  return *reinterpret_cast<const float4*>(src);
}
template <>
__device__ __forceinline__ float4 load4<__nv_bfloat16>(const __nv_bfloat16* src) {
  const uint2 raw = *reinterpret_cast<const uint2*>(src);
  const __nv_bfloat162* p = reinterpret_cast<const __nv_bfloat162*>(&raw);
  const float2 a = __bfloat1622float2(p[0]), b = __bfloat1622float2(p[1]);
  return make_float4(a.x, a.y, b.x, b.y);
}

// rows of at least 1024 elements stage the modulation vectors in shared
// memory (24 KB at d = 3072: 1.25 -> 1.15 ms of LayerNorms per 2-block c5
// call); shorter rows read them directly (staging measured slower at d 384)
__host__ __device__ constexpr bool ln_stage(int nv) { return nv >= 8; }

template <typename T, int NV>
__global__ void ln_mod_kernel(const float* __restrict__ h, int rows, int N, int d,
                              const float* __restrict__ mod, int mod_stride, int shift_off,
                              int scale_off, SlotMap map, T* __restrict__ a) {
  pdl_trigger();
  pdl_wait();
  extern __shared__ float4 ln_sm[];  // shift [d / 4], scale [d / 4] of the block's first scene
  const int row0 = blockIdx.x * (blockDim.x >> 5);
  const int row = row0 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  const int d4 = d >> 2;
  float4 v[NV];
  if (row < rows) load_row<NV>(h + (size_t)row * d, d4, lane, v);
  // Long rows (LN_STAGE): while the rows load, the block stages the shift and
  // scale vectors of its first row's scene once instead of every warp
  // reading them (a block's rows span two scenes only at a scene boundary;
  // rows of the second read theirs from global memory).
  int scene0 = -1;
  if constexpr (ln_stage(NV)) {
    scene0 = map.scene[min(row0, rows - 1) / N];
    const float* m0 = mod + (size_t)scene0 * mod_stride;
    for (int i = threadIdx.x; i < d4; i += blockDim.x) {
      ln_sm[i] = reinterpret_cast<const float4*>(m0 + shift_off)[i];
      ln_sm[d4 + i] = reinterpret_cast<const float4*>(m0 + scale_off)[i];
    }
    __syncthreads();
  }
  if (row >= rows) return;
  float mu, rs;
  row_stats<NV>(v, d, d4, lane, &mu, &rs);
  const int scene = map.scene[row / N];
  const float* mrow = mod + (size_t)scene * mod_stride;
  const float4* sh = scene == scene0 ? ln_sm : reinterpret_cast<const float4*>(mrow + shift_off);
  const float4* sc = scene == scene0 ? ln_sm + d4 : reinterpret_cast<const float4*>(mrow + scale_off);
  T* dst = a + (size_t)row * d;
#pragma unroll
  for (int j = 0; j < NV; ++j) {
    const int i = lane + 32 * j;
    if (i < d4) {
      const float4 s = sh[i], c = sc[i];
      store4<T>(dst + 4 * i, (v[j].x - mu) * rs * (1.f + c.x) + s.x,
                (v[j].y - mu) * rs * (1.f + c.y) + s.y, (v[j].z - mu) * rs * (1.f + c.z) + s.z,
                (v[j].w - mu) * rs * (1.f + c.w) + s.w);
    }
  }
}

// ---------------------------------------------------- interface + Euler

// v_c = sum_e a_e w_f[c][e] + b_f[c] for the modulated, normalised row held
// in registers; lane c < C returns v_c.  The C per-lane partial sums are
// reduced and scattered over the xor butterfly 16, 8, 4, 2, 1 (C - 1 + 5 -
// log2 C shuffles instead of 5 C): at each offset a lane keeps the half of its
// values selected by its lane bit and adds its partner's copy of that half,
// so every sum pairs the same operands in the same order as warp_sum and is
// bitwise the value warp_sum gives.  Lane l ends with channel l / (32 / C).
template <int NV, int C>
__device__ __forceinline__ float head_dot(const float4 (&a)[NV], int d, int d4, int lane,
                                          const float* __restrict__ w_f,
                                          const float* __restrict__ b_f) {
  static_assert(C >= 1 && C <= 32 && (C & (C - 1)) == 0, "C must be a power of two <= 32");
  float s[C];
#pragma unroll
  for (int c = 0; c < C; ++c) {
    const float4* w = reinterpret_cast<const float4*>(w_f + (size_t)c * d);
    float t = 0.f;
#pragma unroll
    for (int j = 0; j < NV; ++j) {
      const int i = lane + 32 * j;
      if (i < d4) {
        const float4 ww = __ldg(w + i);
        t += (a[j].x * ww.x + a[j].y * ww.y) + (a[j].z * ww.z + a[j].w * ww.w);
      }
    }
    s[c] = t;
  }
#pragma unroll
  for (int step = 0; step < 5; ++step) {
    const int off = 16 >> step;
    const int n = C >> step;  // values this lane still holds
    if (n >= 2) {
      const bool upper = (lane & off) != 0;
#pragma unroll
      for (int k = 0; k < n / 2; ++k) {
        const float send = upper ? s[k] : s[k + n / 2];
        const float keep = upper ? s[k + n / 2] : s[k];
        s[k] = keep + __shfl_xor_sync(0xffffffffu, send, off);
      }
    } else {
      s[0] += __shfl_xor_sync(0xffffffffu, s[0], off);
    }
  }
  constexpr int kSpan = 32 / C;  // lanes holding the same channel
  const float v = s[0] + b_f[(lane / kSpan) & (C - 1)];
  return __shfl_sync(0xffffffffu, v, (lane * kSpan) & 31);
}

template <int NV>
__device__ __forceinline__ void modulate(float4 (&v)[NV], float mu, float rs, const float* mrow,
                                         int shift_off, int scale_off, int d4, int lane) {
  const float4* sh = reinterpret_cast<const float4*>(mrow + shift_off);
  const float4* sc = reinterpret_cast<const float4*>(mrow + scale_off);
#pragma unroll
  for (int j = 0; j < NV; ++j) {
    const int i = lane + 32 * j;
    if (i < d4) {
      const float4 s = sh[i], c = sc[i];
      v[j].x = (v[j].x - mu) * rs * (1.f + c.x) + s.x;
      v[j].y = (v[j].y - mu) * rs * (1.f + c.y) + s.y;
      v[j].z = (v[j].z - mu) * rs * (1.f + c.z) + s.z;
      v[j].w = (v[j].w - mu) * rs * (1.f + c.w) + s.w;
    } else {
      v[j] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }
}

// Rows of the interface on the SIMT path (fp32 models, or C != 16).  The
// cache row of a compute step is c = h_L - x W_e^T (the block-stack residual
// plus b_e + pos), so a reuse step forms h = x W_e^T + c.
template <int NV, int C>
__device__ __forceinline__ void embed_latent(const float (&xv)[C], const float* __restrict__ w_eT,
                                             int d, int d4, int lane, float4 (&o)[NV]) {
#pragma unroll
  for (int j = 0; j < NV; ++j) {
    const int i = lane + 32 * j;
    float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
    if (i < d4) {
#pragma unroll
      for (int c = 0; c < C; ++c) {
        const float4 w = __ldg(reinterpret_cast<const float4*>(w_eT + (size_t)c * d) + i);
        a.x += w.x * xv[c]; a.y += w.y * xv[c]; a.z += w.z * xv[c]; a.w += w.w * xv[c];
      }
    }
    o[j] = a;
  }
}

template <typename T, int NV, int C>
__global__ void final_compute_kernel(const float* __restrict__ hL, const float* __restrict__ w_eT,
                                     float* __restrict__ x, float* __restrict__ xj,
                                     T* __restrict__ r, SlotMap map, int N, int d,
                                     const float* __restrict__ mod, int mod_stride, int fin_off,
                                     const float* __restrict__ w_f, const float* __restrict__ b_f,
                                     float dsig, float* __restrict__ vout) {
  pdl_trigger();
  pdl_wait();
  const int row = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;  // slot * N + tok
  const int lane = threadIdx.x & 31;
  if (row >= map.n * N) return;
  const int slot = row / N, tok = row - slot * N;
  const int scene = map.scene[slot];
  const int d4 = d >> 2;
  float4 hv[NV];
  load_row<NV>(hL + (size_t)row * d, d4, lane, hv);
  const float* xr = x + ((size_t)scene * N + tok) * C;
  float xv[C];
#pragma unroll
  for (int c = 0; c < C; ++c) xv[c] = xr[c];
  // cache the reusable backbone output c = h_L - x W_e^T
  {
    float4 ue[NV];
    embed_latent<NV, C>(xv, w_eT, d, d4, lane, ue);
    T* rd = r + ((size_t)scene * N + tok) * d;
#pragma unroll
    for (int j = 0; j < NV; ++j) {
      const int i = lane + 32 * j;
      if (i < d4)
        store4<T>(rd + 4 * i, hv[j].x - ue[j].x, hv[j].y - ue[j].y, hv[j].z - ue[j].z,
                  hv[j].w - ue[j].w);
    }
  }
  float mu, rs;
  row_stats<NV>(hv, d, d4, lane, &mu, &rs);
  modulate<NV>(hv, mu, rs, mod + (size_t)scene * mod_stride, fin_off, fin_off + d, d4, lane);
  const float vc = head_dot<NV, C>(hv, d, d4, lane, w_f, b_f);
  __syncwarp();
  if (lane < C) {
    float xo = xv[0];
#pragma unroll
    for (int c = 1; c < C; ++c)
      if (lane == c) xo = xv[c];
    const size_t xi = ((size_t)scene * N + tok) * C + lane;
    xj[xi] = xo;
    if (vout) vout[xi] = vc;  // the caller combines velocities (guidance)
    else x[xi] = xo + dsig * vc;
  }
}

template <typename T, int NV, int C>
__global__ void final_reuse_kernel(float* __restrict__ x, const T* __restrict__ r,
                                   const float* __restrict__ w_eT, SlotMap map, int N, int d,
                                   const float* __restrict__ mod, int mod_stride, int fin_off,
                                   const float* __restrict__ w_f, const float* __restrict__ b_f,
                                   float dsig, float* __restrict__ vout) {
  pdl_trigger();
  pdl_wait();
  const int row = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (row >= map.n * N) return;
  const int slot = row / N, tok = row - slot * N;
  const int scene = map.scene[slot];
  const int d4 = d >> 2;
  const float* xr = x + ((size_t)scene * N + tok) * C;
  float xv[C];
#pragma unroll
  for (int c = 0; c < C; ++c) xv[c] = xr[c];
  const T* rr = r + ((size_t)scene * N + tok) * d;
  float4 hv[NV];
  embed_latent<NV, C>(xv, w_eT, d, d4, lane, hv);
#pragma unroll
  for (int j = 0; j < NV; ++j) {
    const int i = lane + 32 * j;
    if (i < d4) {
      const float4 rv = load4<T>(rr + 4 * i);
      hv[j].x += rv.x; hv[j].y += rv.y; hv[j].z += rv.z; hv[j].w += rv.w;
    }
  }
  float mu, rs;
  row_stats<NV>(hv, d, d4, lane, &mu, &rs);
  modulate<NV>(hv, mu, rs, mod + (size_t)scene * mod_stride, fin_off, fin_off + d, d4, lane);
  const float vc = head_dot<NV, C>(hv, d, d4, lane, w_f, b_f);
  __syncwarp();
  if (lane < C) {
    float xo = xv[0];
#pragma unroll
    for (int c = 1; c < C; ++c)
      if (lane == c) xo = xv[c];
    const size_t xi = ((size_t)scene * N + tok) * C + lane;
    if (vout) vout[xi] = vc;
    else x[xi] = xo + dsig * vc;
  }
}

// The model's r_j = c_j - b_e - pos_t from the cache row c_j (inspection):
// out [N][d] of the cache type.
template <typename T>
__global__ void cache_to_residual_kernel(const T* __restrict__ c, const float* __restrict__ b_e,
                                         const T* __restrict__ pos, int N, int d, T* __restrict__ out) {
  const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (size_t)N * d) return;
  const int e = (int)(i % d);
  out[i] = from_f<T>(to_f<T>(c[i]) - b_e[e] - to_f<T>(pos[i]));
}

// Guidance: x_s += dsig (v_u + g (v_c - v_u)) with v_c = v[s], v_u = v[B + s].
__global__ void cfg_combine_kernel(float* __restrict__ x, const float* __restrict__ v, int B,
                                   size_t per_scene, float g, float dsig) {
  const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (size_t)B * per_scene) return;
  const float vc = v[i], vu = v[(size_t)B * per_scene + i];
  x[i] = x[i] + dsig * (vu + g * (vc - vu));
}

// ------------------------------------------------------------ drift sums

// Drift sums in Gram form: with u_t = x_t W_e^T + g_t (g_t = b_e + pos_t),
//   ||u_t - u'_t||^2 = dx_t^T G dx_t,   ||u_t||^2 = x_t^T G x_t + 2 x_t . gp_t + gs_t
// where G = W_e^T W_e [C][C], gp_t = W_e^T g_t and gs_t = ||g_t||^2 are fixed
// tables of the model.  One thread per token, fixed token-to-thread mapping
// and fixed reduction trees: the sums are deterministic.
template <int C>
__global__ void drift_partial_kernel(DriftItems items, const float* __restrict__ gram,
                                     const float* __restrict__ gp, const float* __restrict__ gs,
                                     int N, float* __restrict__ partials) {
  __shared__ float sG[C * C];
  __shared__ float red[32][2];
  for (int i = threadIdx.x; i < C * C; i += blockDim.x) sG[i] = gram[i];
  __syncthreads();
  const int part = blockIdx.x, item = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nw = blockDim.x >> 5;
  const int per = (N + kDriftParts - 1) / kDriftParts;
  const int t0 = part * per, t1 = min(N, t0 + per);
  const float4* xn = reinterpret_cast<const float4*>(items.now[item]);
  const float4* xr = reinterpret_cast<const float4*>(items.ref[item]);
  float sd = 0.f, su = 0.f;
  for (int t = t0 + (int)threadIdx.x; t < t1; t += blockDim.x) {
    float xv[C], dv[C], gv[C];
#pragma unroll
    for (int c = 0; c < C / 4; ++c) {
      const float4 a = __ldg(xn + (size_t)t * (C / 4) + c);
      const float4 b = __ldg(xr + (size_t)t * (C / 4) + c);
      const float4 g = __ldg(reinterpret_cast<const float4*>(gp) + (size_t)t * (C / 4) + c);
      xv[4 * c] = a.x; xv[4 * c + 1] = a.y; xv[4 * c + 2] = a.z; xv[4 * c + 3] = a.w;
      dv[4 * c] = a.x - b.x; dv[4 * c + 1] = a.y - b.y; dv[4 * c + 2] = a.z - b.z;
      dv[4 * c + 3] = a.w - b.w;
      gv[4 * c] = g.x; gv[4 * c + 1] = g.y; gv[4 * c + 2] = g.z; gv[4 * c + 3] = g.w;
    }
    float qd = 0.f, qx = 0.f, lin = 0.f;
#pragma unroll
    for (int a = 0; a < C; ++a) {
      float md = 0.f, mx = 0.f;
#pragma unroll
      for (int b = 0; b < C; ++b) {
        md += sG[a * C + b] * dv[b];
        mx += sG[a * C + b] * xv[b];
      }
      qd += dv[a] * md;
      qx += xv[a] * mx;
      lin += xv[a] * gv[a];
    }
    sd += qd;
    su += qx + 2.f * lin + __ldg(gs + t);
  }
  sd = warp_sum(sd);
  su = warp_sum(su);
  if (lane == 0) { red[warp][0] = sd; red[warp][1] = su; }
  __syncthreads();
  if (threadIdx.x == 0) {
    float a = 0.f, b = 0.f;
    for (int w = 0; w < nw; ++w) { a += red[w][0]; b += red[w][1]; }
    partials[((size_t)item * kDriftParts + part) * 2 + 0] = a;
    partials[((size_t)item * kDriftParts + part) * 2 + 1] = b;
  }
}

__global__ void drift_final_kernel(const float* __restrict__ partials, int n, float* __restrict__ out) {
  const int item = blockIdx.x * blockDim.x + threadIdx.x;
  if (item >= n) return;
  float a = 0.f, b = 0.f;
  for (int p = 0; p < kDriftParts; ++p) {
    a += partials[((size_t)item * kDriftParts + p) * 2 + 0];
    b += partials[((size_t)item * kDriftParts + p) * 2 + 1];
  }
  out[2 * item] = a;
  out[2 * item + 1] = b;
}

int nv_for(int d) {
  const int need = (d / 4 + 31) / 32;
  const int opts[] = {1, 2, 3, 4, 6, 8, 9, 12, 16, 24};
  for (int o : opts)
    if (o >= need) return o;
  return -1;
}

#define DC_NV_SWITCH(nv, ...)                        \
  switch (nv) {                                      \
    case 1: { constexpr int NV = 1; __VA_ARGS__; } break;   \
    case 2: { constexpr int NV = 2; __VA_ARGS__; } break;   \
    case 3: { constexpr int NV = 3; __VA_ARGS__; } break;   \
    case 4: { constexpr int NV = 4; __VA_ARGS__; } break;   \
    case 6: { constexpr int NV = 6; __VA_ARGS__; } break;   \
    case 8: { constexpr int NV = 8; __VA_ARGS__; } break;   \
    case 9: { constexpr int NV = 9; __VA_ARGS__; } break;   \
    case 12: { constexpr int NV = 12; __VA_ARGS__; } break; \
    case 16: { constexpr int NV = 16; __VA_ARGS__; } break; \
    case 24: { constexpr int NV = 24; __VA_ARGS__; } break; \
    default: return cudaErrorInvalidValue;           \
  }

}  // namespace

cudaError_t launch_pose_features(const double* poses, int B, int P, float* out, cudaStream_t st) {
  const int n = B * P;
  pose_features_kernel<<<(n + 127) / 128, 128, 0, st>>>(poses, B, P, out);
  return cudaGetLastError();
}

cudaError_t launch_temb_features(const double* sigmas, int K, float* out, cudaStream_t st) {
  temb_features_kernel<<<K, 128, 0, st>>>(sigmas, K, out);
  return cudaGetLastError();
}

template <typename TW>
cudaError_t launch_rows_linear(const float* X, int R, int I, const TW* W, const float* b, int O,
                               float* Y, int in_silu, cudaStream_t st) {
  if (R <= 0 || O <= 0) return cudaSuccess;
  const dim3 grid((unsigned)((O + kRlCols - 1) / kRlCols), (unsigned)((R + kRlRows - 1) / kRlRows));
  rows_linear_kernel<TW><<<grid, 256, 0, st>>>(X, R, I, W, b, O, Y, in_silu);
  return cudaGetLastError();
}
template cudaError_t launch_rows_linear<float>(const float*, int, int, const float*, const float*,
                                               int, float*, int, cudaStream_t);
template cudaError_t launch_rows_linear<__nv_bfloat16>(const float*, int, int, const __nv_bfloat16*,
                                                       const float*, int, float*, int, cudaStream_t);

cudaError_t launch_cond_combine(const float* temb, const float* traj, int K, int B, int d,
                                float* silu_c, cudaStream_t st) {
  const size_t n = (size_t)K * B * d;
  cond_combine_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(temb, traj, K, B, d, silu_c);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_embed(const float* x, const float* w_eT, const float* b_e, const T* pos,
                         const SlotMap& map, int N, int C, int d, float* u, cudaStream_t st) {
  if (map.n <= 0) return cudaSuccess;
  const size_t groups = ((size_t)map.n * N + kEmbedRows - 1) / kEmbedRows;
  const unsigned blocks = (unsigned)((groups * (d / 4) + 255) / 256);
  if (C == 16)
    return launch_pdl(embed_kernel<T, 16>, dim3(blocks), dim3(256), 0, st, x, w_eT, b_e, pos, map,
                      N, d, u);
  if (C == 4)
    return launch_pdl(embed_kernel<T, 4>, dim3(blocks), dim3(256), 0, st, x, w_eT, b_e, pos, map,
                      N, d, u);
  return cudaErrorInvalidValue;
}
template cudaError_t launch_embed<float>(const float*, const float*, const float*, const float*,
                                         const SlotMap&, int, int, int, float*, cudaStream_t);
template cudaError_t launch_embed<__nv_bfloat16>(const float*, const float*, const float*,
                                                 const __nv_bfloat16*, const SlotMap&, int, int,
                                                 int, float*, cudaStream_t);

template <typename T>
cudaError_t launch_ln_mod(const float* h, int rows, int N, int d, const float* mod, int mod_stride,
                          int shift_off, int scale_off, const SlotMap& map, T* a, cudaStream_t st) {
  if (rows <= 0) return cudaSuccess;
  const int threads = 256;
  const int blocks = (int)(((size_t)rows * 32 + threads - 1) / threads);
  DC_NV_SWITCH(nv_for(d), return launch_pdl(ln_mod_kernel<T, NV>, dim3(blocks), dim3(threads),
                                             ln_stage(NV) ? (size_t)2 * d * sizeof(float) : 0, st,
                                             h, rows, N, d, mod, mod_stride, shift_off, scale_off,
                                             map, a));
  return cudaGetLastError();
}
template cudaError_t launch_ln_mod<float>(const float*, int, int, int, const float*, int, int, int,
                                          const SlotMap&, float*, cudaStream_t);
template cudaError_t launch_ln_mod<__nv_bfloat16>(const float*, int, int, int, const float*, int,
                                                  int, int, const SlotMap&, __nv_bfloat16*,
                                                  cudaStream_t);

template <typename T>
cudaError_t launch_final_compute(const float* hL, const float* w_eT, float* x, float* xj, T* r,
                                 const SlotMap& map, int N, int C, int d, const float* mod,
                                 int mod_stride, int fin_off, const float* w_f, const float* b_f,
                                 float dsig, cudaStream_t st, float* vout) {
  if (map.n <= 0) return cudaSuccess;
  const int rows = map.n * N;
  const int threads = 256;
  const int blocks = (int)(((size_t)rows * 32 + threads - 1) / threads);
  if (C == 16) {
    DC_NV_SWITCH(nv_for(d), return launch_pdl(final_compute_kernel<T, NV, 16>, dim3(blocks),
                                               dim3(threads), 0, st, hL, w_eT, x, xj, r, map, N, d,
                                               mod, mod_stride, fin_off, w_f, b_f, dsig, vout));
  } else if (C == 4) {
    DC_NV_SWITCH(nv_for(d), return launch_pdl(final_compute_kernel<T, NV, 4>, dim3(blocks),
                                               dim3(threads), 0, st, hL, w_eT, x, xj, r, map, N, d,
                                               mod, mod_stride, fin_off, w_f, b_f, dsig, vout));
  } else {
    return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}
template cudaError_t launch_final_compute<float>(const float*, const float*, float*, float*, float*,
                                                 const SlotMap&, int, int, int, const float*, int,
                                                 int, const float*, const float*, float, cudaStream_t,
                                                 float*);
template cudaError_t launch_final_compute<__nv_bfloat16>(const float*, const float*, float*, float*,
                                                         __nv_bfloat16*, const SlotMap&, int, int,
                                                         int, const float*, int, int, const float*,
                                                         const float*, float, cudaStream_t, float*);

template <typename T>
cudaError_t launch_final_reuse(float* x, const T* r, const float* w_eT, const SlotMap& map, int N,
                               int C, int d, const float* mod, int mod_stride, int fin_off,
                               const float* w_f, const float* b_f, float dsig, cudaStream_t st,
                               float* vout) {
  if (map.n <= 0) return cudaSuccess;
  const int rows = map.n * N;
  const int threads = 256;
  const int blocks = (int)(((size_t)rows * 32 + threads - 1) / threads);
  if (C == 16) {
    DC_NV_SWITCH(nv_for(d), return launch_pdl(final_reuse_kernel<T, NV, 16>, dim3(blocks),
                                               dim3(threads), 0, st, x, r, w_eT, map, N, d, mod,
                                               mod_stride, fin_off, w_f, b_f, dsig, vout));
  } else if (C == 4) {
    DC_NV_SWITCH(nv_for(d), return launch_pdl(final_reuse_kernel<T, NV, 4>, dim3(blocks),
                                               dim3(threads), 0, st, x, r, w_eT, map, N, d, mod,
                                               mod_stride, fin_off, w_f, b_f, dsig, vout));
  } else {
    return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}
template cudaError_t launch_final_reuse<float>(float*, const float*, const float*, const SlotMap&,
                                               int, int, int, const float*, int, int, const float*,
                                               const float*, float, cudaStream_t, float*);
template cudaError_t launch_final_reuse<__nv_bfloat16>(float*, const __nv_bfloat16*, const float*,
                                                       const SlotMap&, int, int, int, const float*,
                                                       int, int, const float*, const float*, float,
                                                       cudaStream_t, float*);

template <typename T>
cudaError_t launch_cache_to_residual(const T* c, const float* b_e, const T* pos, int N, int d, T* out,
                                     cudaStream_t st) {
  const size_t n = (size_t)N * d;
  if (n == 0) return cudaSuccess;
  cache_to_residual_kernel<T><<<(unsigned)((n + 255) / 256), 256, 0, st>>>(c, b_e, pos, N, d, out);
  return cudaGetLastError();
}
template cudaError_t launch_cache_to_residual<float>(const float*, const float*, const float*, int,
                                                     int, float*, cudaStream_t);
template cudaError_t launch_cache_to_residual<__nv_bfloat16>(const __nv_bfloat16*, const float*,
                                                             const __nv_bfloat16*, int, int,
                                                             __nv_bfloat16*, cudaStream_t);

cudaError_t launch_cfg_combine(float* x, const float* v, int B, size_t per_scene, float g,
                               float dsig, cudaStream_t st) {
  const size_t n = (size_t)B * per_scene;
  if (n == 0) return cudaSuccess;
  cfg_combine_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(x, v, B, per_scene, g, dsig);
  return cudaGetLastError();
}

cudaError_t launch_drift(const DriftItems& items, const float* gram, const float* gp,
                         const float* gs, int N, int C, float* partials, float* out,
                         cudaStream_t st) {
  if (items.n <= 0) return cudaSuccess;
  dim3 grid(kDriftParts, items.n);
  if (C == 16) {
    drift_partial_kernel<16><<<grid, 128, 0, st>>>(items, gram, gp, gs, N, partials);
  } else if (C == 4) {
    drift_partial_kernel<4><<<grid, 128, 0, st>>>(items, gram, gp, gs, N, partials);
  } else {
    return cudaErrorInvalidValue;
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  drift_final_kernel<<<(items.n + 63) / 64, 64, 0, st>>>(partials, items.n, out);
  return cudaGetLastError();
}

}  // namespace dc
