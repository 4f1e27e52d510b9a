// fp32 forward-mode kernels of the synthetic DiT for the joint run responses
// (Eq. 6-7): a primal evaluation at one trace point that keeps what the
// tangents need, and the tangent (Jacobian-vector product) of the velocity
// for a batch of T perturbations of that one point.  The tangent of each op:
//   LayerNorm   y = (x - mu) / sigma,  dy = (dx - mean(dx) - y mean(y dx)) / sigma
//   attention   dS = (dq k^T + q dk^T) / sqrt(dh),  dP = P (dS - rowsum(P dS)),
//               do = dP v + P dv
//   GELU(tanh)  dm = gelu'(z) dz
//   linear      dy = dx W^T;  gated residual dh' = dh + gate (dy)
// (the modulation depends on the step and the trajectory only, so it is a
// constant of the Jacobian).  Everything accumulates in fp32 and reads the
// weights in the model's own type.  Calibration runs once per
// configuration; these kernels favour plain, checkable code over speed.
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace dc {

namespace {

constexpr int kTM = 64, kTN = 64, kTK = 16;  // GEMM tile

template <typename TW>
__device__ __forceinline__ float ldw(const TW* p) { return to_f<TW>(*p); }

__device__ __forceinline__ float gelu_f(float x) {
  const float k0 = 0.7978845608028654f, c = 0.044715f;
  return 0.5f * x * (1.0f + tanhf(k0 * (x + c * x * x * x)));
}
__device__ __forceinline__ float gelu_grad_f(float x) {
  const float k0 = 0.7978845608028654f, c = 0.044715f;
  const float t = tanhf(k0 * (x + c * x * x * x));
  return 0.5f * (1.0f + t) + 0.5f * x * (1.0f - t * t) * k0 * (1.0f + 3.0f * c * x * x);
}

// C[M][N] = A[M][K] W[N][K]^T (fp32 accumulate) + epilogue.  64 x 64 tiles,
// 256 threads with 4 x 4 outputs each; any M, N, K.
template <typename TW>
__global__ void __launch_bounds__(256) gemm_f32w_kernel(const float* __restrict__ A,
                                                        const TW* __restrict__ W, int M, int N,
                                                        int K, JEpi ep) {
  __shared__ float As[kTK][kTM + 4];
  __shared__ float Ws[kTK][kTN + 4];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const int m0 = blockIdx.y * kTM, n0 = blockIdx.x * kTN;
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
  for (int k0 = 0; k0 < K; k0 += kTK) {
    for (int i = threadIdx.x; i < kTM * kTK; i += 256) {
      const int r = i / kTK, kk = i % kTK;
      const int gr = m0 + r, gk = k0 + kk;
      As[kk][r] = (gr < M && gk < K) ? A[(size_t)gr * K + gk] : 0.f;
      const int gn = n0 + r;
      Ws[kk][r] = (gn < N && gk < K) ? ldw(W + (size_t)gn * K + gk) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < kTK; ++kk) {
      float a[4], w[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) w[j] = Ws[kk][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], w[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int r = m0 + ty * 4 + i;
    if (r >= M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int c = n0 + tx * 4 + j;
      if (c >= N) continue;
      const size_t o = (size_t)r * N + c;
      float y = acc[i][j] + (ep.bias ? ep.bias[c] : 0.f);
      switch (ep.mode) {
        case kJStore:
          ep.out[o] = y;
          break;
        case kJGatedAdd:
          ep.out[o] = ep.base[o] + ep.gate[c] * y;
          break;
        case kJGeluPrimal:
          ep.out[o] = y;              // z
          ep.out2[o] = gelu_f(y);     // gelu(z)
          break;
        case kJGeluGrad:
          ep.out[o] = gelu_grad_f(ep.z[(size_t)(r % ep.zrows) * N + c]) * y;
          break;
      }
    }
  }
}

// One warp per row: mean and variance of a d-vector (two passes, fp32).
__device__ __forceinline__ void row_stats(const float* x, int d, float* mu, float* rstd) {
  const int lane = threadIdx.x & 31;
  float s = 0.f;
  for (int i = lane; i < d; i += 32) s += x[i];
  s = warp_sum(s);
  const float m = s / d;
  float v = 0.f;
  for (int i = lane; i < d; i += 32) {
    const float t = x[i] - m;
    v = fmaf(t, t, v);
  }
  v = warp_sum(v);
  *mu = m;
  *rstd = 1.0f / sqrtf(v / d + 1e-6f);
}

// out = LN(h) (1 + scale) + shift, one warp per row.
__global__ void ln_mod_f32_kernel(const float* __restrict__ h, int R, int d,
                                  const float* __restrict__ shift, const float* __restrict__ scale,
                                  float* __restrict__ out) {
  const int row = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (row >= R) return;
  const float* x = h + (size_t)row * d;
  float mu, rs;
  row_stats(x, d, &mu, &rs);
  for (int i = threadIdx.x & 31; i < d; i += 32)
    out[(size_t)row * d + i] = (x[i] - mu) * rs * (1.0f + scale[i]) + shift[i];
}

// out[t][n] = (1 + scale) (dh - mean(dh) - y mean(y dh)) / sigma with y the
// normalised primal row n; one warp per tangent row.
__global__ void ln_jvp_f32_kernel(const float* __restrict__ h, const float* __restrict__ dh, int N,
                                  int T, int d, const float* __restrict__ scale,
                                  float* __restrict__ out) {
  const int row = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (row >= T * N) return;
  const int n = row % N;
  const float* x = h + (size_t)n * d;
  const float* dx = dh + (size_t)row * d;
  float mu, rs;
  row_stats(x, d, &mu, &rs);
  float sd = 0.f, syd = 0.f;
  for (int i = threadIdx.x & 31; i < d; i += 32) {
    sd += dx[i];
    syd = fmaf((x[i] - mu) * rs, dx[i], syd);
  }
  sd = warp_sum(sd) / d;
  syd = warp_sum(syd) / d;
  for (int i = threadIdx.x & 31; i < d; i += 32) {
    const float y = (x[i] - mu) * rs;
    out[(size_t)row * d + i] = (1.0f + scale[i]) * (dx[i] - sd - y * syd) * rs;
  }
}

// u[r][c'] = sum_c x[r][c] W_e^T[c][c'] (+ b_e[c'] + pos[r % N][c'] when primal)
template <typename TP>
__global__ void embed_f32_kernel(const float* __restrict__ x, const float* __restrict__ w_eT,
                                 const float* __restrict__ b_e, const TP* __restrict__ pos, int R,
                                 int N, int C, int d, float* __restrict__ out) {
  const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (size_t)R * d) return;
  const int r = (int)(i / d), j = (int)(i % d);
  float s = 0.f;
  for (int c = 0; c < C; ++c) s = fmaf(x[(size_t)r * C + c], w_eT[(size_t)c * d + j], s);
  if (b_e) s += b_e[j] + to_f<TP>(pos[(size_t)(r % N) * d + j]);
  out[i] = s;
}

// Attention over all tokens of the one primal scene, and (TAN) its tangent
// for T perturbations: qkv [N][3d] primal rows ([q | k | v], heads
// contiguous), dqkv [T][N][3d].  Keys stream in tiles with an online softmax
// (running max m, sum l) and, for the tangent, the running sums
//   b = sum w ds,  Cv = sum w ds v,  Dv = sum w dv   (w = exp(s - m))
// so that do = (Cv - (b / l) A + Dv) / l with A = sum w v.  A block of 128 threads
// takes BQ = 16 RQ query rows of one head (RQ = 4, or 2 at head dim 128) and
// streams the keys in tiles of 32.  Thread t owns rows rg RQ .. rg RQ + RQ-1
// (rg = t / 8) and, with g = t % 8:
//   phase 1  s and ds of its rows against keys 4g .. 4g+3 of the tile
//            (RQ x 4 register block; q, dq, k, dk read as float4 from
//            transposed tiles in shared memory);
//   phase 2  the online softmax of its rows, the tile's row max and sums
//            reduced over the 8 lanes g that share the rows; w and w ds go
//            to shared memory;
//   phase 3  A, Cv, Dv of its rows for head dimensions g, g + 8, g + 16, ...
//            (RQ x DH/8 register block over the tile's 32 keys; the eight
//            lanes g read eight consecutive banks of a value row).
// The lanes that share rows sit in one warp, so the running max m, sum l and
// b = sum w ds live in registers of the same thread in all three phases.
template <int DH, bool TAN>
struct JvpTile {
  static constexpr int RQ = DH >= 128 ? 2 : 4, BQ = 16 * RQ, BK = 32, DG = DH / 8;
  // shared memory (floats): q^T, dq^T [DH][BQ]; k^T, dk^T [DH][BK]; v, dv
  // [BK][DH]; w, w ds [BK][BQ]
  static constexpr int kQ = DH * BQ, kK = DH * BK, kW = BK * BQ;
  static constexpr int kFloats = (TAN ? 2 : 1) * (kQ + 2 * kK) + (TAN ? 2 : 1) * kW;
  static constexpr size_t kBytes = (size_t)kFloats * 4;
};

template <int DH, bool TAN>
__global__ void __launch_bounds__(128) attn_f32_jvp_tiled_kernel(
    const float* __restrict__ qkv, const float* __restrict__ dqkv, int N, int d, float scale,
    float* __restrict__ o, float* __restrict__ dout) {
  using Tl = JvpTile<DH, TAN>;
  constexpr int RQ = Tl::RQ, BQ = Tl::BQ, BK = Tl::BK, DG = Tl::DG;
  extern __shared__ float4 jvp_smem4[];
  float* sm = reinterpret_cast<float*>(jvp_smem4);
  float* sQ = sm;                                  // [DH][BQ]
  float* sK = sQ + Tl::kQ;                         // [DH][BK]
  float* sV = sK + Tl::kK;                         // [BK][DH]
  float* sdQ = sV + Tl::kK;                        // (TAN) [DH][BQ]
  float* sdK = sdQ + (TAN ? Tl::kQ : 0);           // (TAN) [DH][BK]
  float* sdV = sdK + (TAN ? Tl::kK : 0);           // (TAN) [BK][DH]
  float* sW = sdV + (TAN ? Tl::kK : 0);            // [BK][BQ]
  float* sWd = sW + Tl::kW;                        // (TAN) [BK][BQ]
  const int tid = threadIdx.x, rg = tid >> 3, g = tid & 7;
  const int head = blockIdx.y, t = blockIdx.z;
  const int q0 = blockIdx.x * BQ;
  const size_t ld = (size_t)3 * d;
  const float* dbase = TAN ? dqkv + (size_t)t * N * ld : nullptr;
  constexpr int D4 = DH / 4;
  // queries of the block, transposed (row index fastest across threads, so
  // the transposed stores hit distinct banks)
  for (int i = tid; i < BQ * D4; i += 128) {
    const int r = i % BQ, e4 = i / BQ, n = q0 + r;
    const bool in = n < N;
    const size_t at = (size_t)n * ld + head * DH + 4 * e4;
    const float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
    const float4 a = in ? *reinterpret_cast<const float4*>(qkv + at) : z;
    sQ[(4 * e4 + 0) * BQ + r] = a.x; sQ[(4 * e4 + 1) * BQ + r] = a.y;
    sQ[(4 * e4 + 2) * BQ + r] = a.z; sQ[(4 * e4 + 3) * BQ + r] = a.w;
    if (TAN) {
      const float4 da = in ? *reinterpret_cast<const float4*>(dbase + at) : z;
      sdQ[(4 * e4 + 0) * BQ + r] = da.x; sdQ[(4 * e4 + 1) * BQ + r] = da.y;
      sdQ[(4 * e4 + 2) * BQ + r] = da.z; sdQ[(4 * e4 + 3) * BQ + r] = da.w;
    }
  }
  float A[RQ][DG], Cv[RQ][DG], Dv[RQ][DG];
#pragma unroll
  for (int r = 0; r < RQ; ++r)
#pragma unroll
    for (int e = 0; e < DG; ++e) A[r][e] = Cv[r][e] = Dv[r][e] = 0.f;
  float m[RQ], l[RQ], b[RQ];
#pragma unroll
  for (int r = 0; r < RQ; ++r) { m[r] = -INFINITY; l[r] = 0.f; b[r] = 0.f; }

  for (int k0 = 0; k0 < N; k0 += BK) {
    __syncthreads();  // the previous tile's k, v, w are consumed
    const float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int i = tid; i < BK * D4; i += 128) {
      // k, dk transposed: key index fastest across threads
      const int j = i % BK, e4 = i / BK, key = k0 + j;
      const bool in = key < N;
      const size_t at = (size_t)key * ld + d + head * DH + 4 * e4;
      const float4 a = in ? *reinterpret_cast<const float4*>(qkv + at) : z;
      sK[(4 * e4 + 0) * BK + j] = a.x; sK[(4 * e4 + 1) * BK + j] = a.y;
      sK[(4 * e4 + 2) * BK + j] = a.z; sK[(4 * e4 + 3) * BK + j] = a.w;
      if (TAN) {
        const float4 da = in ? *reinterpret_cast<const float4*>(dbase + at) : z;
        sdK[(4 * e4 + 0) * BK + j] = da.x; sdK[(4 * e4 + 1) * BK + j] = da.y;
        sdK[(4 * e4 + 2) * BK + j] = da.z; sdK[(4 * e4 + 3) * BK + j] = da.w;
      }
    }
    for (int i = tid; i < BK * D4; i += 128) {
      // v, dv as rows: head dimension fastest
      const int e4 = i % D4, j = i / D4, key = k0 + j;
      const bool in = key < N;
      const size_t at = (size_t)key * ld + 2 * (size_t)d + head * DH + 4 * e4;
      *reinterpret_cast<float4*>(sV + j * DH + 4 * e4) =
          in ? *reinterpret_cast<const float4*>(qkv + at) : z;
      if (TAN)
        *reinterpret_cast<float4*>(sdV + j * DH + 4 * e4) =
            in ? *reinterpret_cast<const float4*>(dbase + at) : z;
    }
    __syncthreads();
    // phase 1: s, ds for rows rg RQ + r and keys 4 g + c
    float s[RQ][4], ds[RQ][4];
#pragma unroll
    for (int r = 0; r < RQ; ++r)
#pragma unroll
      for (int c = 0; c < 4; ++c) s[r][c] = ds[r][c] = 0.f;
#pragma unroll 4
    for (int e = 0; e < DH; ++e) {
      float qv[RQ], dqv[RQ];
      if constexpr (RQ == 4) {
        const float4 a = *reinterpret_cast<const float4*>(sQ + e * BQ + rg * 4);
        qv[0] = a.x; qv[1] = a.y; qv[2] = a.z; qv[3] = a.w;
        if (TAN) {
          const float4 da = *reinterpret_cast<const float4*>(sdQ + e * BQ + rg * 4);
          dqv[0] = da.x; dqv[1] = da.y; dqv[2] = da.z; dqv[3] = da.w;
        }
      } else {
        const float2 a = *reinterpret_cast<const float2*>(sQ + e * BQ + rg * 2);
        qv[0] = a.x; qv[1] = a.y;
        if (TAN) {
          const float2 da = *reinterpret_cast<const float2*>(sdQ + e * BQ + rg * 2);
          dqv[0] = da.x; dqv[1] = da.y;
        }
      }
      const float4 kv = *reinterpret_cast<const float4*>(sK + e * BK + g * 4);
      const float kk[4] = {kv.x, kv.y, kv.z, kv.w};
      float dkk[4] = {0.f, 0.f, 0.f, 0.f};
      if (TAN) {
        const float4 dk = *reinterpret_cast<const float4*>(sdK + e * BK + g * 4);
        dkk[0] = dk.x; dkk[1] = dk.y; dkk[2] = dk.z; dkk[3] = dk.w;
      }
#pragma unroll
      for (int r = 0; r < RQ; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          s[r][c] = fmaf(qv[r], kk[c], s[r][c]);
          if (TAN) ds[r][c] = fmaf(dqv[r], kk[c], fmaf(qv[r], dkk[c], ds[r][c]));
        }
    }
    // phase 2: online softmax over the tile's 32 keys of each row
#pragma unroll
    for (int r = 0; r < RQ; ++r) {
      float tmax = -INFINITY;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const bool in = k0 + g * 4 + c < N;
        s[r][c] = in ? s[r][c] * scale : -INFINITY;
        ds[r][c] *= scale;
        tmax = fmaxf(tmax, s[r][c]);
      }
      tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 1));
      tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 2));
      tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 4));
      const float mn = fmaxf(m[r], tmax);
      const float cf = m[r] == -INFINITY ? 0.f : expf(m[r] - mn);
      float ls = 0.f, bs = 0.f;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const float w = expf(s[r][c] - mn);  // 0 for masked keys
        ls += w;
        sW[(g * 4 + c) * BQ + rg * RQ + r] = w;
        if (TAN) {
          bs = fmaf(w, ds[r][c], bs);
          sWd[(g * 4 + c) * BQ + rg * RQ + r] = w * ds[r][c];
        }
      }
      ls += __shfl_xor_sync(0xffffffffu, ls, 1);
      ls += __shfl_xor_sync(0xffffffffu, ls, 2);
      ls += __shfl_xor_sync(0xffffffffu, ls, 4);
      l[r] = l[r] * cf + ls;
      if (TAN) {
        bs += __shfl_xor_sync(0xffffffffu, bs, 1);
        bs += __shfl_xor_sync(0xffffffffu, bs, 2);
        bs += __shfl_xor_sync(0xffffffffu, bs, 4);
        b[r] = b[r] * cf + bs;
      }
      m[r] = mn;
#pragma unroll
      for (int e = 0; e < DG; ++e) {
        A[r][e] *= cf;
        if (TAN) { Cv[r][e] *= cf; Dv[r][e] *= cf; }
      }
    }
    __syncwarp();  // w of the 8 lanes g is in shared memory (one warp owns these rows)
    // phase 3: accumulate over the tile's keys
#pragma unroll 2
    for (int j = 0; j < BK; ++j) {
      float wv[RQ], wdv[RQ];
#pragma unroll
      for (int r = 0; r < RQ; ++r) {
        wv[r] = sW[j * BQ + rg * RQ + r];
        if (TAN) wdv[r] = sWd[j * BQ + rg * RQ + r];
      }
#pragma unroll
      for (int e = 0; e < DG; ++e) {
        const float v = sV[j * DH + g + 8 * e];
        const float dv = TAN ? sdV[j * DH + g + 8 * e] : 0.f;
#pragma unroll
        for (int r = 0; r < RQ; ++r) {
          A[r][e] = fmaf(wv[r], v, A[r][e]);
          if (TAN) {
            Cv[r][e] = fmaf(wdv[r], v, Cv[r][e]);
            Dv[r][e] = fmaf(wv[r], dv, Dv[r][e]);
          }
        }
      }
    }
  }
#pragma unroll
  for (int r = 0; r < RQ; ++r) {
    const int n = q0 + rg * RQ + r;
    if (n >= N) continue;
    const float inv = 1.0f / l[r];
    const float beta = b[r] * inv;
#pragma unroll
    for (int e = 0; e < DG; ++e) {
      const int col = head * DH + g + 8 * e;
      if (TAN)
        dout[((size_t)t * N + n) * d + col] = (Cv[r][e] - beta * A[r][e] + Dv[r][e]) * inv;
      else
        o[(size_t)n * d + col] = A[r][e] * inv;
    }
  }
}

// y[i] += a x[i]
__global__ void axpy_f32_kernel(float* __restrict__ y, const float* __restrict__ x, float a,
                                size_t n) {
  const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) y[i] = fmaf(a, x[i], y[i]);
}

// out[i] = a[i] + r[i] (r in the cache type)
template <typename T>
__global__ void add_cache_kernel(const float* __restrict__ a, const T* __restrict__ r,
                                 float* __restrict__ out, size_t n) {
  const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) out[i] = a[i] + to_f<T>(r[i]);
}

// out[i] = s (a[i] - b[i])
__global__ void scaled_diff_kernel(const float* __restrict__ a, const float* __restrict__ b,
                                   float s, float* __restrict__ out, size_t n) {
  const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) out[i] = s * (a[i] - b[i]);
}

unsigned blocks_for(size_t n, int per) { return (unsigned)((n + per - 1) / per); }

}  // namespace

template <typename TW>
cudaError_t launch_gemm_f32w(const float* A, const TW* W, int M, int N, int K, const JEpi& ep,
                             cudaStream_t st) {
  if (M <= 0 || N <= 0) return cudaSuccess;
  dim3 grid((N + kTN - 1) / kTN, (M + kTM - 1) / kTM);
  gemm_f32w_kernel<TW><<<grid, 256, 0, st>>>(A, W, M, N, K, ep);
  return cudaGetLastError();
}
template cudaError_t launch_gemm_f32w<float>(const float*, const float*, int, int, int, const JEpi&,
                                             cudaStream_t);
template cudaError_t launch_gemm_f32w<__nv_bfloat16>(const float*, const __nv_bfloat16*, int, int,
                                                     int, const JEpi&, cudaStream_t);

cudaError_t launch_ln_mod_f32(const float* h, int R, int d, const float* shift, const float* scale,
                              float* out, cudaStream_t st) {
  if (R <= 0) return cudaSuccess;
  ln_mod_f32_kernel<<<blocks_for(R, 8), 256, 0, st>>>(h, R, d, shift, scale, out);
  return cudaGetLastError();
}

cudaError_t launch_ln_jvp_f32(const float* h, const float* dh, int N, int T, int d,
                              const float* scale, float* out, cudaStream_t st) {
  if (N <= 0 || T <= 0) return cudaSuccess;
  ln_jvp_f32_kernel<<<blocks_for((size_t)N * T, 8), 256, 0, st>>>(h, dh, N, T, d, scale, out);
  return cudaGetLastError();
}

template <typename TP>
cudaError_t launch_embed_f32(const float* x, const float* w_eT, const float* b_e, const TP* pos,
                             int R, int N, int C, int d, float* out, cudaStream_t st) {
  if (R <= 0) return cudaSuccess;
  embed_f32_kernel<TP><<<blocks_for((size_t)R * d, 256), 256, 0, st>>>(x, w_eT, b_e, pos, R, N, C,
                                                                       d, out);
  return cudaGetLastError();
}
template cudaError_t launch_embed_f32<float>(const float*, const float*, const float*,
                                             const float*, int, int, int, int, float*,
                                             cudaStream_t);
template cudaError_t launch_embed_f32<__nv_bfloat16>(const float*, const float*, const float*,
                                                     const __nv_bfloat16*, int, int, int, int,
                                                     float*, cudaStream_t);

namespace {
template <int DH, bool TAN>
cudaError_t launch_jvp_tiled(const float* qkv, const float* dqkv, int N, int d, int heads, int T,
                             float scale, float* o, float* dout, cudaStream_t st) {
  using Tl = JvpTile<DH, TAN>;
  static std::atomic<unsigned long long> configured{0};
  const cudaError_t e = configure_once_per_device(configured, [] {
    return cudaFuncSetAttribute(attn_f32_jvp_tiled_kernel<DH, TAN>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Tl::kBytes);
  });
  if (e != cudaSuccess) return e;
  dim3 grid((N + Tl::BQ - 1) / Tl::BQ, heads, T);
  attn_f32_jvp_tiled_kernel<DH, TAN><<<grid, 128, Tl::kBytes, st>>>(qkv, dqkv, N, d, scale, o, dout);
  return cudaGetLastError();
}
}  // namespace

bool attention_f32_jvp_supported(int dh) {
  return dh == 8 || dh == 16 || dh == 32 || dh == 64 || dh == 72 || dh == 128;
}

cudaError_t launch_attention_f32_jvp(const float* qkv, const float* dqkv, int N, int d, int heads,
                                     int dh, int T, float* o, float* dout, cudaStream_t st) {
  if (N <= 0) return cudaSuccess;
  const float scale = 1.0f / sqrtf((float)dh);
  const bool tan = dqkv != nullptr;
#define DC_ATT_JVP(DHV)                                                                      \
  if (dh == DHV) {                                                                           \
    if (tan) return launch_jvp_tiled<DHV, true>(qkv, dqkv, N, d, heads, T, scale, o, dout, st); \
    return launch_jvp_tiled<DHV, false>(qkv, dqkv, N, d, heads, 1, scale, o, dout, st);       \
  }
  DC_ATT_JVP(8)
  DC_ATT_JVP(16)
  DC_ATT_JVP(32)
  DC_ATT_JVP(64)
  DC_ATT_JVP(72)
  DC_ATT_JVP(128)
#undef DC_ATT_JVP
  return cudaErrorInvalidValue;
}

cudaError_t launch_axpy_f32(float* y, const float* x, float a, size_t n, cudaStream_t st) {
  if (n == 0) return cudaSuccess;
  axpy_f32_kernel<<<blocks_for(n, 256), 256, 0, st>>>(y, x, a, n);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_add_cache(const float* a, const T* r, float* out, size_t n, cudaStream_t st) {
  if (n == 0) return cudaSuccess;
  add_cache_kernel<T><<<blocks_for(n, 256), 256, 0, st>>>(a, r, out, n);
  return cudaGetLastError();
}
template cudaError_t launch_add_cache<float>(const float*, const float*, float*, size_t,
                                             cudaStream_t);
template cudaError_t launch_add_cache<__nv_bfloat16>(const float*, const __nv_bfloat16*, float*,
                                                     size_t, cudaStream_t);

cudaError_t launch_scaled_diff(const float* a, const float* b, float s, float* out, size_t n,
                               cudaStream_t st) {
  if (n == 0) return cudaSuccess;
  scaled_diff_kernel<<<blocks_for(n, 256), 256, 0, st>>>(a, b, s, out, n);
  return cudaGetLastError();
}

}  // namespace dc
