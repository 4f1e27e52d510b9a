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
// contiguous), dqkv [T][N][3d].  Four threads per query row, each owning
// DH/4 of the head dimensions; keys in tiles of 16 with an online softmax
// (running max m, sum l) and, for the tangent, the running sums
//   b = sum w ds,  Cv = sum w ds v,  Dv = sum w dv   (w = exp(s - m))
// so that do = (Cv - (b / l) A + Dv) / l with A = sum w v.
template <int DH, bool TAN>
__global__ void __launch_bounds__(128) attn_f32_jvp_kernel(const float* __restrict__ qkv,
                                                           const float* __restrict__ dqkv, int N,
                                                           int d, float scale,
                                                           float* __restrict__ o,
                                                           float* __restrict__ dout) {
  constexpr int D4 = DH / 4, KT = 16;
  __shared__ float sK[KT][DH], sV[KT][DH], sdK[TAN ? KT : 1][DH], sdV[TAN ? KT : 1][DH];
  const int g = threadIdx.x & 3, qi = threadIdx.x >> 2;
  const int head = blockIdx.y, t = blockIdx.z;
  const int n = blockIdx.x * 32 + qi;
  const bool live = n < N;
  const size_t ld = (size_t)3 * d;
  const float* dbase = TAN ? dqkv + (size_t)t * N * ld : nullptr;
  float q[D4], dq[D4], A[D4], Cv[D4], Dv[D4];
#pragma unroll
  for (int e = 0; e < D4; ++e) {
    const int col = head * DH + g * D4 + e;
    q[e] = live ? qkv[(size_t)n * ld + col] : 0.f;
    dq[e] = (TAN && live) ? dbase[(size_t)n * ld + col] : 0.f;
    A[e] = Cv[e] = Dv[e] = 0.f;
  }
  float m = -INFINITY, l = 0.f, b = 0.f;
  for (int k0 = 0; k0 < N; k0 += KT) {
    __syncthreads();
    for (int i = threadIdx.x; i < KT * DH; i += 128) {
      const int kk = i / DH, e = i % DH, key = k0 + kk;
      const bool in = key < N;
      sK[kk][e] = in ? qkv[(size_t)key * ld + d + head * DH + e] : 0.f;
      sV[kk][e] = in ? qkv[(size_t)key * ld + 2 * d + head * DH + e] : 0.f;
      if (TAN) {
        sdK[kk][e] = in ? dbase[(size_t)key * ld + d + head * DH + e] : 0.f;
        sdV[kk][e] = in ? dbase[(size_t)key * ld + 2 * d + head * DH + e] : 0.f;
      }
    }
    __syncthreads();
    float s[KT], ds[KT];
    float tmax = -INFINITY;
#pragma unroll
    for (int kk = 0; kk < KT; ++kk) {
      float a = 0.f, da = 0.f;
#pragma unroll
      for (int e = 0; e < D4; ++e) {
        a = fmaf(q[e], sK[kk][g * D4 + e], a);
        if (TAN) da = fmaf(dq[e], sK[kk][g * D4 + e], fmaf(q[e], sdK[kk][g * D4 + e], da));
      }
      a += __shfl_xor_sync(0xffffffffu, a, 1);
      a += __shfl_xor_sync(0xffffffffu, a, 2);
      if (TAN) {
        da += __shfl_xor_sync(0xffffffffu, da, 1);
        da += __shfl_xor_sync(0xffffffffu, da, 2);
      }
      const bool in = k0 + kk < N;
      s[kk] = in ? a * scale : -INFINITY;
      ds[kk] = da * scale;
      tmax = fmaxf(tmax, s[kk]);
    }
    const float mn = fmaxf(m, tmax);
    const float c = m == -INFINITY ? 0.f : expf(m - mn);
    l *= c;
    b *= c;
#pragma unroll
    for (int e = 0; e < D4; ++e) {
      A[e] *= c;
      Cv[e] *= c;
      Dv[e] *= c;
    }
#pragma unroll
    for (int kk = 0; kk < KT; ++kk) {
      const float w = expf(s[kk] - mn);  // 0 for masked keys
      l += w;
      if (TAN) b = fmaf(w, ds[kk], b);
#pragma unroll
      for (int e = 0; e < D4; ++e) {
        const float v = sV[kk][g * D4 + e];
        A[e] = fmaf(w, v, A[e]);
        if (TAN) {
          Cv[e] = fmaf(w * ds[kk], v, Cv[e]);
          Dv[e] = fmaf(w, sdV[kk][g * D4 + e], Dv[e]);
        }
      }
    }
    m = mn;
  }
  if (!live) return;
  const float inv = 1.0f / l;
  const float beta = b * inv;
#pragma unroll
  for (int e = 0; e < D4; ++e) {
    const int col = head * DH + g * D4 + e;
    if (TAN)
      dout[((size_t)t * N + n) * d + col] = (Cv[e] - beta * A[e] + Dv[e]) * inv;
    else
      o[(size_t)n * d + col] = A[e] * inv;
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

bool attention_f32_jvp_supported(int dh) {
  return dh == 8 || dh == 16 || dh == 32 || dh == 64 || dh == 72 || dh == 128;
}

cudaError_t launch_attention_f32_jvp(const float* qkv, const float* dqkv, int N, int d, int heads,
                                     int dh, int T, float* o, float* dout, cudaStream_t st) {
  if (N <= 0) return cudaSuccess;
  const float scale = 1.0f / sqrtf((float)dh);
  const bool tan = dqkv != nullptr;
  dim3 grid((N + 31) / 32, heads, tan ? T : 1);
#define DC_ATT_JVP(DHV)                                                                     \
  if (dh == DHV) {                                                                          \
    if (tan)                                                                                \
      attn_f32_jvp_kernel<DHV, true><<<grid, 128, 0, st>>>(qkv, dqkv, N, d, scale, o, dout); \
    else                                                                                    \
      attn_f32_jvp_kernel<DHV, false><<<grid, 128, 0, st>>>(qkv, dqkv, N, d, scale, o, dout); \
    return cudaGetLastError();                                                              \
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
