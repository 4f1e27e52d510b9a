// Full (non-causal) spatiotemporal self-attention of the DiT block:
// o = softmax(q k^T / sqrt(dh)) v over all N tokens of a scene, per head.
//
// bf16 path: flash-style streaming over 64-key tiles (online softmax in
// fp32, exp2 with the log2(e)/sqrt(dh) scale folded in), bf16 operands on
// the warp-level tensor-core MMA (m16n8k16), K/V tiles double-buffered with
// cp.async.  64 query rows per CTA (16 per warp).  The head dimension is
// padded to dhp (a multiple of 16; the pad columns of q/k/v are zero) and
// keys beyond N are masked, so any N works.
//
// fp32 path: one warp per query row, SIMT FMA, online softmax per lane then
// a warp merge; dh <= 64.
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace dc {

namespace {

constexpr int kQ = 64;      // query rows per CTA
constexpr int kKV = 64;     // keys per tile
constexpr int kWarps = 4;

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, bool pred) {
  const int n = pred ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(smem)), "l"(gmem),
               "r"(n)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void mma_bf16(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9},"
      " {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 t = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&t);
}

template <int DHP>
__global__ void __launch_bounds__(kWarps * 32)
    attn_bf16_kernel(const __nv_bfloat16* __restrict__ qkv, int slots, int heads, int N, int dh,
                     __nv_bfloat16* __restrict__ o, float scale_log2) {
  constexpr int LD = DHP + 8;  // padded smem row (bank-conflict-free ldmatrix)
  constexpr int CH = DHP / 8;  // 16-byte chunks per row
  extern __shared__ __align__(16) uint8_t smem_raw[];
  __nv_bfloat16* sQ = reinterpret_cast<__nv_bfloat16*>(smem_raw);
  __nv_bfloat16* sK = sQ + kQ * LD;           // [2][kKV][LD]
  __nv_bfloat16* sV = sK + 2 * kKV * LD;      // [2][kKV][LD]

  const int bh = blockIdx.y;  // slot * heads + head
  const int slot = bh / heads, head = bh - slot * heads;
  const int q0 = blockIdx.x * kQ;
  const size_t plane = (size_t)N * DHP;
  const __nv_bfloat16* Qg = qkv + ((size_t)(0 * slots + slot) * heads + head) * plane;
  const __nv_bfloat16* Kg = qkv + ((size_t)(1 * slots + slot) * heads + head) * plane;
  const __nv_bfloat16* Vg = qkv + ((size_t)(2 * slots + slot) * heads + head) * plane;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  for (int c = tid; c < kQ * CH; c += kWarps * 32) {
    const int r = c / CH, cc = c - r * CH;
    const bool ok = q0 + r < N;
    cp_async16(sQ + r * LD + cc * 8, Qg + (size_t)(ok ? q0 + r : 0) * DHP + cc * 8, ok);
  }
  auto load_kv = [&](int tile, int buf) {
    const int k0 = tile * kKV;
    for (int c = tid; c < kKV * CH; c += kWarps * 32) {
      const int r = c / CH, cc = c - r * CH;
      const bool ok = k0 + r < N;
      const size_t g = (size_t)(ok ? k0 + r : 0) * DHP + cc * 8;
      cp_async16(sK + (buf * kKV + r) * LD + cc * 8, Kg + g, ok);
      cp_async16(sV + (buf * kKV + r) * LD + cc * 8, Vg + g, ok);
    }
  };
  const int n_tiles = (N + kKV - 1) / kKV;
  load_kv(0, 0);
  cp_async_commit();

  // Q fragments of this warp's 16 rows
  uint32_t qf[DHP / 16][4];
  float oacc[DHP / 8][4];
#pragma unroll
  for (int i = 0; i < DHP / 8; ++i) oacc[i][0] = oacc[i][1] = oacc[i][2] = oacc[i][3] = 0.f;
  float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};

  for (int t = 0; t < n_tiles; ++t) {
    if (t + 1 < n_tiles) load_kv(t + 1, (t + 1) & 1);
    cp_async_commit();
    cp_async_wait<1>();
    __syncthreads();
    if (t == 0) {
#pragma unroll
      for (int ks = 0; ks < DHP / 16; ++ks) {
        const int i = lane >> 3, r = lane & 7;
        const int row = warp * 16 + (i & 1) * 8 + r;
        const int col = ks * 16 + (i >> 1) * 8;
        ldsm_x4(smem_u32(sQ + row * LD + col), qf[ks][0], qf[ks][1], qf[ks][2], qf[ks][3]);
      }
    }
    const int buf = t & 1;
    const __nv_bfloat16* Kt = sK + buf * kKV * LD;
    const __nv_bfloat16* Vt = sV + buf * kKV * LD;

    float s[kKV / 8][4];
#pragma unroll
    for (int i = 0; i < kKV / 8; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < DHP / 16; ++ks) {
#pragma unroll
      for (int np = 0; np < kKV / 16; ++np) {
        const int i = lane >> 3, r = lane & 7;
        const int key = np * 16 + (i >> 1) * 8 + r;
        const int col = ks * 16 + (i & 1) * 8;
        uint32_t b0, b1, b2, b3;
        ldsm_x4(smem_u32(Kt + key * LD + col), b0, b1, b2, b3);
        mma_bf16(s[2 * np], qf[ks], b0, b1);
        mma_bf16(s[2 * np + 1], qf[ks], b2, b3);
      }
    }
    // scale, mask, online softmax (rows lane/4 and lane/4 + 8 of the warp)
    const int kbase = t * kKV + (lane & 3) * 2;
    float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int nt = 0; nt < kKV / 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = kbase + nt * 8 + (e & 1);
        float v = s[nt][e] * scale_log2;
        if (key >= N) v = -INFINITY;
        s[nt][e] = v;
        mx[e >> 1] = fmaxf(mx[e >> 1], v);
      }
    }
    float corr[2];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      mx[h] = fmaxf(mx[h], __shfl_xor_sync(0xffffffffu, mx[h], 1));
      mx[h] = fmaxf(mx[h], __shfl_xor_sync(0xffffffffu, mx[h], 2));
      const float m_new = fmaxf(m_run[h], mx[h]);
      corr[h] = exp2f(m_run[h] - m_new);
      m_run[h] = m_new;
    }
    float rs[2] = {0.f, 0.f};
#pragma unroll
    for (int nt = 0; nt < kKV / 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float p = exp2f(s[nt][e] - m_run[e >> 1]);
        s[nt][e] = p;
        rs[e >> 1] += p;
      }
    }
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      rs[h] += __shfl_xor_sync(0xffffffffu, rs[h], 1);
      rs[h] += __shfl_xor_sync(0xffffffffu, rs[h], 2);
      l_run[h] = l_run[h] * corr[h] + rs[h];
    }
#pragma unroll
    for (int i = 0; i < DHP / 8; ++i) {
      oacc[i][0] *= corr[0]; oacc[i][1] *= corr[0];
      oacc[i][2] *= corr[1]; oacc[i][3] *= corr[1];
    }
    // O += P V
#pragma unroll
    for (int kk = 0; kk < kKV / 16; ++kk) {
      uint32_t pa[4];
      pa[0] = pack_bf16(s[2 * kk][0], s[2 * kk][1]);
      pa[1] = pack_bf16(s[2 * kk][2], s[2 * kk][3]);
      pa[2] = pack_bf16(s[2 * kk + 1][0], s[2 * kk + 1][1]);
      pa[3] = pack_bf16(s[2 * kk + 1][2], s[2 * kk + 1][3]);
#pragma unroll
      for (int dp = 0; dp < DHP / 16; ++dp) {
        const int i = lane >> 3, r = lane & 7;
        const int key = kk * 16 + (i & 1) * 8 + r;
        const int col = dp * 16 + (i >> 1) * 8;
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(smem_u32(Vt + key * LD + col), b0, b1, b2, b3);
        mma_bf16(oacc[2 * dp], pa, b0, b1);
        mma_bf16(oacc[2 * dp + 1], pa, b2, b3);
      }
    }
    __syncthreads();
  }
  cp_async_wait<0>();

  const float inv0 = 1.f / l_run[0], inv1 = 1.f / l_run[1];
  const int d = heads * dh;
  const int r0 = q0 + warp * 16 + (lane >> 2);
#pragma unroll
  for (int nt = 0; nt < DHP / 8; ++nt) {
    const int c = nt * 8 + (lane & 3) * 2;
    if (c < dh) {
      if (r0 < N) {
        __nv_bfloat162 v = __floats2bfloat162_rn(oacc[nt][0] * inv0, oacc[nt][1] * inv0);
        *reinterpret_cast<__nv_bfloat162*>(o + ((size_t)slot * N + r0) * d + head * dh + c) = v;
      }
      if (r0 + 8 < N) {
        __nv_bfloat162 v = __floats2bfloat162_rn(oacc[nt][2] * inv1, oacc[nt][3] * inv1);
        *reinterpret_cast<__nv_bfloat162*>(o + ((size_t)slot * N + r0 + 8) * d + head * dh + c) = v;
      }
    }
  }
}

template <int DHP>
cudaError_t launch_dhp(const __nv_bfloat16* qkv, int slots, int heads, int N, int dh,
                       __nv_bfloat16* o, cudaStream_t st) {
  constexpr int LD = DHP + 8;
  const size_t smem = (size_t)(kQ + 4 * kKV) * LD * sizeof(__nv_bfloat16);
  static std::atomic<unsigned long long> configured{0};
  cudaError_t e = configure_once_per_device(configured, [&] {
    return cudaFuncSetAttribute(attn_bf16_kernel<DHP>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)smem);
  });
  if (e != cudaSuccess) return e;
  dim3 grid((N + kQ - 1) / kQ, slots * heads);
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)dh);
  attn_bf16_kernel<DHP><<<grid, kWarps * 32, smem, st>>>(qkv, slots, heads, N, dh, o, scale_log2);
  return cudaGetLastError();
}

// ------------------------------------------------------------- fp32 path

template <int DH>
__global__ void attn_f32_kernel(const float* __restrict__ qkv, int slots, int heads, int N,
                                float* __restrict__ o, float scale) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  const int total = slots * heads * N;
  if (warp >= total) return;
  const int qi = warp % N;
  const int bh = warp / N;
  const int slot = bh / heads, head = bh - slot * heads;
  const size_t plane = (size_t)N * DH;
  const float* Q = qkv + ((size_t)(0 * slots + slot) * heads + head) * plane + (size_t)qi * DH;
  const float* Kp = qkv + ((size_t)(1 * slots + slot) * heads + head) * plane;
  const float* Vp = qkv + ((size_t)(2 * slots + slot) * heads + head) * plane;
  float q[DH], acc[DH];
#pragma unroll
  for (int e = 0; e < DH; ++e) { q[e] = Q[e] * scale; acc[e] = 0.f; }
  float m = -INFINITY, l = 0.f;
  for (int key = lane; key < N; key += 32) {
    const float* kr = Kp + (size_t)key * DH;
    float s = 0.f;
#pragma unroll
    for (int e = 0; e < DH; ++e) s += q[e] * kr[e];
    const float m_new = fmaxf(m, s);
    const float c = expf(m - m_new);
    const float p = expf(s - m_new);
    l = l * c + p;
    const float* vr = Vp + (size_t)key * DH;
#pragma unroll
    for (int e = 0; e < DH; ++e) acc[e] = acc[e] * c + p * vr[e];
    m = m_new;
  }
  float mall = m;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) mall = fmaxf(mall, __shfl_xor_sync(0xffffffffu, mall, off));
  const float c = (m == -INFINITY) ? 0.f : expf(m - mall);
  l = warp_sum(l * c);
  const int d = heads * DH;
  float* dst = o + ((size_t)slot * N + qi) * d + head * DH;
#pragma unroll
  for (int e = 0; e < DH; ++e) {
    const float v = warp_sum(acc[e] * c);
    if (lane == 0) dst[e] = v / l;
  }
}

}  // namespace

cudaError_t launch_attention_bf16(const __nv_bfloat16* qkv, int slots, int heads, int N, int dh,
                                  int dhp, __nv_bfloat16* o, cudaStream_t st) {
  if (slots <= 0) return cudaSuccess;
  switch (dhp) {
    case 16: return launch_dhp<16>(qkv, slots, heads, N, dh, o, st);
    case 64: return launch_dhp<64>(qkv, slots, heads, N, dh, o, st);
    case 80: return launch_dhp<80>(qkv, slots, heads, N, dh, o, st);
    case 128: return launch_dhp<128>(qkv, slots, heads, N, dh, o, st);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_attention_f32(const float* qkv, int slots, int heads, int N, int dh, int dhp,
                                 float* o, cudaStream_t st) {
  if (slots <= 0) return cudaSuccess;
  if (dh != dhp) return cudaErrorInvalidValue;
  const int warps = slots * heads * N;
  const int threads = 128;
  const int blocks = (warps * 32 + threads - 1) / threads;
  const float scale = 1.0f / sqrtf((float)dh);
  switch (dh) {
    case 8: attn_f32_kernel<8><<<blocks, threads, 0, st>>>(qkv, slots, heads, N, o, scale); break;
    case 16: attn_f32_kernel<16><<<blocks, threads, 0, st>>>(qkv, slots, heads, N, o, scale); break;
    case 32: attn_f32_kernel<32><<<blocks, threads, 0, st>>>(qkv, slots, heads, N, o, scale); break;
    case 64: attn_f32_kernel<64><<<blocks, threads, 0, st>>>(qkv, slots, heads, N, o, scale); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace dc
