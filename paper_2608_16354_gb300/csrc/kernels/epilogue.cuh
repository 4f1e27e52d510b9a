// Fused GEMM epilogues of the DiT block (shared by the tcgen05 bf16 GEMM and
// the fp32 SIMT GEMM).  Each works on 8 consecutive output columns of one row.
//
//  kEpiQKV  : y = acc + b, scattered head-major into q / k / v
//             [3][slots][heads][tokens][dh_pad]
//  kEpiGELU : y = gelu_tanh(acc + b)             -> [rows][N]
//  kEpiResid: h[row][col] += gate[scene][col] * (acc + b)   (fp32 residual)
#pragma once

#include "common.cuh"

namespace dc {

// Packed fp32x2 arithmetic (one instruction for two lanes of work).
__device__ __forceinline__ float2 f2_fma(float2 a, float2 b, float2 c) {
  float2 r;
  asm("{\n .reg .b64 a, b, c, d;\n mov.b64 a, {%2, %3};\n mov.b64 b, {%4, %5};\n"
      " mov.b64 c, {%6, %7};\n fma.rn.f32x2 d, a, b, c;\n mov.b64 {%0, %1}, d;\n}\n"
      : "=f"(r.x), "=f"(r.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  return r;
}
__device__ __forceinline__ float2 f2_mul(float2 a, float2 b) {
  float2 r;
  asm("{\n .reg .b64 a, b, d;\n mov.b64 a, {%2, %3};\n mov.b64 b, {%4, %5};\n"
      " mul.rn.f32x2 d, a, b;\n mov.b64 {%0, %1}, d;\n}\n"
      : "=f"(r.x), "=f"(r.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return r;
}
__device__ __forceinline__ float2 f2_add(float2 a, float2 b) {
  float2 r;
  asm("{\n .reg .b64 a, b, d;\n mov.b64 a, {%2, %3};\n mov.b64 b, {%4, %5};\n"
      " add.rn.f32x2 d, a, b;\n mov.b64 {%0, %1}, d;\n}\n"
      : "=f"(r.x), "=f"(r.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return r;
}

// gelu_tanh of a pair: x/2 (1 + tanh(x (k0 + k0 c x^2))), packed except the
// two hardware tanh
__device__ __forceinline__ float2 gelu_tanh_pair(float2 x) {
  const float k0 = 0.7978845608028654f, k1 = 0.7978845608028654f * 0.044715f;
  const float2 x2 = f2_mul(x, x);
  const float2 z = f2_mul(x, f2_fma(x2, make_float2(k1, k1), make_float2(k0, k0)));
  const float2 th = make_float2(tanh_approx(z.x), tanh_approx(z.y));
  const float2 hx = f2_mul(x, make_float2(0.5f, 0.5f));
  return f2_fma(hx, th, hx);
}

enum { kEpiQKV = 0, kEpiGELU = 1, kEpiResid = 2 };

struct EpiArgs {
  int M, N;            // valid rows / cols of the product
  int n_tok;           // tokens per slot (row -> slot = row / n_tok)
  const float* bias;   // [N]
  void* out;           // QKV: q/k/v base; GELU: [M][N]
  int d, heads, dh, dhp, nslots;  // QKV layout
  float* h;            // Resid: fp32 residual written [M][N]
  const float* h_in;   // Resid: residual read (== h, or the block-stack input u)
  const float* mod;    // Resid: modulation table of this step [B][mod_stride]
  int mod_stride;      // floats per scene in the table
  int gate_off;        // offset of this block's gate vector inside a scene's row
  int qkv_tma;         // QKV (tcgen05 GEMM): the output map covers q/k/v viewed as
                       // [3 * slots * heads * tokens][dh_pad] with 64 x 128 boxes, and
                       // dh is a multiple of 64: tiles inside one slot go out by TMA
};

template <typename T> struct Pack8;
template <> struct Pack8<__nv_bfloat16> {
  static __device__ __forceinline__ void store(__nv_bfloat16* p, const float* v) {
    __align__(16) __nv_bfloat162 t[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) t[i] = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
    *reinterpret_cast<uint4*>(p) = *reinterpret_cast<const uint4*>(t);
  }
};
template <> struct Pack8<float> {
  static __device__ __forceinline__ void store(float* p, const float* v) {
    reinterpret_cast<float4*>(p)[0] = make_float4(v[0], v[1], v[2], v[3]);
    reinterpret_cast<float4*>(p)[1] = make_float4(v[4], v[5], v[6], v[7]);
  }
};

template <int MODE, typename T>
__device__ __forceinline__ void epilogue8(const EpiArgs& e, const SlotMap& map, int row, int col,
                                          float (&v)[8]) {
  const float4 b0 = *reinterpret_cast<const float4*>(e.bias + col);
  const float4 b1 = *reinterpret_cast<const float4*>(e.bias + col + 4);
  v[0] += b0.x; v[1] += b0.y; v[2] += b0.z; v[3] += b0.w;
  v[4] += b1.x; v[5] += b1.y; v[6] += b1.z; v[7] += b1.w;
  if constexpr (MODE == kEpiQKV) {
    const int which = col / e.d;
    const int within = col - which * e.d;
    const int head = within / e.dh;
    const int c = within - head * e.dh;
    const int slot = row / e.n_tok;
    const int tok = row - slot * e.n_tok;
    T* dst = reinterpret_cast<T*>(e.out) +
             ((((size_t)which * e.nslots + slot) * e.heads + head) * e.n_tok + tok) * e.dhp + c;
    Pack8<T>::store(dst, v);
  } else if constexpr (MODE == kEpiGELU) {
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = sizeof(T) == 2 ? gelu_tanh_bf16(v[i]) : gelu_tanh(v[i]);
    Pack8<T>::store(reinterpret_cast<T*>(e.out) + (size_t)row * e.N + col, v);
  } else {
    const int slot = row / e.n_tok;
    const float* g = e.mod + (size_t)map.scene[slot] * e.mod_stride + e.gate_off + col;
    const float4 g0 = *reinterpret_cast<const float4*>(g);
    const float4 g1 = *reinterpret_cast<const float4*>(g + 4);
    const float4* hi = reinterpret_cast<const float4*>(e.h_in + (size_t)row * e.N + col);
    float4* hp = reinterpret_cast<float4*>(e.h + (size_t)row * e.N + col);
    float4 h0 = hi[0], h1 = hi[1];
    h0.x += g0.x * v[0]; h0.y += g0.y * v[1]; h0.z += g0.z * v[2]; h0.w += g0.w * v[3];
    h1.x += g1.x * v[4]; h1.y += g1.y * v[5]; h1.z += g1.z * v[6]; h1.w += g1.w * v[7];
    hp[0] = h0;
    hp[1] = h1;
  }
}

// Epilogue of one 32 x 32 block staged in shared memory (stg[r * 33 + c],
// r = row within the block, c = column within the block).  The warp writes
// whole rows: fp32 residual rows of 128 B, bf16 rows of 64 B (two rows per
// instruction), so every store and load is coalesced.
template <int MODE>
__device__ __forceinline__ void epilogue_block32(const EpiArgs& e, const SlotMap& map,
                                                 const float* stg, int row0, int col0, int lane) {
  if constexpr (MODE == kEpiResid) {
    // all 32 residual loads are issued before any store (h and h_in may
    // alias, so the compiler would otherwise serialise load -> store pairs)
    const int col = col0 + lane;
    const float b = e.bias[col];
    const int nrow = min(32, e.M - row0);
    const int s_first = row0 / e.n_tok;
    const int s_last = (row0 + nrow - 1) / e.n_tok;
    const float g_first = e.mod[(size_t)map.scene[s_first] * e.mod_stride + e.gate_off + col];
    const float g_last = e.mod[(size_t)map.scene[s_last] * e.mod_stride + e.gate_off + col];
    const int row_split = (s_first + 1) * e.n_tok;  // first row of the next slot
    float hv[32];
#pragma unroll
    for (int r = 0; r < 32; ++r)
      hv[r] = r < nrow ? __ldcs(e.h_in + (size_t)(row0 + r) * e.N + col) : 0.f;
#pragma unroll
    for (int r = 0; r < 32; ++r) {
      if (r < nrow) {
        const float g = row0 + r < row_split ? g_first : g_last;
        e.h[(size_t)(row0 + r) * e.N + col] = hv[r] + g * (stg[r * 33 + lane] + b);
      }
    }
  } else {
    const int cc = 2 * (lane & 15);
    const int col = col0 + cc;
    const float b0 = e.bias[col], b1 = e.bias[col + 1];
    int which = 0, head = 0, c = 0;
    if constexpr (MODE == kEpiQKV) {
      which = col / e.d;
      const int within = col - which * e.d;
      head = within / e.dh;
      c = within - head * e.dh;
    }
    for (int i = 0; i < 16; ++i) {
      const int r = 2 * i + (lane >> 4);
      const int row = row0 + r;
      if (row >= e.M) break;
      float v0 = stg[r * 33 + cc] + b0, v1 = stg[r * 33 + cc + 1] + b1;
      if constexpr (MODE == kEpiGELU) {
        v0 = gelu_tanh(v0);
        v1 = gelu_tanh(v1);
        *reinterpret_cast<__nv_bfloat162*>(reinterpret_cast<__nv_bfloat16*>(e.out) +
                                           (size_t)row * e.N + col) = __floats2bfloat162_rn(v0, v1);
      } else {
        const int slot = row / e.n_tok;
        const int tok = row - slot * e.n_tok;
        __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(e.out) +
                             ((((size_t)which * e.nslots + slot) * e.heads + head) * e.n_tok + tok) *
                                 e.dhp + c;
        *reinterpret_cast<__nv_bfloat162*>(dst) = __floats2bfloat162_rn(v0, v1);
      }
    }
  }
}

}  // namespace dc
