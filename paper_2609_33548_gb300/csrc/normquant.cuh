// Per-token absmax int8 quantisation (with or without RMSNorm) of one row by
// one warp (the norm / quant kernel for rows of up to 3072).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace tmz {

__device__ __forceinline__ float quant_code(float h, float s) {
  float v = rintf(__fmul_rn(h, s));
  return fminf(fmaxf(v, -128.f), 127.f);
}

// The BitLinear GEMM takes an int8 code q as two e4m3 values, hi = 16
// floor(q / 16) in [-128, 112] and lo = q - hi in [0, 15]: both have at most
// four significant bits, so both are exact in e4m3 (1 sign, 4 exponent bits
// with bias 7, 3 mantissa bits), and hi w + lo w = q w exactly.  hi and lo
// are formed exactly in fp32 and converted by the hardware, two per
// instruction (x0 in the low byte).
__device__ __forceinline__ uint32_t e4m3x2(float x0, float x1) {
  uint16_t d;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(d) : "f"(x1), "f"(x0));
  return d;
}
__device__ __forceinline__ float code_hi(float q) { return __fmul_rn(floorf(__fmul_rn(q, 0.0625f)), 16.f); }

// One row by one warp: h_k = (x_k * r) * g_k with r = 1/sqrt(mean(x^2) +
// 1e-5) (gain != null) or h_k = x_k; a = max(max|h|, 1e-5); q_k = rint(h_k *
// (127/a)) stored as its e4m3 pair (qh, ql rows); *deq = a / 127.  Lane l
// holds float4 number i * 32 + l of the row for i < NV (D <= 128 NV, D % 4
// == 0); the sum of squares runs as four fused multiply-add chains (one per
// float4 component) over i in order, added as (x + y) + (z + w), then a
// butterfly over the lanes (float4 past the row's end hold zeros and add
// nothing).  CG: x is read through L2 only (rows other CTAs have just written).
template <int NV, bool CG>
__device__ __forceinline__ void norm_quant_row(const float* __restrict__ xr, const float* __restrict__ gain, int D,
                                               uint8_t* __restrict__ qh8, uint8_t* __restrict__ ql8,
                                               float* __restrict__ deq, int lane) {
  const float4* x4 = reinterpret_cast<const float4*>(xr);
  const float4* gr = reinterpret_cast<const float4*>(gain);
  const int D4 = D >> 2;
  float4 v[NV];
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    const int k = i * 32 + lane;
    v[i] = k < D4 ? (CG ? __ldcg(x4 + k) : x4[k]) : make_float4(0.f, 0.f, 0.f, 0.f);
  }
  if (gain) {
    float sx = 0.f, sy = 0.f, sz = 0.f, sw = 0.f;
#pragma unroll
    for (int i = 0; i < NV; ++i) {
      sx = __fmaf_rn(v[i].x, v[i].x, sx);
      sy = __fmaf_rn(v[i].y, v[i].y, sy);
      sz = __fmaf_rn(v[i].z, v[i].z, sz);
      sw = __fmaf_rn(v[i].w, v[i].w, sw);
    }
    float ss = __fadd_rn(__fadd_rn(sx, sy), __fadd_rn(sz, sw));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ss = __fadd_rn(ss, __shfl_xor_sync(0xffffffffu, ss, o));
    const float r = __fdiv_rn(1.0f, __fsqrt_rn(__fadd_rn(__fdiv_rn(ss, (float)D), 1e-5f)));
#pragma unroll
    for (int i = 0; i < NV; ++i) {
      const int k = i * 32 + lane;
      if (k < D4) {
        const float4 g = gr[k];
        v[i].x = __fmul_rn(__fmul_rn(v[i].x, r), g.x);
        v[i].y = __fmul_rn(__fmul_rn(v[i].y, r), g.y);
        v[i].z = __fmul_rn(__fmul_rn(v[i].z, r), g.z);
        v[i].w = __fmul_rn(__fmul_rn(v[i].w, r), g.w);
      }
    }
  }
  float amax = 0.f;
#pragma unroll
  for (int i = 0; i < NV; ++i)
    amax = fmaxf(fmaxf(fmaxf(amax, fabsf(v[i].x)), fmaxf(fabsf(v[i].y), fabsf(v[i].z))), fabsf(v[i].w));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
  const float a = fmaxf(amax, 1e-5f);
  const float s = __fdiv_rn(127.f, a);
  uint32_t* qh = reinterpret_cast<uint32_t*>(qh8);
  uint32_t* ql = reinterpret_cast<uint32_t*>(ql8);
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    const int k = i * 32 + lane;
    if (k < D4) {
      const float c0 = quant_code(v[i].x, s), c1 = quant_code(v[i].y, s);
      const float c2 = quant_code(v[i].z, s), c3 = quant_code(v[i].w, s);
      const float h0 = code_hi(c0), h1 = code_hi(c1), h2 = code_hi(c2), h3 = code_hi(c3);
      qh[k] = e4m3x2(h0, h1) | (e4m3x2(h2, h3) << 16);
      ql[k] = e4m3x2(__fsub_rn(c0, h0), __fsub_rn(c1, h1)) | (e4m3x2(__fsub_rn(c2, h2), __fsub_rn(c3, h3)) << 16);
    }
  }
  if (lane == 0) *deq = __fdiv_rn(a, 127.f);
}

}  // namespace tmz
