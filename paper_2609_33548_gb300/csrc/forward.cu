// BitNet forward kernels other than the BitLinear GEMM: RMSNorm and
// per-token absmax int8 activation quantisation, squared-ReLU gating,
// 2-bit code expansion, embedding, RoPE, causal GQA attention, and the
// label-token LM head with cross-entropy.
#include <cuda_bf16.h>

#include <cfloat>

#include "common.cuh"
#include "kernels.cuh"
#include "normquant.cuh"

namespace tmz {

namespace {

__device__ __forceinline__ float block_sum(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, o));
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) red[w] = v;
  __syncthreads();
  float t = 0.f;
  for (int i = 0; i < (int)(blockDim.x >> 5); ++i) t = __fadd_rn(t, red[i]);
  return t;
}

__device__ __forceinline__ float block_max(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) red[w] = v;
  __syncthreads();
  float t = 0.f;
  for (int i = 0; i < (int)(blockDim.x >> 5); ++i) t = fmaxf(t, red[i]);
  return t;
}

// One block per row.  h_k = (x_k * r) * g_k with r = 1/sqrt(mean(x^2)+1e-5)
// (RMSNorm) or h_k = x_k; a = max(max|h|, 1e-5); q_k = rint(h_k * (127/a)),
// stored as its e4m3 (hi, lo) pair in q [2, M, D] (hi rows, then lo rows).
// Generic version (any D, any input type): three passes over the row.
template <typename In>
__global__ void k_norm_quant(const In* __restrict__ x, const float* __restrict__ gain, int D,
                             uint8_t* __restrict__ q, float* __restrict__ deq) {
  __shared__ float red[32];
  const size_t row = blockIdx.x;
  const In* xr = x + row * (size_t)D;
  float r = 1.f;
  if (gain) {
    float ss = 0.f;
    for (int k = threadIdx.x; k < D; k += blockDim.x) {
      const float v = (float)xr[k];
      ss = __fadd_rn(ss, __fmul_rn(v, v));
    }
    ss = block_sum(ss, red);
    r = __fdiv_rn(1.0f, __fsqrt_rn(__fadd_rn(__fdiv_rn(ss, (float)D), 1e-5f)));
  }
  float amax = 0.f;
  for (int k = threadIdx.x; k < D; k += blockDim.x) {
    const float v = (float)xr[k];
    const float h = gain ? __fmul_rn(__fmul_rn(v, r), gain[k]) : v;
    amax = fmaxf(amax, fabsf(h));
  }
  const float a = fmaxf(block_max(amax, red), 1e-5f);
  const float s = __fdiv_rn(127.f, a);
  uint8_t* qh = q + row * (size_t)D;
  uint8_t* ql = qh + (size_t)gridDim.x * D;
  for (int k = threadIdx.x; k < D; k += blockDim.x) {
    const float v = (float)xr[k];
    const float h = gain ? __fmul_rn(__fmul_rn(v, r), gain[k]) : v;
    const float c = quant_code(h, s), hi = code_hi(c);
    qh[k] = (uint8_t)(e4m3x2(hi, 0.f) & 0xFFu);
    ql[k] = (uint8_t)(e4m3x2(__fsub_rn(c, hi), 0.f) & 0xFFu);
  }
  if (threadIdx.x == 0) deq[row] = __fdiv_rn(a, 127.f);
}

// Same arithmetic for fp32 rows with D % 4 == 0 and D <= 4 * 256 * VPT: the
// row is read once (float4) and kept in registers.
template <int VPT>
__global__ void __launch_bounds__(256) k_norm_quant_vec(const float* __restrict__ x, const float* __restrict__ gain,
                                                        int D, uint8_t* __restrict__ q, float* __restrict__ deq) {
  __shared__ float red[32];
  grid_dep_wait();
  const size_t row = blockIdx.x;
  const float4* xr = reinterpret_cast<const float4*>(x + row * (size_t)D);
  const float4* gr = reinterpret_cast<const float4*>(gain);
  const int D4 = D >> 2;
  float4 v[VPT];
#pragma unroll
  for (int i = 0; i < VPT; ++i) {
    const int k = i * 256 + threadIdx.x;
    v[i] = k < D4 ? xr[k] : make_float4(0.f, 0.f, 0.f, 0.f);
  }
  float r = 1.f;
  if (gain) {
    float ss = 0.f;
#pragma unroll
    for (int i = 0; i < VPT; ++i) {
      ss = __fadd_rn(ss, __fmul_rn(v[i].x, v[i].x));
      ss = __fadd_rn(ss, __fmul_rn(v[i].y, v[i].y));
      ss = __fadd_rn(ss, __fmul_rn(v[i].z, v[i].z));
      ss = __fadd_rn(ss, __fmul_rn(v[i].w, v[i].w));
    }
    ss = block_sum(ss, red);
    r = __fdiv_rn(1.0f, __fsqrt_rn(__fadd_rn(__fdiv_rn(ss, (float)D), 1e-5f)));
#pragma unroll
    for (int i = 0; i < VPT; ++i) {
      const int k = i * 256 + threadIdx.x;
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
  for (int i = 0; i < VPT; ++i)
    amax = fmaxf(fmaxf(fmaxf(amax, fabsf(v[i].x)), fmaxf(fabsf(v[i].y), fabsf(v[i].z))), fabsf(v[i].w));
  const float a = fmaxf(block_max(amax, red), 1e-5f);
  const float s = __fdiv_rn(127.f, a);
  uint32_t* qh = reinterpret_cast<uint32_t*>(q + row * (size_t)D);
  uint32_t* ql = reinterpret_cast<uint32_t*>(q + ((size_t)gridDim.x + row) * D);
#pragma unroll
  for (int i = 0; i < VPT; ++i) {
    const int k = i * 256 + threadIdx.x;
    if (k < D4) {
      const float c0 = quant_code(v[i].x, s), c1 = quant_code(v[i].y, s);
      const float c2 = quant_code(v[i].z, s), c3 = quant_code(v[i].w, s);
      const float h0 = code_hi(c0), h1 = code_hi(c1), h2 = code_hi(c2), h3 = code_hi(c3);
      qh[k] = e4m3x2(h0, h1) | (e4m3x2(h2, h3) << 16);
      ql[k] = e4m3x2(__fsub_rn(c0, h0), __fsub_rn(c1, h1)) | (e4m3x2(__fsub_rn(c2, h2), __fsub_rn(c3, h3)) << 16);
    }
  }
  if (threadIdx.x == 0) deq[row] = __fdiv_rn(a, 127.f);
}

// Same arithmetic for rows of D <= 128 NV (D % 4 == 0) with one warp per row
// (norm_quant_row): the row's NV float4 per lane are all in flight at once and
// both reductions are warp shuffles, so no CTA barrier stalls the loads (4
// rows per CTA).
template <int NV>
__global__ void __launch_bounds__(128) k_norm_quant_warp(const float* __restrict__ x, const float* __restrict__ gain,
                                                         int D, int M, uint8_t* __restrict__ q,
                                                         float* __restrict__ deq) {
  grid_dep_wait();
  const int row = blockIdx.x * 4 + (threadIdx.x >> 5);
  if (row >= M) return;
  norm_quant_row<NV, false>(x + (size_t)row * D, gain, D, q + (size_t)row * D, q + ((size_t)M + row) * D, deq + row,
                            threadIdx.x & 31);
}

struct Bf16In {
  uint16_t bits;
  __device__ __forceinline__ explicit operator float() const { return __uint_as_float((uint32_t)bits << 16); }
};

// 16 packed codes (2 bits each: 0 -> -1, 1 -> 0, 2 -> +1) -> 16 e4m3 bytes
// (+1 = 0x38, -1 = 0xB8, 0 = 0x00), one 16-byte store.
__device__ __forceinline__ void expand_word(uint32_t w, uint8_t* dst) {
  uint32_t v[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    uint32_t b = 0;
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const uint32_t c = (w >> (8 * j + 2 * e)) & 3u;
      b |= (c == 2u ? 0x38u : (c == 0u ? 0xB8u : 0u)) << (8 * e);
    }
    v[j] = b;
  }
  *reinterpret_cast<uint4*>(dst) = make_uint4(v[0], v[1], v[2], v[3]);
}

// Value of an e4m3 byte (1 sign, 4 exponent bits with bias 7, 3 mantissa
// bits); the codes' halves are integers in [-128, 112] and [0, 15].
__device__ __forceinline__ float e4m3_value(uint32_t b) {
  const int e = (int)((b >> 3) & 15u), m = (int)(b & 7u);
  const float v = e ? ldexpf((float)(8 + m), e - 10) : ldexpf((float)m, -9);
  return (b & 0x80u) ? -v : v;
}

__global__ void k_codes_i8(const uint8_t* __restrict__ q, int M, int K, int8_t* __restrict__ out) {
  const uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const uint64_t n = (uint64_t)M * K;
  if (i >= n) return;
  out[i] = (int8_t)(int)__fadd_rn(e4m3_value(q[i]), e4m3_value(q[n + i]));
}

// One thread per packed word.
__global__ void k_expand_codes(const uint32_t* __restrict__ words, uint64_t n_words, uint8_t* __restrict__ out) {
  const uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n_words) return;
  expand_word(words[i], out + i * 16);
}

// One thread per (interleaved row, word).
__global__ void k_expand_gate_up(const uint32_t* __restrict__ gw, const uint32_t* __restrict__ uw, int F, int wpr,
                                 uint64_t n_words, uint8_t* __restrict__ out) {
  const uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n_words) return;
  const uint64_t r = i / wpr;
  const int jw = (int)(i % wpr);
  const int blk = (int)(r / 256), within = (int)(r % 256);
  const int src = blk * 128 + (within & 127);
  uint32_t w = 0x55555555u;  // code 1 (value 0) in every slot
  if (src < F) w = (within < 128 ? gw : uw)[(size_t)src * wpr + jw];
  expand_word(w, out + i * 16);
}

__global__ void k_embed(const int32_t* __restrict__ tok, const float* __restrict__ embed, int D, int V,
                        float* __restrict__ x, unsigned* err) {
  const size_t t = blockIdx.x;
  int id = tok[t];
  if (id < 0 || id >= V) {
    if (threadIdx.x == 0) atomicOr(err, ERR_BOUNDS);
    id = 0;
  }
  const float* e = embed + (size_t)id * D;
  for (int k = threadIdx.x; k < D; k += blockDim.x) x[t * D + k] = e[k];
}

__global__ void k_rope_tables(int S, int hd, float* cosb, float* sinb) {
  const int half = hd / 2;
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= S * half) return;
  const int pos = i / half, j = i % half;
  const double inv = pow(10000.0, -(2.0 * j) / (double)hd);
  const double ang = (double)pos * inv;
  cosb[i] = (float)cos(ang);
  sinb[i] = (float)sin(ang);
}

// One block per token; threads over (head, j < hd/2) pairs of Q and K, and
// over V elements.
__global__ void k_rope_pack(const float* __restrict__ qkv, const float* __restrict__ cosb,
                            const float* __restrict__ sinb, int S, int H, int KV, int hd,
                            uint16_t* __restrict__ q, uint16_t* __restrict__ k) {
  const int t = blockIdx.x;
  const int b = t / S, pos = t % S;
  const int half = hd / 2;
  const int width = (H + 2 * KV) * hd;
  const float* row = qkv + (size_t)t * width;
  const float* cr = cosb + (size_t)pos * half;
  const float* sr = sinb + (size_t)pos * half;
  for (int i = threadIdx.x; i < (H + KV) * half; i += blockDim.x) {
    const int head = i / half, j = i % half;
    const float* src = row + head * hd;
    const float x1 = src[j], x2 = src[j + half];
    const float c = cr[j], s = sr[j];
    const float o1 = __fsub_rn(__fmul_rn(x1, c), __fmul_rn(x2, s));
    const float o2 = __fadd_rn(__fmul_rn(x2, c), __fmul_rn(x1, s));
    __nv_bfloat16 b1 = __float2bfloat16_rn(o1), b2 = __float2bfloat16_rn(o2);
    uint16_t* dst;
    if (head < H)
      dst = q + (((size_t)b * H + head) * S + pos) * hd;
    else
      dst = k + (((size_t)b * KV + (head - H)) * S + pos) * hd;
    dst[j] = *reinterpret_cast<uint16_t*>(&b1);
    dst[j + half] = *reinterpret_cast<uint16_t*>(&b2);
  }
}

// V [B*S, KV*hd] (inside qkv) -> Vt bf16 [B, KV, hd, S] through a 32x32 tile.
__global__ void k_pack_vt(const float* __restrict__ qkv, int S, int H, int KV, int hd, uint16_t* __restrict__ vt) {
  __shared__ float tile[32][33];
  const int b = blockIdx.z / KV, kvh = blockIdx.z % KV;
  const int s0 = blockIdx.x * 32, d0 = blockIdx.y * 32;
  const int width = (H + 2 * KV) * hd;
  const float* v = qkv + (size_t)(H + KV) * hd + (size_t)kvh * hd;
  for (int r = threadIdx.y; r < 32; r += blockDim.y) {
    const int s = s0 + r, d = d0 + threadIdx.x;
    tile[r][threadIdx.x] = (s < S && d < hd) ? v[((size_t)b * S + s) * width + d] : 0.f;
  }
  __syncthreads();
  for (int r = threadIdx.y; r < 32; r += blockDim.y) {
    const int d = d0 + r, s = s0 + threadIdx.x;
    if (d < hd && s < S) {
      __nv_bfloat16 bv = __float2bfloat16_rn(tile[threadIdx.x][r]);
      vt[(((size_t)b * KV + kvh) * hd + d) * S + s] = *reinterpret_cast<uint16_t*>(&bv);
    }
  }
}

__device__ __forceinline__ void mma_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat16 l = __float2bfloat16_rn(lo), h = __float2bfloat16_rn(hi);
  return (uint32_t)(*reinterpret_cast<uint16_t*>(&l)) | ((uint32_t)(*reinterpret_cast<uint16_t*>(&h)) << 16);
}

__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xFFFF0000u); }

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"((uint32_t)__cvta_generic_to_shared(smem)),
               "l"(gmem)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3, const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"((uint32_t)__cvta_generic_to_shared(p)));
}

// Causal attention, two passes over the keys: pass 1 finds the exact row
// maximum of the scores, pass 2 forms P = bf16(exp(s - max)), l = sum P and
// O = P V / l.  4 warps x 16 query rows per block; bf16 mma.sync tiles fed
// by ldmatrix from a double-buffered cp.async ring of 64-key K / V^T tiles.
template <int HD>
struct AttnSmem {
  static constexpr int KP = HD + 8, VP = 64 + 8;
  static constexpr int K_ELEMS = 64 * KP, V_ELEMS = HD * VP;
  static constexpr int BYTES = 2 * (K_ELEMS + V_ELEMS) * 2;
};

template <int HD>
__global__ void __launch_bounds__(128) k_attention(const uint16_t* __restrict__ Q, const uint16_t* __restrict__ K,
                                                   const uint16_t* __restrict__ Vt, int S, int H, int KV,
                                                   float scale, float* __restrict__ out) {
  using L = AttnSmem<HD>;
  constexpr int KP = L::KP, VP = L::VP;
  extern __shared__ __align__(16) uint16_t att_smem[];
  uint16_t* Ks = att_smem;                      // [2][64][KP]
  uint16_t* Vs = att_smem + 2 * L::K_ELEMS;     // [2][HD][VP]
  const int qblk = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int kvh = h / (H / KV);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, c = lane & 3;
  const int q0 = qblk * 64 + warp * 16;
  const uint16_t* Qp = Q + ((size_t)b * H + h) * S * HD;
  const uint16_t* Kp = K + ((size_t)b * KV + kvh) * S * HD;
  const uint16_t* Vp = Vt + ((size_t)b * KV + kvh) * HD * S;

  uint32_t qa[HD / 16][4];
#pragma unroll
  for (int kk = 0; kk < HD / 16; ++kk) {
    const int col = kk * 16 + 2 * c;
    qa[kk][0] = *reinterpret_cast<const uint32_t*>(Qp + (size_t)(q0 + g) * HD + col);
    qa[kk][1] = *reinterpret_cast<const uint32_t*>(Qp + (size_t)(q0 + g + 8) * HD + col);
    qa[kk][2] = *reinterpret_cast<const uint32_t*>(Qp + (size_t)(q0 + g) * HD + col + 8);
    qa[kk][3] = *reinterpret_cast<const uint32_t*>(Qp + (size_t)(q0 + g + 8) * HD + col + 8);
  }
  const int nkb = qblk + 1;
  const int r0 = q0 + g, r1 = q0 + g + 8;
  float mx0 = -FLT_MAX, mx1 = -FLT_MAX;

  auto load_k = [&](int kb, int buf) {
    uint16_t* dst = Ks + buf * L::K_ELEMS;
    for (int i = threadIdx.x; i < 64 * (HD / 8); i += 128) {
      const int r = i / (HD / 8), c8 = i % (HD / 8);
      cp_async16(&dst[r * KP + c8 * 8], Kp + (size_t)(kb * 64 + r) * HD + c8 * 8);
    }
  };
  auto load_v = [&](int kb, int buf) {
    uint16_t* dst = Vs + buf * L::V_ELEMS;
    for (int i = threadIdx.x; i < HD * 8; i += 128) {
      const int d = i / 8, c8 = i % 8;
      cp_async16(&dst[d * VP + c8 * 8], Vp + (size_t)d * S + kb * 64 + c8 * 8);
    }
  };
  // ldmatrix lane -> row address: lanes 8m..8m+7 address the rows of matrix m.
  const int lm_row = lane & 7, lm_mat = lane >> 3;
  auto scores = [&](const uint16_t* ks, float (&sacc)[8][4]) {
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      sacc[j][0] = sacc[j][1] = sacc[j][2] = sacc[j][3] = 0.f;
#pragma unroll
      for (int kk = 0; kk < HD / 16; kk += 2) {
        // matrices: (kk, lo8), (kk, hi8), (kk+1, lo8), (kk+1, hi8) of key rows j*8..j*8+7
        uint32_t b0, b1, b2, b3;
        ldsm_x4(b0, b1, b2, b3, &ks[(j * 8 + lm_row) * KP + (kk + (lm_mat >> 1)) * 16 + (lm_mat & 1) * 8]);
        mma_16816(sacc[j], qa[kk], b0, b1);
        if (kk + 1 < HD / 16) mma_16816(sacc[j], qa[kk + 1], b2, b3);
      }
    }
  };

  load_k(0, 0);
  cp_async_commit();
  for (int kb = 0; kb < nkb; ++kb) {
    if (kb + 1 < nkb) {
      load_k(kb + 1, (kb + 1) & 1);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    float sacc[8][4];
    scores(Ks + (kb & 1) * L::K_ELEMS, sacc);
#pragma unroll
    for (int j = 0; j < 8; ++j)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = kb * 64 + j * 8 + 2 * c + (e & 1);
        const int row = e < 2 ? r0 : r1;
        if (key <= row) {
          const float s = __fmul_rn(sacc[j][e], scale);
          if (e < 2) mx0 = fmaxf(mx0, s); else mx1 = fmaxf(mx1, s);
        }
      }
    __syncthreads();
  }
#pragma unroll
  for (int o = 1; o <= 2; o <<= 1) {
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, o));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, o));
  }

  float oacc[HD / 8][4];
#pragma unroll
  for (int n = 0; n < HD / 8; ++n) oacc[n][0] = oacc[n][1] = oacc[n][2] = oacc[n][3] = 0.f;
  float l0 = 0.f, l1 = 0.f;
  load_k(0, 0);
  load_v(0, 0);
  cp_async_commit();
  for (int kb = 0; kb < nkb; ++kb) {
    if (kb + 1 < nkb) {
      load_k(kb + 1, (kb + 1) & 1);
      load_v(kb + 1, (kb + 1) & 1);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const uint16_t* vs = Vs + (kb & 1) * L::V_ELEMS;
    float sacc[8][4];
    scores(Ks + (kb & 1) * L::K_ELEMS, sacc);
    uint32_t pf[8][2];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      float pv[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = kb * 64 + j * 8 + 2 * c + (e & 1);
        const int row = e < 2 ? r0 : r1;
        pv[e] = key <= row ? expf(__fsub_rn(__fmul_rn(sacc[j][e], scale), e < 2 ? mx0 : mx1)) : 0.f;
      }
      pf[j][0] = pack_bf16(pv[0], pv[1]);
      pf[j][1] = pack_bf16(pv[2], pv[3]);
      l0 = __fadd_rn(__fadd_rn(l0, bf16_lo(pf[j][0])), bf16_hi(pf[j][0]));
      l1 = __fadd_rn(__fadd_rn(l1, bf16_lo(pf[j][1])), bf16_hi(pf[j][1]));
    }
#pragma unroll
    for (int kc = 0; kc < 4; ++kc) {
      const uint32_t a[4] = {pf[2 * kc][0], pf[2 * kc][1], pf[2 * kc + 1][0], pf[2 * kc + 1][1]};
#pragma unroll
      for (int n = 0; n < HD / 8; n += 2) {
        // matrices: (n, keys lo8), (n, keys hi8), (n+1, lo8), (n+1, hi8) of this key chunk
        uint32_t b0, b1, b2, b3;
        ldsm_x4(b0, b1, b2, b3, &vs[((n + (lm_mat >> 1)) * 8 + lm_row) * VP + kc * 16 + (lm_mat & 1) * 8]);
        mma_16816(oacc[n], a, b0, b1);
        mma_16816(oacc[n + 1], a, b2, b3);
      }
    }
    __syncthreads();
  }
#pragma unroll
  for (int o = 1; o <= 2; o <<= 1) {
    l0 = __fadd_rn(l0, __shfl_xor_sync(0xffffffffu, l0, o));
    l1 = __fadd_rn(l1, __shfl_xor_sync(0xffffffffu, l1, o));
  }
  float* o0 = out + ((size_t)b * S + r0) * (size_t)(H * HD) + h * HD;
  float* o1 = out + ((size_t)b * S + r1) * (size_t)(H * HD) + h * HD;
#pragma unroll
  for (int n = 0; n < HD / 8; ++n) {
    const int col = n * 8 + 2 * c;
    *reinterpret_cast<float2*>(o0 + col) = make_float2(__fdiv_rn(oacc[n][0], l0), __fdiv_rn(oacc[n][1], l0));
    *reinterpret_cast<float2*>(o1 + col) = make_float2(__fdiv_rn(oacc[n][2], l1), __fdiv_rn(oacc[n][3], l1));
  }
}

// Loss mode 0.  One block per sequence: final RMSNorm of the last position,
// h -> bf16, logits over the C label tokens accumulated in float64 (every
// bf16 product is exact in float64), cross-entropy in float64.
__global__ void k_head_ce_last(const float* __restrict__ x, const float* __restrict__ gain,
                               const uint16_t* __restrict__ head, const int32_t* __restrict__ targets, int S,
                               int D, int V, int C, double* __restrict__ per_seq) {
  __shared__ float red[32];
  __shared__ double dred[32];
  __shared__ double logits[64];
  const int b = blockIdx.x;
  const float* xr = x + ((size_t)b * S + (S - 1)) * D;
  float ss = 0.f;
  for (int k = threadIdx.x; k < D; k += blockDim.x) ss = __fadd_rn(ss, __fmul_rn(xr[k], xr[k]));
  ss = block_sum(ss, red);
  const float r = __fdiv_rn(1.0f, __fsqrt_rn(__fadd_rn(__fdiv_rn(ss, (float)D), 1e-5f)));
  for (int cl = 0; cl < C; ++cl) {
    const uint16_t* wr = head + (size_t)(V - C + cl) * D;
    double acc = 0.0;
    for (int k = threadIdx.x; k < D; k += blockDim.x) {
      const float hv = __bfloat162float(__float2bfloat16_rn(__fmul_rn(__fmul_rn(xr[k], r), gain[k])));
      acc += (double)hv * (double)__uint_as_float((uint32_t)wr[k] << 16);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    __syncthreads();
    if ((threadIdx.x & 31) == 0) dred[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
      double t = 0.0;
      for (int i = 0; i < (int)(blockDim.x >> 5); ++i) t += dred[i];
      logits[cl] = t;
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    double m = -DBL_MAX;
    for (int cl = 0; cl < C; ++cl) m = fmax(m, logits[cl]);
    double se = 0.0;
    for (int cl = 0; cl < C; ++cl) se += exp(logits[cl] - m);
    int tg = targets[b];
    tg = tg < 0 ? 0 : (tg >= C ? C - 1 : tg);
    per_seq[b] = m + log(se) - logits[tg];
  }
}

// Final RMSNorm of one row per block, rounded to bf16 (the LM-head operand).
__global__ void k_final_norm_bf16(const float* __restrict__ x, const float* __restrict__ gain, int D,
                                  uint16_t* __restrict__ h) {
  __shared__ float red[32];
  const size_t row = blockIdx.x;
  const float* xr = x + row * (size_t)D;
  float ss = 0.f;
  for (int k = threadIdx.x; k < D; k += blockDim.x) ss = __fadd_rn(ss, __fmul_rn(xr[k], xr[k]));
  ss = block_sum(ss, red);
  const float r = __fdiv_rn(1.0f, __fsqrt_rn(__fadd_rn(__fdiv_rn(ss, (float)D), 1e-5f)));
  for (int k = threadIdx.x; k < D; k += blockDim.x) {
    __nv_bfloat16 v = __float2bfloat16_rn(__fmul_rn(__fmul_rn(xr[k], r), gain[k]));
    h[row * (size_t)D + k] = *reinterpret_cast<uint16_t*>(&v);
  }
}

// One warp per row: log-sum-exp over the tiles' partials in float64.
__global__ void k_ce_rows(const float2* __restrict__ part, int ntiles, const float* __restrict__ tlogit,
                          const int32_t* __restrict__ target, int T, int V, double* __restrict__ tok_loss,
                          unsigned* err) {
  const int row = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= T) return;
  const float2* pr = part + (size_t)row * ntiles;
  float m = -INFINITY;
  for (int j = lane; j < ntiles; j += 32) m = fmaxf(m, pr[j].x);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  double acc = 0.0;
  for (int j = lane; j < ntiles; j += 32) acc += (double)pr[j].y * exp((double)pr[j].x - (double)m);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if (lane == 0) {
    const int tg = target[row];
    if (tg < 0 || tg >= V) {
      atomicOr(err, ERR_BOUNDS);
      tok_loss[row] = 0.0;
    } else {
      tok_loss[row] = (double)m + log(acc) - (double)tlogit[row];
    }
  }
}

// Per-sequence mean of the token losses (fixed order, float64).
__global__ void k_seq_mean(const double* __restrict__ tok_loss, int S, double* __restrict__ per_seq) {
  __shared__ double red[32];
  const int b = blockIdx.x;
  double s = 0.0;
  for (int i = threadIdx.x; i < S; i += blockDim.x) s += tok_loss[(size_t)b * S + i];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += red[w];
    per_seq[b] = t / (double)S;
  }
}

__global__ void k_mean(const double* __restrict__ v, int n, double* __restrict__ out) {
  if (threadIdx.x == 0 && blockIdx.x == 0) {
    double t = 0.0;
    for (int i = 0; i < n; ++i) t += v[i];
    *out = t / (double)n;
  }
}

}  // namespace

uint64_t& kernel_launches() {
  static thread_local uint64_t n = 0;
  return n;
}

void launch_norm_quant(const float* x, const float* gain, int M, int D, uint8_t* q, float* deq, cudaStream_t s) {
  kernel_launches() += 1;
  const int vpt = (D + 1023) / 1024;
  const bool aligned = (D % 4 == 0) && ((uintptr_t)x % 16 == 0) && ((uintptr_t)q % 4 == 0) &&
                       (!gain || (uintptr_t)gain % 16 == 0);
  if (!aligned || vpt > 8) {
    k_norm_quant<float><<<M, 256, 0, s>>>(x, gain, D, q, deq);
    return;
  }
  // rows of up to 3072 (the 2B and 0.7B model widths): one warp per row
  const dim3 wgrid((unsigned)((M + 3) / 4));
  if (D <= 1536) {
    launch_dependent(k_norm_quant_warp<12>, wgrid, dim3(128), 0, s, x, gain, D, M, q, deq);
    return;
  }
  if (D <= 2560) {
    launch_dependent(k_norm_quant_warp<20>, wgrid, dim3(128), 0, s, x, gain, D, M, q, deq);
    return;
  }
  if (D <= 3072) {
    launch_dependent(k_norm_quant_warp<24>, wgrid, dim3(128), 0, s, x, gain, D, M, q, deq);
    return;
  }
  switch (vpt) {
    case 1: launch_dependent(k_norm_quant_vec<1>, dim3(M), dim3(256), 0, s, x, gain, D, q, deq); break;
    case 2: launch_dependent(k_norm_quant_vec<2>, dim3(M), dim3(256), 0, s, x, gain, D, q, deq); break;
    case 3: launch_dependent(k_norm_quant_vec<3>, dim3(M), dim3(256), 0, s, x, gain, D, q, deq); break;
    case 4: launch_dependent(k_norm_quant_vec<4>, dim3(M), dim3(256), 0, s, x, gain, D, q, deq); break;
    case 5: launch_dependent(k_norm_quant_vec<5>, dim3(M), dim3(256), 0, s, x, gain, D, q, deq); break;
    case 6: launch_dependent(k_norm_quant_vec<6>, dim3(M), dim3(256), 0, s, x, gain, D, q, deq); break;
    case 7: launch_dependent(k_norm_quant_vec<7>, dim3(M), dim3(256), 0, s, x, gain, D, q, deq); break;
    default: launch_dependent(k_norm_quant_vec<8>, dim3(M), dim3(256), 0, s, x, gain, D, q, deq); break;
  }
}

void launch_norm_quant_bf16(const uint16_t* x, int M, int D, uint8_t* q, float* deq, cudaStream_t s) {
  kernel_launches() += 1;
  k_norm_quant<Bf16In><<<M, 256, 0, s>>>(reinterpret_cast<const Bf16In*>(x), nullptr, D, q, deq);
}

void launch_codes_i8(const uint8_t* q, int M, int K, int8_t* out, cudaStream_t s) {
  const uint64_t n = (uint64_t)M * K;
  if (!n) return;
  ++kernel_launches();
  k_codes_i8<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(q, M, K, out);
}

void launch_expand_codes(const uint32_t* words, uint64_t rows, int K, uint8_t* out, cudaStream_t s) {
  kernel_launches() += 1;
  const uint64_t n = rows * (uint64_t)(K / 16);
  k_expand_codes<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(words, n, out);
}

void launch_expand_gate_up(const uint32_t* gate_words, const uint32_t* up_words, int F, int K, uint8_t* out,
                           cudaStream_t s) {
  kernel_launches() += 1;
  const int wpr = K / 16;
  const uint64_t rows = 256ull * (uint64_t)((F + 127) / 128);
  const uint64_t n = rows * (uint64_t)wpr;
  k_expand_gate_up<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(gate_words, up_words, F, wpr, n, out);
}

void launch_embed(const int32_t* tok, const float* embed, int T, int D, int V, float* x, unsigned* err,
                  cudaStream_t s) {
  kernel_launches() += 1;
  k_embed<<<T, 256, 0, s>>>(tok, embed, D, V, x, err);
}

void launch_rope_tables(int S, int hd, float* cosb, float* sinb, cudaStream_t s) {
  kernel_launches() += 1;
  const int n = S * hd / 2;
  k_rope_tables<<<(n + 255) / 256, 256, 0, s>>>(S, hd, cosb, sinb);
}

void launch_rope_pack(const float* qkv, const float* cosb, const float* sinb, int B, int S, int H, int KV, int hd,
                      uint16_t* q, uint16_t* k, uint16_t* vt, cudaStream_t s) {
  kernel_launches() += 2;
  k_rope_pack<<<B * S, 256, 0, s>>>(qkv, cosb, sinb, S, H, KV, hd, q, k);
  dim3 grid((S + 31) / 32, (hd + 31) / 32, B * KV);
  k_pack_vt<<<grid, dim3(32, 8), 0, s>>>(qkv, S, H, KV, hd, vt);
}

template <int HD>
void attention_hd(const uint16_t* q, const uint16_t* k, const uint16_t* vt, int B, int S, int H, int KV, float scale,
                  float* out, cudaStream_t s) {
  static bool attr = false;
  if (!attr) {
    cudaFuncSetAttribute(k_attention<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, AttnSmem<HD>::BYTES);
    attr = true;
  }
  dim3 grid(S / 64, H, B);
  k_attention<HD><<<grid, 128, AttnSmem<HD>::BYTES, s>>>(q, k, vt, S, H, KV, scale, out);
}

void launch_attention(const uint16_t* q, const uint16_t* k, const uint16_t* vt, int B, int S, int H, int KV, int hd,
                      float* out, cudaStream_t s) {
  kernel_launches() += 1;
  const float scale = 1.0f / sqrtf((float)hd);
  switch (hd) {
    case 64: attention_hd<64>(q, k, vt, B, S, H, KV, scale, out, s); break;
    case 96: attention_hd<96>(q, k, vt, B, S, H, KV, scale, out, s); break;
    case 128: attention_hd<128>(q, k, vt, B, S, H, KV, scale, out, s); break;
    default: break;
  }
}

void launch_final_norm_bf16(const float* x, const float* gain, int M, int D, uint16_t* h, cudaStream_t s) {
  kernel_launches() += 1;
  k_final_norm_bf16<<<M, 256, 0, s>>>(x, gain, D, h);
}

void launch_ce_reduce(const float2* part, int ntiles, const float* tlogit, const int32_t* target, int B, int S,
                      int V, double* tok_loss, double* per_seq, double* total, unsigned* err, cudaStream_t s) {
  kernel_launches() += 3;
  const int T = B * S;
  k_ce_rows<<<(T + 7) / 8, 256, 0, s>>>(part, ntiles, tlogit, target, T, V, tok_loss, err);
  k_seq_mean<<<B, 256, 0, s>>>(tok_loss, S, per_seq);
  k_mean<<<1, 32, 0, s>>>(per_seq, B, total);
}

void launch_head_ce_last(const float* x, const float* gain, const uint16_t* head, const int32_t* targets, int B,
                         int S, int D, int V, int C, double* per_seq, double* total, cudaStream_t s) {
  kernel_launches() += 2;
  k_head_ce_last<<<B, 256, 0, s>>>(x, gain, head, targets, S, D, V, C, per_seq);
  k_mean<<<1, 32, 0, s>>>(per_seq, B, total);
}

}  // namespace tmz
