// Device helpers shared by the TerMeZO kernels (sm_103a).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace tmz {

typedef unsigned __int128 u128;

// Error bits recorded by kernels in the context's device error word.
enum : unsigned {
  ERR_TIMEOUT = 1u,   // a bounded wait (mbarrier) gave up
  ERR_BOUNDS = 2u,    // an index failed its bounds check
};

// ---------------------------------------------------------------------------
// Exact sum of |w| over fp32 values (the absmean gamma of Sec. 3).
// |w| = m * 2^(e' - 150) with m < 2^24 and e' = max(biased exponent, 1).
// Bucket b = e' >> 6 accumulates m << (e' & 63) (< 2^88) in a 128-bit
// integer, so 2^40 additions cannot overflow.  Integer sums are exact, so
// the total does not depend on the order of accumulation.
// ---------------------------------------------------------------------------
struct ExactSum {
  u128 b[4];
};

__device__ __forceinline__ void es_zero(ExactSum& s) {
#pragma unroll
  for (int i = 0; i < 4; ++i) s.b[i] = 0;
}

__device__ __forceinline__ void es_add_abs(ExactSum& s, float w) {
  uint32_t bits = __float_as_uint(w) & 0x7FFFFFFFu;
  uint32_t e = bits >> 23;
  uint32_t m = bits & 0x7FFFFFu;
  if (e) m |= 0x800000u;
  e = e ? e : 1u;
  const uint32_t bucket = e >> 6;
  const u128 v = ((u128)m) << (e & 63u);
#pragma unroll
  for (int i = 0; i < 4; ++i) s.b[i] += (bucket == (uint32_t)i) ? v : (u128)0;
}

__device__ __forceinline__ void es_merge(ExactSum& a, const ExactSum& o) {
#pragma unroll
  for (int i = 0; i < 4; ++i) a.b[i] += o.b[i];
}

// Per-thread accumulator with a fast path for |w| in [2^-63, 2) (biased
// exponent 64..127, bucket 1): m << (e - 64) is split into two 64-bit words
// (shift < 32, and shift - 32 for the rest, weighted 2^32), flushed into the
// 128-bit bucket every 16 values (16 * 2^55 < 2^63).  Other values take
// es_add_abs.  The result is the same exact integer.
struct ExactAcc {
  ExactSum s;
  uint64_t a0, a1;
  int cnt;
};

__device__ __forceinline__ void ea_zero(ExactAcc& a) {
  es_zero(a.s);
  a.a0 = a.a1 = 0;
  a.cnt = 0;
}

__device__ __forceinline__ void ea_flush(ExactAcc& a) {
  a.s.b[1] += (u128)a.a0 + ((u128)a.a1 << 32);
  a.a0 = a.a1 = 0;
  a.cnt = 0;
}

__device__ __forceinline__ void ea_add_abs(ExactAcc& a, float w) {
  const uint32_t bits = __float_as_uint(w) & 0x7FFFFFFFu;
  const uint32_t e = bits >> 23;
  if (e >= 64u && e < 128u) {
    const uint64_t m = (uint64_t)((bits & 0x7FFFFFu) | 0x800000u);
    const uint32_t sh = e - 64u;
    const uint64_t v = m << (sh & 31u);
    if (sh < 32u) a.a0 += v; else a.a1 += v;
    if (++a.cnt == 16) ea_flush(a);
  } else {
    es_add_abs(a.s, w);
  }
}

__device__ __forceinline__ const ExactSum& ea_result(ExactAcc& a) {
  ea_flush(a);
  return a.s;
}

__device__ __forceinline__ u128 shfl_xor_u128(u128 v, int mask) {
  uint64_t lo = (uint64_t)v, hi = (uint64_t)(v >> 64);
  lo = __shfl_xor_sync(0xffffffffu, lo, mask);
  hi = __shfl_xor_sync(0xffffffffu, hi, mask);
  return ((u128)hi << 64) | lo;
}

// Buckets that are zero in every lane (usually all but bucket 1) are skipped.
__device__ __forceinline__ void es_warp_reduce(ExactSum& s) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    if (!__any_sync(0xffffffffu, s.b[i] != 0)) continue;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s.b[i] += shfl_xor_u128(s.b[i], off);
  }
}

// Block reduction into thread 0's s (blockDim.x a multiple of 32, <= 1024).
// `scratch` holds blockDim.x/32 ExactSum entries of shared memory.
__device__ __forceinline__ void es_block_reduce(ExactSum& s, ExactSum* scratch) {
  es_warp_reduce(s);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) scratch[warp] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w) es_merge(s, scratch[w]);
  }
  __syncthreads();
}

// Correctly rounded (nearest, ties to even) float64 value of the exact sum.
__device__ __forceinline__ double es_to_double(const ExactSum& s) {
  // 384-bit integer L = sum_b s.b[b] * 2^(64 b), little-endian limbs.
  uint64_t L[6] = {0, 0, 0, 0, 0, 0};
  for (int i = 0; i < 4; ++i) {
    const uint64_t add[2] = {(uint64_t)s.b[i], (uint64_t)(s.b[i] >> 64)};
    uint64_t carry = 0;
    for (int j = i; j < 6; ++j) {
      const uint64_t a = (j - i < 2) ? add[j - i] : 0;
      const uint64_t t = L[j] + a;
      const uint64_t c1 = t < a;
      const uint64_t t2 = t + carry;
      const uint64_t c2 = t2 < carry;
      L[j] = t2;
      carry = c1 | c2;  // at most one of the two can be set
    }
  }
  int top = -1;
  for (int i = 5; i >= 0; --i)
    if (L[i]) { top = i; break; }
  if (top < 0) return 0.0;
  const int nbits = 64 * top + (64 - __clzll((long long)L[top]));
  if (nbits <= 53) return ldexp((double)L[0], -150);
  const int shift = nbits - 53;
  auto bits_at = [&](int pos, int count) -> uint64_t {  // count <= 64
    uint64_t r = 0;
    const int li = pos >> 6, bo = pos & 63;
    r = L[li] >> bo;
    if (bo && li + 1 < 6) r |= L[li + 1] << (64 - bo);
    if (count < 64) r &= ((uint64_t)1 << count) - 1;
    return r;
  };
  uint64_t mant = bits_at(shift, 53);
  const uint64_t round = bits_at(shift - 1, 1);
  bool sticky = false;
  {
    const int below = shift - 1;  // bits [0, below) feed the sticky bit
    const int full = below >> 6;
    for (int i = 0; i < full; ++i) sticky |= (L[i] != 0);
    if (below & 63) sticky |= (L[full] & (((uint64_t)1 << (below & 63)) - 1)) != 0;
  }
  int e = shift;
  if (round && (sticky || (mant & 1))) {
    ++mant;
    if (mant == ((uint64_t)1 << 53)) {
      mant >>= 1;
      ++e;
    }
  }
  return ldexp((double)mant, e - 150);
}

// gamma = fl32(fl64(S) / n); tau = 0.5 * fl32(gamma + 1e-5); s_w = gamma + 1e-5.
__device__ __forceinline__ void gamma_tau(const ExactSum& s, uint64_t n, float* gamma, float* tau,
                                          float* sw) {
  const double sd = es_to_double(s);
  const float g = (float)(sd / (double)n);
  const float gs = __fadd_rn(g, 1e-5f);
  *gamma = g;
  *sw = gs;
  *tau = __fmul_rn(0.5f, gs);
}

// ---------------------------------------------------------------------------
// Eq. 2 quantizer (strict inequalities), as the stored 2-bit code q + 1.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t ternary_code(float w, float tau) {
  return w > tau ? 2u : (w < -tau ? 0u : 1u);
}

// Eq. 3 boundary distance min(|w - tau|, |w + tau|) = ||w| - tau| (fp32).
__device__ __forceinline__ float boundary_distance(float w, float tau) {
  return fabsf(__fsub_rn(fabsf(w), tau));
}

// ---------------------------------------------------------------------------
// Philox-4x32-10 (Salmon et al., SC'11) and Box-Muller normals.
// z_i: key (seed lo, seed hi), counter (i/4 lo, i/4 hi, 0, 0), word i mod 4;
// pairs (0,1), (2,3) -> r = sqrt(-2 ln x_a), (r cos 2 pi x_b, r sin 2 pi x_b);
// x = (2 (u >> 9) + 1) 2^-24.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint32_t lo0 = 0xD2511F53u * c.x, hi0 = __umulhi(0xD2511F53u, c.x);
    const uint32_t lo1 = 0xCD9E8D57u * c.z, hi1 = __umulhi(0xCD9E8D57u, c.z);
    c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
  return c;
}

__device__ __forceinline__ float philox_uniform(uint32_t u) {
  return (float)(((u >> 9) << 1) | 1u) * 5.9604644775390625e-08f;  // 2^-24, exact
}

// z for global index i (one Philox evaluation; callers needing the four
// lanes of a group should use normal4).
__device__ __forceinline__ float normal_at(uint64_t seed, uint64_t i) {
  const uint64_t g = i >> 2;
  const uint4 u = philox4x32_10(make_uint4((uint32_t)g, (uint32_t)(g >> 32), 0u, 0u),
                                (uint32_t)seed, (uint32_t)(seed >> 32));
  const int lane = (int)(i & 3);
  const uint32_t ua = (lane < 2) ? u.x : u.z;
  const uint32_t ub = (lane < 2) ? u.y : u.w;
  const float r = sqrtf(__fmul_rn(-2.0f, logf(philox_uniform(ua))));
  float s, c;
  sincospif(__fmul_rn(2.0f, philox_uniform(ub)), &s, &c);
  return (lane & 1) ? __fmul_rn(r, s) : __fmul_rn(r, c);
}

// ---------------------------------------------------------------------------
// Bounded waits: every device-side wait gives up after kWaitNs nanoseconds,
// records ERR_TIMEOUT and lets the kernel finish.
// ---------------------------------------------------------------------------
constexpr uint64_t kWaitNs = 2000000000ull;  // 2 s

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// ---------------------------------------------------------------------------
// Programmatic dependent launch.  The forward's kernels are launched so that
// each starts as soon as every CTA of the kernel before it on the stream has
// exited, without waiting for that grid's completion to be signalled: the
// launch and the set-up (barrier init, tensor-memory allocation, descriptor
// prefetch) overlap the predecessor's completion.  Every thread of such a
// kernel calls grid_dep_wait before its first global-memory access; the wait
// returns once the predecessor has completed and its writes are visible.  A
// grid completes only after all its threads passed the wait, so the ordering
// is transitive along the stream.  No kernel signals its dependents early:
// measured on GB300, successors resident next to a running persistent GEMM
// slowed the forward down (27.8 ms against 27.4 ms without the attribute,
// 27.0 ms with the successors released only as CTAs exit).  Launched without
// the attribute, the wait is a no-op.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void grid_dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

template <typename... KArgs, typename... Args>
cudaError_t launch_dependent(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                             Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

}  // namespace tmz
