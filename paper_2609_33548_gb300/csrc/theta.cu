// Dense perturbation and update of the full-precision parameters theta
// (Algorithm 1 perturbs and updates them with the same seed and g as the
// masked latents): token embeddings and RMSNorm gains in float32, the LM
// head in bfloat16.  Their z is the Philox stream of the seed at global
// indices d + j (after the d latents), j running over the embeddings, then
// the gains, then the head.  Every assignment of Algorithm 1 is rounded to
// the stored precision of the part: float32, and for the head the float32
// result rounded to bfloat16 (nearest even).
//
// One thread handles the four consecutive elements that share one Philox
// counter (d and every part size are multiples of 4), so each Philox call
// serves four parameters; parts are read as float4 (fp32) or 8-byte words
// (4 x bf16).
#include <cuda_bf16.h>

#include "common.cuh"
#include "kernels.cuh"
#include "sparse.cuh"

namespace tmz {

namespace {

constexpr int THETA_TPB = 256;

// The four normals of Philox counter g (global indices 4g .. 4g+3), each
// computed exactly as normal_at computes it.
__device__ __forceinline__ void normal4(uint64_t seed, uint64_t g, float (&z)[4]) {
  const uint4 u = philox4x32_10(make_uint4((uint32_t)g, (uint32_t)(g >> 32), 0u, 0u), (uint32_t)seed,
                                (uint32_t)(seed >> 32));
  const float r0 = sqrtf(__fmul_rn(-2.0f, logf(philox_uniform(u.x))));
  const float r1 = sqrtf(__fmul_rn(-2.0f, logf(philox_uniform(u.z))));
  float s0, c0, s1, c1;
  sincospif(__fmul_rn(2.0f, philox_uniform(u.y)), &s0, &c0);
  sincospif(__fmul_rn(2.0f, philox_uniform(u.w)), &s1, &c1);
  z[0] = __fmul_rn(r0, c0);
  z[1] = __fmul_rn(r0, s0);
  z[2] = __fmul_rn(r1, c1);
  z[3] = __fmul_rn(r1, s1);
}

__device__ __forceinline__ float bf16_to_f32(uint16_t h) { return __uint_as_float((uint32_t)h << 16); }
__device__ __forceinline__ uint16_t f32_to_bf16(float x) {
  const __nv_bfloat16 b = __float2bfloat16_rn(x);
  return *reinterpret_cast<const uint16_t*>(&b);
}

// Loads / stores the four parameters of group q (global theta offset 4q).
struct Quad {
  float v[4];
  int part;  // 0 embeddings, 1 gains, 2 head
  uint64_t off;
};

__device__ __forceinline__ Quad load_quad(const ThetaArgs& t, uint64_t q) {
  Quad Q;
  uint64_t j = 4 * q;
  if (j < t.n_emb) {
    Q.part = 0;
    Q.off = j;
    const float4 x = *reinterpret_cast<const float4*>(t.emb + j);
    Q.v[0] = x.x, Q.v[1] = x.y, Q.v[2] = x.z, Q.v[3] = x.w;
  } else if ((j -= t.n_emb) < t.n_gains) {
    Q.part = 1;
    Q.off = j;
    const float4 x = *reinterpret_cast<const float4*>(t.gains + j);
    Q.v[0] = x.x, Q.v[1] = x.y, Q.v[2] = x.z, Q.v[3] = x.w;
  } else {
    j -= t.n_gains;
    Q.part = 2;
    Q.off = j;
    const uint2 x = *reinterpret_cast<const uint2*>(t.head + j);
    Q.v[0] = bf16_to_f32((uint16_t)(x.x & 0xFFFFu));
    Q.v[1] = bf16_to_f32((uint16_t)(x.x >> 16));
    Q.v[2] = bf16_to_f32((uint16_t)(x.y & 0xFFFFu));
    Q.v[3] = bf16_to_f32((uint16_t)(x.y >> 16));
  }
  return Q;
}

// The stored value of a freshly computed float32 result.
__device__ __forceinline__ float stored(const Quad& Q, float x) {
  return Q.part == 2 ? bf16_to_f32(f32_to_bf16(x)) : x;
}

__device__ __forceinline__ void store_quad(const ThetaArgs& t, const Quad& Q) {
  if (Q.part == 0) {
    *reinterpret_cast<float4*>(t.emb + Q.off) = make_float4(Q.v[0], Q.v[1], Q.v[2], Q.v[3]);
  } else if (Q.part == 1) {
    *reinterpret_cast<float4*>(t.gains + Q.off) = make_float4(Q.v[0], Q.v[1], Q.v[2], Q.v[3]);
  } else {
    uint2 x;
    x.x = (uint32_t)f32_to_bf16(Q.v[0]) | ((uint32_t)f32_to_bf16(Q.v[1]) << 16);
    x.y = (uint32_t)f32_to_bf16(Q.v[2]) | ((uint32_t)f32_to_bf16(Q.v[3]) << 16);
    *reinterpret_cast<uint2*>(t.head + Q.off) = x;
  }
}

// mode 0: theta = theta + e (the + pass and the restore); mode 1: theta =
// theta - 2 e (the - pass); e = fl(eps z).
__global__ void __launch_bounds__(THETA_TPB) k_theta_pm(ThetaArgs t, uint64_t seed, float eps, int mode) {
  const uint64_t nq = (t.n_emb + t.n_gains + t.n_head) / 4;
  for (uint64_t q = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; q < nq; q += (uint64_t)gridDim.x * blockDim.x) {
    Quad Q = load_quad(t, q);
    float z[4];
    normal4(seed, (t.d >> 2) + q, z);
#pragma unroll
    for (int l = 0; l < 4; ++l) {
      const float e = __fmul_rn(eps, z[l]);
      Q.v[l] = stored(Q, mode ? __fsub_rn(Q.v[l], __fmul_rn(2.0f, e)) : __fadd_rn(Q.v[l], e));
    }
    store_quad(t, Q);
  }
}

// The last direction's restore, then theta = theta - fl(c_k z_k) for every
// direction k in order, c_k = (float)((lr / K) g_k).
template <int KM>
__global__ void __launch_bounds__(THETA_TPB) k_theta_update(ThetaArgs t, UpdateDirs d, float eps, float lr,
                                                             const double* g_dev) {
  const double lr_k = (double)lr / (double)d.K;
  float c[KM];
#pragma unroll
  for (int k = 0; k < KM; ++k) c[k] = k < d.K ? (float)(lr_k * g_dev[k]) : 0.f;
  const uint64_t last = KM == 1 ? d.seed[0] : d.last;
  const uint64_t nq = (t.n_emb + t.n_gains + t.n_head) / 4;
  for (uint64_t q = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; q < nq; q += (uint64_t)gridDim.x * blockDim.x) {
    Quad Q = load_quad(t, q);
    const uint64_t g = (t.d >> 2) + q;
    float zl[4];
    normal4(last, g, zl);
#pragma unroll
    for (int l = 0; l < 4; ++l) Q.v[l] = stored(Q, __fadd_rn(Q.v[l], __fmul_rn(eps, zl[l])));
#pragma unroll
    for (int k = 0; k < KM; ++k)
      if (k < d.K) {
        float z[4];
        if (KM == 1 || k == d.K - 1) {
#pragma unroll
          for (int l = 0; l < 4; ++l) z[l] = zl[l];
        } else {
          normal4(d.seed[k], g, z);
        }
#pragma unroll
        for (int l = 0; l < 4; ++l) Q.v[l] = stored(Q, __fsub_rn(Q.v[l], __fmul_rn(c[k], z[l])));
      }
    store_quad(t, Q);
  }
}

int theta_grid(const ThetaArgs& t) {
  static int sms = 0;
  if (!sms) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) !=
                                                   cudaSuccess || sms <= 0)
      sms = 148;
  }
  const uint64_t nq = (t.n_emb + t.n_gains + t.n_head) / 4;
  const uint64_t want = (nq + THETA_TPB - 1) / THETA_TPB;
  const uint64_t cap = (uint64_t)sms * 8;
  return (int)(want < cap ? (want ? want : 1) : cap);
}

}  // namespace

void theta_pm(const ThetaArgs& t, uint64_t seed, float eps, int mode, cudaStream_t s) {
  kernel_launches() += 1;
  k_theta_pm<<<theta_grid(t), THETA_TPB, 0, s>>>(t, seed, eps, mode);
}

void theta_update(const ThetaArgs& t, const UpdateDirs& d, float eps, float lr, const double* g_dev, cudaStream_t s) {
  kernel_launches() += 1;
  if (d.K == 1)
    k_theta_update<1><<<theta_grid(t), THETA_TPB, 0, s>>>(t, d, eps, lr, g_dev);
  else
    k_theta_update<KMAX><<<theta_grid(t), THETA_TPB, 0, s>>>(t, d, eps, lr, g_dev);
}

}  // namespace tmz
