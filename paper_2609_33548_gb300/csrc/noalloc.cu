// Allocation-free variant of the per-projection absmean reduction.
//
// Some callers cannot allocate device memory at all: code embedded in a
// host framework that owns every byte of the GPU (a serving engine that
// reserves the device memory up front, or one that forbids cudaMalloc on
// its hot path because it synchronises the device) cannot size and pass a
// workspace for termezo_create.  termezo_absmean_noalloc gives them the
// exact gamma / tau / s_w of one latent tensor without any allocation: its
// per-block partial sums live in the fixed device array below, which every
// GPU that loads this library holds until the process exits.
#include <cstdio>
#include <mutex>

#include "common.cuh"
#include "termezo.h"

namespace {

constexpr uint32_t kChunk = 4096;  // elements per block (16 per thread)
constexpr uint32_t kMaxBlocks = (uint32_t)(TERMEZO_NOALLOC_MAX_ELEMS / kChunk);
constexpr int kThreads = 256;
constexpr int kMaxDevices = 64;

// Shared by every call on a device; each call overwrites the slots it reads.
static __device__ __align__(256) tmz::ExactSum g_partials[kMaxBlocks];

__global__ void __launch_bounds__(kThreads) k_noalloc_partial(const float* __restrict__ w, uint64_t n,
                                                              tmz::ExactSum* __restrict__ parts) {
  __shared__ tmz::ExactSum red[kThreads / 32];
  tmz::ExactAcc acc;
  tmz::ea_zero(acc);
  const uint64_t start = (uint64_t)blockIdx.x * kChunk;
  for (uint32_t j = threadIdx.x; j < kChunk; j += kThreads) {
    const uint64_t i = start + j;
    if (i < n) tmz::ea_add_abs(acc, w[i]);
  }
  tmz::ExactSum s = tmz::ea_result(acc);
  tmz::es_block_reduce(s, red);
  if (threadIdx.x == 0) parts[blockIdx.x] = s;
}

__global__ void __launch_bounds__(kThreads) k_noalloc_final(const tmz::ExactSum* __restrict__ parts, uint32_t nb,
                                                            uint64_t n, float* __restrict__ out) {
  __shared__ tmz::ExactSum red[kThreads / 32];
  tmz::ExactSum s;
  tmz::es_zero(s);
  for (uint32_t b = threadIdx.x; b < nb; b += kThreads) tmz::es_merge(s, parts[b]);
  tmz::es_block_reduce(s, red);
  if (threadIdx.x == 0) tmz::gamma_tau(s, n, &out[0], &out[1], &out[2]);
}

std::mutex g_mu;
tmz::ExactSum* g_addr[kMaxDevices] = {};

// Device address of g_partials for the current device (looked up once per
// device; host code cannot use the symbol itself as a device pointer).  A
// cudaDeviceReset destroys the context that holds the array, so the cached
// address is void afterwards: callers must not reset a device they keep
// using with this entry point.
tmz::ExactSum* scratch_for_current_device(int* status) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    *status = TERMEZO_ECUDA;
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_partials) != cudaSuccess || !p) {
      *status = TERMEZO_ECUDA;
      return nullptr;
    }
    g_addr[dev] = reinterpret_cast<tmz::ExactSum*>(p);
  }
  *status = TERMEZO_OK;
  return g_addr[dev];
}

}  // namespace

extern "C" int termezo_absmean_noalloc(const float* d_w, uint64_t n, float* d_out, void* stream) {
  if (!d_w || !d_out || n == 0) return TERMEZO_EINVAL;
  if (n > TERMEZO_NOALLOC_MAX_ELEMS) {
    fprintf(stderr,
            "termezo_absmean_noalloc: %llu elements exceed the fixed scratch limit of %llu "
            "(TERMEZO_NOALLOC_MAX_ELEMS)\n",
            (unsigned long long)n, (unsigned long long)TERMEZO_NOALLOC_MAX_ELEMS);
    return TERMEZO_EINVAL;
  }
  int status = TERMEZO_OK;
  tmz::ExactSum* parts = scratch_for_current_device(&status);
  if (!parts) return status;
  uint32_t nb = (uint32_t)((n + kChunk - 1) / kChunk);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  // cudaLaunchKernel reports the error of this launch only: an earlier,
  // unrelated error pending on the thread is neither taken as this call's
  // failure nor cleared from the caller's view.
  void* a1[] = {(void*)&d_w, (void*)&n, (void*)&parts};
  if (cudaLaunchKernel((const void*)k_noalloc_partial, dim3(nb), dim3(kThreads), a1, 0, st) != cudaSuccess)
    return TERMEZO_ECUDA;
  void* a2[] = {(void*)&parts, (void*)&nb, (void*)&n, (void*)&d_out};
  if (cudaLaunchKernel((const void*)k_noalloc_final, dim3(1), dim3(kThreads), a2, 0, st) != cudaSuccess)
    return TERMEZO_ECUDA;
  return TERMEZO_OK;
}
