// Mask selection (Eqs. 2-5) and the sparse perturb / requantise / update
// passes of Algorithm 1 over the sparse latent store.
//
// Dense passes (mask build) read the caller's dense latents in blocks of
// 4096 elements that never straddle two projections.  Sparse passes read
// the active-index list and its fp32 latents; each projection owns a fixed
// number of blocks, each block a contiguous part of the projection's
// segment of the (sorted) active list.  Per-projection sums of |w| are exact
// (ExactSum), so tau and therefore every ternary code is independent of
// the order in which blocks are reduced.
#include <cmath>

#include "common.cuh"
#include "kernels.cuh"
#include "sparse.cuh"

namespace tmz {

namespace {

// e4m3 byte of a stored code (q + 1 in {0, 1, 2}): -1 = 0xB8, 0 = 0x00, +1 = 0x38.
__device__ __forceinline__ uint8_t code_e4m3(uint32_t c) { return c == 2u ? 0x38 : (c == 0u ? 0xB8 : 0x00); }

constexpr int TPB = 256;
constexpr uint32_t DENSE_CHUNK = 4096;  // elements per dense block (16 per thread)

struct DenseRange {
  int proj;
  uint64_t start, end;
};

__device__ __forceinline__ DenseRange dense_range(const MaskArgs& a, uint32_t b) {
  DenseRange r;
  r.proj = a.dproj[b];
  r.start = a.base[r.proj] + (uint64_t)(b - a.dpre[r.proj]) * DENSE_CHUNK;
  const uint64_t e = r.start + DENSE_CHUNK;
  r.end = e < a.base[r.proj + 1] ? e : a.base[r.proj + 1];
  return r;
}

struct SparseRange {
  int proj;
  uint32_t beg, end, seg_beg, seg_end;
};

__device__ __forceinline__ SparseRange sparse_range(const MaskArgs& a, const uint32_t* off, uint32_t b) {
  SparseRange r;
  r.proj = a.sproj[b];
  const uint32_t nb = a.spre[r.proj + 1] - a.spre[r.proj];
  const uint32_t j = b - a.spre[r.proj];
  r.seg_beg = off[r.proj];
  r.seg_end = off[r.proj + 1];
  const uint32_t len = r.seg_end - r.seg_beg;
  const uint32_t chunk = (len + nb - 1) / nb;
  const uint64_t lo = (uint64_t)j * chunk, hi = (uint64_t)(j + 1) * chunk;
  r.beg = r.seg_beg + (uint32_t)(lo < len ? lo : len);
  r.end = r.seg_beg + (uint32_t)(hi < len ? hi : len);
  return r;
}

__device__ __forceinline__ void load16(const float* w, uint64_t i, float (&v)[16]) {
  const float4* p = reinterpret_cast<const float4*>(w + i);
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const float4 t = p[q];
    v[4 * q] = t.x; v[4 * q + 1] = t.y; v[4 * q + 2] = t.z; v[4 * q + 3] = t.w;
  }
}

// Exclusive block scan of one uint32 per thread (blockDim.x == TPB).
__device__ __forceinline__ uint32_t block_excl_scan(uint32_t v, uint32_t* sh, uint32_t* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  __syncthreads();
  if (lane == 31) sh[warp] = x;
  __syncthreads();
  uint32_t wpre = 0, tot = 0;
  for (int i = 0; i < TPB / 32; ++i) {
    if (i < warp) wpre += sh[i];
    tot += sh[i];
  }
  if (total) *total = tot;
  return wpre + x - v;
}

// Loads the 4096-element chunk of a dense block with a coalesced pattern
// (thread t reads float4 number q * 256 + t); for passes where the order of
// elements within the block does not matter.
__device__ __forceinline__ int load16_coalesced(const float* w, const DenseRange& r, float (&v)[16]) {
  int n = 0;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const uint64_t i = r.start + 4ull * (q * TPB + threadIdx.x);
    float4 t = make_float4(0.f, 0.f, 0.f, 0.f);
    if (i < r.end) {
      t = *reinterpret_cast<const float4*>(w + i);
      n = 4 * (q + 1);
    }
    v[4 * q] = t.x; v[4 * q + 1] = t.y; v[4 * q + 2] = t.z; v[4 * q + 3] = t.w;
  }
  return n;  // valid values are a prefix of v (chunk lengths are multiples of 16)
}

// ----------------------------------------------------------- dense passes --

__global__ void __launch_bounds__(TPB) k_dense_sum(MaskArgs a, const float* __restrict__ w) {
  __shared__ ExactSum red[TPB / 32];
  const DenseRange r = dense_range(a, blockIdx.x);
  ExactAcc acc;
  ea_zero(acc);
  float v[16];
  const int n = load16_coalesced(w, r, v);
#pragma unroll
  for (int j = 0; j < 16; ++j)
    if (j < n) ea_add_abs(acc, v[j]);
  ExactSum s = ea_result(acc);
  es_block_reduce(s, red);
  if (threadIdx.x == 0) a.partials[blockIdx.x] = s;
}

// One block per projection: S = sum of the block partials [lo, hi) (+ add
// when non-null), then gamma, tau, s_w of the projection.
__global__ void k_reduce_proj(const ExactSum* __restrict__ parts, const uint32_t* __restrict__ pre, int stride,
                              int slot, const ExactSum* __restrict__ add, const uint64_t* __restrict__ base,
                              ExactSum* __restrict__ out_sum, float* gamma, float* tau, float* sw) {
  __shared__ ExactSum red[TPB / 32];
  const int p = blockIdx.x;
  ExactSum s;
  es_zero(s);
  for (uint32_t b = pre[p] + threadIdx.x; b < pre[p + 1]; b += blockDim.x) es_merge(s, parts[(size_t)b * stride + slot]);
  es_block_reduce(s, red);
  if (threadIdx.x == 0) {
    if (add) es_merge(s, add[p]);
    if (out_sum) out_sum[p] = s;
    if (tau) gamma_tau(s, base[p + 1] - base[p], &gamma[p], &tau[p], &sw[p]);
  }
}

__device__ __forceinline__ bool key_filter(uint32_t key, int pass, uint32_t prefix, uint32_t* bin) {
  if (pass == 0) { *bin = key >> 21; return true; }
  if (pass == 1) { *bin = (key >> 10) & 0x7FFu; return (key >> 21) == prefix; }
  *bin = key & 0x3FFu;
  return (key >> 10) == prefix;
}

// Radix histogram.  Pass 0 (top 10 bits of the key: the distances crowd a
// few exponent bins) counts into per-warp shared histograms to spread the
// shared-memory atomics; passes 1-2 see few matching keys and share one.
__global__ void __launch_bounds__(TPB) k_hist(MaskArgs a, const float* __restrict__ w, int pass) {
  constexpr int NB0 = 1024;  // keys of non-negative floats have bit 31 clear
  __shared__ uint32_t h[(TPB / 32) * NB0];
  const int warp = threadIdx.x >> 5;
  const int nz = pass == 0 ? (TPB / 32) * NB0 : 2048;
  for (int i = threadIdx.x; i < nz; i += TPB) h[i] = 0;
  __syncthreads();
  const DenseRange r = dense_range(a, blockIdx.x);
  const float tau = a.tau_cur[r.proj];
  const int grp = a.groups > 1 ? r.proj : 0;
  const uint32_t prefix = a.sel[grp].prefix;
  unsigned long long* hist = a.hist + (size_t)grp * 2048;
  float v[16];
  const uint64_t i0 = r.start + 16ull * threadIdx.x;
  const int n = i0 < r.end ? 16 : 0;
  if (n) load16(w, i0, v);
  uint32_t* hw = pass == 0 ? h + warp * NB0 : h;
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    uint32_t bin;
    if (j < n && key_filter(__float_as_uint(boundary_distance(v[j], tau)), pass, prefix, &bin))
      atomicAdd(&hw[bin], 1u);
  }
  __syncthreads();
  if (pass == 0) {
    for (int i = threadIdx.x; i < NB0; i += TPB) {
      uint32_t t = 0;
      for (int ww = 0; ww < TPB / 32; ++ww) t += h[ww * NB0 + i];
      if (t) atomicAdd(&hist[i], (unsigned long long)t);
    }
  } else {
    for (int i = threadIdx.x; i < 2048; i += TPB)
      if (h[i]) atomicAdd(&hist[i], (unsigned long long)h[i]);
  }
}

// Picks the radix bin that holds the krem-th smallest key (1-based).
// One block per selection group: the radix bin holding the group's rank.
__global__ void k_select(MaskArgs a, int pass) {
  SelectState* sel = a.sel + blockIdx.x;
  unsigned long long* hist = a.hist + (size_t)blockIdx.x * 2048;
  if (threadIdx.x == 0) {
    const int bins = pass < 2 ? 2048 : 1024;
    const int bits = pass < 2 ? 11 : 10;
    unsigned long long cum = 0, krem = sel->krem;
    int B = bins - 1;
    for (int i = 0; i < bins; ++i) {
      if (cum + hist[i] >= krem) { B = i; break; }
      cum += hist[i];
    }
    sel->krem = krem - cum;
    sel->prefix = pass == 0 ? (uint32_t)B : ((sel->prefix << bits) | (uint32_t)B);
  }
  __syncthreads();
  for (int i = threadIdx.x; i < 2048; i += blockDim.x) hist[i] = 0;
}

// xi_0 of every projection: the key its group's selection ended on.
__global__ void k_xi0(MaskArgs a) {
  for (int p = threadIdx.x; p < a.P; p += blockDim.x) a.xi0p[p] = __uint_as_float(a.sel[a.groups > 1 ? p : 0].prefix);
}

__global__ void __launch_bounds__(TPB) k_count(MaskArgs a, const float* __restrict__ w) {
  __shared__ uint32_t sh[TPB / 32];
  const DenseRange r = dense_range(a, blockIdx.x);
  const float tau = a.tau_cur[r.proj];
  const uint32_t key_p = a.sel[a.groups > 1 ? r.proj : 0].prefix;
  uint32_t less = 0, eq = 0;
  float v[16];
  const uint64_t i0 = r.start + 16ull * threadIdx.x;
  const int n = i0 < r.end ? 16 : 0;
  if (n) load16(w, i0, v);
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    if (j < n) {
      const uint32_t key = __float_as_uint(boundary_distance(v[j], tau));
      less += key < key_p;
      eq += key == key_p;
    }
  }
  uint32_t tl, te;
  block_excl_scan(less, sh, &tl);
  block_excl_scan(eq, sh, &te);
  if (threadIdx.x == 0) {
    a.blk_a[blockIdx.x] = tl;
    a.blk_b[blockIdx.x] = te;
  }
}

// Single block: per dense block b, ties before it (blk_d) and selected
// weights before it (blk_c), selecting the first `krem` ties in index order.
__device__ __forceinline__ unsigned long long scan1024(unsigned long long v, unsigned long long* sh) {
  __syncthreads();
  sh[threadIdx.x] = v;
  __syncthreads();
  for (int o = 1; o < 1024; o <<= 1) {
    const unsigned long long t = threadIdx.x >= (unsigned)o ? sh[threadIdx.x - o] : 0;
    __syncthreads();
    sh[threadIdx.x] += t;
    __syncthreads();
  }
  return sh[threadIdx.x] - v;  // exclusive
}

// Single block over the dense blocks in order: per block b, the selected
// weights before it (blk_c, a position in the sorted store) and the ties of
// its group before it (blk_d); group g selects the first sel[g].krem ties in
// index order.  Groups are runs of consecutive blocks (one projection each,
// or all of them).
__global__ void __launch_bounds__(1024) k_scan_dense(MaskArgs a, uint32_t nblk) {
  __shared__ unsigned long long sh[1024];
  const uint32_t per = (nblk + 1023) / 1024;
  const uint32_t b0 = min(nblk, threadIdx.x * per), b1 = min(nblk, b0 + per);
  auto group = [&](uint32_t b) { return a.groups > 1 ? (int)a.dproj[b] : 0; };
  unsigned long long eq = 0;
  for (uint32_t b = b0; b < b1; ++b) eq += a.blk_b[b];
  const unsigned long long tie_start = scan1024(eq, sh);
  // ties before the first block of each group
  unsigned long long tb = tie_start;
  for (uint32_t b = b0; b < b1; ++b) {
    const int g = group(b);
    if (b == (a.groups > 1 ? a.dpre[g] : 0u)) a.grp_tie0[g] = tb;
    tb += a.blk_b[b];
  }
  __syncthreads();
  unsigned long long sel = 0;
  tb = tie_start;
  for (uint32_t b = b0; b < b1; ++b) {
    const int g = group(b);
    const unsigned long long in = tb - a.grp_tie0[g], ties = a.sel[g].krem, e = a.blk_b[b];
    unsigned long long take = in >= ties ? 0 : (ties - in);
    if (take > e) take = e;
    sel += a.blk_a[b] + take;
    tb += e;
  }
  unsigned long long sel_before = scan1024(sel, sh);
  tb = tie_start;
  for (uint32_t b = b0; b < b1; ++b) {
    const int g = group(b);
    const unsigned long long in = tb - a.grp_tie0[g], ties = a.sel[g].krem, e = a.blk_b[b];
    a.blk_c[b] = (uint32_t)sel_before;
    a.blk_d[b] = (uint32_t)in;
    unsigned long long take = in >= ties ? 0 : (ties - in);
    if (take > e) take = e;
    sel_before += a.blk_a[b] + take;
    tb += e;
  }
}

// Writes S_0 (indices + latents, sorted) and the codes of every weight at tau_0.
__global__ void __launch_bounds__(TPB) k_compact(MaskArgs a, const float* __restrict__ w) {
  __shared__ uint32_t sh[TPB / 32];
  const DenseRange r = dense_range(a, blockIdx.x);
  const float tau = a.tau_cur[r.proj];
  const SelectState sg = a.sel[a.groups > 1 ? r.proj : 0];
  const uint32_t key_p = sg.prefix;
  const unsigned long long ties = sg.krem;
  const uint64_t i0 = r.start + 16ull * threadIdx.x;
  const bool live = i0 < r.end;
  float v[16];
  uint32_t keys[16];
  uint32_t eq = 0, word = 0;
  if (live) {
    load16(w, i0, v);
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      keys[j] = __float_as_uint(boundary_distance(v[j], tau));
      eq += keys[j] == key_p;
      word |= ternary_code(v[j], tau) << (2 * j);
    }
    a.packed[i0 >> 4] = word;
    if (a.wbyte) {
      uint32_t b[4];
#pragma unroll
      for (int q = 0; q < 4; ++q)
        b[q] = code_e4m3((word >> (8 * q)) & 3u) | (code_e4m3((word >> (8 * q + 2)) & 3u) << 8) |
               (code_e4m3((word >> (8 * q + 4)) & 3u) << 16) | (code_e4m3((word >> (8 * q + 6)) & 3u) << 24);
      *reinterpret_cast<uint4*>(a.wbyte + i0) = make_uint4(b[0], b[1], b[2], b[3]);
    }
  }
  unsigned long long tie_rank = (unsigned long long)a.blk_d[blockIdx.x] + block_excl_scan(eq, sh, nullptr);
  uint32_t selmask = 0, nsel = 0;
  if (live) {
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      bool s = keys[j] < key_p;
      if (keys[j] == key_p) {
        s = tie_rank < ties;
        ++tie_rank;
      }
      if (s) { selmask |= 1u << j; ++nsel; }
    }
  }
  uint32_t pos = a.blk_c[blockIdx.x] + block_excl_scan(nsel, sh, nullptr);
  if (live) {
#pragma unroll
    for (int j = 0; j < 16; ++j)
      if (selmask & (1u << j)) {
        a.idx[0][pos] = (uint32_t)(i0 + j);
        a.lat[0][pos] = v[j];
        ++pos;
      }
  }
}

__global__ void k_dense_offsets(MaskArgs a, uint32_t k0) {
  for (int p = threadIdx.x; p <= a.P; p += blockDim.x) a.off[0][p] = p < a.P ? a.blk_c[a.dpre[p]] : k0;
}

// ---------------------------------------------------------- sparse passes --

__global__ void __launch_bounds__(TPB) k_sparse_abs(MaskArgs a, int cur) {
  __shared__ ExactSum red[TPB / 32];
  const SparseRange r = sparse_range(a, a.off[cur], blockIdx.x);
  ExactAcc acc;
  ea_zero(acc);
  for (uint32_t e = r.beg + threadIdx.x; e < r.end; e += TPB) ea_add_abs(acc, a.lat[cur][e]);
  ExactSum s = ea_result(acc);
  es_block_reduce(s, red);
  if (threadIdx.x == 0) a.partials[blockIdx.x] = s;
}

// A = S_total - sum over active (bucket-wise; each bucket of the subset sum
// is at most the bucket of the full sum).
__global__ void k_frozen_init(MaskArgs a) {
  __shared__ ExactSum red[TPB / 32];
  const int p = blockIdx.x;
  ExactSum s;
  es_zero(s);
  for (uint32_t b = a.spre[p] + threadIdx.x; b < a.spre[p + 1]; b += blockDim.x) es_merge(s, a.partials[b]);
  es_block_reduce(s, red);
  if (threadIdx.x == 0) {
    ExactSum f = a.S_total[p];
    for (int i = 0; i < 4; ++i) f.b[i] -= s.b[i];
    a.A_frozen[p] = f;
  }
}

__device__ __forceinline__ void perturbed(float w, float z, float eps, float* wp, float* wm, float* ee) {
  *ee = __fmul_rn(eps, z);
  *wp = __fadd_rn(w, *ee);
  *wm = __fsub_rn(*wp, __fmul_rn(2.0f, *ee));
}

__global__ void __launch_bounds__(TPB, 3) k_sparse_pm_sum(MaskArgs a, int cur, uint64_t seed, float eps) {
  __shared__ ExactSum red[TPB / 32];
  const SparseRange r = sparse_range(a, a.off[cur], blockIdx.x);
  ExactAcc ap, am;
  ea_zero(ap);
  ea_zero(am);
  // four weights per iteration: their Philox chains are independent, so they
  // interleave (the exact sums do not depend on the order of the adds)
  for (uint32_t e0 = r.beg + threadIdx.x; e0 < r.end; e0 += 4 * TPB) {
    uint32_t id[4];
    float wv[4], z[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const uint32_t e = e0 + u * TPB;
      id[u] = e < r.end ? a.idx[cur][e] : 0u;
      wv[u] = e < r.end ? a.lat[cur][e] : 0.f;
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) z[u] = normal_at(seed, id[u]);
#pragma unroll
    for (int u = 0; u < 4; ++u)
      if (e0 + u * TPB < r.end) {
        if (a.zbuf) a.zbuf[e0 + u * TPB] = z[u];
        float wp, wm, ee;
        perturbed(wv[u], z[u], eps, &wp, &wm, &ee);
        ea_add_abs(ap, wp);
        ea_add_abs(am, wm);
      }
  }
  ExactSum sp = ea_result(ap), sm = ea_result(am);
  es_block_reduce(sp, red);
  if (threadIdx.x == 0) a.partials[2 * (size_t)blockIdx.x] = sp;
  es_block_reduce(sm, red);
  if (threadIdx.x == 0) a.partials[2 * (size_t)blockIdx.x + 1] = sm;
}

// Rewrites the codes of the active weights.  sign +1: w + eps z at tau+;
// sign -1: (w + eps z) - 2 eps z at tau- (and counts codes that differ from
// the + pass); sign 0: w at tau_cur.  Phase 1 computes the code of every
// element of the block's range in parallel (into shared memory); phase 2 has
// the first active element of each packed word (the "leader") read-modify-
// write that word, so no two threads write the same word.
constexpr uint32_t RQ_MAX = 4096;  // elements per sparse block (see the host's block plan)

// z of active weight e (global index i): from the z buffer (use_z) or regenerated.
__device__ __forceinline__ float z_of(const MaskArgs& a, bool use_z, uint64_t seed, uint32_t e, uint32_t i) {
  return use_z ? a.zbuf[e] : normal_at(seed, i);
}

__device__ __forceinline__ float requant_codes(const MaskArgs& a, int sign, uint64_t seed, float eps, float tau,
                                               float taup, uint32_t i, uint32_t e, bool use_z, float w,
                                               uint32_t* code, uint32_t* code_p) {
  if (sign == 0) {
    *code = ternary_code(w, tau);
    *code_p = *code;
    return w;
  }
  float wp, wm, ee;
  perturbed(w, z_of(a, use_z, seed, e, i), eps, &wp, &wm, &ee);
  const float ws = sign > 0 ? wp : wm;
  *code = ternary_code(ws, tau);
  *code_p = ternary_code(wp, taup);
  return ws;  // the latent this pass quantises
}

__global__ void __launch_bounds__(TPB) k_sparse_requant(MaskArgs a, int cur, uint64_t seed, float eps, int sign,
                                                        bool use_z) {
  __shared__ uint8_t sc[RQ_MAX];
  __shared__ unsigned long long cnt[4];
  if (threadIdx.x < 4) cnt[threadIdx.x] = 0;
  const SparseRange r = sparse_range(a, a.off[cur], blockIdx.x);
  const uint32_t* idx = a.idx[cur];
  const float* lat = a.lat[cur];
  const float* tau_sel = sign > 0 ? a.tau_plus : (sign < 0 ? a.tau_minus : a.tau_cur);
  const float tau = tau_sel[r.proj];
  const float taup = a.tau_plus[r.proj];
  // Near-threshold test of the oracle's report, | |w| - tau | < 1e-5 s_w in
  // float64: near the threshold |w| - tau is exact in fp32 (Sterbenz), and
  // for an fp32 distance "d < t" with t a float64 equals "d < t rounded up to
  // fp32", so one float64 product per block suffices.
  const float sw_sel = sign > 0 ? a.sw_plus[r.proj] : a.sw_minus[r.proj];
  const float near_thr = sign != 0 ? __double2float_ru(1e-5 * (double)sw_sel) : 0.f;
  const uint32_t n = r.end - r.beg;
  if (n > RQ_MAX) {  // cannot happen with the host's block plan; recorded, never silent
    if (threadIdx.x == 0) atomicOr(a.err, ERR_BOUNDS);
    return;
  }
  uint32_t flips = 0, jumps = 0, words = 0, near = 0;  // words: 32-byte sectors rewritten
  // phase 1: codes of the block's own elements (bits 0-1: this pass, 2-3: + pass)
  for (uint32_t j0 = threadIdx.x; j0 < n; j0 += 4 * TPB) {
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const uint32_t j = j0 + u * TPB;
      if (j < n) {
        uint32_t c, cp;
        const float ws =
            requant_codes(a, sign, seed, eps, tau, taup, idx[r.beg + j], r.beg + j, use_z, lat[r.beg + j], &c, &cp);
        near += boundary_distance(ws, tau) < near_thr;
        sc[j] = (uint8_t)(c | (cp << 2));
        if (a.wbyte) a.wbyte[idx[r.beg + j]] = code_e4m3(c);
      }
    }
  }
  __syncthreads();
  // phase 2: leaders rewrite their words
  for (uint32_t e = r.beg + threadIdx.x; e < r.end; e += TPB) {
    const uint32_t i = idx[e];
    if (e != r.seg_beg && (idx[e - 1] >> 4) == (i >> 4)) continue;  // not the leader
    const uint32_t wi = i >> 4;
    // the first rewritten word of a 32-byte sector (8 words) counts the sector
    if (e == r.seg_beg || (idx[e - 1] >> 7) != (i >> 7)) ++words;
    uint32_t word = a.packed[wi];
    for (uint32_t e2 = e; e2 < r.seg_end; ++e2) {
      const uint32_t i2 = idx[e2];
      if ((i2 >> 4) != wi) break;
      uint32_t code, cp;
      if (e2 < r.end) {
        const uint32_t v = sc[e2 - r.beg];
        code = v & 3u;
        cp = v >> 2;
      } else {  // follower in the next block's range
        requant_codes(a, sign, seed, eps, tau, taup, i2, e2, use_z, lat[e2], &code, &cp);
      }
      if (sign < 0) {
        flips += cp != code;
        jumps += (cp ^ code) == 2u;  // 0 <-> 2 in the stored q+1 form
      }
      const uint32_t sh = 2 * (i2 & 15u);
      word = (word & ~(3u << sh)) | (code << sh);
    }
    a.packed[wi] = word;
  }
  if (flips) atomicAdd(&cnt[0], (unsigned long long)flips);
  if (jumps) atomicAdd(&cnt[1], (unsigned long long)jumps);
  if (words) atomicAdd(&cnt[2], (unsigned long long)words);
  if (near) atomicAdd(&cnt[3], (unsigned long long)near);
  __syncthreads();
  if (threadIdx.x == 0) {
    if (cnt[0]) atomicAdd(&a.counters[0], cnt[0]);
    if (cnt[1]) atomicAdd(&a.counters[1], cnt[1]);
    if (cnt[2]) atomicAdd(&a.counters[3], cnt[2]);
    if (cnt[3]) atomicAdd(&a.counters[4], cnt[3]);
  }
}

// Restore and update: w' = ((w + e) - 2e) + e; w <- w' - fl32(c z) with
// c = (float)(lr * g); accumulates the exact sum of the new |w|.
// Algorithm 1's restore of the last direction followed by its update loop:
// w' = fl(w- + e) with the last direction's z, then for each direction k in
// order w = fl(w - fl(c_k z_k)), z_k regenerated from its seed.  Also the
// exact per-block sums of |w| of the result (the next tau).
template <int KM>
__global__ void __launch_bounds__(TPB) k_sparse_update(MaskArgs a, int cur, UpdateDirs d, float eps, float lr,
                                                       const double* g_dev, double g_host, int use_host, bool use_z) {
  __shared__ ExactSum red[TPB / 32];
  const SparseRange r = sparse_range(a, a.off[cur], blockIdx.x);
  const double lr_k = (double)lr / (double)d.K;
  float c[KM];
#pragma unroll
  for (int k = 0; k < KM; ++k) c[k] = k < d.K ? (float)(lr_k * (use_host ? g_host : g_dev[k])) : 0.f;
  const uint64_t last = KM == 1 ? d.seed[0] : d.last;
  ExactAcc acc;
  ea_zero(acc);
  if (KM == 1) {
    // four weights per iteration (independent Philox chains interleave)
    for (uint32_t e0 = r.beg + threadIdx.x; e0 < r.end; e0 += 4 * TPB) {
      uint32_t id[4];
      float wv[4], zl[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const uint32_t e = e0 + u * TPB;
        id[u] = e < r.end ? a.idx[cur][e] : 0u;
        wv[u] = e < r.end ? a.lat[cur][e] : 0.f;
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) zl[u] = (use_z && e0 + u * TPB < r.end) ? a.zbuf[e0 + u * TPB] : normal_at(last, id[u]);
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const uint32_t e = e0 + u * TPB;
        if (e < r.end) {
          float wp, wm, ee;
          perturbed(wv[u], zl[u], eps, &wp, &wm, &ee);
          const float wn = __fsub_rn(__fadd_rn(wm, ee), __fmul_rn(c[0], zl[u]));
          a.lat[cur][e] = wn;
          ea_add_abs(acc, wn);
        }
      }
    }
  } else {
    for (uint32_t e = r.beg + threadIdx.x; e < r.end; e += TPB) {
      const uint32_t i = a.idx[cur][e];
      const float zl = z_of(a, use_z, last, e, i);
      float wp, wm, ee;
      perturbed(a.lat[cur][e], zl, eps, &wp, &wm, &ee);
      float wn = __fadd_rn(wm, ee);
#pragma unroll
      for (int k = 0; k < KM; ++k)
        if (k < d.K) {
          const float z = (k == d.K - 1) ? zl : normal_at(d.seed[k], i);
          wn = __fsub_rn(wn, __fmul_rn(c[k], z));
        }
      a.lat[cur][e] = wn;
      ea_add_abs(acc, wn);
    }
  }
  ExactSum s = ea_result(acc);
  es_block_reduce(s, red);
  if (threadIdx.x == 0) a.partials[blockIdx.x] = s;
}

// Algorithm 1's restore after a direction that is not the last one.
__global__ void __launch_bounds__(TPB) k_sparse_restore(MaskArgs a, int cur, uint64_t seed, float eps, bool use_z) {
  const SparseRange r = sparse_range(a, a.off[cur], blockIdx.x);
  for (uint32_t e = r.beg + threadIdx.x; e < r.end; e += TPB) {
    float wp, wm, ee;
    perturbed(a.lat[cur][e], use_z ? a.zbuf[e] : normal_at(seed, a.idx[cur][e]), eps, &wp, &wm, &ee);
    a.lat[cur][e] = __fadd_rn(wm, ee);
  }
}

// Eq. 5 at tau_cur: marks dropped weights, writes their code at tau_cur,
// sums their |w| and counts the kept ones per block.  The block's indices
// and latents are staged in shared memory; thread t then owns entries
// t + TPB u, and the leader of a packed word (its first entry in the
// segment) rewrites the word when any of its entries was dropped.
__global__ void __launch_bounds__(TPB) k_shrink_mark(MaskArgs a, int cur) {
  constexpr int PER = RQ_MAX / TPB;
  __shared__ ExactSum red[TPB / 32];
  __shared__ uint32_t sh[TPB / 32];
  __shared__ uint32_t si[RQ_MAX];
  __shared__ float sl[RQ_MAX];
  __shared__ uint32_t s_prev;
  const SparseRange r = sparse_range(a, a.off[cur], blockIdx.x);
  const uint32_t* idx = a.idx[cur];
  const float* lat = a.lat[cur];
  const float tau = a.tau_cur[r.proj];
  const float xi0 = a.xi0p[r.proj];
  const uint32_t n = r.end - r.beg;
  if (n > RQ_MAX) {  // cannot happen with the host's block plan; recorded, never silent
    if (threadIdx.x == 0) atomicOr(a.err, ERR_BOUNDS);
    return;
  }
  ExactAcc acc;
  ea_zero(acc);
  uint32_t kept = 0, dropped = 0;
  if (threadIdx.x == 0) s_prev = r.beg > r.seg_beg ? idx[r.beg - 1] : 0xFFFFFFFFu;
  for (uint32_t j = threadIdx.x; j < n; j += TPB) {
    const float w = lat[r.beg + j];
    si[j] = idx[r.beg + j];
    sl[j] = w;
    if (boundary_distance(w, tau) <= xi0) {
      ++kept;
    } else {
      ++dropped;
      ea_add_abs(acc, w);
    }
  }
  __syncthreads();
#pragma unroll 4
  for (int u = 0; u < PER; ++u) {
    const uint32_t j = threadIdx.x + u * TPB;  // consecutive threads, consecutive entries
    if (j >= n) break;
    const uint32_t i = si[j], prev = j ? si[j - 1] : s_prev;
    if (prev != 0xFFFFFFFFu && (prev >> 4) == (i >> 4)) continue;  // not the leader
    const uint32_t wi = i >> 4;
    uint32_t set = 0, mask = 0;
    for (uint32_t e2 = r.beg + j; e2 < r.seg_end; ++e2) {
      const bool in_block = e2 < r.end;
      const uint32_t i2 = in_block ? si[e2 - r.beg] : idx[e2];
      if ((i2 >> 4) != wi) break;
      const float w2 = in_block ? sl[e2 - r.beg] : lat[e2];
      if (boundary_distance(w2, tau) > xi0) {
        const uint32_t shf = 2 * (i2 & 15u), code = ternary_code(w2, tau);
        mask |= 3u << shf;
        set |= code << shf;
        if (a.wbyte) a.wbyte[i2] = code_e4m3(code);
      }
    }
    if (mask) a.packed[wi] = (a.packed[wi] & ~mask) | set;
  }
  ExactSum s = ea_result(acc);
  es_block_reduce(s, red);
  if (threadIdx.x == 0) a.partials[blockIdx.x] = s;
  uint32_t tk, td;
  block_excl_scan(kept, sh, &tk);
  block_excl_scan(dropped, sh, &td);
  if (threadIdx.x == 0) {
    a.blk_a[blockIdx.x] = tk;
    if (td) atomicAdd(&a.counters[2], (unsigned long long)td);
  }
}

__global__ void k_frozen_add(MaskArgs a) {
  __shared__ ExactSum red[TPB / 32];
  const int p = blockIdx.x;
  ExactSum s;
  es_zero(s);
  for (uint32_t b = a.spre[p] + threadIdx.x; b < a.spre[p + 1]; b += blockDim.x) es_merge(s, a.partials[b]);
  es_block_reduce(s, red);
  if (threadIdx.x == 0) es_merge(a.A_frozen[p], s);
}

// Single block exclusive scan of blk_a[0..n) into blk_c; total into *total.
__global__ void __launch_bounds__(1024) k_scan_simple(MaskArgs a, uint32_t n, uint32_t* total) {
  __shared__ unsigned long long sh[1024];
  const uint32_t per = (n + 1023) / 1024;
  const uint32_t b0 = min(n, threadIdx.x * per), b1 = min(n, b0 + per);
  unsigned long long s = 0;
  for (uint32_t b = b0; b < b1; ++b) s += a.blk_a[b];
  unsigned long long run = scan1024(s, sh);
  if (threadIdx.x == 1023) *total = (uint32_t)(run + s);
  for (uint32_t b = b0; b < b1; ++b) {
    a.blk_c[b] = (uint32_t)run;
    run += a.blk_a[b];
  }
}

// The kept weights of the block, in order, to the other buffer.  Warp w owns
// entries 512 w .. 512 w + 511 (lane l: 512 w + 32 u + l, coalesced); a
// ballot per u ranks the kept entries of 32 consecutive ones, one block scan
// gives the warps their offsets.
__global__ void __launch_bounds__(TPB) k_shrink_scatter(MaskArgs a, int cur) {
  constexpr int PER = RQ_MAX / TPB;
  __shared__ uint32_t sh[TPB / 32];
  const SparseRange r = sparse_range(a, a.off[cur], blockIdx.x);
  const float tau = a.tau_cur[r.proj];
  const float xi0 = a.xi0p[r.proj];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t e0 = r.beg + (uint32_t)warp * 32 * PER + lane;
  uint32_t iv[PER], keep = 0, cnt = 0;
  float wv[PER];
#pragma unroll
  for (int u = 0; u < PER; ++u) {
    const uint32_t e = e0 + 32 * u;
    iv[u] = 0;
    wv[u] = 0.f;
    bool k = false;
    if (e < r.end) {
      wv[u] = a.lat[cur][e];
      iv[u] = a.idx[cur][e];
      k = boundary_distance(wv[u], tau) <= xi0;
    }
    const uint32_t b = __ballot_sync(0xffffffffu, k);
    keep |= (k ? 1u : 0u) << u;
    cnt += __popc(b);  // the warp's kept entries (the same in every lane)
  }
  // warp offsets: an exclusive scan of the warps' counts (lane 0's value)
  uint32_t wcnt = lane == 0 ? cnt : 0u;
  uint32_t woff = block_excl_scan(wcnt, sh, nullptr);
  woff = __shfl_sync(0xffffffffu, woff, 0);
  uint32_t pos = a.blk_c[blockIdx.x] + woff;
  const uint32_t lt = (1u << lane) - 1u;
#pragma unroll
  for (int u = 0; u < PER; ++u) {
    const bool k = keep & (1u << u);
    const uint32_t b = __ballot_sync(0xffffffffu, k);
    if (k) {
      const uint32_t p = pos + __popc(b & lt);
      a.idx[cur ^ 1][p] = iv[u];
      a.lat[cur ^ 1][p] = wv[u];
    }
    pos += __popc(b);
  }
}

__global__ void k_sparse_offsets(MaskArgs a, int out, const uint32_t* total) {
  for (int p = threadIdx.x; p <= a.P; p += blockDim.x) a.off[out][p] = p < a.P ? a.blk_c[a.spre[p]] : *total;
}

__global__ void k_grad(const double* loss, float eps, double* g) {
  if (threadIdx.x == 0) *g = (loss[0] - loss[1]) / (2.0 * (double)eps);
}

__global__ void k_normal(uint64_t seed, const uint32_t* idx, uint64_t n, float* z) {
  const uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) z[i] = normal_at(seed, idx[i]);
}

// -------------------------- mask build, two dense passes and a sampled one --
// The global quantile of Eq. 4 with two reads of the dense latents and a
// sample of a third: (1) the exact absmean sums (k_dense_sum_warp), (2) a fine
// histogram of the distance keys (13 bits: exponent and 5 mantissa bits, 32
// bins an octave) over every HIST_SAMPLE-th dense block (every block of a
// small model), which gives a bin bound holding k0 keys with a margin, (3) the
// order-preserving compaction of the "superset" -- every weight whose key
// falls in that bin or below -- into the second sparse-store buffer, with a
// decoupled look-back scan across blocks, written together with every code
// at tau_0 and counted by fine bin over the two octaves up to the bound.  The
// superset holds every key of those bins, so the counts give the exact bin of
// the k0-th key and the rank within it; the exact xi_0 and the ties are then
// resolved on the superset alone (two 9-bit radix passes over the weights of
// that bin, a count, a scan and an order-preserving scatter into S_0).  When
// the superset holds fewer than k0 weights (the sample missed), does not fit
// its buffer, or the k0-th key lies below the counted bins, the host runs the
// six-pass build instead.

constexpr int FINE_SHIFT = 18;                 // fine bin = key >> 18 (bit 31 of a distance is 0)
constexpr int HIST_DB = 16;                    // dense blocks per CTA of the histogram pass
constexpr uint32_t HIST_SAMPLE = 16;           // the histogram reads one dense block in HIST_SAMPLE ...
constexpr uint32_t HIST_SAMPLE_MIN = 65536;    // ... when the model has at least this many blocks
constexpr int SUP_DB = 8;                      // dense blocks per CTA of the superset compaction
constexpr int SUP_STAGE = 4096;                // superset entries a CTA stages in shared memory

// Pass 1 of the fast build: the exact sum of |w| of each dense block, one
// warp per block (float4 number q * 32 + lane for q < 32, no CTA barrier).
// For |w| in [2^-31, 2) (biased exponent e in [96, 128)) m << (e - 96) < 2^56
// is accumulated in one uint64 (128 values per lane: < 2^63); it is bucket 1
// of the ExactSum shifted by 32 (bucket 1 holds m << (e - 64) for e in
// [64, 128)), so the buckets hold the same integers as es_add_abs would put
// there.  Other values take ea_add_abs.
__global__ void __launch_bounds__(TPB) k_dense_sum_warp(MaskArgs a, const float* __restrict__ w) {
  const int lane = threadIdx.x & 31;
  const uint32_t b = blockIdx.x * (TPB / 32) + (threadIdx.x >> 5);
  if (b >= a.NBD) return;
  const DenseRange r = dense_range(a, b);
  ExactAcc acc;
  ea_zero(acc);
  uint64_t fx0 = 0, fx1 = 0;  // two chains (64 values each: < 2^62)
  auto add = [&](float v, uint64_t& fx) {
    const uint32_t bits = __float_as_uint(v) & 0x7FFFFFFFu;
    const uint32_t sh = (bits >> 23) - 96u;
    if (sh < 32u)
      fx += (uint64_t)((bits & 0x7FFFFFu) | 0x800000u) << sh;
    else if (bits)
      ea_add_abs(acc, v);
  };
  // eight float4 loads in flight per lane before they are summed
  for (int q0 = 0; q0 < (int)(DENSE_CHUNK / 128); q0 += 8) {
    float4 t[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const uint64_t i = r.start + 4ull * ((q0 + u) * 32 + lane);
      t[u] = i < r.end ? *reinterpret_cast<const float4*>(w + i) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      add(t[u].x, fx0);
      add(t[u].y, fx1);
      add(t[u].z, fx0);
      add(t[u].w, fx1);
    }
  }
  ExactSum s = ea_result(acc);
  s.b[1] += (u128)(fx0 + fx1) << 32;
  es_warp_reduce(s);
  if (lane == 0) a.partials[b] = s;
}

constexpr int FINE_BINS = 1 << (31 - FINE_SHIFT);
constexpr uint32_t SUP_CHUNK = 4096;           // superset entries per block of the resolution kernels

__device__ __forceinline__ uint32_t dist_key(float w, float tau) {
  return __float_as_uint(boundary_distance(w, tau));
}

// Projection of global index i (binary search over base[0..P]).
__device__ __forceinline__ int proj_of_index(const MaskArgs& a, uint32_t i) {
  int lo = 0, hi = a.P - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (a.base[mid] <= (uint64_t)i) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// Projections of increasing global indices (a thread's run of the sorted
// superset): one binary search, then a step forward whenever an index
// reaches the next projection's base (base[P] = d bounds every index).
struct ProjWalk {
  int p;
  uint64_t next;
  __device__ __forceinline__ void start(const MaskArgs& a, uint32_t i) {
    p = proj_of_index(a, i);
    next = a.base[p + 1];
  }
  __device__ __forceinline__ int at(const MaskArgs& a, uint32_t i) {
    while ((uint64_t)i >= next) next = a.base[++p + 1];
    return p;
  }
};

// Dense blocks read by the histogram pass: b = stride j + stride / 2.
__host__ __device__ __forceinline__ uint32_t sampled_blocks(uint32_t nbd, uint32_t stride) {
  return nbd > stride / 2 ? (nbd - stride / 2 + stride - 1) / stride : 0u;
}

// Pass 2: fine distance histogram of the sampled dense blocks, HIST_DB of them
// per CTA (one flush of the shared histogram).  Thread t reads float4 number
// q * TPB + t of a block (coalesced).
__global__ void __launch_bounds__(TPB) k_hist_fine(MaskArgs a, const float* __restrict__ w, uint32_t stride) {
  __shared__ uint32_t h[FINE_BINS];
  for (int i = threadIdx.x; i < FINE_BINS; i += TPB) h[i] = 0;
  __syncthreads();
  const uint32_t ns = sampled_blocks(a.NBD, stride);
  const uint32_t j0 = blockIdx.x * HIST_DB, j1 = min(ns, j0 + HIST_DB);
  for (uint32_t j = j0; j < j1; ++j) {
    const DenseRange r = dense_range(a, j * stride + stride / 2);
    const float tau = a.tau_cur[r.proj];
    float4 t[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const uint64_t i = r.start + 4ull * (q * TPB + threadIdx.x);
      t[q] = i < r.end ? *reinterpret_cast<const float4*>(w + i) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const uint64_t i = r.start + 4ull * (q * TPB + threadIdx.x);
      if (i < r.end) {
        atomicAdd(&h[dist_key(t[q].x, tau) >> FINE_SHIFT], 1u);
        atomicAdd(&h[dist_key(t[q].y, tau) >> FINE_SHIFT], 1u);
        atomicAdd(&h[dist_key(t[q].z, tau) >> FINE_SHIFT], 1u);
        atomicAdd(&h[dist_key(t[q].w, tau) >> FINE_SHIFT], 1u);
      }
    }
  }
  __syncthreads();
  for (int i = threadIdx.x; i < FINE_BINS; i += TPB)
    if (h[i]) atomicAdd(&a.hist[i], (unsigned long long)h[i]);
}

// The bin of `bins` (a.hist[0..bins), bins <= 8192) that holds the rank-th
// key, and clears the histogram.  Each thread sums a chunk of bins, thread 0
// finds the chunk and then the bin (the chunk's bins loaded at once).  Modes:
// SEL_RADIX appends the bin's `bits` to the prefix and makes krem the rank
// within it (rank = krem); SEL_BOUND sets the prefix to the first bin whose
// cumulative count reaches `target` (the last bin if none does) and leaves
// krem.
enum { SEL_RADIX = 0, SEL_BOUND = 1 };
__global__ void __launch_bounds__(256) k_select_fast(MaskArgs a, int bins, int bits, int mode,
                                                     unsigned long long target) {
  constexpr int MAXPER = 32;
  __shared__ unsigned long long csum[256];
  const int per = (bins + 255) / 256;
  {
    const int b0 = min(bins, (int)threadIdx.x * per), b1 = min(bins, b0 + per);
    unsigned long long sum = 0;
    for (int i = b0; i < b1; ++i) sum += a.hist[i];
    csum[threadIdx.x] = sum;
  }
  __syncthreads();
  if (threadIdx.x == 0 && per <= MAXPER) {
    SelectState* sel = a.sel;
    const unsigned long long krem = mode == SEL_BOUND ? target : sel->krem;
    unsigned long long cum = 0;
    int chunk = 255;
    for (int c = 0; c < 256; ++c) {
      if (cum + csum[c] >= krem) { chunk = c; break; }
      cum += csum[c];
    }
    const int c0 = chunk * per;
    unsigned long long v[MAXPER];
#pragma unroll
    for (int j = 0; j < MAXPER; ++j) v[j] = (j < per && c0 + j < bins) ? a.hist[c0 + j] : 0ull;
    int B = bins - 1;
    for (int j = 0; j < per && c0 + j < bins; ++j) {
      if (cum + v[j] >= krem) { B = c0 + j; break; }
      cum += v[j];
    }
    if (mode != SEL_BOUND) sel->krem = krem - cum;
    sel->prefix = mode == SEL_RADIX ? ((sel->prefix << bits) | (uint32_t)B) : (uint32_t)B;
  }
  __syncthreads();
  for (int i = threadIdx.x; i < bins; i += blockDim.x) a.hist[i] = 0;
}

__device__ __forceinline__ void st_release_u64(unsigned long long* p, unsigned long long v) {
  asm volatile("st.release.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ unsigned long long ld_acquire_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

// Decoupled look-back by one warp: the exclusive prefix of block b (blocks
// numbered in the order they took a ticket, so every block waits only on
// blocks that run or ran before it).  State words: 1 << 62 | aggregate,
// 2 << 62 | inclusive prefix.  The warp reads the states of 32 predecessors
// at once (lane j: block b - 1 - j, then the next 32 ...), adds the
// aggregates up to the nearest inclusive prefix and stops there.  Each wait
// is bounded (kWaitNs, decided by lane 0 for the whole warp); on time-out
// ERR_TIMEOUT is recorded and the prefix found so far is used.
__device__ unsigned long long lookback_prefix(const MaskArgs& a, uint32_t b, uint32_t total, int lane) {
  constexpr unsigned long long AGG = 1ull << 62, INC = 2ull << 62, VAL = (1ull << 62) - 1;
  if (b == 0) {
    if (lane == 0) st_release_u64(&a.scan_state[0], INC | total);
    return 0;
  }
  if (lane == 0) st_release_u64(&a.scan_state[b], AGG | total);
  unsigned long long excl = 0;
  long long base = (long long)b - 1;
  const uint64_t t0 = globaltimer_ns();
  bool timed_out = false;
  while (!timed_out) {
    const long long j = base - lane;
    unsigned long long sv = j >= 0 ? ld_acquire_u64(&a.scan_state[j]) : INC;  // before block 0: nothing
    while (__any_sync(0xffffffffu, (sv >> 62) == 0)) {
      int late = lane == 0 && globaltimer_ns() - t0 > kWaitNs;
      late = __shfl_sync(0xffffffffu, late, 0);
      if (late) {
        if (lane == 0) atomicOr(a.err, ERR_TIMEOUT);
        timed_out = true;
        break;
      }
      if ((sv >> 62) == 0) sv = ld_acquire_u64(&a.scan_state[j]);
    }
    if (timed_out) break;
    const unsigned inc = __ballot_sync(0xffffffffu, (sv >> 62) == 2);
    const int stop = inc ? __ffs(inc) - 1 : 31;  // the nearest inclusive prefix, or the whole window
    unsigned long long v = lane <= stop ? (sv & VAL) : 0ull;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    excl += v;
    if (inc) break;
    base -= 32;
  }
  if (lane == 0) st_release_u64(&a.scan_state[b], INC | (excl + total));
  return excl;
}

// Pass 3: every weight whose fine bin is at most the bound, in index order,
// into idx[1] / lat[1], and every code at tau_0.  A CTA takes SUP_DB
// consecutive dense blocks (in ticket order), one per warp.  A warp walks its
// block in index order (float4 number q * 32 + lane, q-major), ranks its
// selected weights with three ballots (the bits of each lane's count) per
// float4 and stages them in its share of shared memory, counting them by bin
// in its own row; one barrier gives the warps their offsets, the look-back
// the CTA's global offset, and the warps copy their weights out.  A warp with
// more than its share (a dense mask) makes the CTA read its blocks again and
// write directly.  The CTA with the last ticket stores the superset's size in
// sup[0]; entries past the buffer are not written (the size then exceeds
// sup_cap and the host builds the mask the other way).
constexpr int SUP_WSTAGE = SUP_STAGE / (TPB / 32);  // staged entries per warp
// The compaction also counts its selected weights by fine bin over the
// SUP_WIN bins up to the bound (two octaves) and in one count below them:
// enough to place the k0-th key unless the sample was off about 4-fold.
constexpr int SUP_WIN = 63;

// One warp's dense block b: the selected weights in index order, staged
// (stage) or written at out0 + their rank (!stage), and with stage the codes
// of the block (a packed word of 16 codes from the four lanes of a quad).
// Returns the count.
__device__ __forceinline__ uint32_t superset_warp(const MaskArgs& a, const float* __restrict__ w, uint32_t b,
                                                  uint32_t bmax, int lane, bool stage, uint32_t* st_idx,
                                                  float* st_lat, unsigned long long out0, uint32_t* s_win) {
  const DenseRange r = dense_range(a, b);
  const float tau = a.tau_cur[r.proj];
  const uint32_t lt = (1u << lane) - 1u;
  const uint32_t klim = (bmax + 1u) << FINE_SHIFT;  // fine bin <= bmax  <=>  key < klim (bmax < 8192)
  const uint32_t wlo = bmax >= (uint32_t)(SUP_WIN - 1) ? bmax - (SUP_WIN - 1) : 0u;  // first bin of the window
  uint32_t run = 0;
  for (int q0 = 0; q0 < (int)(DENSE_CHUNK / 128); q0 += 8) {
    float4 t[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const uint64_t i = r.start + 4ull * ((q0 + u) * 32 + lane);
      t[u] = i < r.end ? *reinterpret_cast<const float4*>(w + i) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const uint64_t i = r.start + 4ull * ((q0 + u) * 32 + lane);
      const bool live = i < r.end;  // uniform over a quad (chunk lengths are multiples of 16)
      const float vv[4] = {t[u].x, t[u].y, t[u].z, t[u].w};
      uint32_t m = 0, byte = 0;
      if (live) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          m |= (dist_key(vv[e], tau) < klim ? 1u : 0u) << e;
          byte |= ternary_code(vv[e], tau) << (2 * e);
        }
      }
      if (stage) {  // lane 4k gathers the bytes of lanes 4k .. 4k + 3
        const uint32_t h2 = byte | (__shfl_down_sync(0xffffffffu, byte, 1) << 8);
        const uint32_t wd = h2 | (__shfl_down_sync(0xffffffffu, h2, 2) << 16);
        if (live && (lane & 3) == 0) a.packed[i >> 4] = wd;
        if (live && a.wbyte)
          *reinterpret_cast<uint32_t*>(a.wbyte + i) = code_e4m3(byte & 3u) | (code_e4m3((byte >> 2) & 3u) << 8) |
                                                      (code_e4m3((byte >> 4) & 3u) << 16) |
                                                      (code_e4m3((byte >> 6) & 3u) << 24);
      }
      if (!__any_sync(0xffffffffu, m)) continue;
      // lane l's entries follow every selected entry of lanes < l: the
      // three bits of each lane's count (0 .. 4) by ballot
      const uint32_t c = __popc(m);
      const uint32_t s0 = __ballot_sync(0xffffffffu, c & 1u), s1 = __ballot_sync(0xffffffffu, c & 2u);
      const uint32_t s2 = __ballot_sync(0xffffffffu, c & 4u);
      uint32_t pos = run + __popc(s0 & lt) + 2u * __popc(s1 & lt) + 4u * __popc(s2 & lt);
#pragma unroll
      for (int e = 0; e < 4; ++e)
        if (m & (1u << e)) {
          if (stage) {
            if (pos < SUP_WSTAGE) {
              st_idx[pos] = (uint32_t)i + e;
              st_lat[pos] = vv[e];
            }
            const uint32_t bin = dist_key(vv[e], tau) >> FINE_SHIFT;  // <= bmax
            atomicAdd(&s_win[bin >= wlo ? 1u + (bin - wlo) : 0u], 1u);
          } else if (out0 + pos < a.sup_cap) {
            a.idx[1][out0 + pos] = (uint32_t)i + e;
            a.lat[1][out0 + pos] = vv[e];
          }
          ++pos;
        }
      run += __popc(s0) + 2u * __popc(s1) + 4u * __popc(s2);
    }
  }
  return run;
}

__global__ void __launch_bounds__(TPB, 4) k_superset(MaskArgs a, const float* __restrict__ w) {
  __shared__ uint32_t s_bid;
  __shared__ unsigned long long s_excl;
  __shared__ uint32_t s_wcnt[TPB / 32];
  __shared__ uint32_t st_idx[SUP_STAGE];
  __shared__ float st_lat[SUP_STAGE];
  // per warp: [0] below the window, [1 + j] its bin j (only the warp's own lanes add to its row)
  __shared__ uint32_t s_win[TPB / 32][SUP_WIN + 1];
  if (threadIdx.x == 0) s_bid = atomicAdd(&a.sup[2], 1u);
  for (int j = threadIdx.x; j < (TPB / 32) * (SUP_WIN + 1); j += TPB) (&s_win[0][0])[j] = 0;
  __syncthreads();
  const uint32_t c = s_bid;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t b = c * SUP_DB + warp;
  const uint32_t bmax = a.sel->prefix;
  uint32_t* my_idx = st_idx + warp * SUP_WSTAGE;
  float* my_lat = st_lat + warp * SUP_WSTAGE;
  const uint32_t n = b < a.NBD ? superset_warp(a, w, b, bmax, lane, true, my_idx, my_lat, 0, s_win[warp]) : 0u;
  if (lane == 0) s_wcnt[warp] = n;
  __syncthreads();
  if (threadIdx.x <= SUP_WIN) {
    uint32_t c = 0;
#pragma unroll
    for (int k = 0; k < TPB / 32; ++k) c += s_win[k][threadIdx.x];
    if (c) atomicAdd(&a.hist[threadIdx.x], (unsigned long long)c);
  }
  uint32_t woff = 0, total = 0;
  bool fits = true;
  for (int k = 0; k < TPB / 32; ++k) {
    if (k < warp) woff += s_wcnt[k];
    total += s_wcnt[k];
    fits = fits && s_wcnt[k] <= SUP_WSTAGE;
  }
  if (warp == 0) {
    const unsigned long long e = lookback_prefix(a, c, total, lane);
    if (lane == 0) {
      s_excl = e;
      if (c + 1 == gridDim.x) a.sup[0] = (uint32_t)min(e + total, 0xFFFFFFFFull);
    }
  }
  __syncthreads();
  const unsigned long long base = s_excl + woff;
  if (fits) {
    for (uint32_t j = lane; j < n; j += 32)
      if (base + j < a.sup_cap) {
        a.idx[1][base + j] = my_idx[j];
        a.lat[1][base + j] = my_lat[j];
      }
  } else if (b < a.NBD) {
    superset_warp(a, w, b, bmax, lane, false, my_idx, my_lat, base, s_win[warp]);
  }
}

// After the compaction: sup[1] = 1 when the superset holds fewer than k0
// weights or more than its buffer; otherwise the exact fine bin of the k0-th
// key from the compaction's window counts (hist[0] below the window, hist[1
// + j] in its bin j) -- the superset holds every key of those bins -- into
// the prefix, and the rank within it into krem.  A k0-th key below the
// window also sets sup[1].  Clears the counts.
__global__ void k_sup_window(MaskArgs a, uint32_t k0) {
  if (threadIdx.x == 0) {
    SelectState* sel = a.sel;
    const uint32_t n = a.sup[0], bmax = sel->prefix;
    const uint32_t wlo = bmax >= (uint32_t)(SUP_WIN - 1) ? bmax - (SUP_WIN - 1) : 0u;
    const unsigned long long krem = sel->krem;
    bool ok = n >= k0 && n <= a.sup_cap;
    unsigned long long cum = a.hist[0];
    int B = -1;
    if (cum >= krem) ok = false;
    for (int j = 0; ok && j < SUP_WIN; ++j) {
      const unsigned long long c = a.hist[1 + j];
      if (cum + c >= krem) {
        B = j;
        break;
      }
      cum += c;
    }
    ok = ok && B >= 0;
    if (ok) {
      sel->krem = krem - cum;
      sel->prefix = wlo + (uint32_t)B;
    }
    a.sup[1] = ok ? 0u : 1u;
  }
  __syncthreads();
  for (int i = threadIdx.x; i <= SUP_WIN; i += blockDim.x) a.hist[i] = 0;
}

// Radix passes over the superset's weights in the fine bin: pass 1 keys
// bits 17..9 of those in bin prefix, pass 2 bits 8..0 of those whose top 23
// bits match the prefix.
__global__ void __launch_bounds__(TPB) k_sup_hist(MaskArgs a, int pass) {
  __shared__ uint32_t h[512];
  for (int i = threadIdx.x; i < 512; i += TPB) h[i] = 0;
  __syncthreads();
  const bool live = !a.sup[1];
  const uint32_t n = a.sup[0], prefix = a.sel->prefix;
  const uint32_t e0 = blockIdx.x * TPB + threadIdx.x, step = gridDim.x * TPB;
  ProjWalk pw;
  if (live && e0 < n) pw.start(a, a.idx[1][e0]);
  for (uint32_t e = e0; live && e < n; e += step) {
    const uint32_t key = dist_key(a.lat[1][e], a.tau_cur[pw.at(a, a.idx[1][e])]);
    if (pass == 1 && (key >> FINE_SHIFT) == prefix) atomicAdd(&h[(key >> 9) & 511u], 1u);
    if (pass == 2 && (key >> 9) == prefix) atomicAdd(&h[key & 511u], 1u);
  }
  __syncthreads();
  for (int i = threadIdx.x; i < 512; i += TPB)
    if (h[i]) atomicAdd(&a.hist[i], (unsigned long long)h[i]);
}

// Per superset block: weights below the key of xi_0 (blk_a) and equal to it (blk_b).
__global__ void __launch_bounds__(TPB) k_sup_count(MaskArgs a) {
  __shared__ uint32_t sh[TPB / 32];
  const uint32_t n = a.sup[0], key_p = a.sel->prefix;
  const uint32_t lo = blockIdx.x * SUP_CHUNK, hi = min(n, lo + SUP_CHUNK);
  if (a.sup[1] || lo >= n) return;  // (uniform) blocks past the superset own no scratch entry
  uint32_t less = 0, eq = 0;
  ProjWalk pw;
  if (lo + threadIdx.x < hi) pw.start(a, a.idx[1][lo + threadIdx.x]);
  for (uint32_t e = lo + threadIdx.x; e < hi; e += TPB) {
    const uint32_t key = dist_key(a.lat[1][e], a.tau_cur[pw.at(a, a.idx[1][e])]);
    less += key < key_p;
    eq += key == key_p;
  }
  uint32_t tl, te;
  block_excl_scan(less, sh, &tl);
  block_excl_scan(eq, sh, &te);
  if (threadIdx.x == 0) {
    a.blk_a[blockIdx.x] = tl;
    a.blk_b[blockIdx.x] = te;
  }
}

// Single block over the superset blocks: selected weights before each block
// (blk_c) and ties before it (blk_d); the first krem ties in index order are
// kept.
__global__ void __launch_bounds__(1024) k_scan_sup(MaskArgs a) {
  __shared__ unsigned long long sh[1024];
  const uint32_t nblk = a.sup[1] ? 0u : (a.sup[0] + SUP_CHUNK - 1) / SUP_CHUNK;
  const uint32_t per = (nblk + 1023) / 1024;
  const uint32_t b0 = min(nblk, threadIdx.x * per), b1 = min(nblk, b0 + per);
  const unsigned long long ties = a.sel->krem;
  unsigned long long eq = 0;
  for (uint32_t b = b0; b < b1; ++b) eq += a.blk_b[b];
  unsigned long long tb = scan1024(eq, sh);
  unsigned long long sel = 0, t = tb;
  for (uint32_t b = b0; b < b1; ++b) {
    unsigned long long take = t >= ties ? 0 : ties - t;
    if (take > a.blk_b[b]) take = a.blk_b[b];
    sel += a.blk_a[b] + take;
    t += a.blk_b[b];
  }
  unsigned long long sb = scan1024(sel, sh);
  t = tb;
  for (uint32_t b = b0; b < b1; ++b) {
    a.blk_c[b] = (uint32_t)sb;
    a.blk_d[b] = (uint32_t)t;
    unsigned long long take = t >= ties ? 0 : ties - t;
    if (take > a.blk_b[b]) take = a.blk_b[b];
    sb += a.blk_a[b] + take;
    t += a.blk_b[b];
  }
}

// S_0 from the superset, in index order, into idx[0] / lat[0].  Warp w of a
// block owns its entries 512 w .. 512 w + 511 (lane l: 512 w + 32 u + l,
// coalesced); ballots per u rank the ties and then the selected entries of
// 32 consecutive ones, and two block scans give the warps their offsets.
__global__ void __launch_bounds__(TPB) k_sup_scatter(MaskArgs a, uint32_t k0) {
  constexpr int PER = SUP_CHUNK / TPB;
  __shared__ uint32_t sh[TPB / 32];
  const uint32_t n = a.sup[0], key_p = a.sel->prefix;
  const unsigned long long ties = a.sel->krem;
  const uint32_t lo = blockIdx.x * SUP_CHUNK, hi = min(n, lo + SUP_CHUNK);
  if (a.sup[1] || lo >= n) return;  // (uniform)
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t lt = (1u << lane) - 1u;
  const uint32_t e0 = lo + (uint32_t)warp * 32 * PER + lane;
  uint32_t below = 0, tie = 0, nt = 0;  // bit u: entry e0 + 32 u below / equal to xi_0's key
  ProjWalk pw;
  if (e0 < hi) pw.start(a, a.idx[1][e0]);
#pragma unroll
  for (int u = 0; u < PER; ++u) {
    const uint32_t e = e0 + 32u * u;
    uint32_t key = 0xFFFFFFFFu;
    if (e < hi) key = dist_key(a.lat[1][e], a.tau_cur[pw.at(a, a.idx[1][e])]);
    below |= (key < key_p ? 1u : 0u) << u;
    tie |= (key == key_p ? 1u : 0u) << u;
    nt += __popc(__ballot_sync(0xffffffffu, key == key_p));
  }
  uint32_t t_off = block_excl_scan(lane == 0 ? nt : 0u, sh, nullptr);
  unsigned long long tr = (unsigned long long)a.blk_d[blockIdx.x] + __shfl_sync(0xffffffffu, t_off, 0);
  uint32_t selm = 0, ns = 0;
#pragma unroll
  for (int u = 0; u < PER; ++u) {
    const bool t = (tie >> u) & 1u;
    const uint32_t bt = __ballot_sync(0xffffffffu, t);
    const bool s = ((below >> u) & 1u) || (t && tr + __popc(bt & lt) < ties);
    selm |= (s ? 1u : 0u) << u;
    ns += __popc(__ballot_sync(0xffffffffu, s));
    tr += __popc(bt);
  }
  const uint32_t s_off = block_excl_scan(lane == 0 ? ns : 0u, sh, nullptr);
  uint32_t pos = a.blk_c[blockIdx.x] + __shfl_sync(0xffffffffu, s_off, 0);
#pragma unroll
  for (int u = 0; u < PER; ++u) {
    const bool s = (selm >> u) & 1u;
    const uint32_t bs = __ballot_sync(0xffffffffu, s);
    if (s) {
      const uint32_t p = pos + __popc(bs & lt), e = e0 + 32u * u;
      if (p < k0) {
        a.idx[0][p] = a.idx[1][e];
        a.lat[0][p] = a.lat[1][e];
      } else {
        atomicOr(a.err, ERR_BOUNDS);  // more than k0 selected: never silent
      }
    }
    pos += __popc(bs);
  }
}

// off[0][p]: entries of S_0 below projection p (binary search of base[p]).
__global__ void k_off_search(MaskArgs a, uint32_t k0) {
  for (int p = threadIdx.x; p <= a.P; p += blockDim.x) {
    if (p == a.P) { a.off[0][p] = k0; continue; }
    uint32_t lo = 0, hi = k0;
    while (lo < hi) {
      const uint32_t mid = (lo + hi) >> 1;
      if ((uint64_t)a.idx[0][mid] < a.base[p]) lo = mid + 1; else hi = mid;
    }
    a.off[0][p] = lo;
  }
}

}  // namespace

// ----------------------------------------------------------- host side ----

void mask_build(const MaskArgs& a, const float* w, uint64_t k0, cudaStream_t s) {
  kernel_launches() += 13;
  k_dense_sum<<<a.NBD, TPB, 0, s>>>(a, w);
  k_reduce_proj<<<a.P, TPB, 0, s>>>(a.partials, a.dpre, 1, 0, nullptr, a.base, a.S_total, a.gamma_cur, a.tau_cur,
                                    a.sw_cur);
  for (int pass = 0; pass < 3; ++pass) {
    k_hist<<<a.NBD, TPB, 0, s>>>(a, w, pass);
    k_select<<<a.groups, 256, 0, s>>>(a, pass);
  }
  k_count<<<a.NBD, TPB, 0, s>>>(a, w);
  k_scan_dense<<<1, 1024, 0, s>>>(a, a.NBD);
  k_compact<<<a.NBD, TPB, 0, s>>>(a, w);
  k_dense_offsets<<<1, 256, 0, s>>>(a, (uint32_t)k0);
  k_xi0<<<1, 256, 0, s>>>(a);
}

void mask_build_fast(const MaskArgs& a, const float* w, uint64_t k0, cudaStream_t s) {
  kernel_launches() += 14;
  k_dense_sum_warp<<<(a.NBD + TPB / 32 - 1) / (TPB / 32), TPB, 0, s>>>(a, w);
  k_reduce_proj<<<a.P, TPB, 0, s>>>(a.partials, a.dpre, 1, 0, nullptr, a.base, a.S_total, a.gamma_cur, a.tau_cur,
                                    a.sw_cur);
  // The bound: with every block read, the k0-th key's bin; with a sample of
  // one block in HIST_SAMPLE, the first bin whose sampled count reaches
  // (k0 / HIST_SAMPLE) (1 + 1/100) plus eight binomial standard deviations.
  const uint32_t stride = a.NBD >= HIST_SAMPLE_MIN ? HIST_SAMPLE : 1u;
  const uint32_t ns = sampled_blocks(a.NBD, stride);
  const double ks = (double)k0 / stride;
  const unsigned long long target =
      stride == 1 ? (unsigned long long)k0 : (unsigned long long)(ks * 1.01 + 8.0 * sqrt(ks) + 64.0);
  k_hist_fine<<<(ns + HIST_DB - 1) / HIST_DB, TPB, 0, s>>>(a, w, stride);
  k_select_fast<<<1, 256, 0, s>>>(a, FINE_BINS, 0, SEL_BOUND, target);
  k_superset<<<(a.NBD + SUP_DB - 1) / SUP_DB, TPB, 0, s>>>(a, w);
  const uint32_t nsb = (a.sup_cap + SUP_CHUNK - 1) / SUP_CHUNK;
  const uint32_t nh = nsb < 1024u ? (nsb ? nsb : 1u) : 1024u;
  k_sup_window<<<1, 64, 0, s>>>(a, (uint32_t)k0);
  k_sup_hist<<<nh, TPB, 0, s>>>(a, 1);
  k_select_fast<<<1, 256, 0, s>>>(a, 512, 9, SEL_RADIX, 0);
  k_sup_hist<<<nh, TPB, 0, s>>>(a, 2);
  k_select_fast<<<1, 256, 0, s>>>(a, 512, 9, SEL_RADIX, 0);
  k_sup_count<<<nsb ? nsb : 1u, TPB, 0, s>>>(a);
  k_scan_sup<<<1, 1024, 0, s>>>(a);
  k_sup_scatter<<<nsb ? nsb : 1u, TPB, 0, s>>>(a, (uint32_t)k0);
  k_xi0<<<1, 256, 0, s>>>(a);
}

cudaError_t mask_preload() {
  // CUDA loads a kernel at its first launch; the mask build runs once per
  // context, so its kernels are loaded here instead of inside the build
  const void* kernels[] = {(const void*)k_dense_sum_warp, (const void*)k_reduce_proj, (const void*)k_hist_fine,
                           (const void*)k_select_fast,   (const void*)k_superset,    (const void*)k_sup_window,
                           (const void*)k_sup_hist,      (const void*)k_sup_count,   (const void*)k_scan_sup,
                           (const void*)k_sup_scatter,   (const void*)k_xi0,         (const void*)k_off_search,
                           (const void*)k_sparse_abs,    (const void*)k_frozen_init, (const void*)k_dense_sum,
                           (const void*)k_hist,          (const void*)k_select,      (const void*)k_count,
                           (const void*)k_scan_dense,    (const void*)k_compact,     (const void*)k_dense_offsets};
  for (const void* k : kernels) {
    cudaFuncAttributes at;
    const cudaError_t e = cudaFuncGetAttributes(&at, k);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

void mask_build_fast_offsets(const MaskArgs& a, uint64_t k0, cudaStream_t s) {
  kernel_launches() += 1;
  k_off_search<<<1, 256, 0, s>>>(a, (uint32_t)k0);
}

void mask_finish(const MaskArgs& a, cudaStream_t s) {
  kernel_launches() += 2;
  k_sparse_abs<<<a.NBS, TPB, 0, s>>>(a, 0);
  k_frozen_init<<<a.P, TPB, 0, s>>>(a);
}

void sparse_pm_taus(const MaskArgs& a, int cur, uint64_t seed, float eps, cudaStream_t s) {
  kernel_launches() += 3;
  k_sparse_pm_sum<<<a.NBS, TPB, 0, s>>>(a, cur, seed, eps);
  k_reduce_proj<<<a.P, TPB, 0, s>>>(a.partials, a.spre, 2, 0, a.A_frozen, a.base, nullptr, a.gamma_plus, a.tau_plus,
                                    a.sw_plus);
  k_reduce_proj<<<a.P, TPB, 0, s>>>(a.partials, a.spre, 2, 1, a.A_frozen, a.base, nullptr, a.gamma_minus,
                                    a.tau_minus, a.sw_minus);
}

void sparse_requant(const MaskArgs& a, int cur, uint64_t seed, float eps, int sign, bool use_z, cudaStream_t s) {
  kernel_launches() += 1;
  k_sparse_requant<<<a.NBS, TPB, 0, s>>>(a, cur, seed, eps, sign, use_z && a.zbuf);
}

void sparse_update(const MaskArgs& a, int cur, uint64_t seed, float eps, float lr, const double* g_dev, double g_host,
                   int use_host, bool use_z, cudaStream_t s) {
  kernel_launches() += 2;
  UpdateDirs d{};
  d.seed[0] = d.last = seed;
  d.K = 1;
  k_sparse_update<1><<<a.NBS, TPB, 0, s>>>(a, cur, d, eps, lr, g_dev, g_host, use_host, use_z && a.zbuf);
  k_reduce_proj<<<a.P, TPB, 0, s>>>(a.partials, a.spre, 1, 0, a.A_frozen, a.base, nullptr, a.gamma_cur, a.tau_cur,
                                    a.sw_cur);
}

void sparse_update_dirs(const MaskArgs& a, int cur, const UpdateDirs& d, float eps, float lr, const double* g_dev,
                        bool use_z, cudaStream_t s) {
  use_z = use_z && a.zbuf;
  kernel_launches() += 2;
  if (d.K == 1)
    k_sparse_update<1><<<a.NBS, TPB, 0, s>>>(a, cur, d, eps, lr, g_dev, 0.0, 0, use_z);
  else
    k_sparse_update<KMAX><<<a.NBS, TPB, 0, s>>>(a, cur, d, eps, lr, g_dev, 0.0, 0, use_z);
  k_reduce_proj<<<a.P, TPB, 0, s>>>(a.partials, a.spre, 1, 0, a.A_frozen, a.base, nullptr, a.gamma_cur, a.tau_cur,
                                    a.sw_cur);
}

void sparse_restore(const MaskArgs& a, int cur, uint64_t seed, float eps, bool use_z, cudaStream_t s) {
  kernel_launches() += 1;
  k_sparse_restore<<<a.NBS, TPB, 0, s>>>(a, cur, seed, eps, use_z && a.zbuf);
}

void sparse_shrink(const MaskArgs& a, int cur, uint32_t* d_total, cudaStream_t s) {
  kernel_launches() += 5;
  k_shrink_mark<<<a.NBS, TPB, 0, s>>>(a, cur);
  k_frozen_add<<<a.P, TPB, 0, s>>>(a);
  k_scan_simple<<<1, 1024, 0, s>>>(a, a.NBS, d_total);
  k_shrink_scatter<<<a.NBS, TPB, 0, s>>>(a, cur);
  k_sparse_offsets<<<1, 256, 0, s>>>(a, cur ^ 1, d_total);
}

void launch_grad(const double* loss, float eps, double* g, cudaStream_t s) {
  kernel_launches() += 1; k_grad<<<1, 32, 0, s>>>(loss, eps, g); }

void launch_normal(uint64_t seed, const uint32_t* idx, uint64_t n, float* z, cudaStream_t s) {
  if (n) ++kernel_launches();
  if (n) k_normal<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(seed, idx, n, z);
}

}  // namespace tmz
