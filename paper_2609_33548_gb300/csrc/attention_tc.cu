// Causal attention on the 5th-generation tensor cores (sm_103a), for head
// dims 64, 96 and 128 and sequence lengths that are multiples of 128.
//
// Same arithmetic as the mma.sync kernel: Q, K, V bf16; s = fl(acc * scale);
// pass 1 finds the exact row maximum m over the causal keys; pass 2 forms
// P = bf16(exp(s - m)) (exp on the special-function unit), l = sum P (fp32)
// and O = sum P V (fp32) / l.  Since scale > 0 and rounding is monotone,
// max fl(acc * scale) = fl(max acc * scale), so pass 1 reduces the raw
// accumulators.
//
// Persistent CTAs (one per SM, all 512 TMEM columns) walk a list of work
// items; an item is two 128-query tiles A and B that read the same KV head
// (two heads of a GQA group at the same query tile, or two neighbouring tiles
// of one head), so every K / V^T tile loaded serves both.  Items are ordered
// by decreasing causal length and dealt to the CTAs in a snake order.
// Warp 0 issues TMA loads (Q_A, Q_B; a ring of K and V^T tiles, 128-byte
// swizzle); one thread of warp 1 issues tcgen05.mma: S_t = Q_t K^T into TMEM
// buffer t (M 128, N 128, K hd) and O_t += P_t V (M 128, N hd, K 128) with P_t
// from shared memory.  Warps 4-7 own tile A, warps 8-11 tile B (thread = query
// row): they read S_t with tcgen05.ld, release the buffer at once (so S_t of
// the next key block is computed while they work), reduce the row maximum
// (pass 1) or form bf16 P rows in the swizzled K-major layout (pass 2), and
// hand l to warps 12-15, which divide O_t by l and store it while the softmax
// warps go on to the next item.  While one tile's warps run their softmax the
// tensor core works on the other tile.
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.cuh"
#include "tcgen05.cuh"

namespace tmz {

namespace {

// Registers a thread after setmaxnreg: warp 0 TMA, warp 1 MMA (warps 2-3
// idle) 96; the softmax warps 4-7 (tile A) and 8-11 (tile B) 168; the
// epilogue warps 12-15 80.  128 x 96 + 256 x 168 + 128 x 80 = 512 x 128, the
// registers the block is launched with (the host checks the kernel's register
// count before its first launch: a smaller one would leave setmaxnreg.inc
// waiting).  Of the splits that add up, this one spills least (24 bytes).
constexpr int ATT_THREADS = 512;
constexpr int REG_CTRL = 96, REG_SOFTMAX = 168, REG_EPI = 80, REG_LAUNCH = 128;
static_assert(128 * REG_CTRL + 256 * REG_SOFTMAX + 128 * REG_EPI == ATT_THREADS * REG_LAUNCH, "register split");
constexpr int BQ = 128, BKEY = 128;
constexpr int ATOM = 128 * 128;  // one 128-row x 64-element bf16 swizzle atom block

// A Q or K tile (128 rows x HD) is loaded as 64-column swizzle atoms; at HD
// 96 the second atom is half filled (TMA writes zeros past column 95, and the
// MMAs read only its first 32 columns).  A V^T tile is HD rows x 128 keys.
template <int HD>
struct AttTc {
  static constexpr int QK_ATOMS = (HD + 63) / 64;
  static constexpr int QK_BYTES = QK_ATOMS * ATOM;  // bytes TMA writes for a Q or K tile
  static constexpr int V_ATOM = HD * 128;           // V^T: HD rows x 64 keys
  static constexpr int V_BYTES = 2 * V_ATOM;        // bytes TMA writes for a V^T tile
  static constexpr int TILE = QK_BYTES > V_BYTES ? QK_BYTES : V_BYTES;  // a Q buffer or a ring slot
  static constexpr int NS = HD == 64 ? 6 : 3;       // K / V^T ring slots
  static constexpr int Q_OFF = 0;                  // Q_A, Q_B
  static constexpr int R_OFF = Q_OFF + 2 * TILE;   // ring
  static constexpr int P_OFF = R_OFF + NS * TILE;  // P_A, P_B: 128 x 128 bf16 each
  static constexpr int BAR_OFF = P_OFF + 2 * 2 * ATOM;
  static constexpr int L_OFF = BAR_OFF + 512;      // l of each row of A, B (fp32)
  static constexpr int BYTES = L_OFF + 2 * BQ * 4 + 1024;
};

struct AttItem {
  int b, kvh, qa, ha, qb, hb;  // hb < 0: the item has no tile B
};

// Item i: pair rank p = i / (B KV) over the query tiles of one KV head listed
// by decreasing tile index (then head), so n_A = qa + 1 >= n_B = qb + 1.
__device__ __forceinline__ AttItem att_item(int i, int B, int KV, int G, int NQ) {
  AttItem it;
  const int bk = i % (B * KV), u = 2 * (i / (B * KV));
  it.b = bk / KV;
  it.kvh = bk % KV;
  it.qa = NQ - 1 - u / G;
  it.ha = it.kvh * G + u % G;
  if (u + 1 < G * NQ) {
    it.qb = NQ - 1 - (u + 1) / G;
    it.hb = it.kvh * G + (u + 1) % G;
  } else {
    it.qb = -1;
    it.hb = -1;
  }
  return it;
}

// Snake deal: round r gives CTA c item r * G + c (r even) or r * G + G-1-c.
__device__ __forceinline__ int att_sched(int r, int grid, int c) {
  return r * grid + ((r & 1) ? grid - 1 - c : c);
}

__device__ __forceinline__ void fence_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void tmem_ld32_nowait(uint32_t taddr, uint32_t* r) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
        "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
        "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
        "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}

// Orders later uses of 32 registers after a tcgen05.wait::ld.
__device__ __forceinline__ void tmem_tie32(uint32_t* r) {
  asm volatile(""
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]),
                 "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]),
                 "+r"(r[14]), "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]), "+r"(r[20]),
                 "+r"(r[21]), "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]),
                 "+r"(r[28]), "+r"(r[29]), "+r"(r[30]), "+r"(r[31])::"memory");
}

// Loads NC x 32 consecutive TMEM columns of this warp's 32 lanes.
template <int NC>
__device__ __forceinline__ void tmem_ld_cols(uint32_t taddr, uint32_t* r) {
#pragma unroll
  for (int c = 0; c < NC; ++c) tmem_ld32_nowait(taddr + 32 * c, r + 32 * c);
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int c = 0; c < NC; ++c) tmem_tie32(r + 32 * c);
}

__device__ __forceinline__ float max3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// Paired fp32 arithmetic (one instruction for two lanes of a float2), each
// lane rounded to nearest like its scalar form.
__device__ __forceinline__ float2 mul2(float2 a, float2 b) {
  float2 d;
  asm("{\n .reg .b64 x, y, z;\n mov.b64 x, {%2, %3};\n mov.b64 y, {%4, %5};\n mul.rn.f32x2 z, x, y;\n"
      " mov.b64 {%0, %1}, z;\n}\n"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}
__device__ __forceinline__ float2 sub2(float2 a, float2 b) {
  float2 d;
  asm("{\n .reg .b64 x, y, z;\n mov.b64 x, {%2, %3};\n mov.b64 y, {%4, %5};\n sub.rn.f32x2 z, x, y;\n"
      " mov.b64 {%0, %1}, z;\n}\n"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}
__device__ __forceinline__ float2 add2(float2 a, float2 b) {
  float2 d;
  asm("{\n .reg .b64 x, y, z;\n mov.b64 x, {%2, %3};\n mov.b64 y, {%4, %5};\n add.rn.f32x2 z, x, y;\n"
      " mov.b64 {%0, %1}, z;\n}\n"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}

__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) {
  float2 d;
  asm("{\n .reg .b64 x, y, z, w;\n mov.b64 x, {%2, %3};\n mov.b64 y, {%4, %5};\n mov.b64 z, {%6, %7};\n"
      " fma.rn.f32x2 w, x, y, z;\n mov.b64 {%0, %1}, w;\n}\n"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  return d;
}

// o / l rounded to nearest (Markstein, 1990): with y = RN(1/l), q = RN(o y)
// and the exact residual r = o - l q (one FMA), RN(q + r y) is the correctly
// rounded quotient.  Two lanes at a time.
__device__ __forceinline__ float2 div2(float2 o, float2 l2, float2 y2) {
  const float2 q = mul2(o, y2);
  const float2 r = fma2(make_float2(-q.x, -q.y), l2, o);
  return fma2(r, y2, q);
}

__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, uint32_t src, int x, int y) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];" ::"l"((uint64_t)map),
               "r"(src), "r"(x), "r"(y)
               : "memory");
}

// Keys c > row of the diagonal block are outside the causal window: their
// accumulator becomes -inf, which the maximum ignores and exp maps to 0.
__device__ __forceinline__ void causal_mask(uint32_t* sv, int row) {
#pragma unroll
  for (int c = 0; c < BKEY; ++c) sv[c] = c <= row ? sv[c] : 0xff800000u;
}

// 2^x on the special-function unit.  P uses e^x = 2^(x log2 e) (x <= 0): its
// relative error, a few fp32 ulps for the |x| that carry weight, moves a
// bf16-rounded P to the neighbouring value for about one element in 10^4,
// like any other exp of fp32 accuracy.
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// P for keys c0 .. c0+7 of one row: 4 words of bf16 pairs; l2 += P (fp32).
__device__ __forceinline__ uint4 p_chunk(const uint32_t* sv, int c0, float2 sc, float2 m2, float2& l2) {
  const float2 log2e = make_float2(1.44269504088896341f, 1.44269504088896341f);
  uint32_t w[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float2 x = sub2(mul2(make_float2(__uint_as_float(sv[c0 + 2 * e]), __uint_as_float(sv[c0 + 2 * e + 1])), sc), m2);
    const float2 y = mul2(x, log2e);
    const __nv_bfloat162 b = __floats2bfloat162_rn(ex2_approx(y.x), ex2_approx(y.y));
    w[e] = *reinterpret_cast<const uint32_t*>(&b);
    l2 = add2(l2, make_float2(__uint_as_float(w[e] << 16), __uint_as_float(w[e] & 0xffff0000u)));
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

// Warp-uniform bounded wait (the tcgen05.ld that follows is warp-collective).
__device__ __forceinline__ bool mbar_wait_warp(uint32_t bar, uint32_t parity) {
  return __all_sync(0xffffffffu, mbar_wait(bar, parity));
}

template <int HD>
__global__ void __launch_bounds__(ATT_THREADS, 1)
    k_attention_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                   const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmO, int B, int S,
                   int H, int KV, float scale, unsigned* err) {
  using L = AttTc<HD>;
  constexpr int NS = L::NS;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  const uint32_t sb = smem_u32(smem);
  const uint32_t bar = sb + L::BAR_OFF;
  const uint32_t q_full = bar, q_empty = bar + 8, ring_full = bar + 16, ring_empty = ring_full + 8 * NS,
                 s_full = ring_empty + 8 * NS, s_free = s_full + 16, p_full = s_free + 16, p_free = p_full + 16,
                 o_full = p_free + 16, o_free = o_full + 16, fin = o_free + 16, l_full = fin + 8,
                 st_free = l_full + 16;
  uint32_t* tmem_slot = (uint32_t*)(smem + L::BAR_OFF + 496);
  static_assert(8 * (2 + 2 * (HD == 64 ? 6 : 3) + 12 + 1 + 4) <= 496, "barrier area");

  const int G = H / KV, NQ = S / BQ;
  const int n_items = B * KV * ((G * NQ + 1) / 2);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    mbar_init(q_empty, 1);
    for (int s = 0; s < NS; ++s) {
      mbar_init(ring_full + 8 * s, 1);
      mbar_init(ring_empty + 8 * s, 1);
    }
    for (int t = 0; t < 2; ++t) {
      mbar_init(s_full + 8 * t, 1);
      mbar_init(s_free + 8 * t, 4);
      mbar_init(p_full + 8 * t, 4);
      mbar_init(p_free + 8 * t, 1);
      mbar_init(o_full + 8 * t, 1);
      mbar_init(o_free + 8 * t, 4);
      mbar_init(l_full + 8 * t, 4);
      mbar_init(st_free + 8 * t, 4);
    }
    mbar_init(fin, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0 && lane == 0) {
    asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmQ) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmK) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmV) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmO) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(512));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;
  bool ok = true;
  // Q, K, V^T come from the kernel before this one
  grid_dep_wait();
  if (warp < 4) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(REG_CTRL));
  if (warp == 0) {
    if (lane == 0) {
      uint32_t rp = 0, nq = 0;
      for (int r = 0; ok; ++r) {
        if (r * (int)gridDim.x >= n_items) break;
        const int i = att_sched(r, gridDim.x, blockIdx.x);
        if (i >= n_items) continue;
        const AttItem it = att_item(i, B, KV, G, NQ);
        const int na = it.qa + 1;
        if (nq >= 1 && !(ok = mbar_wait(q_empty, (nq - 1) & 1u))) break;
        mbar_expect_tx(q_full, (it.hb >= 0 ? 2 : 1) * L::QK_BYTES);
        for (int a = 0; a < L::QK_ATOMS; ++a)
          tma_load_2d(sb + L::Q_OFF + a * ATOM, &tmQ, a * 64, (it.b * H + it.ha) * S + it.qa * BQ, q_full);
        if (it.hb >= 0)
          for (int a = 0; a < L::QK_ATOMS; ++a)
            tma_load_2d(sb + L::Q_OFF + L::TILE + a * ATOM, &tmQ, a * 64, (it.b * H + it.hb) * S + it.qb * BQ,
                        q_full);
        ++nq;
        const int rowK = (it.b * KV + it.kvh) * S, rowV = (it.b * KV + it.kvh) * HD;
        auto load = [&](bool v, int j) -> bool {
          const uint32_t slot = rp % NS, use = rp / NS;
          if (use >= 1 && !mbar_wait(ring_empty + 8 * slot, (use - 1) & 1u)) return false;
          const uint32_t dst = sb + L::R_OFF + slot * L::TILE, fb = ring_full + 8 * slot;
          mbar_expect_tx(fb, v ? L::V_BYTES : L::QK_BYTES);
          if (!v)
            for (int a = 0; a < L::QK_ATOMS; ++a) tma_load_2d(dst + a * ATOM, &tmK, a * 64, rowK + j * BKEY, fb);
          else
            for (int a = 0; a < 2; ++a) tma_load_2d(dst + a * L::V_ATOM, &tmV, j * BKEY + a * 64, rowV, fb);
          ++rp;
          return true;
        };
        for (int j = 0; j < na && ok; ++j) ok = load(false, j);  // pass 1: K
        if (ok) ok = load(false, 0);                             // pass 2: K_0, then (K_j+1, V_j)
        for (int j = 0; j < na && ok; ++j) {
          if (j + 1 < na) ok = load(false, j + 1);
          if (ok) ok = load(true, j);
        }
      }
      // copies still in flight land before the CTA exits
      for (uint32_t s = 0; s < (uint32_t)NS; ++s)
        if (rp > s) mbar_wait(ring_full + 8 * s, ((rp - 1 - s) / NS) & 1u);
      if (nq >= 1) mbar_wait(q_full, (nq - 1) & 1u);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t id_s = idesc_bf16(BQ, BKEY), id_o = idesc_bf16(BQ, HD);
      uint32_t rc = 0, nq = 0, cs[2] = {0, 0}, cp[2] = {0, 0}, co[2] = {0, 0};
      auto take = [&](uint32_t& slot) -> bool {
        slot = rc % NS;
        if (!mbar_wait(ring_full + 8 * slot, (rc / NS) & 1u)) return false;
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        return true;
      };
      auto release = [&](uint32_t slot) {
        mma_commit(ring_empty + 8 * slot);
        ++rc;
      };
      auto mma_s = [&](int t, uint32_t slot) -> bool {
        if (cs[t] >= 1 && !mbar_wait(s_free + 8 * t, (cs[t] - 1) & 1u)) return false;
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t q = sb + L::Q_OFF + t * L::TILE, k = sb + L::R_OFF + slot * L::TILE;
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk)
          mma_bf16(tmem + t * BKEY, sw128_desc(q + (kk >> 2) * ATOM) + (uint64_t)(2 * (kk & 3)),
                   sw128_desc(k + (kk >> 2) * ATOM) + (uint64_t)(2 * (kk & 3)), id_s, kk ? 1u : 0u);
        mma_commit(s_full + 8 * t);
        ++cs[t];
        return true;
      };
      auto mma_pv = [&](int t, uint32_t slot, int j) -> bool {
        if (j == 0 && co[t] >= 1 && !mbar_wait(o_free + 8 * t, (co[t] - 1) & 1u)) return false;
        if (!mbar_wait(p_full + 8 * t, cp[t] & 1u)) return false;
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t pa = sb + L::P_OFF + t * 2 * ATOM, v = sb + L::R_OFF + slot * L::TILE;
#pragma unroll
        for (int kk = 0; kk < BKEY / 16; ++kk)
          mma_bf16(tmem + 256 + t * 128, sw128_desc(pa + (kk >> 2) * ATOM) + (uint64_t)(2 * (kk & 3)),
                   sw128_desc(v + (kk >> 2) * L::V_ATOM) + (uint64_t)(2 * (kk & 3)), id_o, (j | kk) ? 1u : 0u);
        mma_commit(p_free + 8 * t);
        ++cp[t];
        return true;
      };
      for (int r = 0; ok; ++r) {
        if (r * (int)gridDim.x >= n_items) break;
        const int i = att_sched(r, gridDim.x, blockIdx.x);
        if (i >= n_items) continue;
        const AttItem it = att_item(i, B, KV, G, NQ);
        const int na = it.qa + 1, nb = it.qb + 1;
        if (!(ok = mbar_wait(q_full, nq & 1u))) break;
        ++nq;
        uint32_t slot;
        for (int j = 0; j < na && ok; ++j) {  // pass 1
          if (!(ok = take(slot))) break;
          ok = mma_s(0, slot) && (j >= nb || mma_s(1, slot));
          release(slot);
        }
        if (ok && (ok = take(slot))) {  // pass 2
          ok = mma_s(0, slot) && (nb < 1 || mma_s(1, slot));
          release(slot);
          if (na == 1) mma_commit(q_empty);  // the last MMA that reads Q
        }
        for (int j = 0; j < na && ok; ++j) {
          if (j + 1 < na) {
            if (!(ok = take(slot))) break;
            ok = mma_s(0, slot) && (j + 1 >= nb || mma_s(1, slot));
            release(slot);
            if (!ok) break;
            if (j + 2 == na) mma_commit(q_empty);
          }
          if (!(ok = take(slot))) break;
          ok = mma_pv(0, slot, j) && (j >= nb || mma_pv(1, slot, j));
          release(slot);
        }
        if (!ok) break;
        mma_commit(o_full);
        ++co[0];
        if (nb >= 1) {
          mma_commit(o_full + 8);
          ++co[1];
        }
      }
      // every MMA issued has completed before TMEM is released
      mma_commit(fin);
      if (!mbar_wait(fin, 0)) ok = false;
    }
  }
  } else if (warp < 12) {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(REG_SOFTMAX));
    // Softmax warps: warp w reads TMEM lanes 32 (w % 4) .. +31; lane = row.
    const int t = warp >= 8 ? 1 : 0;
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;
    const uint32_t lanes = (uint32_t)(quarter * 32) << 16;
    const uint32_t tS = tmem + lanes + t * BKEY;
    const uint32_t sfull = s_full + 8 * t, sfree = s_free + 8 * t, pfull = p_full + 8 * t, pfree = p_free + 8 * t,
                   lfull = l_full + 8 * t, stfree = st_free + 8 * t;
    uint8_t* prow = smem + L::P_OFF + t * 2 * ATOM + row * 128;
    float* lrow = reinterpret_cast<float*>(smem + L::L_OFF) + t * BQ + row;
    uint32_t ns = 0, np = 0, nit = 0;
    auto arrive = [&](uint32_t b) {
      __syncwarp();
      if (lane == 0) mbar_arrive(b);
    };
    for (int r = 0; ok; ++r) {
      if (r * (int)gridDim.x >= n_items) break;
      const int i = att_sched(r, gridDim.x, blockIdx.x);
      if (i >= n_items) continue;
      const AttItem it = att_item(i, B, KV, G, NQ);
      const int qt = t ? it.qb : it.qa, h = t ? it.hb : it.ha;
      if (h < 0) continue;
      const int n = qt + 1;
      uint32_t sv[BKEY];
      // pass 1: maximum of the raw accumulators over the causal keys
      float mx0 = -INFINITY, mx1 = -INFINITY;
      for (int j = 0; j < n; ++j) {
        if (!(ok = mbar_wait_warp(sfull, ns & 1u))) break;
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        tmem_ld_cols<BKEY / 32>(tS, sv);
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        arrive(sfree);
        ++ns;
        if (j + 1 == n) causal_mask(sv, row);
#pragma unroll
        for (int c = 0; c < BKEY; c += 4) {
          mx0 = max3(mx0, __uint_as_float(sv[c]), __uint_as_float(sv[c + 1]));
          mx1 = max3(mx1, __uint_as_float(sv[c + 2]), __uint_as_float(sv[c + 3]));
        }
      }
      if (!ok) break;
      const float m = __fmul_rn(fmaxf(mx0, mx1), scale);
      const float2 sc2 = make_float2(scale, scale), m2 = make_float2(m, m);
      // pass 2: P = bf16(exp(fl(s) - m)), l = sum P, P -> shared memory
      float2 la = make_float2(0.f, 0.f), lb = make_float2(0.f, 0.f);
      for (int j = 0; j < n; ++j) {
        if (!(ok = mbar_wait_warp(sfull, ns & 1u))) break;
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        tmem_ld_cols<BKEY / 32>(tS, sv);
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        arrive(sfree);
        ++ns;
        if (j + 1 == n) causal_mask(sv, row);
        // keys 8 ch .. 8 ch + 7 -> atom ch / 8, 16-byte chunk ch % 8, swizzled by row % 8
        uint4 pk[8];
#pragma unroll
        for (int ch = 0; ch < 8; ++ch) pk[ch] = p_chunk(sv, 8 * ch, sc2, m2, (ch & 1) ? lb : la);
        // P of the item's first block overwrites the epilogue's staging of
        // the previous item; later blocks wait for the P V that read P last
        if (j == 0 && nit >= 1 && !(ok = mbar_wait_warp(stfree, (nit - 1) & 1u))) break;
        if (np >= 1 && !(ok = mbar_wait_warp(pfree, (np - 1) & 1u))) break;
#pragma unroll
        for (int ch = 0; ch < 8; ++ch) *reinterpret_cast<uint4*>(prow + (((ch & 7) ^ (row & 7)) * 16)) = pk[ch];
#pragma unroll
        for (int ch = 8; ch < 16; ++ch)
          *reinterpret_cast<uint4*>(prow + ATOM + (((ch & 7) ^ (row & 7)) * 16)) =
              p_chunk(sv, 8 * ch, sc2, m2, (ch & 1) ? lb : la);
        fence_async_smem();
        arrive(pfull);
        ++np;
      }
      if (!ok) break;
      *lrow = __fadd_rn(__fadd_rn(la.x, la.y), __fadd_rn(lb.x, lb.y));
      arrive(lfull);
      ++nit;
    }
  } else {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(REG_EPI));
    // Epilogue warps 12-15: warp w reads TMEM lanes 32 (w % 4) .. +31; lane =
    // row.  Per item, tile A then tile B: O / l staged through the tile's P
    // buffer (free once the item's last P V has completed) in the 128-byte
    // swizzled layout; each warp writes its own 32 rows with TMA stores of
    // 32 x 32 fp32 boxes.  The softmax warps meanwhile start the next item.
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;
    const uint32_t lanes = (uint32_t)(quarter * 32) << 16;
    uint32_t ne[2] = {0, 0};
    auto arrive = [&](uint32_t b) {
      __syncwarp();
      if (lane == 0) mbar_arrive(b);
    };
    for (int r = 0; ok; ++r) {
      if (r * (int)gridDim.x >= n_items) break;
      const int i = att_sched(r, gridDim.x, blockIdx.x);
      if (i >= n_items) continue;
      const AttItem it = att_item(i, B, KV, G, NQ);
      for (int t = 0; t < 2 && ok; ++t) {
        const int qt = t ? it.qb : it.qa, h = t ? it.hb : it.ha;
        if (h < 0) continue;
        if (!(ok = mbar_wait_warp(l_full + 8 * t, ne[t] & 1u))) break;
        if (!(ok = mbar_wait_warp(o_full + 8 * t, ne[t] & 1u))) break;
        ++ne[t];
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const float l = reinterpret_cast<const float*>(smem + L::L_OFF)[t * BQ + row];
        const float2 l2 = make_float2(l, l), y2 = make_float2(__frcp_rn(l), __frcp_rn(l));
        const int orow = it.b * S + qt * BQ + quarter * 32, ocol0 = h * HD;
        const uint32_t tO = tmem + lanes + 256 + t * 128;
        uint8_t* prow = smem + L::P_OFF + t * 2 * ATOM + row * 128;
        const uint32_t wbase = sb + L::P_OFF + t * 2 * ATOM + quarter * 32 * 128;
        constexpr int RD = (HD + 63) / 64;  // rounds of up to 64 columns (two 32-column boxes)
#pragma unroll 1
        for (int rd = 0; rd < RD; ++rd) {
          if (rd > 0) {
            if (lane == 0) asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
            __syncwarp();
          }
#pragma unroll
          for (int cc = 0; cc < 2; ++cc) {
            if (64 * rd + 32 * cc >= HD) break;
            uint32_t ov[32];
            tmem_ld_cols<1>(tO + 64 * rd + 32 * cc, ov);
#pragma unroll
            for (int k = 0; k < 8; ++k) {
              const float2 a = div2(make_float2(__uint_as_float(ov[4 * k]), __uint_as_float(ov[4 * k + 1])), l2, y2);
              const float2 b =
                  div2(make_float2(__uint_as_float(ov[4 * k + 2]), __uint_as_float(ov[4 * k + 3])), l2, y2);
              *reinterpret_cast<float4*>(prow + cc * ATOM + ((k ^ (row & 7)) * 16)) = make_float4(a.x, a.y, b.x, b.y);
            }
          }
          if (rd + 1 == RD) {
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            arrive(o_free + 8 * t);
          }
          fence_async_smem();
          __syncwarp();
          if (lane == 0) {
            tma_store_2d(&tmO, wbase, ocol0 + 64 * rd, orow);
            if (64 * rd + 32 < HD) tma_store_2d(&tmO, wbase + ATOM, ocol0 + 64 * rd + 32, orow);
            asm volatile("cp.async.bulk.commit_group;" ::: "memory");
          }
        }
        // the staging (the tile's P buffer) is P again once the stores read it
        if (lane == 0) asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
        arrive(st_free + 8 * t);
      }
    }
    if (lane == 0) asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
  }
  if (!ok && err) atomicOr(err, ERR_TIMEOUT);
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 1) {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(512));
  }
}

PFN_cuTensorMapEncodeTiled_v12000 att_encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = (PFN_cuTensorMapEncodeTiled_v12000)ptr;
  }
  return fn;
}

bool encode_2d(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_cols,
               uint32_t box_rows, bool fp32 = false) {
  auto fn = att_encode_fn();
  const uint64_t esz = fp32 ? 4 : 2;
  if (!fn || (cols * esz) % 16 || ((uintptr_t)base & 15)) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * esz};
  cuuint32_t box[2] = {box_cols, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, fp32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base),
            dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int sm_count() {
  static int sms = 0;
  if (!sms) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) !=
                                                   cudaSuccess || sms <= 0)
      sms = 148;
  }
  return sms;
}

template <int HD>
cudaError_t launch_tc(const AttnPlan& p, int B, int S, int H, int KV, unsigned* err, cudaStream_t s) {
  static bool attr = false;
  constexpr int smem = AttTc<HD>::BYTES;
  if (!attr) {
    // the warpgroups' setmaxnreg split adds up to exactly the registers of a
    // launch at REG_LAUNCH per thread: any other count is refused here
    cudaFuncAttributes fa;
    cudaError_t e = cudaFuncGetAttributes(&fa, k_attention_tc<HD>);
    if (e != cudaSuccess) return e;
    if (fa.numRegs != REG_LAUNCH) return cudaErrorInvalidConfiguration;
    e = cudaFuncSetAttribute(k_attention_tc<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  const int G = H / KV, NQ = S / BQ;
  const long long items = (long long)B * KV * ((G * NQ + 1) / 2);
  const int grid = (int)(items < sm_count() ? items : sm_count());
  return launch_dependent(k_attention_tc<HD>, dim3(grid), dim3(ATT_THREADS), smem, s, p.q, p.k, p.v, p.o, B, S, H, KV,
                          1.0f / sqrtf((float)HD), err);
}

}  // namespace

bool attention_tc_supported(int S, int hd) { return (hd == 64 || hd == 96 || hd == 128) && S % 128 == 0; }

bool attention_tc_plan(AttnPlan* p, const uint16_t* q, const uint16_t* k, const uint16_t* vt, float* out, int B,
                       int S, int H, int KV, int hd) {
  return encode_2d(&p->q, q, (uint64_t)B * H * S, hd, 64, BQ) &&
         encode_2d(&p->k, k, (uint64_t)B * KV * S, hd, 64, BKEY) &&
         encode_2d(&p->v, vt, (uint64_t)B * KV * hd, S, 64, hd) &&
         encode_2d(&p->o, out, (uint64_t)B * S, (uint64_t)H * hd, 32, 32, true);
}

cudaError_t attention_tc_launch(const AttnPlan& p, int B, int S, int H, int KV, int hd, unsigned* err,
                                cudaStream_t s) {
  kernel_launches() += 1;
  return hd == 64 ? launch_tc<64>(p, B, S, H, KV, err, s)
                  : (hd == 96 ? launch_tc<96>(p, B, S, H, KV, err, s) : launch_tc<128>(p, B, S, H, KV, err, s));
}

}  // namespace tmz
