// BitLinear GEMM on the 5th-generation tensor cores (sm_103a).
//
// acc[m, n] = sum_k q[m, k] * c[n, k] with q the int8 activation codes and c
// the ternary codes.  The int8 MMA kind does not exist on sm_103a (ptxas:
// "Feature '.kind::i8' not supported on .target 'sm_103a'"), so the codes
// travel as e4m3: each q as the pair hi = 16 floor(q/16), lo = q - hi (both
// exact in e4m3), each ternary code as itself.  Two kind::f8f6f4 MMAs per
// k-step, A_hi B and A_lo B, accumulate into one fp32 accumulator; every
// product is an integer and every partial sum an integer of magnitude
// <= 128 * K < 2^24, so the accumulator holds the int32 dot product exactly.
// The same kernel with bf16 operands (kind::f16, one MMA per k-step) serves
// the LM head, whose operands are not integers.
//
// Structure: a persistent grid (one CTA per SM) walks 128 x BN output tiles
// (BN 256, 192, 160 or 128, picked per shape to fill the last wave; the last
// wave's tiles split along N or K); warp 0 issues TMA loads with 128-byte
// swizzle into a ring whose stages hold 128 bytes of K per row (A hi, A lo and
// B for 128 K elements, or A and B for 64 bf16); one thread of warp 1 issues
// tcgen05.mma (M = 128, N = BN) into one of two fp32 accumulators in tensor
// memory; warps 2-5 read the other accumulator back with tcgen05.ld and write
// y = acc * (a/127)[m] * s_w[n] (stored, added into the residual stream,
// fused with RoPE or with the squared-ReLU gating, or reduced to the LM
// head's log-sum-exp partials).
#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.cuh"
#include "tcgen05.cuh"

namespace tmz {

namespace {

constexpr int BM = 128;
constexpr int BK = 64;  // bf16 elements per k-block (128 bytes)
constexpr int GEMM_THREADS = 192;

constexpr int EPI_WARPS = 4;
constexpr int EPI_LD = 33;  // staging row stride (floats): conflict-free transpose

// A ring stage holds one k-block of 128 bytes per row: 64 bf16 elements, or
// 128 e4m3 elements with A as two tiles (the hi and lo halves of the codes).
template <int BN, bool F8>
struct GemmSmem {
  static constexpr int KE = F8 ? 128 : BK;            // K elements per k-block
  static constexpr int A_TILE = BM * 128;
  static constexpr int A_BYTES = F8 ? 2 * A_TILE : A_TILE;
  static constexpr int B_BYTES = BN * 128;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  // as many ring stages as fit next to the epilogue staging (at most 6)
  // epilogue staging: per warp two 32 x 32 fp32 tiles (128-byte swizzle) for
  // the TMA output path, or one 32 x 33 transpose block for the others
  static constexpr int EPI_BYTES = EPI_WARPS * 2 * 4096;
  static_assert(EPI_BYTES >= EPI_WARPS * 32 * (EPI_LD + 1) * 4, "staging");
  static constexpr int FIT = (232448 - 1280 - EPI_BYTES) / STAGE_BYTES;
  static constexpr int STAGES = FIT < 6 ? FIT : 6;
  static constexpr int EPI_OFF = STAGES * STAGE_BYTES;
  static constexpr int BAR_OFF = EPI_OFF + EPI_BYTES;
  static constexpr int BYTES = BAR_OFF + 256 + 1024;  // barriers + alignment slack
  // tensor memory: two accumulators of BN columns in a power-of-two allocation,
  // the second at half of it
  static constexpr uint32_t TMEM_COLS = 2 * BN <= 256 ? 256 : 512;
  static constexpr uint32_t ACC_STRIDE = TMEM_COLS / 2;
};

// Work units: the tiles of the full waves, then the tiles of the last,
// partial wave either split into split_s ranges of k-blocks (split_s > 1) or
// into nsplit ranges of BN / nsplit columns (nsplit > 1).  The accumulator is
// an exact integer (< 2^24) in fp32, so partial accumulators add up exactly
// and a split tile equals the unsplit one bit for bit; a column range is a
// narrower tile computed whole.
struct Unit {
  int tile, kb0, kb1, tail, split;  // tail: index among the K-split tiles, -1 for a whole tile
  int c0, nw;                       // the unit's columns n0 + c0 .. n0 + c0 + nw - 1 of its tile
};

template <int BN>
__device__ __forceinline__ Unit unit_of(const GemmArgs& p, int u, int KB) {
  Unit w;
  w.c0 = 0, w.nw = BN;
  if (p.nsplit > 1 && u >= p.full_units) {
    const int v = u - p.full_units;
    w.tile = p.full_units + v / p.nsplit;
    w.nw = BN / p.nsplit;
    w.c0 = (v % p.nsplit) * w.nw;
    w.kb0 = 0, w.kb1 = KB, w.tail = -1, w.split = 0;
  } else if (p.split_s <= 1 || u < p.full_units) {
    w.tile = u, w.kb0 = 0, w.kb1 = KB, w.tail = -1, w.split = 0;
  } else {
    const int v = u - p.full_units;
    w.tail = v / p.split_s;
    w.split = v % p.split_s;
    w.tile = p.full_units + w.tail;
    w.kb0 = w.split * KB / p.split_s;
    w.kb1 = (w.split + 1) * KB / p.split_s;
  }
  return w;
}

// Persistent: CTA c processes units c, c + gridDim.x, ...  With m fastest the
// CTAs running together share B tiles and sweep A through L2; with n fastest
// (an A too large for L2, a B that fits) they share A tiles, so A streams from
// HBM once.  The
// accumulator is double-buffered in tensor memory (2 x BN columns) so that
// the epilogue of one tile overlaps the main loop of the next.
// Named barrier 1 over the four epilogue warps (128 threads).  Every epilogue
// warp reaches each use in the same unit and chunk: the loop over units is
// uniform, and a failed wait is made uniform first (epi_all).
__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }
__device__ __forceinline__ bool epi_all(bool v) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.and.pred q, 1, 128, p;\n selp.u32 %0, 1, 0, q;\n}\n"
      : "=r"(r)
      : "r"((uint32_t)v)
      : "memory");
  return r != 0;
}

template <int BN, bool F8>
__global__ void __launch_bounds__(GEMM_THREADS, 1)
    k_bitlinear_gemm(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmA2,
                     const __grid_constant__ CUtensorMap tmB, const __grid_constant__ CUtensorMap tmBn,
                     const __grid_constant__ CUtensorMap tmBu, const __grid_constant__ CUtensorMap tmO,
                     const __grid_constant__ CUtensorMap tmO32, const __grid_constant__ CUtensorMap tmQ,
                     const __grid_constant__ CUtensorMap tmK, GemmArgs p) {
  using L = GemmSmem<BN, F8>;
  constexpr int STAGES = L::STAGES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  const uint32_t sbase = smem_u32(smem);
  const uint32_t bar_full = sbase + L::BAR_OFF;        // STAGES x 8 B
  const uint32_t bar_empty = bar_full + STAGES * 8;    // STAGES x 8 B
  const uint32_t bar_tfull = bar_empty + STAGES * 8;   // 2 x 8 B: accumulator ready
  const uint32_t bar_tempty = bar_tfull + 16;          // 2 x 8 B: accumulator drained
  uint32_t* tmem_slot = (uint32_t*)(smem + L::BAR_OFF + 2 * STAGES * 8 + 32);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_mt = (p.M + BM - 1) / BM, n_nt = (p.N + BN - 1) / BN;
  const int tiles = n_mt * n_nt;
  const int KB = (p.K + L::KE - 1) / L::KE;
  const int units = p.split_s > 1   ? p.full_units + (tiles - p.full_units) * p.split_s
                    : p.nsplit > 1 ? p.full_units + (tiles - p.full_units) * p.nsplit
                                   : tiles;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(bar_full + 8 * s, 1);
      mbar_init(bar_empty + 8 * s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(bar_tfull + 8 * b, 1);
      mbar_init(bar_tempty + 8 * b, EPI_WARPS);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0 && lane == 0) {
    asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmA) : "memory");
    if (F8) asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmA2) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmB) : "memory");
    if (p.nsplit > 1) asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmBn) : "memory");
    if (p.gu_split) asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmBu) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(L::TMEM_COLS));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;
  bool ok = true;
  // everything above touched only this CTA's own resources; A, the output
  // and the residual stream belong to the kernels before this one
  grid_dep_wait();

  if (warp == 0) {
    if (lane == 0) {
      uint32_t it = 0;
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
        const Unit w = unit_of<BN>(p, u, KB);
        const int tile = w.tile;
        const int m0 = (p.n_fast ? tile / n_nt : tile % n_mt) * BM;
        const int n0 = (p.n_fast ? tile % n_nt : tile / n_mt) * BN;
        const bool narrow = w.nw < BN;
        for (int kb = w.kb0; kb < w.kb1; ++kb, ++it) {
          const uint32_t s = it % STAGES, use = it / STAGES;
          if (it >= (uint32_t)STAGES && !(ok = mbar_wait(bar_empty + 8 * s, (use & 1u) ^ 1u))) break;
          const uint32_t sa = sbase + s * L::STAGE_BYTES;
          mbar_expect_tx(bar_full + 8 * s, narrow ? L::A_BYTES + w.nw * 128 : L::STAGE_BYTES);
          tma_load_2d(sa, &tmA, kb * L::KE, m0, bar_full + 8 * s);
          if (F8) tma_load_2d(sa + L::A_TILE, &tmA2, kb * L::KE, m0, bar_full + 8 * s);
          if (p.gu_split) {
            // gate rows 128 j.. then up rows 128 j.. of tile j (BN 256)
            tma_load_2d(sa + L::A_BYTES, &tmB, kb * L::KE, n0 / 2, bar_full + 8 * s);
            tma_load_2d(sa + L::A_BYTES + 128 * 128, &tmBu, kb * L::KE, n0 / 2, bar_full + 8 * s);
          } else {
            tma_load_2d(sa + L::A_BYTES, narrow ? &tmBn : &tmB, kb * L::KE, n0 + w.c0, bar_full + 8 * s);
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const int n_narrow = BN / (p.nsplit > 1 ? p.nsplit : 1);
      const uint32_t idesc_full = F8 ? idesc_e4m3(BM, BN) : idesc_bf16(BM, BN);
      const uint32_t idesc_narrow = F8 ? idesc_e4m3(BM, n_narrow) : idesc_bf16(BM, n_narrow);
      uint32_t it = 0, local = 0;
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x, ++local) {
        const Unit w = unit_of<BN>(p, u, KB);
        const uint32_t b = local & 1u, j = local >> 1;
        if (j >= 1 && !(ok = mbar_wait(bar_tempty + 8 * b, (j & 1u) ^ 1u))) break;
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t d = tmem + b * L::ACC_STRIDE;
        const uint32_t idesc = w.nw < BN ? idesc_narrow : idesc_full;
        for (int kb = w.kb0; kb < w.kb1; ++kb, ++it) {
          const uint32_t s = it % STAGES;
          if (!(ok = mbar_wait(bar_full + 8 * s, (it / STAGES) & 1u))) break;
          asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
          const uint32_t sa = sbase + s * L::STAGE_BYTES;
          const uint64_t da = sw128_desc(sa), db = sw128_desc(sa + L::A_BYTES);
          // each MMA step reads 32 bytes of every row: 16 bf16 or 32 e4m3
          // elements; the e4m3 path adds hi B and lo B into one accumulator
          if (F8) {
            const uint64_t dl = sw128_desc(sa + L::A_TILE);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              mma_e4m3(d, da + (uint64_t)(2 * k), db + (uint64_t)(2 * k), idesc, (kb > w.kb0 || k) ? 1u : 0u);
              mma_e4m3(d, dl + (uint64_t)(2 * k), db + (uint64_t)(2 * k), idesc, 1u);
            }
          } else {
#pragma unroll
            for (int k = 0; k < 4; ++k)
              mma_bf16(d, da + (uint64_t)(2 * k), db + (uint64_t)(2 * k), idesc, (kb > w.kb0 || k) ? 1u : 0u);
          }
          mma_commit(bar_empty + 8 * s);
        }
        if (!ok) break;
        mma_commit(bar_tfull + 8 * b);
      }
    }
  } else {
    // Epilogue warps 2..5: warp w may access TMEM lanes 32*(w % 4) .. +31.
    // Lane l owns row row0 + l when reading TMEM and column col0 + l when
    // writing: the 32 x 32 block is transposed through shared memory so that
    // every store (and residual load) is one coalesced 128-byte row segment.
    const int quarter = warp & 3;
    float* stage = reinterpret_cast<float*>(smem + L::EPI_OFF) + (warp - 2) * 32 * (EPI_LD + 1);
    // TMA output path: this warp's two swizzled 32 x 32 staging tiles
    uint8_t* otile = smem + L::EPI_OFF + (warp - 2) * 2 * 4096;
    uint32_t n_out_tiles = 0;
    // TMA output of whole tiles: the four warps stage one 128-row x 32-column
    // fp32 block (16 KB, two buffers) and one thread issues its store or
    // reduce-add, so the epilogue takes 8 TMA operations a tile instead of 32
    // and leaves the TMA unit to the operand loads
    uint8_t* gbuf = smem + L::EPI_OFF;
    const bool issuer = warp == 2 && lane == 0;
    uint32_t n_grp = 0;
    bool drained = false;
    float* dqs = stage + 32 * EPI_LD;  // the 32 rows' activation scales
    const float s0 = p.sw[0], s1 = p.sw[1], s2 = p.sw[2];
    uint32_t local = 0;
    for (int u = blockIdx.x; u < units; u += gridDim.x, ++local) {
      const Unit w = unit_of<BN>(p, u, KB);
      const int tile = w.tile;
      const int m0 = (p.n_fast ? tile / n_nt : tile % n_mt) * BM;
      // a narrow unit's accumulator columns 0 .. nw-1 are output columns n0 ..
      const int n0 = (p.n_fast ? tile % n_nt : tile / n_mt) * BN + w.c0;
      const int ncols = w.nw;
      const uint32_t b = local & 1u, j = local >> 1;
      const int row0 = m0 + quarter * 32;
      const int nrows = min(32, p.M - row0);
      const bool tma_path = p.tma_out && !p.relu2 && !p.lse && !p.rope;
      const float dq_row = (lane < nrows && p.deq) ? p.deq[row0 + lane] : 0.f;
      // dqs shares shared memory with the TMA staging tiles: only the
      // transposing paths use it
      if (!tma_path && !p.rope) dqs[lane] = dq_row;
      // residual mode without the TMA path: the first chunk's residual rows are
      // loaded before the accumulator is ready, those of chunk c + 1 while
      // chunk c is written
      const bool resid = p.out && p.mode && !p.tma_out && !p.relu2 && !p.lse && nrows > 0;
      float prev[32];
      if (resid) {
        const int col = n0 + lane;
#pragma unroll
        for (int rr = 0; rr < 32; ++rr)
          prev[rr] = (rr < nrows && col < p.N) ? p.out[(size_t)(row0 + rr) * p.ldo + col] : 0.f;
      }
      ok = epi_all(mbar_wait(bar_tfull + 8 * b, j & 1u));
      if (!ok) break;
      // a K-split tail unit stages per warp (each warp decides alone whether
      // it finishes its rows): the whole-tile buffers must be read out first
      if (tma_path && w.tail >= 0 && n_grp > 0 && !drained) {
        if (issuer) asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
        epi_bar();
        drained = true;
      }
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const uint32_t tacc = tmem + ((uint32_t)(quarter * 32) << 16) + b * L::ACC_STRIDE;
      // split partials: [unit][quarter][column / 4][lane] float4 (columns 4k .. 4k+3 of the
      // lane's row): every warp access is 512 contiguous bytes
      auto part_at = [&](int split, int col) {
        return reinterpret_cast<float4*>(p.split_ws) +
               (((size_t)(w.tail * p.split_s + split) * 4 + quarter) * (BN / 4) + col / 4) * 32 + lane;
      };
      if (w.tail >= 0) {
        // a split of a tail tile: its partial accumulator goes to the
        // workspace; the last split to finish these 32 rows keeps its own in
        // TMEM and adds the others
        for (int c = 0; c < BN / 32; ++c) {
          uint32_t r[32];
          tmem_ld32(tacc + (uint32_t)(c * 32), r);
          float4* dst = part_at(w.split, 32 * c);
#pragma unroll
          for (int q4 = 0; q4 < 8; ++q4)
            dst[32 * q4] = make_float4(__uint_as_float(r[4 * q4]), __uint_as_float(r[4 * q4 + 1]),
                                       __uint_as_float(r[4 * q4 + 2]), __uint_as_float(r[4 * q4 + 3]));
        }
        __threadfence();
        unsigned prev = 0;
        if (lane == 0) prev = atomicAdd(p.split_cnt + w.tail * 4 + quarter, 1u);
        prev = __shfl_sync(0xffffffffu, prev, 0);
        if (prev + 1 != (unsigned)p.split_s) {
          asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
          __syncwarp();
          if (lane == 0) mbar_arrive(bar_tempty + 8 * b);
          continue;
        }
        __threadfence();
        if (lane == 0) p.split_cnt[w.tail * 4 + quarter] = 0;  // ready for the next launch
        // the other splits' partials added into this split's accumulator,
        // 16 columns at a time with all of their loads issued before the
        // first add (one L2 round trip each); integers below 2^24, so the
        // fp32 sum is exact in any order
        for (int c = 0; c < BN / 32; ++c) {
          uint32_t r[32];
          tmem_ld32(tacc + (uint32_t)(c * 32), r);
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            float4 pv[3][4];
#pragma unroll
            for (int t = 0; t < 3; ++t) {
              const int sp = t + (t >= w.split ? 1 : 0);  // the t-th split other than this one
              if (sp < p.split_s) {
                const float4* src = part_at(sp, 32 * c + 16 * h);
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) pv[t][q4] = __ldcg(src + 32 * q4);
              }
            }
#pragma unroll
            for (int t = 0; t < 3; ++t) {
              const int sp = t + (t >= w.split ? 1 : 0);
              if (sp < p.split_s) {
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) {
                  uint32_t* rr = r + 16 * h + 4 * q4;
                  rr[0] = __float_as_uint(__fadd_rn(__uint_as_float(rr[0]), pv[t][q4].x));
                  rr[1] = __float_as_uint(__fadd_rn(__uint_as_float(rr[1]), pv[t][q4].y));
                  rr[2] = __float_as_uint(__fadd_rn(__uint_as_float(rr[2]), pv[t][q4].z));
                  rr[3] = __float_as_uint(__fadd_rn(__uint_as_float(rr[3]), pv[t][q4].w));
                }
              }
            }
          }
          tmem_st32(tacc + (uint32_t)(c * 32), r);
        }
        asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
      }
      // 32 accumulator columns col .. col+31 of this thread's row
      auto load_acc = [&](int col, uint32_t(&r)[32]) { tmem_ld32(tacc + (uint32_t)col, r); };
      if (p.lse) {
        // lane = row: running max and sum of exp over this tile's columns
        const int row = row0 + lane;
        const int tg = (lane < nrows) ? p.target[row] : -1;
        float m = -INFINITY, se = 0.f;
        for (int c = 0; c < BN / 32; ++c) {
          uint32_t r[32];
          tmem_ld32(tmem + ((uint32_t)(quarter * 32) << 16) + b * L::ACC_STRIDE + (uint32_t)(c * 32), r);
          const int col0 = n0 + c * 32;
          float cm = -INFINITY;
#pragma unroll
          for (int q = 0; q < 32; ++q)
            if (col0 + q < p.N) cm = fmaxf(cm, __uint_as_float(r[q]));
          const float mn = fmaxf(m, cm);
          if (mn != -INFINITY) {
            float t = (m == -INFINITY) ? 0.f : __fmul_rn(se, expf(__fsub_rn(m, mn)));
#pragma unroll
            for (int q = 0; q < 32; ++q)
              if (col0 + q < p.N) t = __fadd_rn(t, expf(__fsub_rn(__uint_as_float(r[q]), mn)));
            se = t;
            m = mn;
          }
          if (tg >= col0 && tg < col0 + 32) {
            float tv = 0.f;
#pragma unroll
            for (int q = 0; q < 32; ++q)
              if (col0 + q == tg) tv = __uint_as_float(r[q]);
            p.tlogit[row] = tv;
          }
        }
        if (lane < nrows) p.part[(size_t)row * n_nt + (n0 / BN)] = make_float2(m, se);
      } else if (p.relu2) {
        // TMEM columns [0, BN/2) hold gate features f0.., [BN/2, BN) the up
        // features f0..; lane = row: hid = relu(g)^2 * u, then transposed.
        const int f0 = (n0 / BN) * (BN / 2);
        const float dql = dqs[lane];
        for (int c = 0; c < BN / 64; ++c) {
          {
            uint32_t g[32], u[32];
            const uint32_t tb = tmem + ((uint32_t)(quarter * 32) << 16) + b * L::ACC_STRIDE;
            tmem_ld32(tb + (uint32_t)(c * 32), g);
            tmem_ld32(tb + (uint32_t)(BN / 2 + c * 32), u);
#pragma unroll
            for (int q = 0; q < 32; ++q) {
              const float gv = fmaxf(__fmul_rn(__fmul_rn(__uint_as_float(g[q]), dql), s0), 0.f);
              const float uv = __fmul_rn(__fmul_rn(__uint_as_float(u[q]), dql), s1);
              stage[lane * EPI_LD + q] = __fmul_rn(__fmul_rn(gv, gv), uv);
            }
          }
          __syncwarp();
          const int col = f0 + c * 32 + lane;
          if (col < p.n_out && nrows > 0) {
            float* o = p.out + (size_t)row0 * p.ldo + col;
#pragma unroll 8
            for (int rr = 0; rr < 32; ++rr)
              if (rr < nrows) o[(size_t)rr * p.ldo] = stage[rr * EPI_LD + lane];
          }
          __syncwarp();
        }
      }
      if (p.rope) {
        // lane = row = token at position pos of sequence sb; the tile's
        // columns are whole heads of hd (q heads, then k, then v)
        const float dq = dq_row;
        const int sb = row0 / p.S, pos0 = row0 - sb * p.S, pos = pos0 + lane;
        const int half = p.hd >> 1;
        for (int hb = 0; hb < ncols / p.hd; ++hb) {
          const int col0 = n0 + hb * p.hd;
          if (col0 >= p.N) break;
          const int head = col0 / p.hd;
          const int hc = hb * p.hd;  // this head's first accumulator column
          if (head >= p.H + p.KV) {
            // v: bf16 into vt[b, kvh, d, pos]; the warp's 32 positions of
            // one d are 64 contiguous bytes
            uint16_t* vcol = p.vt + ((size_t)(sb * p.KV + head - p.H - p.KV) * p.hd) * p.S + pos;
            for (int c = 0; c < p.hd / 32; ++c) {
              uint32_t r[32];
              load_acc(hc + c * 32, r);
#pragma unroll
              for (int q = 0; q < 32; ++q) {
                const __nv_bfloat16 v = __float2bfloat16_rn(__fmul_rn(__fmul_rn(__uint_as_float(r[q]), dq), s2));
                vcol[(size_t)(c * 32 + q) * p.S] = *reinterpret_cast<const uint16_t*>(&v);
              }
            }
            continue;
          }
          const bool isq = head < p.H;
          const float sw = isq ? s0 : s1;
          // both staging tiles are rewritten: the previous head's stores must
          // have read them
          if (n_out_tiles) {
            if (lane == 0) asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
            __syncwarp();
          }
          for (int c = 0; c < half / 32; ++c) {
            uint32_t r1[32], r2[32];
            load_acc(hc + c * 32, r1);
            load_acc(hc + half + c * 32, r2);
            const float4* cr = reinterpret_cast<const float4*>(p.cosb + (size_t)pos * half + c * 32);
            const float4* sr = reinterpret_cast<const float4*>(p.sinb + (size_t)pos * half + c * 32);
            uint32_t w1[16], w2[16];
#pragma unroll
            for (int g = 0; g < 8; ++g) {
              const float4 cv = cr[g], sv = sr[g];
              const float cs[4] = {cv.x, cv.y, cv.z, cv.w}, sn[4] = {sv.x, sv.y, sv.z, sv.w};
              float o1[4], o2[4];
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const float x1 = __fmul_rn(__fmul_rn(__uint_as_float(r1[4 * g + e]), dq), sw);
                const float x2 = __fmul_rn(__fmul_rn(__uint_as_float(r2[4 * g + e]), dq), sw);
                o1[e] = __fsub_rn(__fmul_rn(x1, cs[e]), __fmul_rn(x2, sn[e]));
                o2[e] = __fadd_rn(__fmul_rn(x2, cs[e]), __fmul_rn(x1, sn[e]));
              }
              __nv_bfloat162 a0 = __floats2bfloat162_rn(o1[0], o1[1]), a1 = __floats2bfloat162_rn(o1[2], o1[3]);
              __nv_bfloat162 c0 = __floats2bfloat162_rn(o2[0], o2[1]), c1 = __floats2bfloat162_rn(o2[2], o2[3]);
              w1[2 * g] = *reinterpret_cast<uint32_t*>(&a0);
              w1[2 * g + 1] = *reinterpret_cast<uint32_t*>(&a1);
              w2[2 * g] = *reinterpret_cast<uint32_t*>(&c0);
              w2[2 * g + 1] = *reinterpret_cast<uint32_t*>(&c1);
            }
            // bf16 columns 32c.. (first half) and half + 32c.. (second half)
            // of the head -> 64-column swizzled tiles
#pragma unroll
            for (int t = 0; t < 4; ++t) {
              const int c1c = c * 32 + 8 * t, c2c = half + c * 32 + 8 * t;
              *reinterpret_cast<uint4*>(otile + (c1c >> 6) * 4096 + lane * 128 + ((((c1c & 63) >> 3) ^ (lane & 7)) * 16)) =
                  make_uint4(w1[4 * t], w1[4 * t + 1], w1[4 * t + 2], w1[4 * t + 3]);
              *reinterpret_cast<uint4*>(otile + (c2c >> 6) * 4096 + lane * 128 + ((((c2c & 63) >> 3) ^ (lane & 7)) * 16)) =
                  make_uint4(w2[4 * t], w2[4 * t + 1], w2[4 * t + 2], w2[4 * t + 3]);
            }
          }
          asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
          __syncwarp();
          if (lane == 0) {
            const int hidx = isq ? head : head - p.H;
            const int yrow = (sb * (isq ? p.H : p.KV) + hidx) * p.S + pos0;
            for (int bx = 0; bx < p.hd / 64; ++bx)
              asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                               (uint64_t)(isq ? &tmQ : &tmK)),
                           "r"(smem_u32(otile + bx * 4096)), "r"(bx * 64), "r"(yrow)
                           : "memory");
            asm volatile("cp.async.bulk.commit_group;" ::: "memory");
          }
          ++n_out_tiles;
        }
      }
      if (tma_path) {
        // lane = row: y = acc (a/127)[row] s_w[col] through shared memory with
        // a TMA store, or added into the residual stream with a TMA
        // reduce-add (one fp32 add, rounded to nearest, per element: the same
        // value as out + y); whole tiles as 128 x 32 blocks of the four warps,
        // K-split tail units as 32 x 32 blocks of each warp
        const float dq = dq_row;
        const int row = row0 + lane;
        const bool group = w.tail < 0;
        for (int c = 0; c < ncols / 32; ++c) {
          const int col0 = n0 + c * 32;
          if (col0 >= p.N) break;
          uint32_t r[32];
          load_acc(c * 32, r);
          if (p.acc_out && lane < nrows) {
#pragma unroll
            for (int q = 0; q < 32; ++q)
              if (col0 + q < p.N) p.acc_out[(size_t)row * p.N + col0 + q] = __float2int_rn(__uint_as_float(r[q]));
          }
          uint8_t* ot;
          if (group) {
            // the buffer was last read by the store of two blocks ago
            if (issuer && n_grp >= 2) asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
            epi_bar();
            ot = gbuf + (n_grp & 1u) * 16384 + quarter * 4096;
          } else {
            ot = otile + (n_out_tiles & 1u) * 4096;
            if (n_out_tiles >= 2) {
              if (lane == 0) asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
              __syncwarp();
            }
          }
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            float v[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const int col = col0 + 4 * k + e;
              const float sw = col < p.n1 ? s0 : (col < p.n2 ? s1 : s2);
              v[e] = __fmul_rn(__fmul_rn(__uint_as_float(r[4 * k + e]), dq), sw);
            }
            *reinterpret_cast<float4*>(ot + lane * 128 + ((k ^ (lane & 7)) * 16)) = make_float4(v[0], v[1], v[2], v[3]);
          }
          asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
          if (group) {
            epi_bar();
          } else {
            __syncwarp();
          }
          const CUtensorMap* map = group ? &tmO : &tmO32;
          const int y0 = group ? row0 - quarter * 32 : row0;
          if (group ? issuer : lane == 0) {
            const uint32_t src = smem_u32(group ? gbuf + (n_grp & 1u) * 16384 : ot);
            if (p.mode)
              asm volatile(
                  "cp.reduce.async.bulk.tensor.2d.global.shared::cta.add.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                      (uint64_t)map),
                  "r"(src), "r"(col0), "r"(y0)
                  : "memory");
            else
              asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                               (uint64_t)map),
                           "r"(src), "r"(col0), "r"(y0)
                           : "memory");
            asm volatile("cp.async.bulk.commit_group;" ::: "memory");
          }
          if (group)
            ++n_grp;
          else
            ++n_out_tiles;
        }
      }
      for (int c = 0; c < ((p.relu2 || p.lse || p.tma_out || p.rope) ? 0 : ncols / 32); ++c) {
        {
          uint32_t r[32];
          tmem_ld32(tmem + ((uint32_t)(quarter * 32) << 16) + b * L::ACC_STRIDE + (uint32_t)(c * 32), r);
#pragma unroll
          for (int q = 0; q < 32; ++q) stage[lane * EPI_LD + q] = __uint_as_float(r[q]);
        }
        __syncwarp();
        const int col = n0 + c * 32 + lane;
        if (col < p.N && nrows > 0) {
          if (p.acc_out) {
            int32_t* ao = p.acc_out + (size_t)row0 * p.N + col;
#pragma unroll 8
            for (int rr = 0; rr < 32; ++rr)
              if (rr < nrows) ao[(size_t)rr * p.N] = __float2int_rn(stage[rr * EPI_LD + lane]);
          }
          if (p.out) {
            const float sw = col < p.n1 ? s0 : (col < p.n2 ? s1 : s2);
            float* o = p.out + (size_t)row0 * p.ldo + col;
            if (p.mode) {
              float nxt[32];
              const int ncol = col + 32;
              const bool more = c + 1 < ncols / 32 && ncol < p.N;
#pragma unroll
              for (int rr = 0; rr < 32; ++rr) nxt[rr] = (more && rr < nrows) ? o[(size_t)rr * p.ldo + 32] : 0.f;
#pragma unroll
              for (int rr = 0; rr < 32; ++rr)
                if (rr < nrows)
                  o[(size_t)rr * p.ldo] =
                      __fadd_rn(prev[rr], __fmul_rn(__fmul_rn(stage[rr * EPI_LD + lane], dqs[rr]), sw));
#pragma unroll
              for (int rr = 0; rr < 32; ++rr) prev[rr] = nxt[rr];
            } else {
#pragma unroll 8
              for (int rr = 0; rr < 32; ++rr)
                if (rr < nrows) o[(size_t)rr * p.ldo] = __fmul_rn(__fmul_rn(stage[rr * EPI_LD + lane], dqs[rr]), sw);
            }
          }
        }
        __syncwarp();
      }
      asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
      __syncwarp();
      if (lane == 0) mbar_arrive(bar_tempty + 8 * b);
    }
    // the TMA writes complete before the kernel does
    if (lane == 0 && (n_out_tiles || (issuer && n_grp))) asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
  }
  if (!ok && p.err) atomicOr(p.err, ERR_TIMEOUT);
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 1) {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(L::TMEM_COLS));
  }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
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

}  // namespace

constexpr int GEMM_BN = 256;  // fixed for the fused gate/up and LM-head modes

// K-major operand [rows, k] (bf16 or bytes) with boxes of 128 bytes x
// box_rows, 128-byte swizzle; columns past k read as zero.
bool encode_kmajor(CUtensorMap* map, const void* base, uint64_t rows, uint64_t k, uint32_t box_rows, bool bytes) {
  auto fn = encode_fn();
  const uint64_t esz = bytes ? 1 : 2;
  if (!fn || (k * esz) % 16 != 0 || ((uintptr_t)base & 15)) return false;
  cuuint64_t dims[2] = {k, rows};
  cuuint64_t strides[1] = {k * esz};
  cuuint32_t box[2] = {(cuuint32_t)(128 / esz), box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, bytes ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                  const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

namespace {

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

}  // namespace

int gemm_pick_bn(int M, int N, int sms) {
  // A persistent CTA's time is (tiles it walks) x (one tile's main loop, ~BN).
  // Smaller tiles fill the last wave better, but each k-step then holds less
  // MMA work to cover the load latency of the ring: measured on GB300 at
  // K 2560-6912, a 160-column tile costs ~1.4x per column what a 256-column
  // one does.
  static const int bns[4] = {256, 192, 160, 128};
  static const double cost_per_col[4] = {1.0, 1.2, 1.4, 1.6};
  const long long m_tiles = (M + BM - 1) / BM;
  int best = 256;
  double best_cost = 0;
  for (int i = 0; i < 4; ++i) {
    const long long tiles = m_tiles * ((N + bns[i] - 1) / bns[i]);
    const long long waves = (tiles + sms - 1) / sms;
    const double cost = (double)waves * bns[i] * cost_per_col[i];
    if (i == 0 || cost < best_cost * 0.999) {
      best = bns[i];
      best_cost = cost;
    }
  }
  return best;
}

namespace {

bool make_plan(GemmPlan* plan, const void* a, int M, int K, const void* b, int N, bool any_bn, bool f8) {
  plan->M = M;
  plan->N = N;
  plan->K = K;
  plan->f8 = f8 ? 1 : 0;
  plan->bn = (any_bn && f8) ? gemm_pick_bn(M, N, sm_count()) : GEMM_BN;
  plan->o_ptr = nullptr;
  plan->o_ld = 0;
  plan->rope = 0;
  // n fastest when A (2 bytes per element either way) is too large to stay
  // in L2 and B is not
  const double a_bytes = 2.0 * M * K, b_bytes = (f8 ? 1.0 : 2.0) * N * K;
  plan->n_fast = (a_bytes > 64e6 && b_bytes < a_bytes) ? 1 : 0;
  if (!encode_kmajor(&plan->a, a, (uint64_t)M, (uint64_t)K, BM, f8) ||
      !encode_kmajor(&plan->b, b, (uint64_t)N, (uint64_t)K, (uint32_t)plan->bn, f8))
    return false;
  plan->a2 = plan->a;
  plan->b_up = plan->b;
  plan->gu_split = 0;
  if (f8 && !encode_kmajor(&plan->a2, (const uint8_t*)a + (size_t)M * K, (uint64_t)M, (uint64_t)K, BM, true))
    return false;
  // narrow units of the last wave: whole 32-column epilogue chunks, at least
  // 64 columns (an MMA of N 64 still reads all of A per k-step)
  plan->narrow_ok = 0;
  for (int f = 2; f <= 4; f *= 2) {
    const int w = plan->bn / f;
    if (w % 32 == 0 && w >= 64 &&
        encode_kmajor(f == 2 ? &plan->b2 : &plan->b4, b, (uint64_t)N, (uint64_t)K, (uint32_t)w, f8))
      plan->narrow_ok |= f;
  }
  return true;
}

}  // namespace

bool gemm_make_plan(GemmPlan* plan, const uint16_t* a, int M, int K, const uint16_t* b, int N, bool any_bn) {
  return make_plan(plan, a, M, K, b, N, any_bn, false);
}

bool gemm_make_plan_f8(GemmPlan* plan, const uint8_t* a, int M, int K, const uint8_t* b, int N, bool any_bn) {
  return make_plan(plan, a, M, K, b, N, any_bn, true);
}

bool gemm_make_plan_f8_gu(GemmPlan* plan, const uint8_t* a, int M, int K, const uint8_t* gate, const uint8_t* up,
                          int F) {
  if (!make_plan(plan, a, M, K, gate, 256 * ((F + 127) / 128), false, true)) return false;
  // B boxes of 128 rows from each matrix; no narrow last-wave units
  plan->narrow_ok = 0;
  plan->gu_split = 1;
  return encode_kmajor(&plan->b, gate, (uint64_t)F, (uint64_t)K, 128, true) &&
         encode_kmajor(&plan->b_up, up, (uint64_t)F, (uint64_t)K, 128, true);
}

int gemm_col_tiles(int N) { return (N + GEMM_BN - 1) / GEMM_BN; }

bool gemm_plan_rope(GemmPlan* plan, uint16_t* q, uint16_t* k, int B, int S, int H, int KV, int hd) {
  if ((hd != 64 && hd != 128) || S % 32 || plan->bn % hd || (long long)B * S != plan->M ||
      plan->N != (H + 2 * KV) * hd)
    return false;
  CUtensorMap mq, mk;
  auto enc = [&](CUtensorMap* m, uint16_t* base, uint64_t rows) {
    auto fn = encode_fn();
    if (!fn || ((uintptr_t)base & 15)) return false;
    cuuint64_t dims[2] = {(cuuint64_t)hd, rows};
    cuuint64_t strides[1] = {(cuuint64_t)hd * 2};
    cuuint32_t box[2] = {64, 32};
    cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
              CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
  };
  if (!enc(&mq, q, (uint64_t)B * H * S) || !enc(&mk, k, (uint64_t)B * KV * S)) return false;
  plan->q = mq;
  plan->k = mk;
  plan->rope = 1;
  return true;
}

bool gemm_plan_output(GemmPlan* plan, float* out, int ldo) {
  plan->o_ptr = nullptr;
  auto fn = encode_fn();
  if (!fn || !out || ldo < plan->N || ((uintptr_t)out & 15) || ((size_t)ldo * 4) % 16) return false;
  cuuint64_t dims[2] = {(cuuint64_t)plan->N, (cuuint64_t)plan->M};
  cuuint64_t strides[1] = {(cuuint64_t)ldo * 4};
  cuuint32_t estr[2] = {1, 1};
  // 32 columns x 128 rows (a whole tile's block) and x 32 rows (one warp's)
  for (int v = 0; v < 2; ++v) {
    cuuint32_t box[2] = {32, v ? 32u : 128u};
    if (fn(v ? &plan->o32 : &plan->o, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, out, dims, strides, box, estr,
           CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
           CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return false;
  }
  plan->o_ptr = out;
  plan->o_ld = ldo;
  return true;
}

namespace {

template <int BN, bool F8>
cudaError_t launch_bn(const GemmPlan& plan, const GemmArgs& args, cudaStream_t stream) {
  static bool attr_set = false;
  constexpr int smem = GemmSmem<BN, F8>::BYTES;
  static_assert(smem <= 232448, "shared memory");
  if (!attr_set) {
    cudaError_t e =
        cudaFuncSetAttribute(k_bitlinear_gemm<BN, F8>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  const int sms = sm_count();
  const int tiles = ((plan.N + BN - 1) / BN) * ((plan.M + BM - 1) / BM);
  dim3 grid(tiles < sms ? tiles : sms);
  // the last, partial wave: its tiles split along K so that all CTAs finish
  // together (store / residual / fused-RoPE epilogues only; measured on GB300
  // to pay off for K >= 4096)
  GemmArgs a = args;
  a.split_s = 1;
  a.full_units = tiles;
  const int full = (tiles / (int)grid.x) * (int)grid.x, rem = tiles - full;
  const int KB = (plan.K + GemmSmem<BN, F8>::KE - 1) / GemmSmem<BN, F8>::KE;
  // (only long reductions, K >= 4096: for K of a few thousand a tile's main
  // loop is short next to the cost of writing and re-reading the partials)
  if (a.split_ws && a.split_cnt && rem > 0 && full > 0 && plan.K >= 4096 && !a.relu2 && !a.lse &&
      (a.tma_out || a.rope)) {
    int S = (int)grid.x / rem;
    if (S > 4) S = 4;
    if (S > KB) S = KB;
    if (S >= 2 && rem * S <= a.split_cap) {
      a.split_s = S;
      a.full_units = full;
    }
  }
  // otherwise split the last wave's tiles along N, as finely as the idle CTAs
  // allow (fused RoPE: whole heads per unit; not for the gate/up and
  // LM-head epilogues, whose tiles pair or reduce columns)
  a.nsplit = 1;
  const CUtensorMap* bn_map = &plan.b;
  if (a.split_s == 1 && rem > 0 && full > 0 && !a.relu2 && !a.lse) {
    for (int f = 4; f >= 2; f /= 2) {
      if (!(plan.narrow_ok & f) || rem * f > (int)grid.x || (a.rope && (BN / f) % a.hd)) continue;
      a.nsplit = f;
      a.full_units = full;
      bn_map = f == 2 ? &plan.b2 : &plan.b4;
      break;
    }
  }
  return launch_dependent(k_bitlinear_gemm<BN, F8>, grid, dim3(GEMM_THREADS), smem, stream, plan.a, plan.a2, plan.b,
                          *bn_map, plan.b_up, plan.o, plan.o32, plan.q, plan.k, a);
}

}  // namespace

cudaError_t gemm_launch(const GemmPlan& plan, GemmArgs args, cudaStream_t stream) {
  args.M = plan.M;
  args.N = plan.N;
  args.K = plan.K;
  args.n_fast = plan.n_fast;
  args.gu_split = plan.gu_split;
  if (plan.gu_split && (!args.relu2 || plan.bn != 256)) return cudaErrorInvalidValue;
  if (args.rope && (!plan.rope || plan.bn % args.hd)) return cudaErrorInvalidValue;
  args.tma_out = (plan.o_ptr && args.out == plan.o_ptr && args.ldo == plan.o_ld && !args.relu2 && !args.lse) ? 1 : 0;
  if ((args.relu2 || args.lse) && plan.bn != GEMM_BN) return cudaErrorInvalidValue;
  if (!args.sw) return cudaErrorInvalidValue;  // every epilogue reads sw[0..2]
  ++kernel_launches();
  if (!plan.f8) return plan.bn == 256 ? launch_bn<256, false>(plan, args, stream) : cudaErrorInvalidValue;
  switch (plan.bn) {
    case 256: return launch_bn<256, true>(plan, args, stream);
    case 192: return launch_bn<192, true>(plan, args, stream);
    case 160: return launch_bn<160, true>(plan, args, stream);
    case 128: return launch_bn<128, true>(plan, args, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace tmz
