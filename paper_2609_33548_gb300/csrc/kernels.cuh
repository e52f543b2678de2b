// Declarations shared by the TerMeZO translation units (host side).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "common.cuh"

namespace tmz {

// Kernels launched by the calling thread (every launcher adds its count).
uint64_t& kernel_launches();

// ---------------------------------------------------------------- GEMM ----
struct GemmArgs {
  int M, N, K;          // filled from the plan
  float* out;           // fp32 [M, ldo] output (nullable)
  int ldo;
  int mode;             // 0: out = y; 1: out += y (residual stream)
  int32_t* acc_out;     // raw int32 accumulators [M, N] (nullable)
  const float* deq;     // [M] per-row activation scale a/127
  const float* sw;      // three column-segment weight scales sw[0..2]
  int n1, n2;           // segment bounds: [0,n1) sw[0], [n1,n2) sw[1], [n2,N) sw[2]
  int relu2;            // fused gate/up: B rows interleave 128 gate and 128 up rows per
                        // 256-row tile; out[m, f] = relu(g)^2 * u with g scaled by sw[0],
                        // u by sw[1]; f < n_out (out is [M, ldo])
  int n_out;
  int lse;              // LM-head cross-entropy partials instead of an output matrix:
                        // part[m * ceil(N/BN) + j] = (max, sum exp(acc - max)) over the
                        // columns n < N of tile j; tlogit[m] = acc[m, target[m]]
  float2* part;
  float* tlogit;
  const int32_t* target;
  unsigned* err;        // device error word
  int n_fast;           // filled from the plan: tile order walks n fastest
  int tma_out;          // filled at launch: out / ldo match the plan's output map
  // fused RoPE + pack of the attention projections (q, k, v heads of hd
  // columns, the plan made by gemm_plan_rope): q, k rotated at position
  // (row mod S) with the cos / sin tables [S, hd/2], rounded to bf16 and
  // stored as [B, H, S, hd] / [B, KV, S, hd]; v rounded to bf16 into vt
  // [B, KV, hd, S].  out is not written.
  // split K of the last wave (set in gemm_launch from the split workspace):
  // split_ws fp32 [split_cap x 128 x 256] partial accumulators, split_cnt
  // [split_cap x 4] counters (zero between launches), split_s 1: no split
  float* split_ws;
  unsigned* split_cnt;
  int split_cap;
  int split_s, full_units;
  // split N of the last wave (set at launch; exclusive with split_s > 1):
  // its tiles become nsplit units of BN / nsplit columns each (1: no split)
  int nsplit;
  int gu_split;  // filled from the plan: gate and up rows from two B maps
  int rope;
  const float* cosb;
  const float* sinb;
  uint16_t* vt;
  int S, H, KV, hd;
};

// Column tiles of the GEMM (the stride of GemmArgs::part).
int gemm_col_tiles(int N);

struct GemmPlan {
  CUtensorMap a, b;
  CUtensorMap a2;      // e4m3 plans: the lo matrix of A (a holds hi)
  CUtensorMap b2, b4;  // B with boxes of bn / 2 and bn / 4 rows (the narrow last-wave units)
  int narrow_ok;       // bit 1: b2 valid, bit 2: b4 valid
  int f8;              // 1: e4m3 operands, kind::f8f6f4 (BitLinear); 0: bf16, kind::f16
  CUtensorMap b_up;    // gu_split: B tile rows 0..127 from b (gate), 128..255 from b_up
  int gu_split;
  int M, N, K, bn;  // bn: output tile width (columns of B per tile)
  int n_fast;       // tile order: n fastest (A streamed once, B kept in L2)
  CUtensorMap o;    // fp32 output [M, N] (row stride o_ld): TMA store / reduce-add, 32 x 128 boxes
  CUtensorMap o32;  // the same output, 32 x 32 boxes (one warp's rows)
  float* o_ptr;     // the output the map was made for (null: none)
  int o_ld;
  CUtensorMap q, k;  // fused RoPE outputs (gemm_plan_rope)
  int rope;
};

// Tensor maps of the bf16 Q [B*H*S, hd] and K [B*KV*S, hd] for the fused
// RoPE epilogue.  Needs a plan with 256-column tiles, hd 64 or 128, S a
// multiple of 32 and M = B*S; false (plan unchanged) otherwise.
bool gemm_plan_rope(GemmPlan* plan, uint16_t* q, uint16_t* k, int B, int S, int H, int KV, int hd);

// Records a TMA map of the fp32 output out [M, ldo] in the plan; launches
// whose GemmArgs::out / ldo match it write through TMA (store, or reduce-add
// in residual mode).  False (and no map) when the layout does not allow it.
bool gemm_plan_output(GemmPlan* plan, float* out, int ldo);

// any_bn: the plan may use any tile width (store / residual-add epilogues);
// otherwise 256 (fused gate/up and LM-head epilogues).
// bf16 operands (the LM head): A [M, K], B [N, K]; 256-column tiles only.
bool gemm_make_plan(GemmPlan* plan, const uint16_t* a, int M, int K, const uint16_t* b, int N, bool any_bn);
// BitLinear: A the e4m3 (hi, lo) code pair [2, M, K] of launch_norm_quant, B
// e4m3 ternary weights [N, K] (launch_expand_*); K a multiple of 16.  Every
// product is an integer and every partial sum below 2^24, so the fp32
// accumulator is the exact int32 dot product.
bool gemm_make_plan_f8(GemmPlan* plan, const uint8_t* a, int M, int K, const uint8_t* b, int N, bool any_bn);
// The fused gate/up projection straight from two e4m3 weight matrices gate,
// up [F, K]: tile j pairs gate rows 128 j .. 128 j + 127 with the same up rows
// (the layout launch_expand_gate_up writes; rows past F read as zero).
bool gemm_make_plan_f8_gu(GemmPlan* plan, const uint8_t* a, int M, int K, const uint8_t* gate, const uint8_t* up,
                          int F);
int gemm_pick_bn(int M, int N, int sms);
cudaError_t gemm_launch(const GemmPlan& plan, GemmArgs args, cudaStream_t stream);

// ------------------------------------------------------------ forward ----
// Per-row absmax int8 quantisation of h = RMSNorm(x) (gain != nullptr) or
// of h = x (gain == nullptr), deq[m] = a / 127.  Each code q is stored as the
// e4m3 pair hi = 16 floor(q/16), lo = q - hi (both exact): q [2, M, D] bytes,
// the hi matrix then the lo matrix (ld = D).
void launch_norm_quant(const float* x, const float* gain, int M, int D, uint8_t* q, float* deq,
                       cudaStream_t s);
// The int8 activation codes held as e4m3 (hi, lo) pairs in q [2, M, K] (the
// layout launch_norm_quant writes) -> int8 out [M, K] (hi + lo).
void launch_codes_i8(const uint8_t* q, int M, int K, int8_t* out, cudaStream_t s);
// Packed 2-bit codes [rows, K/16] -> e4m3 {-1, 0, +1} [rows, K] bytes.
void launch_expand_codes(const uint32_t* words, uint64_t rows, int K, uint8_t* out, cudaStream_t s);
// gate, up codes (two [F, K/16] word matrices) -> e4m3 [256 * ceil(F/128), K]
// with 256-row tiles [gate rows 128b..128b+127 | up rows 128b..128b+127]
// (rows beyond F are zero).
void launch_expand_gate_up(const uint32_t* gate_words, const uint32_t* up_words, int F, int K, uint8_t* out,
                           cudaStream_t s);
// x[t] = embed[tok[t]].
void launch_embed(const int32_t* tok, const float* embed, int T, int D, int V, float* x, unsigned* err,
                  cudaStream_t s);
// Per-row absmax int8 quantisation of raw bf16 activations (no norm); q as
// for launch_norm_quant.
void launch_norm_quant_bf16(const uint16_t* x, int M, int D, uint8_t* q, float* deq, cudaStream_t s);
// RoPE tables cos/sin fp32 [S, hd/2] computed in float64, rounded to fp32.
void launch_rope_tables(int S, int hd, float* cosb, float* sinb, cudaStream_t s);
// qkv fp32 [B*S, (H + 2 KV) hd] -> Q bf16 [B, H, S, hd] (RoPE), K bf16
// [B, KV, S, hd] (RoPE), Vt bf16 [B, KV, hd, S] (transposed).
void launch_rope_pack(const float* qkv, const float* cosb, const float* sinb, int B, int S, int H, int KV,
                      int hd, uint16_t* q, uint16_t* k, uint16_t* vt, cudaStream_t s);
// Causal GQA attention -> out fp32 [B*S, H*hd].
void launch_attention(const uint16_t* q, const uint16_t* k, const uint16_t* vt, int B, int S, int H, int KV,
                      int hd, float* out, cudaStream_t s);
// Final RMSNorm of every row, rounded to bf16: h bf16 [M, D].
void launch_final_norm_bf16(const float* x, const float* gain, int M, int D, uint16_t* h, cudaStream_t s);
// Loss mode 1: combines the per-tile (max, sum exp) partials of each row into
// the log-sum-exp (float64), subtracts the target logit, and averages the
// token losses of each sequence (per_seq[b], float64) and of the batch.
void launch_ce_reduce(const float2* part, int ntiles, const float* tlogit, const int32_t* target, int B, int S,
                      int V, double* tok_loss, double* per_seq, double* total, unsigned* err, cudaStream_t s);
// tcgen05 attention (hd 64 / 128, S % 128 == 0): tensor maps of Q
// [B*H*S, hd], K [B*KV*S, hd] and V^T [B*KV*hd, S] (bf16) and of the
// output [B*S, H*hd] (fp32).
struct AttnPlan {
  CUtensorMap q, k, v, o;
};
bool attention_tc_supported(int S, int hd);
bool attention_tc_plan(AttnPlan* p, const uint16_t* q, const uint16_t* k, const uint16_t* vt, float* out, int B, int S,
                       int H, int KV, int hd);
cudaError_t attention_tc_launch(const AttnPlan& p, int B, int S, int H, int KV, int hd, unsigned* err, cudaStream_t s);
// Final RMSNorm + LM head over the label tokens at the last position and
// cross-entropy (loss mode 0): per_seq[b] (fp64), total = mean (fp64).
void launch_head_ce_last(const float* x, const float* gain, const uint16_t* head, const int32_t* targets,
                         int B, int S, int D, int V, int C, double* per_seq, double* total, cudaStream_t s);

// ------------------------------------------------------ mask / sparse ----
struct ProjTable {
  int P;                      // number of projections
  const uint64_t* base;       // [P+1] global base index of each projection (base[P] = d)
  const uint32_t* blk_prefix; // [P+1] prefix of dense blocks per projection
};

}  // namespace tmz
