/*
 * termezo.h -- C ABI of libtermezo.so, a GB300 (sm_103a) implementation of
 * the TerMeZO training step: sparse zeroth-order fine-tuning of a ternary
 * BitNet model (Sifaou, Katti, Rajendran, Simeone, arXiv 2609.33548).
 *
 * Conventions shared by every call
 *  - Pointers named d_* are device pointers owned by the caller; h_* are
 *    host pointers owned by the caller.  The library allocates no device
 *    memory at run time: every buffer of a context is carved from the one
 *    workspace the caller passes to termezo_create, and the only device
 *    memory of its own is the fixed 4 MiB array that
 *    termezo_absmean_noalloc uses.
 *  - All device work is ordered on the stream given to termezo_create (a
 *    cudaStream_t passed as void*; NULL = legacy default stream).  Calls
 *    that return host values synchronise that stream before returning.
 *  - Return value: TERMEZO_OK (0), a positive warning, or a negative error
 *    code; termezo_strerror gives a message.  After TERMEZO_ECUDA or
 *    TERMEZO_ETIMEOUT the context must be destroyed.
 *  - Latent layout ("global order"): layer 0..L-1; within a layer the
 *    projections q, k, v, o, gate, up, down; each a row-major [N_out, K_in]
 *    fp32 matrix, concatenated.  q: [H*hd, D]; k, v: [KV*hd, D];
 *    o: [D, H*hd]; gate, up: [F, D]; down: [D, F]; hd = D / H.
 *  - Packed ternary store: code q + 1 of global weight i (q in {-1,0,1},
 *    Eq. 2) in bits 2*(i mod 16) of uint32 word i / 16.
 */
#ifndef TERMEZO_H
#define TERMEZO_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define TERMEZO_OK 0
#define TERMEZO_WMASKFIXED 1   /* density differs from the built mask; ignored */
#define TERMEZO_EINVAL (-1)    /* bad shape, null pointer, density outside (0,1] */
#define TERMEZO_ESTATE (-2)    /* call out of order (e.g. step before build_mask) */
#define TERMEZO_ENOMEM (-3)    /* workspace smaller than termezo_workspace_bytes */
#define TERMEZO_ECUDA (-4)     /* a CUDA call failed */
#define TERMEZO_ETIMEOUT (-5)  /* a bounded device-side wait gave up */

typedef struct termezo_ctx termezo_ctx;

/* Shape of the BitNet decoder and of one minibatch.
 * layers == 0 selects the single-projection ("BitLinear op") context: one
 * ternary projection of shape [ffn, hidden] and seq*batch activation rows;
 * termezo_step and termezo_forward_loss are then unavailable.
 * loss_mode 0: cross-entropy of the last position over the n_labels label
 * tokens vocab-n_labels .. vocab-1 (targets = class ids [batch]).
 * loss_mode 1: token-level cross-entropy over the full vocabulary at every
 * position (targets = token ids [batch, seq]).
 * weight_cache != 0 (decoder contexts): the workspace also holds every
 * weight's ternary code as one e4m3 byte (d bytes), kept equal to the packed
 * 2-bit store by every call that rewrites codes, and the forward's GEMMs read
 * it directly instead of expanding the packed codes of each projection
 * before its GEMM.  It trades d bytes of device memory (not part of the
 * paper's memory equation) for the expansion work.  Ignored for layers == 0.
 * z_cache != 0: the workspace also holds one float per active weight (the
 * sparse store's capacity, 4 k bytes, not part of the paper's memory
 * equation): the perturbation sums of a direction write z there in store
 * order and the requantisations, the restore and the update of the same
 * direction read it instead of regenerating z by Philox (the values are the
 * same).  0: every pass regenerates z (Algorithm 1 draws z from the seed). */
typedef struct {
  int32_t layers, hidden, heads, kv_heads, ffn, vocab, seq, batch;
  int32_t loss_mode;
  int32_t n_labels;
  int32_t weight_cache;
  int32_t z_cache;
} termezo_model_cfg;

/* Per-step report (Algorithm 1 with K = 1; counters of Eq. 11). */
typedef struct {
  double loss_plus;   /* F+ = minibatch loss at w + eps m.z            */
  double loss_minus;  /* F- = minibatch loss at w - eps m.z            */
  double g;           /* projected gradient (F+ - F-) / (2 eps)        */
  uint64_t k_active;  /* k_t = |S_t| after this step's shrink (Eq. 5)  */
  uint64_t n_flipped; /* active codes that differ between the two passes */
  uint64_t n_jumps;   /* active codes that moved -1 <-> +1 between them  */
  uint64_t n_dropped; /* weights frozen by this step's shrink           */
  uint64_t n_near_threshold; /* active latents within 1e-5 s_w of +-tau (Eq. 2
                        thresholds) in the + pass plus those in the - pass:
                        the codes excluded from bit-exact comparison, the
                        distance | |w| - tau | taken in float64          */
} termezo_step_out;

/* Bytes of device workspace a context needs for cfg and mask density
 * rho_0 (the sparse store holds floor(rho_0 * d) weights).  Host only. */
int termezo_workspace_bytes(const termezo_model_cfg* cfg, double density, size_t* bytes);

/* Device memory of a context, by part (Sec. 5's memory equation): the
 * paper gives the TerMeZO footprint as the MeZO footprint minus
 * d (1 - rho_0)(B - B_Q) plus rho_0 d B_Q plus the mask, M_mask =
 * min(ceil(d / 8), ceil(rho_0 d ceil(log2 d) / 8)).  This library stores the
 * active latents in float32 (B = 4) with 32-bit indices, both in two buffers
 * (the order-preserving shrink writes the second), and every code packed at
 * B_Q = 2/8.  All sizes in bytes; host only, no device call. */
typedef struct {
  uint64_t d;               /* ternary latents */
  uint64_t k_cap;           /* active latents the store holds (k0) */
  uint64_t packed;          /* 2-bit codes of all d latents */
  uint64_t sparse_index;    /* active index lists (two buffers) */
  uint64_t sparse_latents;  /* fp32 active latents (two buffers) */
  uint64_t mask_state;      /* exact sums, partials, histograms, counters, losses */
  uint64_t forward;         /* forward activations and GEMM operands */
  uint64_t workspace;       /* all of the above: termezo_workspace_bytes */
  uint64_t theta;           /* the caller's embeddings (fp32), norm gains (fp32), LM head (bf16) */
  uint64_t mask_bitmask;    /* the paper's dense bit-mask option, ceil(d / 8) */
  uint64_t mask_index_list; /* the paper's index-list option, ceil(rho_0 d ceil(log2 d) / 8) */
  uint64_t weight_cache;    /* e4m3 copy of the codes (weight_cache != 0), d bytes; else 0 */
  uint64_t z_cache;         /* z of the active weights (z_cache != 0), 4 k_cap bytes; else 0 */
} termezo_memory_out;

int termezo_memory(const termezo_model_cfg* cfg, double density, termezo_memory_out* out);

/* Creates a context over a caller-owned device workspace of `bytes` bytes
 * (>= termezo_workspace_bytes(cfg, density)); 256-byte aligned.  `stream`
 * is a cudaStream_t.  The workspace must outlive the context.  The kernels
 * of the mask build are loaded here (CUDA loads a kernel at its first launch
 * otherwise), so termezo_build_mask's one run is not charged their loading.
 * Returns TERMEZO_ECUDA when that loading fails. */
int termezo_create(const termezo_model_cfg* cfg, double density, void* d_workspace,
                   size_t bytes, void* stream, termezo_ctx** out);

/* Registers the parameters (device pointers, read by later calls; they
 * must stay valid until termezo_build_mask returns, and d_embed, d_gains,
 * d_head for the life of the context).  d_latents is read by
 * termezo_build_mask only: once it returns successfully the context forgets
 * the pointer (the caller may release the dense latents; another build
 * needs another termezo_load_params, else it returns TERMEZO_ESTATE):
 *   d_latents fp32 [d]       dense latent weights w_0, global order;
 *   d_embed   fp32 [V, D]    token embeddings (theta);
 *   d_gains   fp32 [2L+1, D] RMSNorm gains: 2l = attention input of layer l,
 *                            2l+1 = MLP input, 2L = final norm;
 *   d_head    bf16 [V, D]    LM head, raw bfloat16 bits.
 * For a single-projection context d_embed, d_gains, d_head may be NULL. */
int termezo_load_params(termezo_ctx* ctx, const float* d_latents, const float* d_embed,
                        const float* d_gains, const uint16_t* d_head);

/* The initial mask of Algorithm 1 (Eqs. 2-4): per projection gamma = mean |w|
 * (exact sum), tau_0 = (gamma + 1e-5) / 2, distances d_i = min(|w_i - tau|,
 * |w_i + tau|) of all weights of all projections, xi_0 the lower
 * rho_0-quantile: exactly k0 = floor(rho_0 d) weights with the smallest
 * (d_i, i) pairs form S_0 (ties at xi_0 go to the lower global index).
 * Writes the sparse store (sorted active indices + fp32 latents) and the
 * packed codes of every weight at tau_0.  Host outputs k0, xi0 (nullable).
 * density must not exceed the one given to termezo_create.  Synchronises. */
int termezo_build_mask(termezo_ctx* ctx, double density, uint64_t* k0, float* xi0);

/* Mask rules: the global quantile of Eq. 4 (termezo_build_mask), or its
 * per-tensor variant, in which every projection l keeps its own
 * floor(rho_0 n_l) smallest (d_i, i) pairs (ties to the lower index) and has
 * its own xi_0^l, used by its shrink (Eq. 5). */
enum { TERMEZO_MASK_GLOBAL = 0, TERMEZO_MASK_PER_TENSOR = 1 };

/* termezo_build_mask with a mask rule.  Host outputs: k0 (the total kept),
 * xi0: one float for TERMEZO_MASK_GLOBAL, [n_proj] floats (xi_0 of every
 * projection, 0 where a projection keeps none) for TERMEZO_MASK_PER_TENSOR;
 * nullable.  Synchronises. */
int termezo_build_mask_rule(termezo_ctx* ctx, double density, int32_t rule, uint64_t* k0, float* xi0);

/* Minibatch loss F(Q(w_t), theta; B) (Eqs. 6-7) at the current latents:
 * requantises the active weights, runs the BitNet forward.  d_tokens int32
 * [batch, seq]; d_targets int32 (see loss_mode).  Host outputs: loss, and
 * per_seq[batch] (nullable) the loss of each sequence.  Synchronises. */
int termezo_forward_loss(termezo_ctx* ctx, const int32_t* d_tokens, const int32_t* d_targets,
                         double* loss, double* per_seq);

/* Intermediates of one decoder layer of the forward (Sec. 3 BitNet block;
 * Eqs. 6-7 evaluate it at the perturbed codes), for layer-by-layer parity
 * checks.  Every pointer is a caller-owned device buffer that the call fills,
 * or NULL to skip it; T = batch * seq rows, D = hidden, Hq = heads * hd,
 * F = ffn.  Activation codes are the int8 values q of the per-token absmax
 * quantiser that the BitLinear GEMM consumes, with deq = a / 127 per row.
 *   x_in       fp32 [T, D]   residual stream entering the layer
 *   codes_attn int8 [T, D], deq_attn fp32 [T]   codes of RMSNorm(x_in)
 *   q          bf16 [B, H, S, hd]   RoPE-rotated queries (raw bits)
 *   k          bf16 [B, KV, S, hd]  RoPE-rotated keys
 *   vt         bf16 [B, KV, hd, S]  values, transposed
 *   attn       fp32 [T, Hq]  causal attention output
 *   codes_o    int8 [T, Hq], deq_o fp32 [T]     codes of attn
 *   x_mid      fp32 [T, D]   x_in + o(attn)
 *   codes_mlp  int8 [T, D], deq_mlp fp32 [T]    codes of RMSNorm(x_mid)
 *   hid        fp32 [T, F]   relu(gate)^2 * up
 *   codes_down int8 [T, F], deq_down fp32 [T]   codes of hid
 *   x_out      fp32 [T, D]   x_mid + down(hid)
 * For layer == layers only x_in is filled: the residual stream after the last
 * layer, which the final RMSNorm and the LM head read. */
typedef struct {
  float* x_in;
  int8_t* codes_attn;
  float* deq_attn;
  uint16_t *q, *k, *vt;
  float* attn;
  int8_t* codes_o;
  float* deq_o;
  float* x_mid;
  int8_t* codes_mlp;
  float* deq_mlp;
  float* hid;
  int8_t* codes_down;
  float* deq_down;
  float* x_out;
} termezo_layer_trace;

/* The BitNet forward and minibatch loss at the codes now in the packed store
 * (those of the last termezo_build_mask, termezo_requantize or step, with
 * their weight scales; nothing is requantised), copying the intermediates of
 * `layer` (0 <= layer <= layers) into `trace`.  A test and diagnostic call:
 * the copies cost a device-to-device copy per buffer.  loss, per_seq as
 * termezo_forward_loss (nullable).  Synchronises. */
int termezo_forward_trace(termezo_ctx* ctx, const int32_t* d_tokens, const int32_t* d_targets, int32_t layer,
                          const termezo_layer_trace* trace, double* loss, double* per_seq);

/* One TerMeZO iteration (Algorithm 1 loop body, K = 1):
 *   t >= 1: tau_t recomputed, S_t = {i in S_{t-1}: d_i(w_t) <= xi_0} (Eq. 5);
 *   z_i ~ N(0,1) regenerated from (seed, i) by Philox-4x32-10 + Box-Muller;
 *   w += eps m.z -> requantise (Eq. 2) -> F+;  w -= 2 eps m.z -> F-;
 *   w += eps m.z (restore); g = (F+ - F-) / (2 eps) (Eq. 1);
 *   w -= lr g m.z with the same z.
 * density: the mask's rho_0 is fixed after build (xi_0 is fixed, Eq. 5); a
 * different value returns TERMEZO_WMASKFIXED and is otherwise ignored.
 * out: host report (required); per_seq_plus / per_seq_minus: host [batch]
 * per-sequence losses of the two passes (nullable).  Synchronises once, at
 * the end, where it also reads back the active set's per-projection offsets
 * and re-plans the split of the sparse store into blocks of at most 4096
 * active weights for the next call (the results do not depend on it). */
int termezo_step(termezo_ctx* ctx, uint64_t seed, float eps, float lr, double density,
                 const int32_t* d_tokens, const int32_t* d_targets, termezo_step_out* out,
                 double* per_seq_plus, double* per_seq_minus);

/* One TerMeZO iteration of Algorithm 1 with K directions (1 <= K <= 8; the
 * paper's experiments use K = 5):
 *   t >= 1: the mask shrinks once (Eq. 5), as in termezo_step;
 *   for k = 0..K-1 with z_k regenerated from seeds[k]:
 *     w += eps m.z_k -> F+_k;  w -= 2 eps m.z_k -> F-_k;  w += eps m.z_k
 *     (restore: the next direction starts from the restored latents);
 *     g_k = (F+_k - F-_k) / (2 eps);
 *   then for k = 0..K-1: w -= (lr / K) g_k m.z_k, with (lr / K) g_k formed in
 *   float64 and rounded to float32.
 * seeds: host [K].  out: host report (required; loss_plus, loss_minus and g
 * are those of the last direction, the counters are summed over the
 * directions); losses: host [2K] F+_0, F-_0, F+_1, ... (nullable); g: host
 * [K] (nullable).  K = 1 is termezo_step.  Synchronises once. */
int termezo_step_k(termezo_ctx* ctx, const uint64_t* seeds, int32_t K, float eps, float lr, double density,
                   const int32_t* d_tokens, const int32_t* d_targets, termezo_step_out* out, double* losses,
                   double* g);

/* Algorithm 1 as written: termezo_step_k over the masked latents and the
 * full-precision parameters theta together.  Each direction perturbs theta
 * densely with the same seed (+eps z, -2 eps z, restore +eps z, each pass
 * next to the latents' requantisation), and the update applies
 * theta -= (lr / K) g_k z_k.  theta is the embeddings (fp32), norm gains
 * (fp32) and LM head (bf16) given to termezo_load_params, which must be
 * writable: they are updated in place, every assignment rounded to the
 * stored precision (the head: the float32 result rounded to bfloat16).
 * theta's z is the Philox stream of the seed at global indices d + j, j over
 * the embeddings, then the gains, then the head.  Needs D % 4 == 0,
 * 16-byte aligned embeddings and gains and an 8-byte aligned head, else
 * TERMEZO_EINVAL.  Arguments and report as termezo_step_k. */
int termezo_step_joint(termezo_ctx* ctx, const uint64_t* seeds, int32_t K, float eps, float lr, double density,
                       const int32_t* d_tokens, const int32_t* d_targets, termezo_step_out* out, double* losses,
                       double* g);

/* Pieces of the step, for the single-projection context and for tests.
 * termezo_shrink: Eq. 5 at the current latents (no-op before the first
 *   update); host output n_dropped (nullable).
 * termezo_requantize: sign = +1 writes the codes of w + eps z, sign = -1
 *   the codes of (w + eps z) - 2 eps z, sign = 0 the codes of w, each at
 *   the tau of the perturbed projection (Eq. 2); active weights only.
 * termezo_update: restore (+eps z) and w -= (float)(lr * g) z (Algorithm 1).
 * None of these synchronises. */
int termezo_shrink(termezo_ctx* ctx, uint64_t* n_dropped);
int termezo_requantize(termezo_ctx* ctx, uint64_t seed, float eps, int sign);
int termezo_update(termezo_ctx* ctx, uint64_t seed, float eps, float lr, double g);

/* BitLinear of projection `proj` (global order index) on activations
 * d_x bf16 [M, K_in] (raw bits, row-major): per row a = max(max|x|, 1e-5),
 * int8 codes q = clamp(rint(x * (127/a)), -128, 127) decided in fp32,
 * acc = q . codes^T (exact int32), y = acc * (a/127) * s_w with
 * s_w = gamma + 1e-5 of the current codes.  Outputs (device, nullable):
 * d_acc int32 [M, N_out], d_y fp32 [M, N_out].  M <= seq * batch. */
int termezo_bitlinear(termezo_ctx* ctx, int32_t proj, const uint16_t* d_x, int32_t M,
                      int32_t* d_acc, float* d_y);

/* Sizes of the state: d (latent count), k_active (current |S_t|),
 * n_proj (projection count).  Host outputs, each nullable.  Synchronises. */
int termezo_state_sizes(termezo_ctx* ctx, uint64_t* d, uint64_t* k_active, int32_t* n_proj);

/* Copies the state to host buffers (each nullable): h_idx uint32 [k_active]
 * sorted active global indices; h_latents fp32 [k_active] their latents;
 * h_packed uint32 [d/16] the packed codes; h_tau fp32 [3 * n_proj] the
 * thresholds tau of the current latents, of the + pass and of the - pass.
 * Synchronises. */
int termezo_export_state(termezo_ctx* ctx, uint32_t* h_idx, float* h_latents, uint32_t* h_packed,
                         float* h_tau);

/* z_i for n global indices d_idx (uint32, device) with key `seed`, written
 * to d_z fp32 [n].  Stateless; ordered on `stream`. */
int termezo_normal(uint64_t seed, const uint32_t* d_idx, uint64_t n, float* d_z, void* stream);

/* Allocation-free absmean.  The paper has no counterpart: this is an
 * interface for callers that cannot allocate device memory -- code inside a
 * host framework that owns all of the GPU's memory (a serving engine that
 * reserves it up front, or one that forbids cudaMalloc on its hot path
 * because it synchronises the device) and so cannot pass a workspace to
 * termezo_create.
 * Computes, for one fp32 latent tensor d_w[n] (device), the exact
 * gamma = mean |w| (Sec. 3, same arithmetic as termezo_build_mask),
 * tau = 0.5 (gamma + 1e-5) and s_w = gamma + 1e-5, written to the device
 * floats d_out[0], d_out[1], d_out[2], ordered on `stream`.
 * Scratch: a fixed array of TERMEZO_NOALLOC_MAX_ELEMS / 4096 partial sums
 * (4 MiB) inside the library; every GPU that loads the library holds it
 * until the process exits.  n > TERMEZO_NOALLOC_MAX_ELEMS returns
 * TERMEZO_EINVAL (with a message on stderr).  The first call on a device
 * looks up that device's address of the array; make it before any stream
 * capture.  The address is kept for the life of the process, so a
 * cudaDeviceReset of that device voids it: do not reset a device that is
 * still used with this call.  Calls share the array: calls that overlap on
 * the GPU race.
 * Each call overwrites every partial sum it reads.  Allocates nothing. */
#define TERMEZO_NOALLOC_MAX_ELEMS (1ull << 28)
int termezo_absmean_noalloc(const float* d_w, uint64_t n, float* d_out, void* stream);

/* Kernel timing of a context.  enable = n >= 1 resets the totals and starts
 * recording CUDA events (on the context's stream) around every n-th launch of
 * each kind: BitLinear GEMM, attention, sparse pass (n = 1: all of them; a
 * prime n such as 13 samples the four GEMM shapes of a layer and the five
 * sparse passes of a step in turn, and leaves most launches free of the
 * events, which also cut the programmatic overlap of the launches around
 * them); enable = 0 stops recording; enable = -1 leaves the state unchanged.  When out is non-NULL the stream
 * is synchronised and the totals since the last reset are written.
 * Algorithmic work: GEMM 2*M*N*K flops; attention 4*B*H*hd*S(S+1)/2 flops
 * (QK^T and PV over the causal half); sparse passes, by kind (pass_*):
 *   0 perturbation sums (k_sparse_pm_sum + the tau+- reductions): 8 B per
 *     active weight (index + latent) read;
 *   1 requantisation (one sign): 8 B per active weight read, plus every
 *     32-byte sector of the packed store that holds an active weight, read
 *     and written (64 B per sector);
 *   2 restore + update: 8 B per active weight read, 4 B written;
 *   3 shrink (Eq. 5): 8 B per active weight read twice, 8 B per kept weight
 *     written (counted as 24 B per active weight);
 *   4 theta perturbation / update (termezo_step_joint): each parameter read
 *     and written in its stored precision.
 * sparse_* are the totals over the kinds. */
#define TERMEZO_PASS_KINDS 5
typedef struct {
  uint64_t launches;        /* kernels launched by this thread since the reset */
  uint64_t gemm_launches;
  double gemm_ms, gemm_flops;
  uint64_t attn_launches;
  double attn_ms, attn_flops;
  uint64_t sparse_launches; /* timed sparse passes (each 1-5 kernels) */
  double sparse_ms, sparse_bytes;
  uint64_t gemm_seen, attn_seen, sparse_seen; /* launches of each kind while recording (timed or not) */
  uint64_t pass_launches[TERMEZO_PASS_KINDS], pass_seen[TERMEZO_PASS_KINDS];
  double pass_ms[TERMEZO_PASS_KINDS], pass_bytes[TERMEZO_PASS_KINDS];
} termezo_profile_out;

int termezo_profile(termezo_ctx* ctx, int enable, termezo_profile_out* out);

/* Causal attention of the BitNet forward on its own (the kernel
 * termezo_step uses), for tests and benchmarks.  d_q bf16 [B, H, S, hd],
 * d_k bf16 [B, KV, S, hd], d_vt bf16 [B, KV, hd, S] (V transposed); head h
 * reads KV head h / (H / KV); scores scaled by 1/sqrt(hd); P = exp(s -
 * row max) rounded to bf16; d_out fp32 [B*S, H*hd] = (P V) / sum P.
 * S % 64 == 0, hd in {64, 96, 128}, H % KV == 0.  Runs on the tcgen05
 * tensor cores when S % 128 == 0, else on mma.sync.
 * Stateless; on `stream`. */
int termezo_attention(const uint16_t* d_q, const uint16_t* d_k, const uint16_t* d_vt, int32_t B, int32_t S,
                      int32_t H, int32_t KV, int32_t hd, float* d_out, void* stream);

/* Releases the host-side context (the workspace stays the caller's). */
void termezo_destroy(termezo_ctx* ctx);

const char* termezo_strerror(int status);

#ifdef __cplusplus
}
#endif

#endif /* TERMEZO_H */
