// Device state of the mask and of the sparse latent store (host side view).
#pragma once

#include <cuda_runtime.h>

#include <cstdint>

#include "common.cuh"

namespace tmz {

struct SelectState {
  unsigned long long krem;  // rank still to find (1-based); after the last pass: ties to take
  uint32_t prefix;          // radix prefix found so far; after the last pass: the key of xi_0
  uint32_t pad;
};

// Everything the mask / sparse kernels touch.  Passed by value to kernels.
struct MaskArgs {
  int P;                        // projections
  const uint64_t* base;         // [P+1] first global index of each projection
  const uint32_t* dpre;         // [P+1] dense-block prefix (4096 elements per block)
  const uint16_t* dproj;        // [NBD] projection of each dense block
  uint32_t NBD;                 // dense blocks
  const uint32_t* spre;         // [P+1] sparse-block prefix
  const uint16_t* sproj;        // [NBS] projection of each sparse block
  uint32_t NBS;                 // sparse blocks
  uint32_t* packed;             // [d/16] 2-bit codes
  uint8_t* wbyte;               // [d] the same codes as e4m3 bytes (+1, 0, -1), or null: every
                                // kernel that writes packed codes writes these bytes too
  uint32_t* idx[2];             // active global indices (double buffer)
  float* lat[2];                // active latents
  uint32_t* off[2];             // [P+1] segment offsets into idx/lat
  ExactSum* S_total;            // [P] exact sum of |w_0|
  ExactSum* A_frozen;           // [P] exact sum of |w| over frozen weights
  ExactSum* partials;           // per-block partial sums
  float *gamma_cur, *tau_cur, *sw_cur;       // [P+2] of the current latents
  float *gamma_plus, *tau_plus, *sw_plus;    // [P+2] of w + eps z
  float *gamma_minus, *tau_minus, *sw_minus; // [P+2] of w - eps z
  int groups;                   // selection groups: 1 (the global quantile of Eq. 4) or P
                                // (one per projection: the per-tensor variant)
  unsigned long long* hist;     // [max(groups x 2048, 8192)]
  SelectState* sel;             // [groups]
  unsigned long long* grp_tie0; // [P] ties before the first dense block of each group
  float* xi0p;                  // [P] xi_0 of each projection (Eq. 5)
  uint32_t *blk_a, *blk_b, *blk_c, *blk_d;   // per-block scratch
  float* zbuf;                  // [k_cap] z of the active weights of the current direction, in
                                // store order (written by the perturbation sums), or null: every
                                // pass regenerates z
  uint32_t sup_cap;             // entries idx[1] / lat[1] hold (the superset of mask_build_fast)
  unsigned long long* scan_state; // [NBD] decoupled look-back words of the superset compaction
  uint32_t* sup;                // [4] superset size, overflow flag, block ticket, unused
  unsigned long long* counters; // [0] flipped, [1] jumps, [2] dropped, [3] 32-byte sectors of the packed store rewritten,
                                // [4] active latents within 1e-5 s_w of +-tau in the +/- passes
  unsigned* err;
};

// Selects S_0 (the a.groups groups' select states must hold their k) and
// writes the sparse store, the codes at tau_0 and xi0p.
void mask_build(const MaskArgs& a, const float* w, uint64_t k0, cudaStream_t s);
// The global quantile (groups == 1, 0 < k0) in two dense passes and a
// sampled one.  hist [8192], sup and scan_state must be zero and sel hold k0.
// Afterwards sup[1] != 0 means the superset held fewer than k0 weights or did
// not fit in idx[1] / lat[1], and nothing but the codes at tau_0 was written
// (run mask_build instead); otherwise S_0, xi0p and the codes are written and
// mask_build_fast_offsets writes off[0].
void mask_build_fast(const MaskArgs& a, const float* w, uint64_t k0, cudaStream_t s);
void mask_build_fast_offsets(const MaskArgs& a, uint64_t k0, cudaStream_t s);
// Loads every kernel of the mask build (done when a context is created).
cudaError_t mask_preload();
void mask_finish(const MaskArgs& a, cudaStream_t s);
void sparse_pm_taus(const MaskArgs& a, int cur, uint64_t seed, float eps, cudaStream_t s);
// use_z: read z from zbuf (filled by sparse_pm_taus for this seed and store
// order) instead of regenerating it.
void sparse_requant(const MaskArgs& a, int cur, uint64_t seed, float eps, int sign, bool use_z, cudaStream_t s);
// Directions of one step (Algorithm 1 with K <= KMAX perturbations).
constexpr int KMAX = 8;
struct UpdateDirs {
  uint64_t seed[KMAX];
  uint64_t last;  // seed[K - 1]
  int K;
};
// The full-precision parameters theta (device pointers the caller owns):
// embeddings fp32 [n_emb], norm gains fp32 [n_gains], LM head bf16 [n_head];
// all sizes and d multiples of 4, fp32 parts 16-byte and the head 8-byte
// aligned.
struct ThetaArgs {
  float* emb;
  uint64_t n_emb;
  float* gains;
  uint64_t n_gains;
  uint16_t* head;
  uint64_t n_head;
  uint64_t d;  // latents: theta's z is the Philox stream at indices d + j
};
// theta += e (mode 0: the + pass and the restore) or theta -= 2 e (mode 1).
void theta_pm(const ThetaArgs& t, uint64_t seed, float eps, int mode, cudaStream_t s);
// The last direction's restore, then theta -= (lr / K) g_k z_k for each k.
void theta_update(const ThetaArgs& t, const UpdateDirs& d, float eps, float lr, const double* g_dev, cudaStream_t s);

// Restore after direction seed: w = fl(fl(fl(w + e) - 2 e) + e), e = fl(eps z).
void sparse_restore(const MaskArgs& a, int cur, uint64_t seed, float eps, bool use_z, cudaStream_t s);
// Restore after the last direction, then w = fl(w - fl(c_k z_k)) for k = 0..K-1
// with c_k = (float)((lr / K) g_k), g_k = g_dev[k]; exact sums of the result.
void sparse_update_dirs(const MaskArgs& a, int cur, const UpdateDirs& d, float eps, float lr, const double* g_dev,
                        bool use_z, cudaStream_t s);
void sparse_update(const MaskArgs& a, int cur, uint64_t seed, float eps, float lr, const double* g_dev,
                   double g_host, int use_host, bool use_z, cudaStream_t s);
void sparse_shrink(const MaskArgs& a, int cur, uint32_t* d_total, cudaStream_t s);
void launch_grad(const double* loss, float eps, double* g, cudaStream_t s);
void launch_normal(uint64_t seed, const uint32_t* idx, uint64_t n, float* z, cudaStream_t s);

}  // namespace tmz
