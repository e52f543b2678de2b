// C ABI of libtermezo.so: context, workspace layout and the host-side
// orchestration of Algorithm 1 (declarations and contracts in termezo.h).
#include <cmath>
#include <cstdio>
#include <cstring>
#include <new>
#include <vector>

#include "kernels.cuh"
#include "sparse.cuh"
#include "termezo.h"

using tmz::ExactSum;
using tmz::GemmArgs;
using tmz::GemmPlan;
using tmz::MaskArgs;

namespace {

constexpr uint32_t DENSE_CHUNK = 4096;
constexpr uint32_t SPARSE_CHUNK = 4096;

struct Shape {
  bool op;
  bool wcache;  // e4m3 weight cache (decoder contexts)
  bool zcache;  // z of the active weights kept between the passes of a direction
  int L, D, H, KV, hd, F, V, S, B, T, C, mode;
  int P;
  std::vector<uint64_t> base;  // [P+1]
  std::vector<int> N, K;       // [P]
  uint64_t d;
};

int make_shape(const termezo_model_cfg* c, Shape* s) {
  if (!c) return TERMEZO_EINVAL;
  s->op = c->layers == 0;
  s->wcache = !s->op && c->weight_cache != 0;
  s->zcache = c->z_cache != 0;
  s->L = c->layers;
  s->D = c->hidden;
  s->F = c->ffn;
  s->S = c->seq;
  s->B = c->batch;
  s->T = c->seq * c->batch;
  s->mode = c->loss_mode;
  s->C = c->n_labels;
  s->V = c->vocab;
  s->H = c->heads;
  s->KV = c->kv_heads;
  if (c->layers < 0 || c->hidden <= 0 || c->ffn <= 0 || c->seq <= 0 || c->batch <= 0) return TERMEZO_EINVAL;
  if (c->hidden % 16 || c->ffn % 16) return TERMEZO_EINVAL;
  s->base.assign(1, 0);
  s->N.clear();
  s->K.clear();
  if (s->op) {
    s->P = 1;
    s->N.push_back(c->ffn);
    s->K.push_back(c->hidden);
    s->hd = 0;
  } else {
    if (c->heads <= 0 || c->kv_heads <= 0 || c->hidden % c->heads || c->heads % c->kv_heads) return TERMEZO_EINVAL;
    s->hd = c->hidden / c->heads;
    if (s->hd != 64 && s->hd != 96 && s->hd != 128) return TERMEZO_EINVAL;
    if (c->seq % 64) return TERMEZO_EINVAL;
    if (c->vocab <= 0) return TERMEZO_EINVAL;
    if (c->loss_mode != 0 && c->loss_mode != 1) return TERMEZO_EINVAL;
    if (c->loss_mode == 0 && (c->n_labels < 1 || c->n_labels > 64 || c->n_labels > c->vocab)) return TERMEZO_EINVAL;
    const int Hq = s->H * s->hd, Hkv = s->KV * s->hd;
    const int n[7] = {Hq, Hkv, Hkv, s->D, s->F, s->F, s->D};
    const int k[7] = {s->D, s->D, s->D, Hq, s->D, s->D, s->F};
    s->P = 7 * s->L;
    for (int l = 0; l < s->L; ++l)
      for (int j = 0; j < 7; ++j) {
        s->N.push_back(n[j]);
        s->K.push_back(k[j]);
      }
  }
  for (int p = 0; p < s->P; ++p) s->base.push_back(s->base.back() + (uint64_t)s->N[p] * (uint64_t)s->K[p]);
  s->d = s->base.back();
  if (s->d >= (1ull << 32) || s->P > 65535) return TERMEZO_EINVAL;
  return TERMEZO_OK;
}

uint64_t keep_count(double density, uint64_t d) { return (uint64_t)std::floor(density * (double)d); }

// Bump allocator over the workspace; with base == nullptr it only measures.
// Workspace sections, for the memory report.
// Sparse pass kinds of termezo_profile_out::pass_* (see termezo.h).
enum { PASS_PM = 0, PASS_REQUANT = 1, PASS_UPDATE = 2, PASS_SHRINK = 3, PASS_THETA = 4 };
static_assert(PASS_THETA + 1 == TERMEZO_PASS_KINDS, "pass kinds");

enum Section { SEC_PACKED, SEC_INDEX, SEC_LATENTS, SEC_MASK, SEC_FORWARD, SEC_WCACHE, SEC_ZCACHE, SEC_COUNT };

struct Carver {
  uint8_t* base;
  size_t off = 0;
  int sec = SEC_MASK;
  size_t bytes[SEC_COUNT] = {};
  template <typename T>
  T* take(size_t count) {
    const size_t start = (off + 255) & ~(size_t)255;
    T* p = base ? reinterpret_cast<T*>(base + start) : nullptr;
    bytes[sec] += start + count * sizeof(T) - off;
    off = start + count * sizeof(T);
    return p;
  }
};

// The QKV projection writes RoPE-rotated bf16 Q, K and V^T directly (fused
// epilogue) for head dims 64 / 128 and S a multiple of 32; other shapes go
// through an fp32 QKV buffer and a separate RoPE pass.
bool rope_fused_shape(const Shape& s) { return !s.op && (s.hd == 64 || s.hd == 128) && s.S % 32 == 0; }

}  // namespace

struct termezo_ctx {
  Shape sh;
  double density = 0;
  uint64_t k_cap = 0;
  cudaStream_t stream = nullptr;
  MaskArgs ma{};
  uint32_t NBS_max = 0;
  uint32_t* d_total = nullptr;
  std::vector<uint32_t> dpre;
  std::vector<uint32_t> off_host, spre_host;  // sparse-store offsets read back, block plan uploaded
  std::vector<uint16_t> sproj_host;
  int cur = 0;
  bool built = false;
  int t = 0;
  bool updated = false;
  float xi0 = 0.f;
  uint64_t k0 = 0, k_active = 0;
  const float* latents = nullptr;
  const float* embed = nullptr;
  const float* gains = nullptr;
  const uint16_t* head = nullptr;
  // forward buffers
  float* x = nullptr;
  uint8_t* xq = nullptr;  // e4m3 (hi, lo) activation codes [2, T, K]
  float* deq = nullptr;
  float* qkv = nullptr;
  uint16_t *qb = nullptr, *kb = nullptr, *vt = nullptr;
  float* attn = nullptr;
  float* gu = nullptr;
  uint8_t* wexp = nullptr;
  uint8_t* wbyte = nullptr;  // weight cache: e4m3 code of every weight [d]
  std::vector<GemmPlan> cplan;  // weight cache: per layer the q,k,v / o / gate,up / down plans
  float *cosb = nullptr, *sinb = nullptr;
  double* per_seq = nullptr;  // [2B]
  double* loss = nullptr;     // [2]
  double* g = nullptr;        // [KMAX]: g of each direction of a step
  double* lossk = nullptr;    // [2 KMAX]: F+, F- of each direction
  GemmPlan plan_qkv{}, plan_o{}, plan_gu{}, plan_down{}, plan_head{};
  tmz::AttnPlan att_plan{};
  bool att_tc = false;
  bool head_plan_ok = false;
  // loss mode 1 (token-level cross-entropy over the vocabulary)
  uint16_t* hfin = nullptr;   // bf16 [T, D]
  float2* part = nullptr;     // [T, ceil(V/256)]
  float* tlogit = nullptr;    // [T]
  double* tok_loss = nullptr; // [T]
  const float* code_sw = nullptr;  // s_w array matching the codes now in the packed store
  uint64_t pm_seed = 0;
  float pm_eps = 0.f;
  bool pm_valid = false;
  // kernel timing (termezo_profile)
  struct ProfRec {
    int cat;  // 0 GEMM, 1 attention, 2 + PASS_* a sparse pass
    cudaEvent_t a, b;
    double work;
  };
  bool prof_on = false;
  int prof_stride = 1;
  uint64_t prof_seq[2 + TERMEZO_PASS_KINDS] = {};
  std::vector<ProfRec> prof;
  std::vector<cudaEvent_t> ev_pool;
  // weight expansion overlapped with the previous GEMM: a side stream and two
  // e4m3 weight buffers (q,k,v and gate,up in wexp; o and down in wexp2)
  uint8_t* wexp2 = nullptr;
  float* split_ws = nullptr;     // GEMM tail-wave split-K partial tiles
  unsigned* split_cnt = nullptr;
  int split_cap = 0;
  cudaStream_t xstream = nullptr;
  cudaEvent_t ev_free[2] = {nullptr, nullptr};   // buffer b no longer read
  cudaEvent_t ev_ready[2] = {nullptr, nullptr};  // buffer b holds the next group's weights
  cudaEvent_t ev_codes = nullptr;                // the codes of this forward are final
  size_t ev_used = 0;
  uint64_t launch_base = 0;
  // termezo_forward_trace: the layer whose intermediates run_forward copies
  const termezo_layer_trace* trace = nullptr;
  int trace_layer = -1;
  ~termezo_ctx() {
    for (cudaEvent_t e : ev_pool) cudaEventDestroy(e);
    for (cudaEvent_t e : {ev_free[0], ev_free[1], ev_ready[0], ev_ready[1], ev_codes})
      if (e) cudaEventDestroy(e);
    if (xstream) cudaStreamDestroy(xstream);
  }
};

namespace {

size_t xq_cols(const Shape& s) {
  if (s.op) return (size_t)s.D;
  size_t m = s.D;
  if ((size_t)s.H * s.hd > m) m = (size_t)s.H * s.hd;
  if ((size_t)s.F > m) m = s.F;
  return m;
}

// Partial-tile slots of the GEMM's tail-wave split (at most one wave of
// 128-row tiles, and no more than the context's GEMMs can have).
int split_slots(const Shape& s) {
  const size_t mt = ((size_t)s.T + 127) / 128;
  const size_t nmax = s.op ? (size_t)s.F : (size_t)(s.H + 2 * s.KV) * s.hd + 2 * (size_t)s.F + s.D;
  const size_t tiles = mt * ((nmax + 127) / 128);
  return (int)(tiles < 192 ? tiles : 192);
}

size_t wexp_elems(const Shape& s) {
  size_t m = 0;
  if (s.op) return (size_t)s.N[0] * s.K[0];
  const size_t qkv = (size_t)(s.H + 2 * s.KV) * s.hd * s.D, o = (size_t)s.D * s.H * s.hd,
               gu = (size_t)256 * ((s.F + 127) / 128) * s.D,
               dn = (size_t)s.D * s.F;
  m = qkv;
  if (o > m) m = o;
  if (gu > m) m = gu;
  if (dn > m) m = dn;
  return m;
}

void carve(termezo_ctx* c, Carver& cv) {
  const Shape& s = c->sh;
  const int P = s.P;
  MaskArgs& a = c->ma;
  a.P = P;
  a.base = cv.take<uint64_t>(P + 1);
  a.dpre = cv.take<uint32_t>(P + 1);
  a.spre = cv.take<uint32_t>(P + 1);
  a.dproj = cv.take<uint16_t>(c->dpre.empty() ? 1 : c->dpre.back());
  a.sproj = cv.take<uint16_t>(c->NBS_max);
  cv.sec = SEC_PACKED;
  a.packed = cv.take<uint32_t>(s.d / 16);
  // The second buffer is followed by k_cap / 8 + 4096 spare entries (mask
  // state): the fast mask build stages its superset of S_0 there (about k0
  // (1 + 1/100 + 1/45) plus the sampling margin).
  const size_t spare = c->k_cap / 8 + 4096;
  for (int i = 0; i < 2; ++i) {
    cv.sec = SEC_INDEX;
    a.idx[i] = cv.take<uint32_t>(c->k_cap);
    const size_t idx_end = cv.off;
    cv.sec = SEC_MASK;
    if (i == 1) cv.take<uint32_t>(spare);
    const size_t idx_room = (cv.off - idx_end) / sizeof(uint32_t) + c->k_cap;
    cv.sec = SEC_LATENTS;
    a.lat[i] = cv.take<float>(c->k_cap);
    const size_t lat_end = cv.off;
    cv.sec = SEC_MASK;
    if (i == 1) cv.take<float>(spare);
    const size_t lat_room = (cv.off - lat_end) / sizeof(float) + c->k_cap;
    if (i == 1) {
      // entries that fit below the next buffer (alignment gaps included)
      const size_t room = idx_room < lat_room ? idx_room : lat_room;
      a.sup_cap = (uint32_t)(room < 0xFFFFFFFFull ? room : 0xFFFFFFFFull);
    }
    a.off[i] = cv.take<uint32_t>(P + 1);
  }
  if (s.zcache) {
    cv.sec = SEC_ZCACHE;
    a.zbuf = cv.take<float>(c->k_cap);
    cv.sec = SEC_MASK;
  }
  a.S_total = cv.take<ExactSum>(P);
  a.A_frozen = cv.take<ExactSum>(P);
  const size_t nbd = c->dpre.empty() ? 0 : c->dpre.back();
  const size_t nblk = nbd > c->NBS_max ? nbd : c->NBS_max;
  a.partials = cv.take<ExactSum>(nbd > 2 * (size_t)c->NBS_max ? nbd : 2 * (size_t)c->NBS_max);
  float** fl[9] = {&a.gamma_cur, &a.tau_cur, &a.sw_cur, &a.gamma_plus, &a.tau_plus,
                   &a.sw_plus,   &a.gamma_minus, &a.tau_minus, &a.sw_minus};
  for (auto f : fl) *f = cv.take<float>(P + 2);
  a.hist = cv.take<unsigned long long>(2048 * (size_t)P > 8192 ? 2048 * (size_t)P : 8192);
  a.scan_state = cv.take<unsigned long long>(nbd ? nbd : 1);
  a.sup = cv.take<uint32_t>(4);
  a.sel = cv.take<tmz::SelectState>(P);
  a.grp_tie0 = cv.take<unsigned long long>(P);
  a.xi0p = cv.take<float>(P);
  a.blk_a = cv.take<uint32_t>(nblk);
  a.blk_b = cv.take<uint32_t>(nblk);
  a.blk_c = cv.take<uint32_t>(nblk);
  a.blk_d = cv.take<uint32_t>(nblk);
  a.counters = cv.take<unsigned long long>(8);
  a.err = cv.take<unsigned>(1);
  c->d_total = cv.take<uint32_t>(1);
  const size_t T = s.T;
  cv.sec = SEC_FORWARD;
  c->xq = cv.take<uint8_t>(2 * T * xq_cols(s));
  c->deq = cv.take<float>(T);
  // expansion buffers, or (weight cache) one e4m3 byte per weight
  c->wexp = s.wcache ? nullptr : cv.take<uint8_t>(wexp_elems(s));
  c->wexp2 = (s.op || s.wcache) ? nullptr : cv.take<uint8_t>(wexp_elems(s));
  if (s.wcache) {
    cv.sec = SEC_WCACHE;
    c->wbyte = cv.take<uint8_t>(s.d);
    cv.sec = SEC_FORWARD;
  }
  a.wbyte = c->wbyte;
  c->split_cap = split_slots(s);
  c->split_ws = cv.take<float>((size_t)c->split_cap * 128 * 256);
  c->split_cnt = cv.take<unsigned>((size_t)c->split_cap * 4);
  if (!s.op) {
    const size_t hq = (size_t)s.H * s.hd, hkv = (size_t)s.KV * s.hd;
    c->x = cv.take<float>(T * s.D);
    c->qkv = rope_fused_shape(s) ? nullptr : cv.take<float>(T * (hq + 2 * hkv));
    c->qb = cv.take<uint16_t>(T * hq);
    c->kb = cv.take<uint16_t>(T * hkv);
    c->vt = cv.take<uint16_t>(T * hkv);
    c->attn = cv.take<float>(T * hq);
    c->gu = cv.take<float>(T * (size_t)s.F);  // hid = relu(gate)^2 up
    c->cosb = cv.take<float>((size_t)s.S * s.hd / 2);
    c->sinb = cv.take<float>((size_t)s.S * s.hd / 2);
    if (s.mode == 1) {
      c->hfin = cv.take<uint16_t>(T * s.D);
      c->part = cv.take<float2>(T * (size_t)tmz::gemm_col_tiles(s.V));
      c->tlogit = cv.take<float>(T);
      c->tok_loss = cv.take<double>(T);
    }
  }
  cv.sec = SEC_MASK;
  c->per_seq = cv.take<double>(2 * (size_t)s.B);
  c->loss = cv.take<double>(2);
  c->g = cv.take<double>(tmz::KMAX);
  c->lossk = cv.take<double>(2 * tmz::KMAX);
}

void plan_sizes(termezo_ctx* c, double density) {
  const Shape& s = c->sh;
  c->density = density;
  c->k_cap = keep_count(density, s.d);
  if (c->k_cap == 0) c->k_cap = 1;
  c->dpre.assign(1, 0);
  for (int p = 0; p < s.P; ++p) {
    const uint64_t n = s.base[p + 1] - s.base[p];
    c->dpre.push_back(c->dpre.back() + (uint32_t)((n + DENSE_CHUNK - 1) / DENSE_CHUNK));
  }
  c->NBS_max = (uint32_t)(2 * s.P + c->k_cap / SPARSE_CHUNK + 1);
}

int cuda_status(termezo_ctx* c) {
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    fprintf(stderr, "termezo: CUDA error %s\n", cudaGetErrorString(e));
    return TERMEZO_ECUDA;
  }
  (void)c;
  return TERMEZO_OK;
}

int sync_status(termezo_ctx* c) {
  cudaError_t e = cudaStreamSynchronize(c->stream);
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) {
    fprintf(stderr, "termezo: CUDA error %s\n", cudaGetErrorString(e));
    return TERMEZO_ECUDA;
  }
  unsigned err = 0;
  if (cudaMemcpy(&err, c->ma.err, sizeof(unsigned), cudaMemcpyDeviceToHost) != cudaSuccess) return TERMEZO_ECUDA;
  if (err & tmz::ERR_TIMEOUT) return TERMEZO_ETIMEOUT;
  if (err & tmz::ERR_BOUNDS) {
    cudaMemsetAsync(c->ma.err, 0, sizeof(unsigned), c->stream);
    return TERMEZO_EINVAL;
  }
  return TERMEZO_OK;
}

int proj_of(const Shape& s, int layer, int j) { return 7 * layer + j; }

cudaEvent_t ev_get(termezo_ctx* c) {
  if (c->ev_used == c->ev_pool.size()) {
    cudaEvent_t e;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    c->ev_pool.push_back(e);
  }
  return c->ev_pool[c->ev_used++];
}

// Records CUDA events around the launches made during its lifetime when
// profiling is on.
struct ProfScope {
  termezo_ctx* c;
  int cat;
  double work;
  cudaEvent_t a = nullptr;
  ProfScope(termezo_ctx* ctx, int category, double w) : c(ctx), cat(category), work(w) {
    // every prof_stride-th launch of each category (a stride prime to the
    // four GEMMs of a layer and the five sparse passes of a step samples
    // every kind in turn)
    if (c->prof_on && c->prof_seq[category]++ % c->prof_stride == 0 && (a = ev_get(c))) cudaEventRecord(a, c->stream);
  }
  ~ProfScope() {
    if (!a) return;
    cudaEvent_t b = ev_get(c);
    if (!b) return;
    cudaEventRecord(b, c->stream);
    c->prof.push_back({cat, a, b, work});
  }
};

double gemm_flops(const GemmPlan& p) { return 2.0 * p.M * (double)p.N * p.K; }

// BitNet forward at the codes now in the packed store, with weight scales
// sw[] (one per projection); writes per_seq[slot*B ..] and loss[slot].
int run_forward(termezo_ctx* c, const int32_t* tokens, const int32_t* targets, const float* sw, int slot) {
  const Shape& s = c->sh;
  cudaStream_t st = c->stream;
  const int T = s.T, D = s.D, F = s.F, hq = s.H * s.hd, hkv = s.KV * s.hd;
  tmz::launch_embed(tokens, c->embed, T, D, s.V, c->x, c->ma.err, st);
  // Projection group g of layer l (0 q,k,v; 1 o; 2 gate,up; 3 down) is
  // expanded to e4m3 on the side stream into buffer g % 2 while the GEMM of
  // the group before it runs; the GEMM waits for its weights, and the next
  // expansion into a buffer waits for the GEMM that read it last.  With the
  // weight cache the GEMMs read the cached codes and nothing is expanded.
  const bool cached = c->wbyte != nullptr;
  uint8_t* wbuf[2] = {c->wexp, c->wexp2};
  // termezo_forward_trace copies (stream-ordered, between the kernels)
  const termezo_layer_trace* tr = c->trace;
  auto tr_copy = [&](void* dst, const void* src, size_t bytes) {
    if (dst) cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDeviceToDevice, st);
  };
  auto tr_codes = [&](int8_t* codes, float* deq, int K) {
    if (codes) tmz::launch_codes_i8(c->xq, T, K, codes, st);
    tr_copy(deq, c->deq, (size_t)T * sizeof(float));
  };
  cudaStream_t xs = c->xstream;
  auto expand = [&](int l, int g) {
    const int b = g & 1;
    cudaStreamWaitEvent(xs, c->ev_free[b], 0);
    const uint32_t* pk = c->ma.packed;
    if (g == 0)
      tmz::launch_expand_codes(pk + s.base[proj_of(s, l, 0)] / 16, (uint64_t)(hq + 2 * hkv), D, wbuf[b], xs);
    else if (g == 1)
      tmz::launch_expand_codes(pk + s.base[proj_of(s, l, 3)] / 16, (uint64_t)D, hq, wbuf[b], xs);
    else if (g == 2)
      tmz::launch_expand_gate_up(pk + s.base[proj_of(s, l, 4)] / 16, pk + s.base[proj_of(s, l, 5)] / 16, F, D,
                                 wbuf[b], xs);
    else
      tmz::launch_expand_codes(pk + s.base[proj_of(s, l, 6)] / 16, (uint64_t)D, F, wbuf[b], xs);
    cudaEventRecord(c->ev_ready[b], xs);
  };
  auto plan_of = [&](int l, int g) -> const GemmPlan& {
    if (cached) return c->cplan[(size_t)4 * l + g];
    return g == 0 ? c->plan_qkv : g == 1 ? c->plan_o : g == 2 ? c->plan_gu : c->plan_down;
  };
  auto gemm = [&](int l, int g, GemmArgs a, double flops) -> bool {
    const GemmPlan& plan = plan_of(l, g);
    a.split_ws = c->split_ws;
    a.split_cnt = c->split_cnt;
    a.split_cap = c->split_cap;
    if (!cached) cudaStreamWaitEvent(st, c->ev_ready[g & 1], 0);
    {
      ProfScope ps(c, 0, flops > 0 ? flops : gemm_flops(plan));
      if (tmz::gemm_launch(plan, a, st) != cudaSuccess) return false;
    }
    if (cached) return true;
    cudaEventRecord(c->ev_free[g & 1], st);
    const int nl = g == 3 ? l + 1 : l, ng = (g + 1) & 3;
    if (nl < s.L) expand(nl, ng);
    return true;
  };
  if (!cached) {
    cudaEventRecord(c->ev_codes, st);
    cudaStreamWaitEvent(xs, c->ev_codes, 0);
    expand(0, 0);
  }
  for (int l = 0; l < s.L; ++l) {
    const int pq = proj_of(s, l, 0), po = proj_of(s, l, 3), pg = proj_of(s, l, 4), pd = proj_of(s, l, 6);
    const termezo_layer_trace* lt = (tr && c->trace_layer == l) ? tr : nullptr;
    // attention block
    if (lt) tr_copy(lt->x_in, c->x, (size_t)T * D * sizeof(float));
    tmz::launch_norm_quant(c->x, c->gains + (size_t)(2 * l) * D, T, D, c->xq, c->deq, st);
    if (lt) tr_codes(lt->codes_attn, lt->deq_attn, D);
    GemmArgs a{};
    a.out = c->qkv;
    a.ldo = hq + 2 * hkv;
    a.mode = 0;
    a.deq = c->deq;
    a.sw = sw + pq;
    a.n1 = hq;
    a.n2 = hq + hkv;
    a.err = c->ma.err;
    const bool rope = plan_of(l, 0).rope != 0;
    if (rope) {
      a.rope = 1;
      a.cosb = c->cosb;
      a.sinb = c->sinb;
      a.vt = c->vt;
      a.S = s.S;
      a.H = s.H;
      a.KV = s.KV;
      a.hd = s.hd;
    }
    if (!gemm(l, 0, a, 0.0)) return TERMEZO_ECUDA;
    if (!rope)
      tmz::launch_rope_pack(c->qkv, c->cosb, c->sinb, s.B, s.S, s.H, s.KV, s.hd, c->qb, c->kb, c->vt, st);
    if (lt) {
      tr_copy(lt->q, c->qb, (size_t)T * hq * sizeof(uint16_t));
      tr_copy(lt->k, c->kb, (size_t)T * hkv * sizeof(uint16_t));
      tr_copy(lt->vt, c->vt, (size_t)T * hkv * sizeof(uint16_t));
    }
    a.rope = 0;  // the remaining projections of the layer reuse a
    {
      ProfScope ps(c, 1, 4.0 * s.B * s.H * (double)s.hd * (0.5 * s.S * (s.S + 1.0)));
      if (c->att_tc) {
        if (tmz::attention_tc_launch(c->att_plan, s.B, s.S, s.H, s.KV, s.hd, c->ma.err, st) != cudaSuccess)
          return TERMEZO_ECUDA;
      } else {
        tmz::launch_attention(c->qb, c->kb, c->vt, s.B, s.S, s.H, s.KV, s.hd, c->attn, st);
      }
    }
    if (lt) tr_copy(lt->attn, c->attn, (size_t)T * hq * sizeof(float));
    tmz::launch_norm_quant(c->attn, nullptr, T, hq, c->xq, c->deq, st);
    if (lt) tr_codes(lt->codes_o, lt->deq_o, hq);
    a.out = c->x;
    a.ldo = D;
    a.mode = 1;
    a.sw = sw + po;
    a.n1 = a.n2 = D;
    if (!gemm(l, 1, a, 0.0)) return TERMEZO_ECUDA;
    // MLP block
    if (lt) tr_copy(lt->x_mid, c->x, (size_t)T * D * sizeof(float));
    tmz::launch_norm_quant(c->x, c->gains + (size_t)(2 * l + 1) * D, T, D, c->xq, c->deq, st);
    if (lt) tr_codes(lt->codes_mlp, lt->deq_mlp, D);
    a.out = c->gu;  // hid = relu(gate)^2 * up, fp32 [T, F]
    a.ldo = F;
    a.mode = 0;
    a.sw = sw + pg;
    a.n1 = a.n2 = a.N;
    a.relu2 = 1;
    a.n_out = F;
    if (!gemm(l, 2, a, 2.0 * T * (2.0 * F) * D)) return TERMEZO_ECUDA;
    a.relu2 = 0;
    if (lt) tr_copy(lt->hid, c->gu, (size_t)T * F * sizeof(float));
    tmz::launch_norm_quant(c->gu, nullptr, T, F, c->xq, c->deq, st);
    if (lt) tr_codes(lt->codes_down, lt->deq_down, F);
    a.out = c->x;
    a.ldo = D;
    a.mode = 1;
    a.sw = sw + pd;
    a.n1 = a.n2 = D;
    if (!gemm(l, 3, a, 0.0)) return TERMEZO_ECUDA;
    if (lt) tr_copy(lt->x_out, c->x, (size_t)T * D * sizeof(float));
  }
  if (tr && c->trace_layer == s.L) tr_copy(tr->x_in, c->x, (size_t)T * D * sizeof(float));
  if (s.mode == 0) {
    tmz::launch_head_ce_last(c->x, c->gains + (size_t)(2 * s.L) * D, c->head, targets, s.B, s.S, D, s.V, s.C,
                             c->per_seq + (size_t)slot * s.B, c->loss + slot, st);
  } else {
    if (!c->head_plan_ok) return TERMEZO_ESTATE;
    tmz::launch_final_norm_bf16(c->x, c->gains + (size_t)(2 * s.L) * D, T, D, c->hfin, st);
    GemmArgs h{};
    h.lse = 1;
    h.part = c->part;
    h.tlogit = c->tlogit;
    h.target = targets;
    h.sw = sw;  // unused by the cross-entropy epilogue
    h.err = c->ma.err;
    {
      ProfScope ps(c, 0, gemm_flops(c->plan_head));
      if (tmz::gemm_launch(c->plan_head, h, st) != cudaSuccess) return TERMEZO_ECUDA;
    }
    tmz::launch_ce_reduce(c->part, tmz::gemm_col_tiles(s.V), c->tlogit, targets, s.B, s.S, s.V, c->tok_loss,
                          c->per_seq + (size_t)slot * s.B, c->loss + slot, c->ma.err, st);
  }
  return cuda_status(c);
}

// The z buffer holds the z of `seed` in the current store order (written by
// the perturbation sums of that seed since the last shrink or update).
bool z_ready(const termezo_ctx* c, uint64_t seed) {
  return c->ma.zbuf && c->pm_valid && c->pm_seed == seed;
}

void ensure_pm(termezo_ctx* c, uint64_t seed, float eps) {
  if (c->pm_valid && c->pm_seed == seed && c->pm_eps == eps) return;
  tmz::sparse_pm_taus(c->ma, c->cur, seed, eps, c->stream);
  c->pm_seed = seed;
  c->pm_eps = eps;
  c->pm_valid = true;
}

// Splits each projection's segment of the sparse store (off[p] .. off[p+1])
// into ceil(count / SPARSE_CHUNK) blocks, at least one, and uploads that plan
// (spre, sproj) for the sparse kernels, which split each segment evenly over
// its blocks from the offsets on the device.  The mask only shrinks, so a plan
// made from earlier counts keeps every block at most SPARSE_CHUNK long; the
// step re-plans after each read-back so that the blocks stay full as the
// active set shrinks.  Every per-block result (exact sums, counts, the words
// rewritten by their leaders) is independent of the partition.
int plan_sparse_blocks(termezo_ctx* c, const uint32_t* off) {
  const int P = c->sh.P;
  std::vector<uint32_t>& spre = c->spre_host;
  spre.assign(P + 1, 0);
  for (int p = 0; p < P; ++p) {
    const uint32_t cnt = off[p + 1] - off[p];
    const uint32_t nb = (cnt + SPARSE_CHUNK - 1) / SPARSE_CHUNK;
    spre[p + 1] = spre[p] + (nb ? nb : 1);
  }
  if (spre[P] > c->NBS_max) return TERMEZO_ECUDA;
  c->ma.NBS = spre[P];
  c->sproj_host.resize(spre[P]);
  for (int p = 0; p < P; ++p)
    for (uint32_t b = spre[p]; b < spre[p + 1]; ++b) c->sproj_host[b] = (uint16_t)p;
  cudaMemcpyAsync((void*)c->ma.spre, spre.data(), (P + 1) * sizeof(uint32_t), cudaMemcpyHostToDevice, c->stream);
  cudaMemcpyAsync((void*)c->ma.sproj, c->sproj_host.data(), spre[P] * sizeof(uint16_t), cudaMemcpyHostToDevice,
                  c->stream);
  return cuda_status(c);
}

int do_shrink(termezo_ctx* c) {
  ProfScope ps(c, 2 + PASS_SHRINK, 3.0 * 8.0 * (double)c->k_active);
  tmz::sparse_shrink(c->ma, c->cur, c->d_total, c->stream);
  c->cur ^= 1;
  c->pm_valid = false;
  return cuda_status(c);
}

}  // namespace

extern "C" {

int termezo_workspace_bytes(const termezo_model_cfg* cfg, double density, size_t* bytes) {
  if (!bytes || !(density > 0.0 && density <= 1.0)) return TERMEZO_EINVAL;
  termezo_ctx tmp;
  int rc = make_shape(cfg, &tmp.sh);
  if (rc) return rc;
  plan_sizes(&tmp, density);
  Carver cv{nullptr};
  carve(&tmp, cv);
  *bytes = cv.off + 256;
  return TERMEZO_OK;
}

int termezo_memory(const termezo_model_cfg* cfg, double density, termezo_memory_out* out) {
  if (!out || !(density > 0.0 && density <= 1.0)) return TERMEZO_EINVAL;
  termezo_ctx tmp;
  int rc = make_shape(cfg, &tmp.sh);
  if (rc) return rc;
  plan_sizes(&tmp, density);
  Carver cv{nullptr};
  carve(&tmp, cv);
  const Shape& s = tmp.sh;
  out->d = s.d;
  out->k_cap = tmp.k_cap;
  out->packed = cv.bytes[SEC_PACKED];
  out->sparse_index = cv.bytes[SEC_INDEX];
  out->sparse_latents = cv.bytes[SEC_LATENTS];
  out->mask_state = cv.bytes[SEC_MASK];
  out->forward = cv.bytes[SEC_FORWARD];
  out->weight_cache = cv.bytes[SEC_WCACHE];
  out->z_cache = cv.bytes[SEC_ZCACHE];
  out->workspace = cv.off + 256;
  out->theta = s.op ? 0
                    : (uint64_t)s.V * s.D * 4 + (uint64_t)(2 * s.L + 1) * s.D * 4 + (uint64_t)s.V * s.D * 2;
  uint64_t lg = 0;
  while ((1ull << lg) < s.d) ++lg;
  const uint64_t k0 = keep_count(density, s.d);
  out->mask_bitmask = (s.d + 7) / 8;
  out->mask_index_list = (k0 * lg + 7) / 8;
  return TERMEZO_OK;
}

int termezo_create(const termezo_model_cfg* cfg, double density, void* d_workspace, size_t bytes, void* stream,
                   termezo_ctx** out) {
  if (!out || !d_workspace || !(density > 0.0 && density <= 1.0)) return TERMEZO_EINVAL;
  if ((uintptr_t)d_workspace & 255) return TERMEZO_EINVAL;
  *out = nullptr;
  termezo_ctx* c = new (std::nothrow) termezo_ctx();
  if (!c) return TERMEZO_ENOMEM;
  int rc = make_shape(cfg, &c->sh);
  if (rc) {
    delete c;
    return rc;
  }
  plan_sizes(c, density);
  Carver cv{reinterpret_cast<uint8_t*>(d_workspace)};
  carve(c, cv);
  if (cv.off > bytes) {
    delete c;
    return TERMEZO_ENOMEM;
  }
  c->stream = reinterpret_cast<cudaStream_t>(stream);
  const Shape& s = c->sh;
  c->ma.NBD = c->dpre.back();
  cudaStream_t st = c->stream;
  cudaMemcpyAsync((void*)c->ma.base, s.base.data(), (s.P + 1) * sizeof(uint64_t), cudaMemcpyHostToDevice, st);
  cudaMemcpyAsync((void*)c->ma.dpre, c->dpre.data(), (s.P + 1) * sizeof(uint32_t), cudaMemcpyHostToDevice, st);
  {
    std::vector<uint16_t> dproj(c->dpre.back());
    for (int p = 0; p < s.P; ++p)
      for (uint32_t b = c->dpre[p]; b < c->dpre[p + 1]; ++b) dproj[b] = (uint16_t)p;
    cudaMemcpy((void*)c->ma.dproj, dproj.data(), dproj.size() * sizeof(uint16_t), cudaMemcpyHostToDevice);
  }
  cudaMemsetAsync(c->ma.err, 0, sizeof(unsigned), st);
  cudaMemsetAsync(c->split_cnt, 0, (size_t)c->split_cap * 4 * sizeof(unsigned), st);
  cudaMemsetAsync(c->ma.counters, 0, 8 * sizeof(unsigned long long), st);
  for (float* f : {c->ma.gamma_cur, c->ma.tau_cur, c->ma.sw_cur, c->ma.gamma_plus, c->ma.tau_plus, c->ma.sw_plus,
                   c->ma.gamma_minus, c->ma.tau_minus, c->ma.sw_minus})
    cudaMemsetAsync(f, 0, (s.P + 2) * sizeof(float), st);
  if (tmz::mask_preload() != cudaSuccess) {
    delete c;
    return TERMEZO_ECUDA;
  }
  if (!s.op) {
    tmz::launch_rope_tables(s.S, s.hd, c->cosb, c->sinb, st);
    const int T = s.T, D = s.D, F = s.F, hq = s.H * s.hd, hkv = s.KV * s.hd;
    const bool rope_fused = rope_fused_shape(s);
    // the expansion buffers' plans, or (weight cache) every layer's own
    bool ok = s.wcache ||
              (tmz::gemm_make_plan_f8(&c->plan_qkv, c->xq, T, D, c->wexp, hq + 2 * hkv, !rope_fused) &&
               tmz::gemm_make_plan_f8(&c->plan_o, c->xq, T, hq, c->wexp2, D, true) &&
               tmz::gemm_make_plan_f8(&c->plan_gu, c->xq, T, D, c->wexp, 256 * ((F + 127) / 128), false) &&
               tmz::gemm_make_plan_f8(&c->plan_down, c->xq, T, F, c->wexp2, D, true));
    if (s.wcache) {
      c->cplan.resize((size_t)4 * s.L);
      for (int l = 0; l < s.L && ok; ++l) {
        GemmPlan* p = &c->cplan[(size_t)4 * l];
        const uint8_t* w = c->wbyte;
        ok = tmz::gemm_make_plan_f8(&p[0], c->xq, T, D, w + s.base[proj_of(s, l, 0)], hq + 2 * hkv, !rope_fused) &&
             tmz::gemm_make_plan_f8(&p[1], c->xq, T, hq, w + s.base[proj_of(s, l, 3)], D, true) &&
             tmz::gemm_make_plan_f8_gu(&p[2], c->xq, T, D, w + s.base[proj_of(s, l, 4)], w + s.base[proj_of(s, l, 5)],
                                       F) &&
             tmz::gemm_make_plan_f8(&p[3], c->xq, T, F, w + s.base[proj_of(s, l, 6)], D, true);
      }
    }
    ok = ok && cudaStreamCreateWithFlags(&c->xstream, cudaStreamNonBlocking) == cudaSuccess;
    for (cudaEvent_t* e : {&c->ev_free[0], &c->ev_free[1], &c->ev_ready[0], &c->ev_ready[1], &c->ev_codes})
      ok = ok && cudaEventCreateWithFlags(e, cudaEventDisableTiming) == cudaSuccess;
    if (!ok) {
      delete c;
      return TERMEZO_ECUDA;
    }
    // TMA output maps (a layout that does not allow one keeps the plain stores)
    // q, k, v written by the QKV GEMM's epilogue (RoPE fused) where the head
    // layout allows it
    const int n_sets = s.wcache ? s.L : 1;
    for (int l = 0; l < n_sets; ++l) {
      GemmPlan *pq = s.wcache ? &c->cplan[(size_t)4 * l] : &c->plan_qkv,
               *po = s.wcache ? pq + 1 : &c->plan_o, *pd = s.wcache ? pq + 3 : &c->plan_down;
      if (rope_fused) {
        // the workspace has no fp32 QKV buffer for these shapes
        if (!tmz::gemm_plan_rope(pq, c->qb, c->kb, s.B, s.S, s.H, s.KV, s.hd)) {
          delete c;
          return TERMEZO_ECUDA;
        }
      } else {
        tmz::gemm_plan_output(pq, c->qkv, hq + 2 * hkv);
      }
      tmz::gemm_plan_output(po, c->x, D);
      tmz::gemm_plan_output(pd, c->x, D);
    }
    c->att_tc = tmz::attention_tc_supported(s.S, s.hd) &&
                tmz::attention_tc_plan(&c->att_plan, c->qb, c->kb, c->vt, c->attn, s.B, s.S, s.H, s.KV, s.hd);
  }
  c->code_sw = c->ma.sw_cur;
  rc = sync_status(c);
  if (rc) {
    delete c;
    return rc;
  }
  *out = c;
  return TERMEZO_OK;
}

int termezo_load_params(termezo_ctx* c, const float* d_latents, const float* d_embed, const float* d_gains,
                        const uint16_t* d_head) {
  if (!c || !d_latents) return TERMEZO_EINVAL;
  if (!c->sh.op && (!d_embed || !d_gains || !d_head)) return TERMEZO_EINVAL;
  if ((uintptr_t)d_latents & 15) return TERMEZO_EINVAL;
  c->latents = d_latents;
  c->embed = d_embed;
  c->gains = d_gains;
  c->head = d_head;
  if (!c->sh.op && c->sh.mode == 1) {
    c->head_plan_ok = tmz::gemm_make_plan(&c->plan_head, c->hfin, c->sh.T, c->sh.D, d_head, c->sh.V, false);
    if (!c->head_plan_ok) return TERMEZO_EINVAL;  // head must be 16-byte aligned
  }
  return TERMEZO_OK;
}

int termezo_build_mask(termezo_ctx* c, double density, uint64_t* k0_out, float* xi0_out) {
  return termezo_build_mask_rule(c, density, TERMEZO_MASK_GLOBAL, k0_out, xi0_out);
}

int termezo_build_mask_rule(termezo_ctx* c, double density, int32_t rule, uint64_t* k0_out, float* xi0_out) {
  if (!c) return TERMEZO_EINVAL;
  if (!c->latents) return TERMEZO_ESTATE;
  if (!(density > 0.0 && density <= 1.0)) return TERMEZO_EINVAL;
  if (rule != TERMEZO_MASK_GLOBAL && rule != TERMEZO_MASK_PER_TENSOR) return TERMEZO_EINVAL;
  const Shape& s = c->sh;
  // one selection group for the global quantile, one per projection else
  std::vector<tmz::SelectState> groups;
  uint64_t k0 = 0;
  if (rule == TERMEZO_MASK_GLOBAL) {
    k0 = keep_count(density, s.d);
    groups.push_back(tmz::SelectState{k0, 0u, 0u});
  } else {
    for (int p = 0; p < s.P; ++p) {
      const uint64_t kp = keep_count(density, s.base[p + 1] - s.base[p]);
      groups.push_back(tmz::SelectState{kp, 0u, 0u});
      k0 += kp;
    }
  }
  if (k0 > keep_count(c->density, s.d)) return TERMEZO_EINVAL;
  cudaStream_t st = c->stream;
  c->ma.groups = (int)groups.size();
  std::vector<tmz::SelectState> sel_h = groups;
  cudaMemcpyAsync(c->ma.sel, sel_h.data(), groups.size() * sizeof(tmz::SelectState), cudaMemcpyHostToDevice, st);
  int rc = TERMEZO_OK;
  bool built_fast = false;
  if (rule == TERMEZO_MASK_GLOBAL && k0 > 0) {
    // two dense passes and a sampled one (tmz::mask_build_fast); the six-pass
    // build when the superset of S_0 misses k0 or does not fit its buffer
    cudaMemsetAsync(c->ma.hist, 0, 8192 * sizeof(unsigned long long), st);
    cudaMemsetAsync(c->ma.sup, 0, 4 * sizeof(uint32_t), st);
    cudaMemsetAsync(c->ma.scan_state, 0, (size_t)c->ma.NBD * sizeof(unsigned long long), st);
    tmz::mask_build_fast(c->ma, c->latents, k0, st);
    uint32_t sup[4] = {0, 0, 0, 0};
    cudaMemcpyAsync(sup, c->ma.sup, sizeof(sup), cudaMemcpyDeviceToHost, st);
    rc = sync_status(c);
    if (rc) return rc;
    if (!sup[1]) {
      tmz::mask_build_fast_offsets(c->ma, k0, st);
      built_fast = true;
    } else {
      cudaMemcpyAsync(c->ma.sel, sel_h.data(), groups.size() * sizeof(tmz::SelectState), cudaMemcpyHostToDevice,
                      st);
    }
  }
  if (!built_fast) {
    cudaMemsetAsync(c->ma.hist, 0, groups.size() * 2048 * sizeof(unsigned long long), st);
    tmz::mask_build(c->ma, c->latents, k0, st);
  }
  rc = cuda_status(c);
  if (rc) return rc;
  std::vector<uint32_t> off(s.P + 1);
  std::vector<float> xi0p(s.P);
  cudaMemcpyAsync(off.data(), c->ma.off[0], (s.P + 1) * sizeof(uint32_t), cudaMemcpyDeviceToHost, st);
  cudaMemcpyAsync(xi0p.data(), c->ma.xi0p, s.P * sizeof(float), cudaMemcpyDeviceToHost, st);
  rc = sync_status(c);
  if (rc) return rc;
  if (off[s.P] != k0) {
    fprintf(stderr, "termezo: mask build selected %u weights, expected %llu\n", off[s.P], (unsigned long long)k0);
    return TERMEZO_ECUDA;
  }
  rc = plan_sparse_blocks(c, off.data());
  if (rc) return rc;
  tmz::mask_finish(c->ma, st);
  c->cur = 0;
  c->k0 = k0;
  c->k_active = k0;
  c->xi0 = rule == TERMEZO_MASK_GLOBAL ? xi0p[0] : 0.f;
  c->t = 0;
  c->updated = false;
  c->pm_valid = false;
  c->code_sw = c->ma.sw_cur;
  rc = sync_status(c);
  if (rc) return rc;
  c->built = true;
  // the dense latents are not read again: the caller may release them
  c->latents = nullptr;
  if (k0_out) *k0_out = k0;
  if (xi0_out) {
    if (rule == TERMEZO_MASK_GLOBAL)
      *xi0_out = xi0p[0];
    else
      for (int p = 0; p < s.P; ++p) xi0_out[p] = xi0p[p];
  }
  return TERMEZO_OK;
}

int termezo_forward_loss(termezo_ctx* c, const int32_t* d_tokens, const int32_t* d_targets, double* loss,
                         double* per_seq) {
  if (!c || !d_tokens || !d_targets) return TERMEZO_EINVAL;
  if (c->sh.op || !c->built) return TERMEZO_ESTATE;
  tmz::sparse_requant(c->ma, c->cur, 0, 0.f, 0, false, c->stream);
  c->code_sw = c->ma.sw_cur;
  int rc = run_forward(c, d_tokens, d_targets, c->ma.sw_cur, 0);
  if (rc) return rc;
  double l = 0;
  cudaMemcpyAsync(&l, c->loss, sizeof(double), cudaMemcpyDeviceToHost, c->stream);
  if (per_seq)
    cudaMemcpyAsync(per_seq, c->per_seq, c->sh.B * sizeof(double), cudaMemcpyDeviceToHost, c->stream);
  rc = sync_status(c);
  if (rc) return rc;
  if (loss) *loss = l;
  return TERMEZO_OK;
}

int termezo_forward_trace(termezo_ctx* c, const int32_t* d_tokens, const int32_t* d_targets, int32_t layer,
                          const termezo_layer_trace* trace, double* loss, double* per_seq) {
  if (!c || !d_tokens || !d_targets || !trace) return TERMEZO_EINVAL;
  if (c->sh.op || !c->built) return TERMEZO_ESTATE;
  if (layer < 0 || layer > c->sh.L) return TERMEZO_EINVAL;
  c->trace = trace;
  c->trace_layer = layer;
  int rc = run_forward(c, d_tokens, d_targets, c->code_sw, 0);
  c->trace = nullptr;
  c->trace_layer = -1;
  if (rc) return rc;
  double l = 0;
  cudaMemcpyAsync(&l, c->loss, sizeof(double), cudaMemcpyDeviceToHost, c->stream);
  if (per_seq)
    cudaMemcpyAsync(per_seq, c->per_seq, c->sh.B * sizeof(double), cudaMemcpyDeviceToHost, c->stream);
  rc = sync_status(c);
  if (rc) return rc;
  if (loss) *loss = l;
  return TERMEZO_OK;
}

namespace {

// Algorithm 1's loop body with K directions: shrink (t >= 1); for each
// direction k: pm taus, requantise at +eps z_k, forward, requantise at
// -eps z_k, forward, g_k, and (k < K-1) restore; then the last restore and
// the K-term update in one pass.
int step_impl(termezo_ctx* c, const uint64_t* seeds, int K, float eps, float lr, double density,
              const int32_t* d_tokens, const int32_t* d_targets, termezo_step_out* out, double* losses, double* gs,
              double* per_seq_plus, double* per_seq_minus, bool theta) {
  if (!c || !seeds || !d_tokens || !d_targets || !out) return TERMEZO_EINVAL;
  if (K < 1 || K > tmz::KMAX) return TERMEZO_EINVAL;
  if (c->sh.op || !c->built) return TERMEZO_ESTATE;
  tmz::ThetaArgs th{};
  if (theta) {
    // theta is updated in place in the caller's buffers of termezo_load_params
    const Shape& s = c->sh;
    if (!c->embed || !c->gains || !c->head || s.D % 4 || ((uintptr_t)c->embed & 15) || ((uintptr_t)c->gains & 15) ||
        ((uintptr_t)c->head & 7) || s.d % 4)
      return TERMEZO_EINVAL;
    th.emb = const_cast<float*>(c->embed);
    th.n_emb = (uint64_t)s.V * s.D;
    th.gains = const_cast<float*>(c->gains);
    th.n_gains = (uint64_t)(2 * s.L + 1) * s.D;
    th.head = const_cast<uint16_t*>(c->head);
    th.n_head = (uint64_t)s.V * s.D;
    th.d = s.d;
  }
  const double theta8 = theta ? 2.0 * (4.0 * (th.n_emb + th.n_gains) + 2.0 * th.n_head) : 0.0;
  if (!(eps > 0.f) || !std::isfinite(lr)) return TERMEZO_EINVAL;
  const int warn = (density != c->density) ? TERMEZO_WMASKFIXED : TERMEZO_OK;
  cudaStream_t st = c->stream;
  cudaMemsetAsync(c->ma.counters, 0, 3 * sizeof(unsigned long long), st);
  cudaMemsetAsync(c->ma.counters + 4, 0, sizeof(unsigned long long), st);
  int rc;
  if (c->updated) {
    rc = do_shrink(c);
    if (rc) return rc;
  }
  c->pm_valid = false;
  const double k8 = 8.0 * (double)c->k_active;
  tmz::UpdateDirs dirs{};
  dirs.K = K;
  for (int k = 0; k < K; ++k) {
    const uint64_t seed = seeds[k];
    dirs.seed[k] = seed;
    {
      ProfScope ps(c, 2 + PASS_PM, k8);
      ensure_pm(c, seed, eps);
    }
    {
      ProfScope ps(c, 2 + PASS_REQUANT, k8);
      tmz::sparse_requant(c->ma, c->cur, seed, eps, +1, z_ready(c, seed), st);
    }
    if (theta) {
      ProfScope ps(c, 2 + PASS_THETA, theta8);
      tmz::theta_pm(th, seed, eps, 0, st);
    }
    rc = run_forward(c, d_tokens, d_targets, c->ma.sw_plus, 0);
    if (rc) return rc;
    {
      ProfScope ps(c, 2 + PASS_REQUANT, k8);
      tmz::sparse_requant(c->ma, c->cur, seed, eps, -1, z_ready(c, seed), st);
    }
    if (theta) {
      ProfScope ps(c, 2 + PASS_THETA, theta8);
      tmz::theta_pm(th, seed, eps, 1, st);
    }
    rc = run_forward(c, d_tokens, d_targets, c->ma.sw_minus, 1);
    if (rc) return rc;
    c->code_sw = c->ma.sw_minus;
    tmz::launch_grad(c->loss, eps, c->g + k, st);
    if (K > 1) cudaMemcpyAsync(c->lossk + 2 * k, c->loss, 2 * sizeof(double), cudaMemcpyDeviceToDevice, st);
    if (k + 1 < K) {
      ProfScope ps(c, 2 + PASS_UPDATE, 1.5 * k8);
      tmz::sparse_restore(c->ma, c->cur, seed, eps, z_ready(c, seed), st);
      c->pm_valid = false;
      if (theta) tmz::theta_pm(th, seed, eps, 0, st);
    }
  }
  dirs.last = seeds[K - 1];
  {
    ProfScope ps(c, 2 + PASS_UPDATE, 1.5 * k8);
    tmz::sparse_update_dirs(c->ma, c->cur, dirs, eps, lr, c->g, z_ready(c, dirs.last), st);
  }
  if (theta) {
    ProfScope ps(c, 2 + PASS_THETA, theta8);
    tmz::theta_update(th, dirs, eps, lr, c->g, st);
  }
  c->pm_valid = false;
  struct {
    double loss[2 * tmz::KMAX];
    double g[tmz::KMAX];
    unsigned long long cnt[5];
    uint32_t k;
  } h{};
  cudaMemcpyAsync(h.loss, K > 1 ? c->lossk : c->loss, 2 * K * sizeof(double), cudaMemcpyDeviceToHost, st);
  cudaMemcpyAsync(h.g, c->g, K * sizeof(double), cudaMemcpyDeviceToHost, st);
  cudaMemcpyAsync(h.cnt, c->ma.counters, 5 * sizeof(unsigned long long), cudaMemcpyDeviceToHost, st);
  c->off_host.resize(c->sh.P + 1);
  cudaMemcpyAsync(c->off_host.data(), c->ma.off[c->cur], (c->sh.P + 1) * sizeof(uint32_t), cudaMemcpyDeviceToHost,
                  st);
  if (per_seq_plus)
    cudaMemcpyAsync(per_seq_plus, c->per_seq, c->sh.B * sizeof(double), cudaMemcpyDeviceToHost, st);
  if (per_seq_minus)
    cudaMemcpyAsync(per_seq_minus, c->per_seq + c->sh.B, c->sh.B * sizeof(double), cudaMemcpyDeviceToHost, st);
  rc = sync_status(c);
  if (rc) return rc;
  h.k = c->off_host[c->sh.P];
  rc = plan_sparse_blocks(c, c->off_host.data());
  if (rc) return rc;
  c->updated = true;
  c->t += 1;
  c->k_active = h.k;
  out->loss_plus = h.loss[2 * (K - 1)];
  out->loss_minus = h.loss[2 * (K - 1) + 1];
  out->g = h.g[K - 1];
  out->k_active = h.k;
  out->n_flipped = h.cnt[0];
  out->n_jumps = h.cnt[1];
  out->n_dropped = h.cnt[2];
  out->n_near_threshold = h.cnt[4];
  if (losses)
    for (int i = 0; i < 2 * K; ++i) losses[i] = h.loss[i];
  if (gs)
    for (int k = 0; k < K; ++k) gs[k] = h.g[k];
  return warn;
}

}  // namespace

int termezo_step(termezo_ctx* c, uint64_t seed, float eps, float lr, double density, const int32_t* d_tokens,
                 const int32_t* d_targets, termezo_step_out* out, double* per_seq_plus, double* per_seq_minus) {
  return step_impl(c, &seed, 1, eps, lr, density, d_tokens, d_targets, out, nullptr, nullptr, per_seq_plus,
                   per_seq_minus, false);
}

int termezo_step_k(termezo_ctx* c, const uint64_t* seeds, int32_t K, float eps, float lr, double density,
                   const int32_t* d_tokens, const int32_t* d_targets, termezo_step_out* out, double* losses,
                   double* g) {
  return step_impl(c, seeds, K, eps, lr, density, d_tokens, d_targets, out, losses, g, nullptr, nullptr, false);
}

int termezo_step_joint(termezo_ctx* c, const uint64_t* seeds, int32_t K, float eps, float lr, double density,
                       const int32_t* d_tokens, const int32_t* d_targets, termezo_step_out* out, double* losses,
                       double* g) {
  return step_impl(c, seeds, K, eps, lr, density, d_tokens, d_targets, out, losses, g, nullptr, nullptr, true);
}

int termezo_shrink(termezo_ctx* c, uint64_t* n_dropped) {
  if (!c) return TERMEZO_EINVAL;
  if (!c->built) return TERMEZO_ESTATE;
  if (!c->updated) {
    if (n_dropped) *n_dropped = 0;
    return TERMEZO_OK;
  }
  cudaMemsetAsync(c->ma.counters + 2, 0, sizeof(unsigned long long), c->stream);
  int rc = do_shrink(c);
  if (rc) return rc;
  c->updated = false;
  if (n_dropped) {
    unsigned long long d = 0;
    uint32_t k = 0;
    cudaMemcpyAsync(&d, c->ma.counters + 2, sizeof(d), cudaMemcpyDeviceToHost, c->stream);
    cudaMemcpyAsync(&k, c->ma.off[c->cur] + c->sh.P, sizeof(k), cudaMemcpyDeviceToHost, c->stream);
    rc = sync_status(c);
    if (rc) return rc;
    *n_dropped = d;
    c->k_active = k;
  }
  return TERMEZO_OK;
}

int termezo_requantize(termezo_ctx* c, uint64_t seed, float eps, int sign) {
  if (!c || sign < -1 || sign > 1) return TERMEZO_EINVAL;
  if (!c->built) return TERMEZO_ESTATE;
  if (sign != 0) {
    if (!(eps > 0.f)) return TERMEZO_EINVAL;
    ensure_pm(c, seed, eps);
  }
  tmz::sparse_requant(c->ma, c->cur, seed, eps, sign, sign != 0 && z_ready(c, seed), c->stream);
  c->code_sw = sign > 0 ? c->ma.sw_plus : (sign < 0 ? c->ma.sw_minus : c->ma.sw_cur);
  return cuda_status(c);
}

int termezo_update(termezo_ctx* c, uint64_t seed, float eps, float lr, double g) {
  if (!c) return TERMEZO_EINVAL;
  if (!c->built) return TERMEZO_ESTATE;
  if (!(eps > 0.f) || !std::isfinite(lr) || !std::isfinite(g)) return TERMEZO_EINVAL;
  tmz::sparse_update(c->ma, c->cur, seed, eps, lr, nullptr, g, 1, z_ready(c, seed), c->stream);
  c->updated = true;
  c->pm_valid = false;
  c->t += 1;
  return cuda_status(c);
}

int termezo_bitlinear(termezo_ctx* c, int32_t proj, const uint16_t* d_x, int32_t M, int32_t* d_acc, float* d_y) {
  if (!c || !d_x || proj < 0 || proj >= c->sh.P || M <= 0 || M > c->sh.T) return TERMEZO_EINVAL;
  if (!c->built) return TERMEZO_ESTATE;
  const int N = c->sh.N[proj], K = c->sh.K[proj];
  if ((size_t)K > xq_cols(c->sh) || (size_t)N * K > wexp_elems(c->sh)) return TERMEZO_EINVAL;
  cudaStream_t st = c->stream;
  tmz::launch_norm_quant_bf16(d_x, M, K, c->xq, c->deq, st);
  tmz::launch_expand_codes(c->ma.packed + c->sh.base[proj] / 16, (uint64_t)N, K, c->wexp, st);
  GemmPlan plan;
  if (!tmz::gemm_make_plan_f8(&plan, c->xq, M, K, c->wexp, N, true)) return TERMEZO_ECUDA;
  if (d_y) tmz::gemm_plan_output(&plan, d_y, N);
  GemmArgs a{};
  a.out = d_y;
  a.ldo = N;
  a.mode = 0;
  a.acc_out = d_acc;
  a.split_ws = c->split_ws;
  a.split_cnt = c->split_cnt;
  a.split_cap = c->split_cap;
  a.deq = c->deq;
  a.sw = c->code_sw + proj;
  a.n1 = a.n2 = N;
  a.err = c->ma.err;
  if (tmz::gemm_launch(plan, a, st) != cudaSuccess) return TERMEZO_ECUDA;
  return cuda_status(c);
}

int termezo_state_sizes(termezo_ctx* c, uint64_t* d, uint64_t* k_active, int32_t* n_proj) {
  if (!c) return TERMEZO_EINVAL;
  uint32_t k = 0;
  if (c->built) {
    cudaMemcpyAsync(&k, c->ma.off[c->cur] + c->sh.P, sizeof(k), cudaMemcpyDeviceToHost, c->stream);
    int rc = sync_status(c);
    if (rc) return rc;
  }
  if (d) *d = c->sh.d;
  if (k_active) *k_active = k;
  if (n_proj) *n_proj = c->sh.P;
  return TERMEZO_OK;
}

int termezo_export_state(termezo_ctx* c, uint32_t* h_idx, float* h_latents, uint32_t* h_packed, float* h_tau) {
  if (!c) return TERMEZO_EINVAL;
  if (!c->built) return TERMEZO_ESTATE;
  cudaStream_t st = c->stream;
  uint32_t k = 0;
  cudaMemcpyAsync(&k, c->ma.off[c->cur] + c->sh.P, sizeof(k), cudaMemcpyDeviceToHost, st);
  int rc = sync_status(c);
  if (rc) return rc;
  if (h_idx && k) cudaMemcpyAsync(h_idx, c->ma.idx[c->cur], k * sizeof(uint32_t), cudaMemcpyDeviceToHost, st);
  if (h_latents && k) cudaMemcpyAsync(h_latents, c->ma.lat[c->cur], k * sizeof(float), cudaMemcpyDeviceToHost, st);
  if (h_packed) cudaMemcpyAsync(h_packed, c->ma.packed, c->sh.d / 16 * sizeof(uint32_t), cudaMemcpyDeviceToHost, st);
  if (h_tau) {
    const int P = c->sh.P;
    cudaMemcpyAsync(h_tau, c->ma.tau_cur, P * sizeof(float), cudaMemcpyDeviceToHost, st);
    cudaMemcpyAsync(h_tau + P, c->ma.tau_plus, P * sizeof(float), cudaMemcpyDeviceToHost, st);
    cudaMemcpyAsync(h_tau + 2 * P, c->ma.tau_minus, P * sizeof(float), cudaMemcpyDeviceToHost, st);
  }
  return sync_status(c);
}

int termezo_normal(uint64_t seed, const uint32_t* d_idx, uint64_t n, float* d_z, void* stream) {
  if (n && (!d_idx || !d_z)) return TERMEZO_EINVAL;
  tmz::launch_normal(seed, d_idx, n, d_z, reinterpret_cast<cudaStream_t>(stream));
  return cudaGetLastError() == cudaSuccess ? TERMEZO_OK : TERMEZO_ECUDA;
}

int termezo_profile(termezo_ctx* c, int enable, termezo_profile_out* out) {
  if (!c || enable < -1 || enable > 1000) return TERMEZO_EINVAL;
  if (enable >= 1) {
    int rc = sync_status(c);
    if (rc) return rc;
    c->prof.clear();
    c->ev_used = 0;
    c->prof_stride = enable;
    for (auto& q : c->prof_seq) q = 0;
    c->launch_base = tmz::kernel_launches();
    cudaMemsetAsync(c->ma.counters + 3, 0, sizeof(unsigned long long), c->stream);
    c->prof_on = true;
  } else if (enable == 0) {
    c->prof_on = false;
  }
  if (out) {
    int rc = sync_status(c);
    if (rc) return rc;
    memset(out, 0, sizeof(*out));
    out->launches = tmz::kernel_launches() - c->launch_base;
    for (const auto& r : c->prof) {
      float ms = 0.f;
      if (cudaEventElapsedTime(&ms, r.a, r.b) != cudaSuccess) return TERMEZO_ECUDA;
      if (r.cat == 0) {
        out->gemm_launches++;
        out->gemm_ms += ms;
        out->gemm_flops += r.work;
      } else if (r.cat == 1) {
        out->attn_launches++;
        out->attn_ms += ms;
        out->attn_flops += r.work;
      } else {
        const int k = r.cat - 2;
        out->pass_launches[k]++;
        out->pass_ms[k] += ms;
        out->pass_bytes[k] += r.work;
      }
    }
    out->gemm_seen = c->prof_seq[0];
    out->attn_seen = c->prof_seq[1];
    for (int k = 0; k < TERMEZO_PASS_KINDS; ++k) out->pass_seen[k] = c->prof_seq[2 + k];
    // the 32-byte sectors of the packed store that the requantisations
    // rewrote (read and written), in the proportion of the timed passes
    unsigned long long sectors = 0;
    cudaMemcpy(&sectors, c->ma.counters + 3, sizeof(sectors), cudaMemcpyDeviceToHost);
    if (out->pass_seen[PASS_REQUANT])
      out->pass_bytes[PASS_REQUANT] += 64.0 * (double)sectors * (double)out->pass_launches[PASS_REQUANT] /
                                       (double)out->pass_seen[PASS_REQUANT];
    for (int k = 0; k < TERMEZO_PASS_KINDS; ++k) {
      out->sparse_launches += out->pass_launches[k];
      out->sparse_seen += out->pass_seen[k];
      out->sparse_ms += out->pass_ms[k];
      out->sparse_bytes += out->pass_bytes[k];
    }
  }
  return TERMEZO_OK;
}

int termezo_attention(const uint16_t* d_q, const uint16_t* d_k, const uint16_t* d_vt, int32_t B, int32_t S,
                      int32_t H, int32_t KV, int32_t hd, float* d_out, void* stream) {
  if (!d_q || !d_k || !d_vt || !d_out || B <= 0 || S <= 0 || S % 64 || H <= 0 || KV <= 0 || H % KV) return TERMEZO_EINVAL;
  if (hd != 64 && hd != 96 && hd != 128) return TERMEZO_EINVAL;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  tmz::AttnPlan plan;
  if (tmz::attention_tc_supported(S, hd) && tmz::attention_tc_plan(&plan, d_q, d_k, d_vt, d_out, B, S, H, KV, hd))
    return tmz::attention_tc_launch(plan, B, S, H, KV, hd, nullptr, st) == cudaSuccess ? TERMEZO_OK
                                                                                             : TERMEZO_ECUDA;
  tmz::launch_attention(d_q, d_k, d_vt, B, S, H, KV, hd, d_out, st);
  return cudaGetLastError() == cudaSuccess ? TERMEZO_OK : TERMEZO_ECUDA;
}

void termezo_destroy(termezo_ctx* c) { delete c; }

const char* termezo_strerror(int status) {
  switch (status) {
    case TERMEZO_OK: return "ok";
    case TERMEZO_WMASKFIXED: return "mask density is fixed after termezo_build_mask; the new value was ignored";
    case TERMEZO_EINVAL: return "invalid argument (shape, pointer, density or token id)";
    case TERMEZO_ESTATE: return "call out of order for this context";
    case TERMEZO_ENOMEM: return "workspace smaller than termezo_workspace_bytes";
    case TERMEZO_ECUDA: return "CUDA error";
    case TERMEZO_ETIMEOUT: return "a bounded device wait timed out";
    default: return "unknown status";
  }
}

}  // extern "C"
