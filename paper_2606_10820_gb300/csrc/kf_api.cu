// Host runtime behind the C ABI (include/kforcing.h): context and weight
// upload, the paged KV pool and its page allocator, chunked prefill, the
// decode step (Alg. 1 loop body) replayed as one CUDA graph per
// (batch, pending, k) shape, and per-kernel profiling.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <map>
#include <string>
#include <tuple>
#include <vector>

#include "kf_internal.cuh"

using namespace kf;

namespace kf {
thread_local bool g_pdl = false;
thread_local int g_gemm_flags = 0;
}

namespace kf {
void launch_convert_f32(bool bf16, const float* src, void* dst, size_t n, cudaStream_t s);
}

struct LayerW {
  void* wqkv;
  void* wo;
  void* w_up;
  void* w_down;
  const float* attn_norm;
  const float* mlp_norm;
};

struct kf_ctx {
  kf_config cfg{};
  int dev = 0;
  cudaStream_t stream = nullptr;
  bool own_stream = false;
  bool bf16 = false;
  size_t esz = 4;
  int d = 0, H = 0, hd = 64, L = 0, F = 0, V = 0, NH = 0, V_pad = 0, max_k = 1, num_sms = 148;
  std::vector<void*> allocs;
  // weights
  void* tok_emb = nullptr;
  float* pos_emb = nullptr;
  std::vector<LayerW> layers;
  float* final_norm = nullptr;
  void* w_head = nullptr;
  void* w_mtp = nullptr;        // [mtp_k][V_pad][d] MTP heads (mtp_k > 0)
  int mtp_k = 0;
  bool last_mtp = false;        // the last step decoded with the MTP heads
  void* ne_w1 = nullptr;
  float* ne_b1 = nullptr;
  void* ne_w2 = nullptr;
  float* ne_b2 = nullptr;
  float* rope_cos = nullptr;
  float* rope_sin = nullptr;
  float* noise_freq = nullptr;   // [d/2]: exp(-ln(1e4) t / (d/2)), rounded to fp32
  float* tau_feat = nullptr;     // [d]: cos | sin of (noise_scale * tau) * noise_freq, in fp32
  // paged KV
  void* kv = nullptr;
  int n_pages = 0, max_pages = 0;
  int32_t* d_page_table = nullptr;
  int32_t* h_page_table = nullptr;  // pinned mirror
  std::vector<int> free_pages;
  std::vector<int> n_alloc;
  // sequence state
  bool have_batch = false, have_step = false;
  bool admitted = false;        // kf_admit since the last kf_prefill (no rewind snapshot)
  int B = 0, P = 0, last_nh = 0;
  std::vector<int> h_len, h_len0;
  int32_t *d_len = nullptr, *d_len0 = nullptr, *d_pending = nullptr, *d_pending0 = nullptr;
  // decode attention visits the sequences longest first (d_order: a
  // permutation of 0..B-1 by decreasing cached length, ties by index); every
  // step adds the same count to every length, so only prefill, admit and
  // rewind change it
  int32_t* d_order = nullptr;
  std::vector<int32_t> h_order;
  bool order_dirty = true;
  int pend_stride = 8;
  // workspaces
  int R_cap = 0, NR_cap = 0, prefill_rows = 0;
  bool fused = false;     // RMSNorm fused into the tcgen05 GEMMs (bf16, head_dim 64)
  // The projections of the layers being enqueued run as skinny warp-MMA
  // kernels (at most 64 rows, fused path): their norm consumers take the
  // RMSNorm from their A rows, so no producer writes per-slot sums.
  bool skinny = false;
  float* ss = nullptr;    // [rows][d/64] sums of squares of the residual stream
  float* x = nullptr;
  void *xn = nullptr, *qkv = nullptr, *attn = nullptr, *hmid = nullptr;
  float* q = nullptr;
  void *nfeat = nullptr, *nhid = nullptr, *head_in = nullptr;
  HeadRec* rec = nullptr;
  int nchunk = 0;
  int32_t* tokens = nullptr;
  int32_t* t_out = nullptr;     // kf_teacher_step: [B][k] tokens of the k AR sub-steps
  float* noise = nullptr;
  int32_t *row_seq = nullptr, *row_pos = nullptr, *noise_map = nullptr, *head_map = nullptr;
  int32_t* row_tok = nullptr;
  int4* groups = nullptr;
  float* part_o = nullptr;
  float2* part_ml = nullptr;
  int* split_count = nullptr;   // [max groups][H] split counters of the warp-MMA attention
  size_t part_units = 0;
  int* d_err = nullptr;
  // graphs
  std::map<std::tuple<int, int, int>, cudaGraphExec_t> graphs;
  // profiling
  bool prof = false;
  bool launch_failed = false;   // a launch refused on the host (e.g. a TMA descriptor)
  std::vector<cudaEvent_t> ev;
  std::vector<int> ev_kind;
  int ev_used = 0;
  std::string err;
};

static thread_local std::string g_err;

namespace kf {
void set_global_error(const std::string& msg) { g_err = msg; }
}

static int fail(kf_ctx* c, int code, const std::string& msg) {
  if (c) c->err = msg;
  else g_err = msg;
  return code;
}

static int cuda_fail(kf_ctx* c, cudaError_t e, const char* what) {
  std::string m = std::string(what) + ": " + cudaGetErrorString(e);
  return fail(c, KF_E_CUDA, m);
}

#define KF_CUDA(call)                                       \
  do {                                                      \
    cudaError_t e_ = (call);                                \
    if (e_ != cudaSuccess) return cuda_fail(c, e_, #call);  \
  } while (0)

// status of the launches enqueued since the last call: a CUDA error, or a
// launch the host refused to make
static cudaError_t enqueue_status(kf_ctx* c) {
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess && c->launch_failed) e = cudaErrorInvalidValue;
  c->launch_failed = false;
  return e;
}

static bool is_device_ptr(const void* p) {
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

template <typename T>
static int dalloc(kf_ctx* c, T** p, size_t bytes, bool zero = true) {
  void* v = nullptr;
  if (bytes == 0) bytes = 16;
  cudaError_t e = cudaMalloc(&v, bytes);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return fail(c, KF_E_OOM, "cudaMalloc of " + std::to_string(bytes) + " bytes failed");
  }
  c->allocs.push_back(v);
  if (zero) {
    e = cudaMemset(v, 0, bytes);
    if (e != cudaSuccess) return cuda_fail(c, e, "cudaMemset");
  }
  *p = reinterpret_cast<T*>(v);
  return KF_OK;
}

#define KF_TRY(call)              \
  do {                            \
    int r_ = (call);              \
    if (r_ != KF_OK) return r_;   \
  } while (0)

// ------------------------------------------------------------- launches
// programmatic dependent launch for the kernels enqueued in this scope
struct PdlScope {
  bool prev;
  explicit PdlScope(bool on) : prev(g_pdl) { g_pdl = on; }
  ~PdlScope() { g_pdl = prev; }
};

static void prof_begin(kf_ctx* c, int kind) {
  if (!c->prof) return;
  if (c->ev_used + 2 > (int)c->ev.size()) return;
  // recorded while the profiled step is captured: an event record node
  cudaEventRecordWithFlags(c->ev[c->ev_used], c->stream, cudaEventRecordExternal);
  c->ev_kind[c->ev_used / 2] = kind;
}
static void prof_end(kf_ctx* c) {
  if (!c->prof) return;
  if (c->ev_used + 2 > (int)c->ev.size()) return;
  cudaEventRecordWithFlags(c->ev[c->ev_used + 1], c->stream, cudaEventRecordExternal);
  c->ev_used += 2;
}

static void gemm(kf_ctx* c, int kind, int M, int N, int K, const void* A, int lda, const void* W,
                 int ldw, const Epi& e, const void* l2_next = nullptr, size_t l2_bytes = 0) {
  if (M == 0) return;
  GemmDesc g{M, N, K, A, lda, W, ldw, e};
  g.l2_next = l2_next;
  g.l2_bytes = l2_bytes;
  prof_begin(c, kind);
  bool use_tc = c->bf16 && !(c->cfg.flags & KF_FLAG_SIMT_GEMM) && tc_gemm_supported(g);
  g_gemm_flags = (c->cfg.flags & KF_FLAG_NO_PERSISTENT_GEMM) ? kGemmNoPersist : 0;
  if (c->skinny && e.kind != EPI_HEAD && e.kind != EPI_LOGITS) {
    // every projection of a skinny enqueue must take this path: the fused
    // RMSNorm's producers and consumers agree on it
    if (!skinny_gemm_supported(g) || launch_gemm_skinny(g, c->d_err, c->stream) != 0) c->launch_failed = true;
  } else if (use_tc) {
    if (launch_gemm_tc(g, c->d_err, c->stream) != 0) c->launch_failed = true;
  }
  else
    launch_gemm_simt(c->bf16, g, c->stream);
  prof_end(c);
}

// attention split count: enough CTAs to cover the SMs twice, and at most
// max_keys keys per CTA
static void attn_plan(kf_ctx* c, int n_groups, int R, int max_keys, int* n_split, int* kps) {
  int ctas = n_groups * c->H;
  int max_split = ceil_div(c->cfg.max_len, 64);
  int s = std::max(1, std::min(max_split, ceil_div(2 * c->num_sms, std::max(1, ctas))));
  s = std::max(s, ceil_div(c->cfg.max_len, max_keys));
  while (s > 1 && (size_t)s * R * c->H > c->part_units && ceil_div(c->cfg.max_len, s - 1) <= max_keys)
    --s;
  *n_split = s;
  *kps = round_up(ceil_div(c->cfg.max_len, s), 64);
}

// warp-MMA attention: split the keys only while the (group, head) CTAs
// leave SMs idle, into at most 4 splits, and only into splits of more than
// one tile (those CTAs merge their own splits; measured on OWT-shaped
// decode: 1 and 8 sequences gain 10-14%, 32 and more lose with any split)
static void attn_plan_mma(kf_ctx* c, int n_groups, int R, int* n_split, int* kps) {
  const int L = c->cfg.max_len;
  const int ctas = n_groups * c->H;
  int s = ctas >= c->num_sms ? 1 : std::min(4, ceil_div(c->num_sms, std::max(1, ctas)));
  while (s > 1 && (round_up(ceil_div(L, s), kPage) <= 128 || (size_t)s * R * c->H > c->part_units)) --s;
  *n_split = s;
  *kps = round_up(ceil_div(L, s), kPage);
}

// L decoder layers over R rows (Table 4): pre-norm attention and MLP blocks.
// On the fused tensor-core path (c->fused) the pre-norms run inside the
// GEMMs: xn holds bf16(x), ss the per-64-column sums of squares written by
// the producers of x, and the QKV and MLP-up epilogues scale their rows (the
// gains are folded into wqkv and w_up).  Otherwise an RMSNorm kernel writes
// the normed rows into xn.
static void enqueue_layers(kf_ctx* c, int R, int n_groups, const int4* groups, int uniform_rows) {
  const int d = c->d, H = c->H, F = c->F;
  cudaStream_t s = c->stream;
  // Attention: the warp-MMA kernel for the bf16 cache with head_dim 64; the
  // FP32-FMA kernel otherwise (fp32 cache, head_dim 32).
  const int rows = groups ? kMaxGroupRows : uniform_rows;
  const bool mma_attn = attention_mma_supported(c->bf16, c->hd, rows);
  int n_split, kps;
  if (mma_attn) attn_plan_mma(c, n_groups, R, &n_split, &kps);
  else attn_plan(c, n_groups, R, 1 << 30, &n_split, &kps);
  auto norm_in = [&](Epi& e) {
    e.ss_in = c->ss; e.nslot = d / 64; e.inv_d = 1.0f / d; e.eps = c->cfg.rms_eps;
  };
  auto norm_out = [&](Epi& e) {
    e.xb_out = c->xn; e.nslot = d / 64;
    if (!c->skinny) e.ss_out = c->ss;
  };
  // In one 128-row tile the projections stream their weights with few rows
  // to multiply them by: each prefetches the next projection's weights into
  // L2 (the last layer's MLP-down the first 32 MiB of the LM head).  Measured
  // on OWT-shaped decode at k = 4: batch 1 53.1 -> 48.4 ms per generation;
  // at 256 rows and more it cost 2-5 %.
  const bool pf = R <= 128 && c->fused;
  const size_t e2 = c->esz;
  for (int l = 0; l < c->L; ++l) {
    const LayerW& w = c->layers[l];
    const bool last = l + 1 == c->L;
    const void* next_qkv = last ? c->w_head : c->layers[l + 1].wqkv;
    const size_t next_qkv_bytes = last ? std::min((size_t)c->V_pad * d * e2, (size_t)32 << 20) : (size_t)3 * d * d * e2;
    if (!c->fused) {
      prof_begin(c, KF_KIND_RMSNORM);
      launch_rmsnorm(c->bf16, R, nullptr, c->x, d, w.attn_norm, c->cfg.rms_eps, c->xn, s);
      prof_end(c);
    }
    // QKV projection; on the tensor-core path RoPE and the KV append run in
    // its epilogue, otherwise in a separate kernel
    if (c->fused) {
      Epi eq;
      eq.kind = EPI_QKV; eq.q_out = c->q; eq.kv = c->kv; eq.layer = l; eq.n_pages = c->n_pages;
      eq.H = H; eq.max_pages = c->max_pages; eq.dsec = d; eq.row_seq = c->row_seq;
      eq.row_pos = c->row_pos; eq.page_table = c->d_page_table;
      eq.cos_t = c->cfg.pos_kind == KF_POS_ROPE ? c->rope_cos : nullptr; eq.sin_t = c->rope_sin;
      eq.d_err = c->d_err;
      if (!groups) { eq.seq_len = c->d_len; eq.rows_per_seq = uniform_rows; }
      norm_in(eq);
      gemm(c, KF_KIND_GEMM_QKV, R, 3 * d, d, c->xn, d, w.wqkv, d, eq, pf ? w.wo : nullptr, (size_t)d * d * e2);
    } else {
      Epi e;
      e.kind = EPI_STORE; e.out = c->qkv; e.ldo = 3 * d;
      gemm(c, KF_KIND_GEMM_QKV, R, 3 * d, d, c->xn, d, w.wqkv, d, e);
      prof_begin(c, KF_KIND_ROPE_KV);
      launch_rope_append(c->bf16, R, c->qkv, d, H, c->hd, c->row_seq, c->row_pos,
                         c->cfg.pos_kind == KF_POS_ROPE ? c->rope_cos : nullptr, c->rope_sin,
                         c->q, c->kv, l, c->n_pages, c->d_page_table, c->max_pages, c->d_err, s);
      prof_end(c);
    }
    AttnArgs a{};
    a.q = c->q; a.kv = c->kv; a.layer = l; a.n_pages = c->n_pages; a.H = H; a.hd = c->hd;
    a.page_table = c->d_page_table; a.max_pages = c->max_pages;
    a.row_seq = c->row_seq; a.row_pos = c->row_pos; a.groups = groups;
    a.uniform_rows = uniform_rows; a.out = c->attn; a.part_o = c->part_o; a.part_ml = c->part_ml;
    a.R = R; a.n_split = n_split; a.keys_per_split = kps; a.d_err = c->d_err;
    a.len = groups ? nullptr : c->d_len;   // decode: keys below it are stable during the step
    a.order = groups || !mma_attn ? nullptr : c->d_order;   // longest sequences first
    a.split_count = c->split_count;
    prof_begin(c, KF_KIND_ATTENTION);
    bool merged = false;
    if (mma_attn) {
      if (launch_attention_mma(a, n_groups, rows, c->cfg.max_len, s, &merged) != 0) c->launch_failed = true;
    }
    else launch_attention(c->bf16, a, n_groups, c->cfg.max_len, s);
    prof_end(c);
    if (n_split > 1 && !merged) {
      prof_begin(c, KF_KIND_ATTN_COMBINE);
      launch_attn_combine(c->bf16, a, s);
      prof_end(c);
    }
    Epi eo;
    eo.kind = EPI_RESID; eo.x = c->x; eo.ldx = d;
    if (c->fused) norm_out(eo);
    gemm(c, KF_KIND_GEMM_O, R, d, d, c->attn, d, w.wo, d, eo, pf ? w.w_up : nullptr, (size_t)F * d * e2);
    if (!c->fused) {
      prof_begin(c, KF_KIND_RMSNORM);
      launch_rmsnorm(c->bf16, R, nullptr, c->x, d, w.mlp_norm, c->cfg.rms_eps, c->xn, s);
      prof_end(c);
    }
    Epi eu;
    eu.kind = EPI_BIAS_GELU; eu.out = c->hmid; eu.ldo = F;
    if (c->fused) norm_in(eu);
    gemm(c, KF_KIND_GEMM_UP, R, F, d, c->xn, d, w.w_up, d, eu, pf ? w.w_down : nullptr, (size_t)d * F * e2);
    Epi ed;
    ed.kind = EPI_RESID; ed.x = c->x; ed.ldx = d;
    if (c->fused) norm_out(ed);
    gemm(c, KF_KIND_GEMM_DOWN, R, d, F, c->hmid, F, w.w_down, F, ed, pf ? next_qkv : nullptr, next_qkv_bytes);
  }
}

// Calls of at most 16 rows run their projections as skinny warp-MMA kernels
// (weights staged before the dependency wait, no 128-row tcgen05 tiles).
// Measured on the OWT-shaped model, microseconds per decode call, skinny vs
// tcgen05 (same box): 2 sequences at k = 4 (16 rows) 374.7 vs 388.3, AR step
// of 16 sequences 382.4 vs 396.3; but 32 rows 470.7 vs 401.0 and 64 rows
// 564.0 vs 442.8 (a 16-column CTA re-reads the A rows once per 16 columns).
constexpr int kSkinnyMaxRows = 16;
static bool use_skinny(const kf_ctx* c, int R) {
  return c->fused && R <= kSkinnyMaxRows && !(c->cfg.flags & KF_FLAG_NO_SKINNY);
}

// One decode step on the device: no host data dependence, so it can be
// captured once per (B, P, k) and replayed.
static void enqueue_step(kf_ctx* c, int B, int P, int k, const float* noise) {
  cudaStream_t s = c->stream;
  PdlScope pdl(!c->prof && !(c->cfg.flags & KF_FLAG_NO_PDL));
  const int d = c->d;
  // standard MTP (Sec. 3.3): one noise-conditioning token per sequence whose
  // NoiseEnc input is the k values' features side by side; k heads decode it
  const bool mtp = c->mtp_k > 0 && k > 0;
  const int kz = mtp ? 1 : k;                      // noise rows per sequence
  const int S = P + kz, R = B * S, nout = k > 0 ? k : 1, nh = mtp ? B : B * nout;
  c->skinny = use_skinny(c, R);
  // row maps, pending-token embeddings and noise features: one launch
  prof_begin(c, KF_KIND_EMBED);
  launch_step_prologue(c->bf16, B, P, kz, c->d_len, c->d_pending, c->pend_stride, c->tok_emb,
                       c->pos_emb, c->V, d, c->x, c->fused ? c->xn : nullptr,
                       c->fused ? c->ss : nullptr, c->d_err, c->row_seq, c->row_pos, c->noise_map,
                       c->head_map, k > 0 ? B * k : 0, noise, c->noise_freq, c->tau_feat,
                       c->cfg.noise_scale, c->nfeat, s);
  prof_end(c);
  if (k > 0) {
    // h_z = NoiseEnc(z): W2 . gelu(W1 s(z, tau) + b1) + b2, written into the noise rows
    // (MTP: the B rows of k * d features, [B][k][d] as laid out by the feature kernel)
    const int ne_in = mtp ? k * d : d;
    Epi e1;
    e1.kind = EPI_BIAS_GELU; e1.out = c->nhid; e1.ldo = c->NH; e1.bias = c->ne_b1;
    const bool pf = R <= 128 && c->fused;
    gemm(c, KF_KIND_NOISE_GEMM, B * kz, c->NH, ne_in, c->nfeat, ne_in, c->ne_w1, ne_in, e1,
         pf ? c->ne_w2 : nullptr, (size_t)d * c->NH * c->esz);
    Epi e2;
    e2.kind = EPI_NOISE_OUT; e2.x = c->x; e2.ldx = d; e2.bias = c->ne_b2;
    e2.row_map = c->noise_map; e2.row_pos = c->row_pos; e2.pos_emb = c->pos_emb;
    if (c->fused) {
      e2.xb_out = c->xn; e2.nslot = d / 64;
      if (!c->skinny) e2.ss_out = c->ss;
    }
    gemm(c, KF_KIND_NOISE_GEMM, B * kz, d, c->NH, c->nhid, c->NH, c->ne_w2, c->NH, e2,
         pf ? c->layers[0].wqkv : nullptr, (size_t)3 * d * d * c->esz);
  }
  enqueue_layers(c, R, B, nullptr, S);
  prof_begin(c, KF_KIND_HEAD_NORM);
  launch_rmsnorm(c->bf16, nh, c->head_map, c->x, d, c->final_norm, c->cfg.rms_eps, c->head_in, s);
  prof_end(c);
  if (mtp) {
    // head j over the B noise rows; its chunk records at rows j * B + b
    for (int j = 0; j < k; ++j) {
      Epi eh;
      eh.kind = EPI_HEAD; eh.inv_tau = 1.0f / c->cfg.tau; eh.n_valid = c->V;
      eh.rec = c->rec + (size_t)j * B * c->nchunk; eh.nchunk = c->nchunk;
      gemm(c, KF_KIND_GEMM_HEAD, B, c->V_pad, d, c->head_in, d,
           static_cast<const char*>(c->w_mtp) + (size_t)j * c->V_pad * d * c->esz, d, eh);
    }
  } else {
    Epi eh;
    eh.kind = EPI_HEAD; eh.inv_tau = 1.0f / c->cfg.tau; eh.n_valid = c->V; eh.rec = c->rec;
    eh.nchunk = c->nchunk;
    gemm(c, KF_KIND_GEMM_HEAD, nh, c->V_pad, d, c->head_in, d, c->w_head, d, eh);
  }
  // the noise -> token map, which also commits the step (the emitted tokens
  // become the pending ids, the lengths grow by P)
  StepCommit cm;
  cm.pending = c->d_pending; cm.pend_stride = c->pend_stride; cm.len = c->d_len; cm.P = P;
  cm.nout = nout;
  prof_begin(c, KF_KIND_HEAD_SELECT);
  launch_head_select(c->bf16, B * nout, c->rec, c->nchunk, c->head_in, d, mtp ? c->w_mtp : c->w_head,
                     c->V, 1.0f / c->cfg.tau, c->cfg.map_kind, noise, c->tokens, mtp ? B : 0,
                     (size_t)c->V_pad * d, c->d_err, cm, s);
  prof_end(c);
}

// ------------------------------------------------------------- pages
static void reset_pages(kf_ctx* c) {
  c->free_pages.clear();
  for (int p = c->n_pages - 1; p >= 0; --p) c->free_pages.push_back(p);
  std::fill(c->n_alloc.begin(), c->n_alloc.end(), 0);
  for (size_t i = 0; i < (size_t)c->cfg.max_batch * c->max_pages; ++i) c->h_page_table[i] = -1;
}

// make sequence b's pages cover positions 0 .. upto
static int ensure_pages(kf_ctx* c, int b, int upto, bool* dirty) {
  int need = upto / kPage + 1;
  if (need > c->max_pages) return fail(c, KF_E_CAPACITY, "sequence longer than max_len");
  while (c->n_alloc[b] < need) {
    if (c->free_pages.empty()) return fail(c, KF_E_CAPACITY, "KV page pool exhausted");
    int p = c->free_pages.back();
    c->free_pages.pop_back();
    c->h_page_table[(size_t)b * c->max_pages + c->n_alloc[b]] = p;
    c->n_alloc[b]++;
    *dirty = true;
  }
  return KF_OK;
}

static int upload_page_row(kf_ctx* c, int b) {
  size_t off = (size_t)b * c->max_pages;
  KF_CUDA(cudaMemcpyAsync(c->d_page_table + off, c->h_page_table + off, c->max_pages * 4,
                          cudaMemcpyHostToDevice, c->stream));
  return KF_OK;
}

// ------------------------------------------------------------- C ABI
extern "C" {

int kf_init(const kf_config* cfg_in, const kf_weights* w, void* stream, kf_ctx** out) {
  kf_ctx* c = nullptr;
  if (!out) return fail(nullptr, KF_E_ARG, "out is NULL");
  *out = nullptr;
  if (!cfg_in || !w) return fail(nullptr, KF_E_ARG, "cfg or weights is NULL");
  kf_config cfg = *cfg_in;
  if (cfg.noise_hidden == 0) cfg.noise_hidden = 4 * cfg.d_model;
  if (cfg.prefill_rows == 0) cfg.prefill_rows = 4096;
  const char* bad = nullptr;
  if (cfg.n_layer < 1) bad = "n_layer < 1";
  else if (cfg.n_head < 1 || cfg.d_model % cfg.n_head ||
           (cfg.d_model / cfg.n_head != 32 && cfg.d_model / cfg.n_head != 64))
    bad = "head_dim = d_model / n_head must be 32 or 64";
  else if (cfg.d_ff < 64 || cfg.d_ff % 64) bad = "d_ff must be a positive multiple of 64";
  else if (cfg.noise_hidden < 64 || cfg.noise_hidden % 64) bad = "noise_hidden must be a multiple of 64";
  else if (cfg.vocab < 2) bad = "vocab < 2";
  else if (cfg.max_len < 2) bad = "max_len < 2";
  else if (cfg.max_k < 1 || cfg.max_k > 8) bad = "max_k must be in 1..8";
  else if (cfg.max_batch < 1) bad = "max_batch < 1";
  else if (cfg.page_size != kPage) bad = "page_size must be 16";
  else if (cfg.pos_kind != KF_POS_ROPE && cfg.pos_kind != KF_POS_LEARNED) bad = "bad pos_kind";
  else if (cfg.dtype != KF_DTYPE_FP32 && cfg.dtype != KF_DTYPE_BF16) bad = "bad dtype";
  else if (cfg.map_kind != KF_MAP_ICDF && cfg.map_kind != KF_MAP_ARGMAX) bad = "bad map_kind";
  else if (!(cfg.tau > 0.f)) bad = "tau must be > 0";
  else if (!(cfg.rms_eps >= 0.f)) bad = "rms_eps must be >= 0";
  else if (cfg.n_pages < 0 || cfg.prefill_rows < 16) bad = "bad n_pages / prefill_rows";
  else if (cfg.mtp_k < 0 || cfg.mtp_k > cfg.max_k) bad = "mtp_k must be in 0..max_k";
  else if (cfg.mtp_k > 0 && !w->w_mtp) bad = "w_mtp is NULL with mtp_k > 0";
  else if (!w->tok_emb || !w->attn_norm || !w->wqkv || !w->wo || !w->mlp_norm || !w->w_up ||
           !w->w_down || !w->final_norm || !w->w_head || !w->ne_w1 || !w->ne_b1 || !w->ne_w2 ||
           !w->ne_b2)
    bad = "a weight pointer is NULL";
  else if (cfg.pos_kind == KF_POS_LEARNED && !w->pos_emb) bad = "pos_emb is NULL";
  if (bad) return fail(nullptr, KF_E_ARG, bad);

  c = new kf_ctx();
  c->cfg = cfg;
  cudaError_t e = cudaGetDevice(&c->dev);
  if (e != cudaSuccess) {
    std::string m = std::string("no CUDA device: ") + cudaGetErrorString(e);
    delete c;
    return fail(nullptr, KF_E_CUDA, m);
  }
  int r = KF_OK;
  auto bail = [&](int code) {
    g_err = c->err;
    kf_free(c);
    return code;
  };
  cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, c->dev);
  if (stream) {
    c->stream = (cudaStream_t)stream;
  } else {
    // a blocking stream keeps implicit ordering with the legacy default stream
    e = cudaStreamCreate(&c->stream);
    if (e != cudaSuccess) { cuda_fail(c, e, "cudaStreamCreate"); return bail(KF_E_CUDA); }
    c->own_stream = true;
  }
  c->bf16 = cfg.dtype == KF_DTYPE_BF16;
  c->esz = c->bf16 ? 2 : 4;
  c->d = cfg.d_model; c->H = cfg.n_head; c->hd = cfg.d_model / cfg.n_head; c->L = cfg.n_layer; c->F = cfg.d_ff; c->V = cfg.vocab;
  c->NH = cfg.noise_hidden; c->V_pad = round_up(cfg.vocab, 256); c->max_k = cfg.max_k;
  c->mtp_k = cfg.mtp_k;
  c->nchunk = ceil_div(cfg.vocab, kChunk);
  const int d = c->d, L = c->L, F = c->F, V = c->V, NH = c->NH;
  const bool dev_w = is_device_ptr(w->tok_emb);

  // -- weights: staged through one fp32 device buffer, converted to storage type
  const int ne_in = d * std::max(1, cfg.mtp_k);   // NoiseEnc input width
  size_t max_elems = std::max({(size_t)V * d, (size_t)L * 3 * d * d, (size_t)L * F * d,
                               (size_t)NH * ne_in, (size_t)cfg.max_len * d});
  float* stage = nullptr;
  if ((r = dalloc(c, &stage, max_elems * 4, false))) return bail(r);
  const float* fold_gain = nullptr;   // gains to fold into the columns being uploaded
  int fold_rows = 0;
  auto upload = [&](const float* src, size_t n, void* dst, bool convert) -> int {
    e = cudaMemcpyAsync(stage, src, n * 4, dev_w ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice,
                        c->stream);
    if (e != cudaSuccess) return cuda_fail(c, e, "weight copy");
    if (fold_gain) launch_scale_cols(stage, fold_gain, fold_rows, d, n, c->stream);
    if (convert) launch_convert_f32(c->bf16, stage, dst, n, c->stream);
    else launch_convert_f32(false, stage, dst, n, c->stream);
    e = cudaStreamSynchronize(c->stream);
    if (e != cudaSuccess) return cuda_fail(c, e, "weight convert");
    return KF_OK;
  };
  auto wbuf = [&](void** p, size_t n) { return dalloc(c, p, n * c->esz); };
  auto fbuf = [&](float** p, size_t n) { return dalloc(c, p, n * 4); };
  void *wqkv, *wo, *wup, *wdown;
  float *an, *mn;
  if ((r = wbuf(&c->tok_emb, (size_t)V * d)) || (r = upload(w->tok_emb, (size_t)V * d, c->tok_emb, true)))
    return bail(r);
  if (cfg.pos_kind == KF_POS_LEARNED) {
    if ((r = fbuf(&c->pos_emb, (size_t)cfg.max_len * d)) ||
        (r = upload(w->pos_emb, (size_t)cfg.max_len * d, c->pos_emb, false)))
      return bail(r);
  }
  // the fused path folds the pre-norm gains into the consuming projections:
  // rmsnorm(x) W^T = rinv(x) * (x (W diag(g))^T)
  c->fused = c->bf16 && !(cfg.flags & KF_FLAG_SIMT_GEMM) && c->hd == 64 && d % 64 == 0;
  auto upload_fold = [&](const float* src, size_t n, void* dst, const float* gains,
                         int rows_per_layer) -> int {
    fold_gain = gains;
    fold_rows = rows_per_layer;
    int rr = upload(src, n, dst, true);
    fold_gain = nullptr;
    return rr;
  };
  if ((r = fbuf(&an, (size_t)L * d)) || (r = upload(w->attn_norm, (size_t)L * d, an, false)) ||
      (r = fbuf(&mn, (size_t)L * d)) || (r = upload(w->mlp_norm, (size_t)L * d, mn, false)) ||
      (r = wbuf(&wqkv, (size_t)L * 3 * d * d)) ||
      (r = upload_fold(w->wqkv, (size_t)L * 3 * d * d, wqkv, c->fused ? an : nullptr, 3 * d)) ||
      (r = wbuf(&wo, (size_t)L * d * d)) || (r = upload(w->wo, (size_t)L * d * d, wo, true)) ||
      (r = wbuf(&wup, (size_t)L * F * d)) ||
      (r = upload_fold(w->w_up, (size_t)L * F * d, wup, c->fused ? mn : nullptr, F)) ||
      (r = wbuf(&wdown, (size_t)L * d * F)) || (r = upload(w->w_down, (size_t)L * d * F, wdown, true)) ||
      (r = fbuf(&c->final_norm, d)) || (r = upload(w->final_norm, d, c->final_norm, false)) ||
      (r = wbuf(&c->w_head, (size_t)c->V_pad * d)) ||
      (r = upload(w->w_head, (size_t)V * d, c->w_head, true)) ||
      (r = wbuf(&c->ne_w1, (size_t)NH * ne_in)) || (r = upload(w->ne_w1, (size_t)NH * ne_in, c->ne_w1, true)) ||
      (r = fbuf(&c->ne_b1, NH)) || (r = upload(w->ne_b1, NH, c->ne_b1, false)) ||
      (r = wbuf(&c->ne_w2, (size_t)d * NH)) || (r = upload(w->ne_w2, (size_t)d * NH, c->ne_w2, true)) ||
      (r = fbuf(&c->ne_b2, d)) || (r = upload(w->ne_b2, d, c->ne_b2, false)))
    return bail(r);
  if (c->mtp_k > 0) {
    // MTP heads, each padded to V_pad zero rows like w_head
    if ((r = wbuf(&c->w_mtp, (size_t)c->mtp_k * c->V_pad * d))) return bail(r);
    for (int j = 0; j < c->mtp_k; ++j)
      if ((r = upload(w->w_mtp + (size_t)j * V * d, (size_t)V * d,
                      static_cast<char*>(c->w_mtp) + (size_t)j * c->V_pad * d * c->esz, true)))
        return bail(r);
  }
  for (int l = 0; l < L; ++l) {
    LayerW lw;
    lw.wqkv = (char*)wqkv + (size_t)l * 3 * d * d * c->esz;
    lw.wo = (char*)wo + (size_t)l * d * d * c->esz;
    lw.w_up = (char*)wup + (size_t)l * F * d * c->esz;
    lw.w_down = (char*)wdown + (size_t)l * d * F * c->esz;
    lw.attn_norm = an + (size_t)l * d;
    lw.mlp_norm = mn + (size_t)l * d;
    c->layers.push_back(lw);
  }

  // -- position and noise-feature tables, formed in fp64 on the host
  {
    const int half = c->hd / 2;
    std::vector<float> cs((size_t)cfg.max_len * half), sn((size_t)cfg.max_len * half);
    for (int p = 0; p < cfg.max_len; ++p)
      for (int i = 0; i < half; ++i) {
        double ang = (double)p * std::pow((double)cfg.rope_theta, -2.0 * i / c->hd);
        cs[(size_t)p * half + i] = (float)std::cos(ang);
        sn[(size_t)p * half + i] = (float)std::sin(ang);
      }
    if ((r = fbuf(&c->rope_cos, cs.size())) || (r = fbuf(&c->rope_sin, sn.size()))) return bail(r);
    // the noise encoding's frequencies in fp32, and the temperature's
    // encoding with the oracle's fp32 arithmetic: (scale * tau) * freq
    std::vector<float> fr(d / 2);
    for (int t = 0; t < d / 2; ++t) fr[t] = (float)std::exp(-std::log(1e4) * t / (d / 2));
    std::vector<float> tf(d);
    const float st = cfg.noise_scale * cfg.tau;
    for (int t = 0; t < d / 2; ++t) {
      const float ang = st * fr[t];
      tf[t] = std::cos(ang);
      tf[d / 2 + t] = std::sin(ang);
    }
    if ((r = fbuf(&c->noise_freq, fr.size())) || (r = fbuf(&c->tau_feat, tf.size()))) return bail(r);
    if (cudaMemcpy(c->rope_cos, cs.data(), cs.size() * 4, cudaMemcpyHostToDevice) != cudaSuccess ||
        cudaMemcpy(c->rope_sin, sn.data(), sn.size() * 4, cudaMemcpyHostToDevice) != cudaSuccess ||
        cudaMemcpy(c->noise_freq, fr.data(), fr.size() * 4, cudaMemcpyHostToDevice) != cudaSuccess ||
        cudaMemcpy(c->tau_feat, tf.data(), tf.size() * 4, cudaMemcpyHostToDevice) != cudaSuccess) {
      cuda_fail(c, cudaGetLastError(), "table upload");
      return bail(KF_E_CUDA);
    }
  }

  // -- paged KV pool and page table
  c->max_pages = ceil_div(cfg.max_len, kPage);
  c->n_pages = cfg.n_pages ? cfg.n_pages : cfg.max_batch * c->max_pages;
  size_t kv_bytes = (size_t)L * c->n_pages * 2 * c->H * kPage * c->hd * c->esz;
  if ((r = dalloc(c, &c->kv, kv_bytes))) return bail(r);
  if ((r = dalloc(c, &c->d_page_table, (size_t)cfg.max_batch * c->max_pages * 4))) return bail(r);
  e = cudaMallocHost(&c->h_page_table, (size_t)cfg.max_batch * c->max_pages * 4);
  if (e != cudaSuccess) { cuda_fail(c, e, "cudaMallocHost"); return bail(KF_E_OOM); }
  c->n_alloc.assign(cfg.max_batch, 0);
  reset_pages(c);

  // -- state and workspaces
  const int MB = cfg.max_batch, MK = cfg.max_k;
  c->pend_stride = MK;
  c->NR_cap = round_up(MB * MK, 128);
  c->prefill_rows = round_up(cfg.prefill_rows, 128);
  c->R_cap = std::max(round_up(MB * 2 * MK, 128), c->prefill_rows);
  const int R = c->R_cap;
  if ((r = dalloc(c, &c->d_len, MB * 4)) || (r = dalloc(c, &c->d_len0, MB * 4)) ||
      (r = dalloc(c, &c->d_order, MB * 4)) ||
      (r = dalloc(c, &c->d_pending, (size_t)MB * MK * 4)) ||
      (r = dalloc(c, &c->d_pending0, (size_t)MB * MK * 4)) ||
      (r = dalloc(c, &c->x, (size_t)R * d * 4)) || (r = wbuf(&c->xn, (size_t)R * d)) ||
      (r = dalloc(c, &c->ss, (size_t)R * (d / 64 + 1) * 4)) ||
      (r = wbuf(&c->qkv, (size_t)R * 3 * d)) || (r = dalloc(c, &c->q, (size_t)R * d * 4)) ||
      (r = wbuf(&c->attn, (size_t)R * d)) || (r = wbuf(&c->hmid, (size_t)R * F)) ||
      (r = wbuf(&c->nfeat, (size_t)c->NR_cap * d)) || (r = wbuf(&c->nhid, (size_t)c->NR_cap * NH)) ||
      (r = wbuf(&c->head_in, (size_t)c->NR_cap * d)) ||
      (r = dalloc(c, &c->rec, (size_t)c->NR_cap * c->nchunk * sizeof(HeadRec))) ||
      (r = dalloc(c, &c->tokens, (size_t)c->NR_cap * 4)) ||
      (r = dalloc(c, &c->t_out, (size_t)c->NR_cap * 4)) ||
      (r = dalloc(c, &c->noise, (size_t)c->NR_cap * 4)) ||
      (r = dalloc(c, &c->row_seq, (size_t)R * 4)) || (r = dalloc(c, &c->row_pos, (size_t)R * 4)) ||
      (r = dalloc(c, &c->row_tok, (size_t)R * 4)) ||
      (r = dalloc(c, &c->noise_map, (size_t)c->NR_cap * 4)) ||
      (r = dalloc(c, &c->head_map, (size_t)c->NR_cap * 4)) ||
      (r = dalloc(c, &c->groups, (size_t)R * sizeof(int4))) || (r = dalloc(c, &c->d_err, 4)))
    return bail(r);
  // split-KV partials: small batches split to fill the SMs
  c->part_units = (size_t)4 * c->num_sms * kMaxGroupRows;
  if ((r = dalloc(c, &c->part_o, c->part_units * c->hd * 4)) ||
      (r = dalloc(c, &c->part_ml, c->part_units * sizeof(float2))) ||
      (r = dalloc(c, &c->split_count, (size_t)std::max(R, cfg.max_batch) * c->H * sizeof(int))))
    return bail(r);
  e = cudaDeviceSynchronize();
  if (e != cudaSuccess) { cuda_fail(c, e, "init"); return bail(KF_E_CUDA); }
  *out = c;
  return KF_OK;
}

// Prefill: the KV of each listed slot's first n tokens (positions 0..n-1),
// in row chunks of up to prefill_rows, attention groups of <= 16 rows per
// sequence.  The slots' pages must be allocated and uploaded.
struct PrefillSeq {
  int slot;
  const int32_t* tok;
  int n;
};
static int prefill_rows(kf_ctx* c, const std::vector<PrefillSeq>& seqs) {
  std::vector<int32_t> r_tok, r_seq, r_pos;
  std::vector<int4> grp;
  auto flush = [&]() -> int {
    int R = (int)r_tok.size();
    if (R == 0) return KF_OK;
    KF_CUDA(cudaMemcpyAsync(c->row_tok, r_tok.data(), R * 4, cudaMemcpyHostToDevice, c->stream));
    KF_CUDA(cudaMemcpyAsync(c->row_seq, r_seq.data(), R * 4, cudaMemcpyHostToDevice, c->stream));
    KF_CUDA(cudaMemcpyAsync(c->row_pos, r_pos.data(), R * 4, cudaMemcpyHostToDevice, c->stream));
    KF_CUDA(cudaMemcpyAsync(c->groups, grp.data(), grp.size() * sizeof(int4), cudaMemcpyHostToDevice,
                            c->stream));
    {
      PdlScope pdl(!(c->cfg.flags & KF_FLAG_NO_PDL));
      c->skinny = use_skinny(c, R);
      launch_embed_tokens(c->bf16, R, c->row_tok, c->tok_emb, c->pos_emb, c->row_pos, c->V, c->d,
                          c->x, c->fused ? c->xn : nullptr, c->fused ? c->ss : nullptr, c->d_err,
                          c->stream);
      enqueue_layers(c, R, (int)grp.size(), c->groups, 0);
    }
    KF_CUDA(enqueue_status(c));
    // the host vectors are reused: wait until the copies have consumed them
    KF_CUDA(cudaStreamSynchronize(c->stream));
    r_tok.clear(); r_seq.clear(); r_pos.clear(); grp.clear();
    return KF_OK;
  };
  for (const PrefillSeq& q : seqs) {
    int p = 0;
    while (p < q.n) {
      if ((int)r_tok.size() == c->prefill_rows) KF_TRY(flush());
      int take = std::min({q.n - p, kMaxGroupRows, c->prefill_rows - (int)r_tok.size()});
      grp.push_back(make_int4(q.slot, (int)r_tok.size(), take, 0));
      for (int i = 0; i < take; ++i) {
        r_tok.push_back(q.tok[p + i]);
        r_seq.push_back(q.slot);
        r_pos.push_back(p + i);
      }
      p += take;
    }
  }
  return flush();
}

int kf_prefill(kf_ctx* c, int32_t B, const int32_t* tokens, const int32_t* lens) {
  if (!c) return fail(nullptr, KF_E_ARG, "ctx is NULL");
  if (B < 1 || B > c->cfg.max_batch) return fail(c, KF_E_ARG, "B out of range 1..max_batch");
  if (!tokens || !lens) return fail(c, KF_E_ARG, "tokens or lens is NULL");
  std::vector<int> ln(B);
  size_t total = 0;
  for (int b = 0; b < B; ++b) {
    ln[b] = lens[b];
    if (ln[b] < 1) return fail(c, KF_E_ARG, "prompt length < 1");
    if (ln[b] + 1 > c->cfg.max_len) return fail(c, KF_E_CAPACITY, "prompt longer than max_len - 1");
    total += ln[b];
  }
  // Host prompts are checked here; device-resident prompts are checked where
  // the embedding kernel reads them (an id outside [0, V) embeds as id 0 and
  // flags the device error word: the call then returns KF_E_DEVICE).
  std::vector<int32_t> tok(total);
  const bool dev_tok = is_device_ptr(tokens);
  if (dev_tok) {
    KF_CUDA(cudaMemcpy(tok.data(), tokens, total * 4, cudaMemcpyDeviceToHost));
  } else {
    memcpy(tok.data(), tokens, total * 4);
    for (size_t i = 0; i < total; ++i)
      if (tok[i] < 0 || tok[i] >= c->V) return fail(c, KF_E_ARG, "token id out of range");
  }
  KF_CUDA(cudaStreamSynchronize(c->stream));
  c->have_batch = false;
  c->have_step = false;
  // a new batch starts with a clear device error word
  KF_CUDA(cudaMemsetAsync(c->d_err, 0, 4, c->stream));
  reset_pages(c);
  for (int b = 0; b < B; ++b) {
    bool dirty = false;
    if (ln[b] > 1) KF_TRY(ensure_pages(c, b, ln[b] - 2, &dirty));
  }
  KF_CUDA(cudaMemcpyAsync(c->d_page_table, c->h_page_table,
                          (size_t)c->cfg.max_batch * c->max_pages * 4, cudaMemcpyHostToDevice,
                          c->stream));
  // rows: every prompt token but the last
  std::vector<PrefillSeq> seqs;
  {
    size_t o = 0;
    for (int b = 0; b < B; ++b) {
      seqs.push_back({b, tok.data() + o, ln[b] - 1});
      o += ln[b];
    }
  }
  KF_TRY(prefill_rows(c, seqs));
  // state: cached = N - 1, one pending token (the prompt's last)
  c->B = B;
  c->P = 1;
  c->h_len.assign(B, 0);
  std::vector<int32_t> pend((size_t)B * c->pend_stride, 0);
  size_t off = 0;
  for (int b = 0; b < B; ++b) {
    c->h_len[b] = ln[b] - 1;
    pend[(size_t)b * c->pend_stride] = tok[off + ln[b] - 1];
    off += ln[b];
  }
  c->h_len0 = c->h_len;
  c->order_dirty = true;
  std::vector<int32_t> hl(c->h_len.begin(), c->h_len.end());
  KF_CUDA(cudaMemcpyAsync(c->d_len, hl.data(), B * 4, cudaMemcpyHostToDevice, c->stream));
  KF_CUDA(cudaMemcpyAsync(c->d_len0, hl.data(), B * 4, cudaMemcpyHostToDevice, c->stream));
  KF_CUDA(cudaMemcpyAsync(c->d_pending, pend.data(), pend.size() * 4, cudaMemcpyHostToDevice, c->stream));
  KF_CUDA(cudaMemcpyAsync(c->d_pending0, pend.data(), pend.size() * 4, cudaMemcpyHostToDevice, c->stream));
  KF_CUDA(cudaStreamSynchronize(c->stream));
  int err = 0;
  KF_CUDA(cudaMemcpy(&err, c->d_err, 4, cudaMemcpyDeviceToHost));
  if (err) return fail(c, KF_E_DEVICE, "device error flag " + std::to_string(err) + " in prefill");
  c->have_batch = true;
  c->admitted = false;
  return KF_OK;
}

int kf_admit(kf_ctx* c, int32_t n, const int32_t* slots, const int32_t* tokens, const int32_t* lens) {
  if (!c) return fail(nullptr, KF_E_ARG, "ctx is NULL");
  if (!c->have_batch) return fail(c, KF_E_STATE, "admit before prefill");
  if (n < 1 || n > c->B) return fail(c, KF_E_ARG, "n out of range 1..B");
  if (!slots || !tokens || !lens) return fail(c, KF_E_ARG, "slots, tokens or lens is NULL");
  const int P = c->P;
  std::vector<int> sl(n), ln(n);
  std::vector<char> seen(c->B, 0);
  size_t total = 0;
  for (int i = 0; i < n; ++i) {
    sl[i] = slots[i];
    ln[i] = lens[i];
    if (sl[i] < 0 || sl[i] >= c->B) return fail(c, KF_E_ARG, "slot out of range 0..B-1");
    if (seen[sl[i]]) return fail(c, KF_E_ARG, "slot listed twice");
    seen[sl[i]] = 1;
    if (ln[i] < 1 || ln[i] < P) return fail(c, KF_E_ARG, "prompt shorter than the batch's pending count");
    if (ln[i] + 1 > c->cfg.max_len) return fail(c, KF_E_CAPACITY, "prompt longer than max_len - 1");
    total += ln[i];
  }
  std::vector<int32_t> tok(total);
  if (is_device_ptr(tokens)) {
    KF_CUDA(cudaMemcpy(tok.data(), tokens, total * 4, cudaMemcpyDeviceToHost));
  } else {
    memcpy(tok.data(), tokens, total * 4);
  }
  for (size_t i = 0; i < total; ++i)
    if (tok[i] < 0 || tok[i] >= c->V) return fail(c, KF_E_ARG, "token id out of range");
  // steps in flight still read these slots' pages and the page-table mirror
  KF_CUDA(cudaStreamSynchronize(c->stream));
  // evict: the slots' pages return to the pool
  for (int i = 0; i < n; ++i) {
    const size_t row = (size_t)sl[i] * c->max_pages;
    for (int j = 0; j < c->n_alloc[sl[i]]; ++j) {
      c->free_pages.push_back(c->h_page_table[row + j]);
      c->h_page_table[row + j] = -1;
    }
    c->n_alloc[sl[i]] = 0;
  }
  // insert: the first len - P tokens cached, the last P pending (the batch's
  // pending count stays uniform)
  std::vector<PrefillSeq> seqs;
  std::vector<int32_t> pend((size_t)n * P), nl(n);
  size_t off = 0;
  for (int i = 0; i < n; ++i) {
    const int m = ln[i] - P;
    bool dirty = true;
    if (m > 0) KF_TRY(ensure_pages(c, sl[i], m - 1, &dirty));
    KF_TRY(upload_page_row(c, sl[i]));
    if (m > 0) seqs.push_back({sl[i], tok.data() + off, m});
    for (int j = 0; j < P; ++j) pend[(size_t)i * P + j] = tok[off + m + j];
    nl[i] = m;
    off += ln[i];
  }
  KF_TRY(prefill_rows(c, seqs));
  for (int i = 0; i < n; ++i) {
    KF_CUDA(cudaMemcpyAsync(c->d_pending + (size_t)sl[i] * c->pend_stride, pend.data() + (size_t)i * P,
                            (size_t)P * 4, cudaMemcpyHostToDevice, c->stream));
    KF_CUDA(cudaMemcpyAsync(c->d_len + sl[i], nl.data() + i, 4, cudaMemcpyHostToDevice, c->stream));
    c->h_len[sl[i]] = nl[i];
    c->order_dirty = true;
  }
  KF_CUDA(cudaStreamSynchronize(c->stream));
  int err = 0;
  KF_CUDA(cudaMemcpy(&err, c->d_err, 4, cudaMemcpyDeviceToHost));
  if (err) return fail(c, KF_E_DEVICE, "device error flag " + std::to_string(err) + " in admit");
  c->admitted = true;
  c->have_step = false;
  return KF_OK;
}

// the attention's sequence order for the current lengths (uploaded when
// prefill, admit or rewind changed them)
static int sync_order(kf_ctx* c) {
  if (!c->order_dirty) return KF_OK;
  const int B = c->B;
  c->h_order.resize(B);
  for (int b = 0; b < B; ++b) c->h_order[b] = b;
  std::stable_sort(c->h_order.begin(), c->h_order.end(),
                   [&](int32_t x, int32_t y) { return c->h_len[x] > c->h_len[y]; });
  KF_CUDA(cudaMemcpyAsync(c->d_order, c->h_order.data(), (size_t)B * 4, cudaMemcpyHostToDevice, c->stream));
  // the copy reads pageable memory: it has been staged when it returns
  c->order_dirty = false;
  return KF_OK;
}

int kf_teacher_step(kf_ctx* c, int32_t B, int32_t k, const float* noise, int32_t* out_tokens) {
  if (!c) return fail(nullptr, KF_E_ARG, "ctx is NULL");
  if (!c->have_batch) return fail(c, KF_E_STATE, "decode before prefill");
  if (B != c->B) return fail(c, KF_E_ARG, "B differs from the prefilled batch");
  if (k < 1 || k > c->max_k) return fail(c, KF_E_ARG, "k out of range 1..max_k");
  if (!noise || !out_tokens) return fail(c, KF_E_ARG, "noise or out_tokens is NULL");
  const int P = c->P;
  for (int b = 0; b < B; ++b)
    if (c->h_len[b] + P + k > c->cfg.max_len) return fail(c, KF_E_CAPACITY, "step would pass max_len");
  for (int b = 0; b < B; ++b) {
    bool dirty = false;
    KF_TRY(ensure_pages(c, b, c->h_len[b] + P + k - 1, &dirty));
    if (dirty) KF_TRY(upload_page_row(c, b));
  }
  KF_TRY(sync_order(c));
  // noise [B][k] -> [k][B]: sub-step j reads a contiguous column
  for (int j = 0; j < k; ++j)
    KF_CUDA(cudaMemcpy2DAsync(c->noise + (size_t)j * B, 4, noise + j, (size_t)k * 4, 4, B, cudaMemcpyDefault,
                              c->stream));
  // k AR sub-steps (Eq. 1 with k = 1, sequentially: the G* teacher of the
  // k-token joint), each token copied into column j of t_out
  auto enqueue = [&]() {
    for (int j = 0; j < k; ++j) {
      enqueue_step(c, B, j == 0 ? P : 1, 0, c->noise + (size_t)j * B);
      cudaMemcpy2DAsync(c->t_out + j, (size_t)k * 4, c->tokens, 4, 4, B, cudaMemcpyDeviceToDevice, c->stream);
    }
  };
  if (!(c->cfg.flags & KF_FLAG_NO_GRAPH)) {
    auto key = std::make_tuple((int)B, P, -(int)k);
    auto it = c->graphs.find(key);
    cudaGraphExec_t exec = nullptr;
    if (it == c->graphs.end()) {
      cudaGraph_t g = nullptr;
      KF_CUDA(cudaStreamBeginCapture(c->stream, cudaStreamCaptureModeThreadLocal));
      enqueue();
      cudaError_t e1 = enqueue_status(c);
      cudaError_t e2 = cudaStreamEndCapture(c->stream, &g);
      if (e1 != cudaSuccess) return cuda_fail(c, e1, "capture launch");
      if (e2 != cudaSuccess) return cuda_fail(c, e2, "cudaStreamEndCapture");
      cudaError_t e3 = cudaGraphInstantiate(&exec, g, 0);
      cudaGraphDestroy(g);
      if (e3 != cudaSuccess) return cuda_fail(c, e3, "cudaGraphInstantiate");
      c->graphs[key] = exec;
    } else {
      exec = it->second;
    }
    KF_CUDA(cudaGraphLaunch(exec, c->stream));
  } else {
    enqueue();
    KF_CUDA(enqueue_status(c));
  }
  KF_CUDA(cudaMemcpyAsync(out_tokens, c->t_out, (size_t)B * k * 4, cudaMemcpyDefault, c->stream));
  for (int b = 0; b < B; ++b) c->h_len[b] += P + k - 1;
  c->P = 1;
  c->last_nh = B;
  c->last_mtp = false;
  c->have_step = true;
  if (!is_device_ptr(out_tokens)) {
    KF_CUDA(cudaStreamSynchronize(c->stream));
    int err = 0;
    KF_CUDA(cudaMemcpy(&err, c->d_err, 4, cudaMemcpyDeviceToHost));
    if (err) return fail(c, KF_E_DEVICE, "device error flag " + std::to_string(err));
  }
  return KF_OK;
}

static int step_common(kf_ctx* c, int32_t B, int32_t k, const float* noise, int32_t* out_tokens,
                       bool profile) {
  if (!c) return fail(nullptr, KF_E_ARG, "ctx is NULL");
  if (!c->have_batch) return fail(c, KF_E_STATE, "decode before prefill");
  if (B != c->B) return fail(c, KF_E_ARG, "B differs from the prefilled batch");
  if (k < 0 || k > c->max_k) return fail(c, KF_E_ARG, "k out of range 0..max_k");
  if (c->mtp_k > 0 && k > 0 && k != c->mtp_k) return fail(c, KF_E_ARG, "an MTP model steps with k = 0 or mtp_k");
  if (!noise || !out_tokens) return fail(c, KF_E_ARG, "noise or out_tokens is NULL");
  const int P = c->P, nout = k > 0 ? k : 1;
  for (int b = 0; b < B; ++b)
    if (c->h_len[b] + P + k > c->cfg.max_len)
      return fail(c, KF_E_CAPACITY, "step would pass max_len");
  for (int b = 0; b < B; ++b) {
    bool dirty = false;
    KF_TRY(ensure_pages(c, b, c->h_len[b] + P + k - 1, &dirty));
    if (dirty) KF_TRY(upload_page_row(c, b));
  }
  KF_TRY(sync_order(c));
  KF_CUDA(cudaMemcpyAsync(c->noise, noise, (size_t)B * nout * 4, cudaMemcpyDefault, c->stream));
  bool use_graph = !profile && !(c->cfg.flags & KF_FLAG_NO_GRAPH);
  if (use_graph) {
    auto key = std::make_tuple((int)B, P, (int)k);
    auto it = c->graphs.find(key);
    cudaGraphExec_t exec = nullptr;
    if (it == c->graphs.end()) {
      cudaGraph_t g = nullptr;
      KF_CUDA(cudaStreamBeginCapture(c->stream, cudaStreamCaptureModeThreadLocal));
      enqueue_step(c, B, P, k, c->noise);
      cudaError_t e1 = enqueue_status(c);
      cudaError_t e2 = cudaStreamEndCapture(c->stream, &g);
      if (e1 != cudaSuccess) return cuda_fail(c, e1, "capture launch");
      if (e2 != cudaSuccess) return cuda_fail(c, e2, "cudaStreamEndCapture");
      cudaError_t e3 = cudaGraphInstantiate(&exec, g, 0);
      cudaGraphDestroy(g);
      if (e3 != cudaSuccess) return cuda_fail(c, e3, "cudaGraphInstantiate");
      c->graphs[key] = exec;
    } else {
      exec = it->second;
    }
    KF_CUDA(cudaGraphLaunch(exec, c->stream));
  } else {
    if (profile) {
      c->prof = true;
      c->ev_used = 0;
      if (c->ev.empty()) {
        c->ev.resize(4096);
        c->ev_kind.resize(2048);
        for (auto& ev : c->ev) KF_CUDA(cudaEventCreate(&ev));
      }
      // the profiled step replays as a graph with the event records as nodes,
      // so each event pair brackets its kernel and not the host's launch work
      cudaGraph_t g = nullptr;
      cudaGraphExec_t exec = nullptr;
      KF_CUDA(cudaStreamBeginCapture(c->stream, cudaStreamCaptureModeThreadLocal));
      enqueue_step(c, B, P, k, c->noise);
      c->prof = false;
      cudaError_t e1 = enqueue_status(c);
      cudaError_t e2 = cudaStreamEndCapture(c->stream, &g);
      if (e1 != cudaSuccess && g) cudaGraphDestroy(g);
      if (e1 != cudaSuccess) return cuda_fail(c, e1, "profile capture");
      if (e2 != cudaSuccess) return cuda_fail(c, e2, "profile cudaStreamEndCapture");
      cudaError_t e3 = cudaGraphInstantiate(&exec, g, 0);
      cudaGraphDestroy(g);
      if (e3 != cudaSuccess) return cuda_fail(c, e3, "profile cudaGraphInstantiate");
      cudaError_t e4 = cudaGraphLaunch(exec, c->stream);
      cudaError_t e5 = cudaStreamSynchronize(c->stream);
      cudaGraphExecDestroy(exec);
      if (e4 != cudaSuccess) return cuda_fail(c, e4, "profile cudaGraphLaunch");
      if (e5 != cudaSuccess) return cuda_fail(c, e5, "profile step");
    } else {
      enqueue_step(c, B, P, k, c->noise);
      KF_CUDA(enqueue_status(c));
    }
  }
  KF_CUDA(cudaMemcpyAsync(out_tokens, c->tokens, (size_t)B * nout * 4, cudaMemcpyDefault, c->stream));
  for (int b = 0; b < B; ++b) c->h_len[b] += P;
  c->P = nout;
  c->last_nh = B * nout;
  c->last_mtp = c->mtp_k > 0 && k > 0;
  c->have_step = true;
  if (!is_device_ptr(out_tokens)) {
    KF_CUDA(cudaStreamSynchronize(c->stream));
    int err = 0;
    KF_CUDA(cudaMemcpy(&err, c->d_err, 4, cudaMemcpyDeviceToHost));
    if (err) return fail(c, KF_E_DEVICE, "device error flag " + std::to_string(err));
  }
  return KF_OK;
}

int kf_decode_step(kf_ctx* c, int32_t B, int32_t k, const float* noise, int32_t* out_tokens) {
  return step_common(c, B, k, noise, out_tokens, false);
}

int kf_profile_step(kf_ctx* c, int32_t B, int32_t k, const float* noise, int32_t* out_tokens,
                    float* ms_per_kind, int32_t* launches_per_kind) {
  if (!c) return fail(nullptr, KF_E_ARG, "ctx is NULL");
  if (!ms_per_kind || !launches_per_kind) return fail(c, KF_E_ARG, "profile outputs are NULL");
  int r = step_common(c, B, k, noise, out_tokens, true);
  if (r != KF_OK) return r;
  KF_CUDA(cudaStreamSynchronize(c->stream));
  for (int i = 0; i < KF_KIND_COUNT; ++i) { ms_per_kind[i] = 0.f; launches_per_kind[i] = 0; }
  for (int i = 0; i < c->ev_used / 2; ++i) {
    float ms = 0.f;
    KF_CUDA(cudaEventElapsedTime(&ms, c->ev[2 * i], c->ev[2 * i + 1]));
    int kd = c->ev_kind[i];
    ms_per_kind[kd] += ms;
    launches_per_kind[kd] += 1;
  }
  return KF_OK;
}

int kf_debug_logits(kf_ctx* c, float* out) {
  if (!c) return fail(nullptr, KF_E_ARG, "ctx is NULL");
  if (!c->have_step) return fail(c, KF_E_STATE, "no decode step yet");
  if (!out) return fail(c, KF_E_ARG, "out is NULL");
  const int nh = c->last_nh;
  float* dst = out;
  float* tmp = nullptr;
  bool dev = is_device_ptr(out);
  if (!dev) {
    KF_CUDA(cudaMalloc(&tmp, (size_t)nh * c->V * 4));
    dst = tmp;
  }
  if (c->last_mtp) {
    // head j of the B noise rows -> out[b][j][V]
    const int kk = nh / c->B;
    for (int j = 0; j < kk; ++j) {
      Epi e;
      e.kind = EPI_LOGITS; e.outf = dst + (size_t)j * c->V; e.ldo = kk * c->V;
      e.inv_tau = 1.0f / c->cfg.tau; e.n_valid = c->V;
      gemm(c, KF_KIND_GEMM_HEAD, c->B, c->V_pad, c->d, c->head_in, c->d,
           static_cast<const char*>(c->w_mtp) + (size_t)j * c->V_pad * c->d * c->esz, c->d, e);
    }
  } else {
    Epi e;
    e.kind = EPI_LOGITS; e.outf = dst; e.ldo = c->V; e.inv_tau = 1.0f / c->cfg.tau; e.n_valid = c->V;
    gemm(c, KF_KIND_GEMM_HEAD, nh, c->V_pad, c->d, c->head_in, c->d, c->w_head, c->d, e);
  }
  cudaError_t err = enqueue_status(c);
  if (err == cudaSuccess && !dev)
    err = cudaMemcpyAsync(out, tmp, (size_t)nh * c->V * 4, cudaMemcpyDeviceToHost, c->stream);
  if (err == cudaSuccess) err = cudaStreamSynchronize(c->stream);
  if (tmp) cudaFree(tmp);
  if (err != cudaSuccess) return cuda_fail(c, err, "debug logits");
  return KF_OK;
}

int kf_rewind(kf_ctx* c) {
  if (!c) return fail(nullptr, KF_E_ARG, "ctx is NULL");
  if (!c->have_batch) return fail(c, KF_E_STATE, "rewind before prefill");
  if (c->admitted) return fail(c, KF_E_STATE, "rewind after kf_admit (no snapshot of admitted slots)");
  KF_CUDA(cudaMemcpyAsync(c->d_len, c->d_len0, c->B * 4, cudaMemcpyDeviceToDevice, c->stream));
  KF_CUDA(cudaMemcpyAsync(c->d_pending, c->d_pending0, (size_t)c->B * c->pend_stride * 4,
                          cudaMemcpyDeviceToDevice, c->stream));
  c->h_len = c->h_len0;
  c->order_dirty = true;
  c->P = 1;
  c->have_step = false;
  return KF_OK;
}

int kf_get_lengths(const kf_ctx* c, int32_t* lens_out) {
  if (!c || !lens_out) return fail(nullptr, KF_E_ARG, "NULL argument");
  for (int b = 0; b < c->B; ++b) lens_out[b] = c->h_len[b];
  return KF_OK;
}

int kf_set_stream(kf_ctx* c, void* stream) {
  if (!c) return fail(nullptr, KF_E_ARG, "ctx is NULL");
  KF_CUDA(cudaStreamSynchronize(c->stream));
  if (c->own_stream) cudaStreamDestroy(c->stream);
  c->own_stream = false;
  if (stream) {
    c->stream = (cudaStream_t)stream;
  } else {
    KF_CUDA(cudaStreamCreate(&c->stream));
    c->own_stream = true;
  }
  return KF_OK;
}

int kf_sync(kf_ctx* c) {
  if (!c) return fail(nullptr, KF_E_ARG, "ctx is NULL");
  KF_CUDA(cudaStreamSynchronize(c->stream));
  int err = 0;
  KF_CUDA(cudaMemcpy(&err, c->d_err, 4, cudaMemcpyDeviceToHost));
  if (err) return fail(c, KF_E_DEVICE, "device error flag " + std::to_string(err));
  return KF_OK;
}

int kf_free(kf_ctx* c) {
  if (!c) return KF_OK;
  if (c->stream) cudaStreamSynchronize(c->stream);
  for (auto& kv : c->graphs) cudaGraphExecDestroy(kv.second);
  for (auto ev : c->ev) cudaEventDestroy(ev);
  for (void* p : c->allocs) cudaFree(p);
  if (c->h_page_table) cudaFreeHost(c->h_page_table);
  if (c->own_stream && c->stream) cudaStreamDestroy(c->stream);
  delete c;
  return KF_OK;
}

const char* kf_last_error(const kf_ctx* c) {
  if (c) return c->err.c_str();
  return g_err.c_str();
}

}  // extern "C"
