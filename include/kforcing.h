/*
 * kforcing.h - C ABI of the GB300 (sm_103a) K-Forcing decode library.
 *
 * The library runs the batched joint next-k-token decode step of a
 * push-forward causal Transformer (Sec. 3.1: G_theta maps a context and k
 * i.i.d. U(0,1) noise values to k tokens in one forward pass; Sec. 3.3: the
 * fully causal architecture, one noise token per slot, shared head; App. C.1,
 * Alg. 1: KV-cached inference where each step feeds the P pending committed
 * tokens plus k noise tokens, keeps the context KV and discards the noise KV).
 *
 * Conventions for every call:
 *   - Return value: KF_OK (0) or a negative KF_E_* status.  On error
 *     kf_last_error() describes it.  Argument errors are detected on the host
 *     before anything is enqueued.
 *   - All GPU work is enqueued on the stream given to kf_init (or
 *     kf_set_stream).  Caller buffers are borrowed for the duration of the
 *     call only; the library copies what it keeps.
 *   - Pointers marked "host or device" are classified with
 *     cudaPointerGetAttributes: device (or managed) memory is read/written by
 *     the GPU directly; host memory is copied inside the call, and a call that
 *     writes host memory synchronises the stream before returning.
 *   - A context is not thread-safe; one host thread drives it at a time.
 */
#ifndef KFORCING_H
#define KFORCING_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* status codes */
#define KF_OK 0
#define KF_E_ARG (-1)            /* bad argument (checked on the host)          */
#define KF_E_CAPACITY (-2)       /* a sequence would pass max_len, or no pages  */
#define KF_E_OOM (-3)            /* device allocation failed                    */
#define KF_E_CUDA (-4)           /* a CUDA runtime call failed                  */
#define KF_E_DEVICE (-5)         /* a kernel flagged an invalid index / timeout */
#define KF_E_STATE (-6)          /* call out of order (e.g. decode before prefill) */

/* kf_config.pos_kind */
#define KF_POS_ROPE 0            /* rotary positions on q, k (Table 4)          */
#define KF_POS_LEARNED 1         /* learned absolute position table             */
/* kf_config.dtype: storage type of weights, activations fed to GEMMs and KV */
#define KF_DTYPE_FP32 0          /* fp32 everywhere (exact-token parity mode)   */
#define KF_DTYPE_BF16 1          /* bf16 storage, fp32 accumulation/softmax     */
/* kf_config.map_kind: the noise -> token map at the noise slots */
#define KF_MAP_ICDF 0            /* inverse CDF of softmax(logits/tau), Eq. 1   */
#define KF_MAP_ARGMAX 1          /* greedy head of the learned PFLM (Alg. 1)    */
/* kf_config.flags */
#define KF_FLAG_NO_GRAPH 1       /* launch kernels eagerly instead of replaying a CUDA graph */
#define KF_FLAG_SIMT_GEMM 2      /* bf16 mode: use the SIMT GEMM, not tcgen05   */
#define KF_FLAG_NO_PDL 4         /* launch without programmatic dependent launch */
#define KF_FLAG_NO_PERSISTENT_GEMM 16 /* bf16: one CTA per output tile even when the
                                    tiles exceed a wave (no persistent tile loop) */
#define KF_FLAG_NO_SKINNY 32     /* bf16: keep the tcgen05 GEMMs for calls of at most
                                    64 rows (no skinny warp-MMA projections)     */

/*
 * Model and runtime configuration.  Table 4 gives the backbone (pre-norm
 * RMSNorm decoder, RoPE d_rot = head_dim = 64) and the noise encoder
 * (sinusoidal encoding of z and tau, then a two-layer GELU MLP).
 */
typedef struct kf_config {
  int32_t n_layer;      /* L                                                  */
  int32_t d_model;      /* d; head_dim = d_model / n_head must be 32 or 64    */
  int32_t n_head;       /* H                                                  */
  int32_t d_ff;         /* MLP width F                                        */
  int32_t vocab;        /* V                                                  */
  int32_t max_len;      /* longest sequence, prompt + generated (positions)   */
  int32_t noise_hidden; /* NoiseEnc hidden width; 0 => 4 * d_model            */
  int32_t pos_kind;     /* KF_POS_*                                           */
  int32_t dtype;        /* KF_DTYPE_*                                         */
  int32_t map_kind;     /* KF_MAP_*                                           */
  int32_t max_batch;    /* most sequences in one batch                        */
  int32_t max_k;        /* most noise slots per step, 1..8                    */
  int32_t page_size;    /* tokens per KV page; must be 16                     */
  int32_t n_pages;      /* KV pool size in pages; 0 => enough for max_batch
                           sequences of max_len tokens                        */
  int32_t prefill_rows; /* rows per prefill chunk; 0 => 4096                  */
  int32_t flags;        /* KF_FLAG_*                                          */
  float tau;            /* temperature: logits are divided by tau (> 0)       */
  float rms_eps;        /* RMSNorm epsilon                                    */
  float rope_theta;     /* RoPE base                                          */
  float noise_scale;    /* sinusoid argument = noise_scale * z                */
  int32_t mtp_k;        /* 0: the fully causal model (k noise tokens, one
                           shared head); > 0: the standard MTP variant (Sec.
                           3.3) with mtp_k heads: a k-step (k = mtp_k) feeds
                           one noise-conditioning token whose NoiseEnc input
                           is the k values' sinusoidal features concatenated
                           (k * d wide), and head j maps its hidden state
                           with noise[b][j].  mtp_k <= max_k.               */
} kf_config;

/*
 * Weights, fp32, row-major, nn.Linear layout ([out_features][in_features]).
 * Host or device pointers (all of one kind).  kf_init copies and converts
 * them (to bf16 with round-to-nearest-even in bf16 mode); the caller keeps
 * ownership.  wqkv rows are [q; k; v], head h of each at rows h*64..h*64+63.
 */
typedef struct kf_weights {
  const float* tok_emb;     /* [V][d]                                  */
  const float* pos_emb;     /* [max_len][d]; NULL unless KF_POS_LEARNED */
  const float* attn_norm;   /* [L][d]                                  */
  const float* wqkv;        /* [L][3d][d]                              */
  const float* wo;          /* [L][d][d]                               */
  const float* mlp_norm;    /* [L][d]                                  */
  const float* w_up;        /* [L][F][d]                               */
  const float* w_down;      /* [L][d][F]                               */
  const float* final_norm;  /* [d]                                     */
  const float* w_head;      /* [V][d] (untied)                         */
  const float* ne_w1;       /* [noise_hidden][d] ([noise_hidden][mtp_k d] for MTP) */
  const float* ne_b1;       /* [noise_hidden]                          */
  const float* ne_w2;       /* [d][noise_hidden]                       */
  const float* ne_b2;       /* [d]                                     */
  const float* w_mtp;       /* [mtp_k][V][d], the MTP heads; NULL unless mtp_k > 0 */
} kf_weights;

typedef struct kf_ctx kf_ctx;

/*
 * Create a context on the current CUDA device: validate cfg, allocate the
 * weights, the paged KV pool and all workspaces, and copy w.  stream is a
 * cudaStream_t (NULL = legacy default stream).  *out receives the context
 * (NULL on failure).  Errors: KF_E_ARG, KF_E_OOM, KF_E_CUDA.
 */
int kf_init(const kf_config* cfg, const kf_weights* w, void* stream,
            kf_ctx** out);

/*
 * Start B sequences (Alg. 1 REQUIRE: prompt tokens x_{1:N}).  tokens is the
 * concatenation of the B prompts (host or device, int32 ids in [0, V)),
 * lens[b] >= 1 their lengths (host).  The KV of every prompt token but the
 * last is computed and cached; the last token of each prompt becomes its one
 * pending token.  Any earlier batch is dropped, and the context's device
 * error word is cleared (collect earlier asynchronous errors with kf_sync
 * first).  Synchronises.  Host prompts are range-checked before any launch
 * (KF_E_ARG); device-resident prompts are checked by the embedding kernel:
 * an id outside [0, V) is embedded as id 0, flags the error word, and the
 * call returns KF_E_DEVICE (the batch is then unusable until the next
 * kf_prefill).  Errors: KF_E_ARG, KF_E_CAPACITY (a prompt is longer than
 * max_len - 1, or the pool is full), KF_E_CUDA, KF_E_DEVICE.
 */
int kf_prefill(kf_ctx* ctx, int32_t B, const int32_t* tokens,
               const int32_t* lens);

/*
 * One decode step (Alg. 1 loop body) for all B sequences of the batch.
 *   k >= 1: the push-forward step.  Each sequence feeds its P pending tokens
 *           and k noise slots; slot j's token is the noise -> token map of
 *           its logits with noise[b][j].  Emits k tokens per sequence.
 *   k == 0: the AR teacher step (Eq. 1 with one token): the last pending
 *           row's logits mapped with noise[b][0].  Emits 1 token.
 *   MTP models (mtp_k > 0): k must be 0 or mtp_k; the k-step feeds the P
 *           pending tokens and one noise token, and head j maps the noise
 *           token's hidden state with noise[b][j].  Emits k tokens.
 * noise:      [B][max(k,1)] fp32 in [0,1), host or device.
 * out_tokens: [B][max(k,1)] int32, host or device, caller-owned.
 * Afterwards each sequence's cache holds P more tokens and the emitted tokens
 * are its pending tokens (fixed stride, App. C.1).  B must equal the prefilled
 * batch and k <= max_k.  Errors: KF_E_ARG, KF_E_STATE, KF_E_CAPACITY,
 * KF_E_CUDA, KF_E_DEVICE.  A call with host out_tokens synchronises and
 * reports the device error word; with device out_tokens it returns after
 * enqueueing, and kf_sync reports the word.  Once a kernel has flagged an
 * error (a bounded wait ran out, an invalid page or token id), the token
 * map writes -1 for every slot of that and every later step until the next
 * kf_prefill.
 */
int kf_decode_step(kf_ctx* ctx, int32_t B, int32_t k, const float* noise,
                   int32_t* out_tokens);

/*
 * The k-pass teacher G* (App. B, Eq. sequential-icdf): k AR steps (Eq. 1
 * with one token each) in one call, the j-th mapping the AR distribution
 * conditioned on the cache, the pending tokens and the j-1 tokens drawn
 * before it with noise[b][j].  The first sub-step feeds the P pending
 * tokens, the later ones the token just drawn.  This is the target map the
 * push-forward step learns; a caller uses it to produce teacher samples or to
 * compare the joint step with the AR chain on the same noise.
 * noise:      [B][k] fp32 in [0,1), host or device.
 * out_tokens: [B][k] int32, host or device, caller-owned.
 * Afterwards each cache holds P + k - 1 more tokens and the last drawn token
 * is the one pending token.  1 <= k <= max_k.  Tokens equal those of k
 * kf_decode_step calls with k = 0 on the same noise columns.  Errors as
 * kf_decode_step.
 */
int kf_teacher_step(kf_ctx* ctx, int32_t B, int32_t k, const float* noise,
                    int32_t* out_tokens);

/*
 * Continuous batching (App. C.1, KV-cached inference): at a step boundary,
 * replace the n sequences slots[0..n) (distinct, 0 <= slot < B) by new
 * prompts.  tokens is the concatenation of the n prompts (host or device),
 * lens[i] their lengths (host).  The replaced sequences' KV pages return to
 * the pool (recycled by later allocations); each new prompt is admitted with
 * its first len - P tokens cached (one chunked prefill pass over all of
 * them) and its last P tokens pending, P being the batch's current pending
 * count, so every sequence keeps the same stride and the next kf_decode_step
 * serves it like the others.  Synchronises.  lens[i] >= max(1, P).  After
 * an admission kf_rewind is refused (KF_E_STATE) until the next kf_prefill.
 * Errors: KF_E_ARG, KF_E_STATE, KF_E_CAPACITY (pool exhausted, or a prompt
 * longer than max_len - 1), KF_E_CUDA, KF_E_DEVICE.
 */
int kf_admit(kf_ctx* ctx, int32_t n, const int32_t* slots, const int32_t* tokens,
             const int32_t* lens);

/*
 * Parity aid: recompute the last decode step's head logits (logits / tau,
 * fp32) for its B * max(k,1) mapped rows into out [B][max(k,1)][V] (host or
 * device).  The logits come from the same normalised rows and head weights
 * the step used.  Errors: KF_E_STATE (no step yet), KF_E_ARG.
 */
int kf_debug_logits(kf_ctx* ctx, float* out);

/*
 * Restore every sequence to the state right after the last kf_prefill
 * (lengths and pending tokens).  The prompt's cached KV is reused: decode
 * steps only write positions at or after each prompt's last token, whose KV
 * is recomputed identically.  Lets a caller replay a generation.
 */
int kf_rewind(kf_ctx* ctx);

/* Cached lengths (tokens whose KV is in the cache) of the B sequences. */
int kf_get_lengths(const kf_ctx* ctx, int32_t* lens_out);

/* Enqueue subsequent work on another stream (cudaStream_t). */
int kf_set_stream(kf_ctx* ctx, void* stream);

/* Synchronise the context's stream and report any device-side error flag. */
int kf_sync(kf_ctx* ctx);

/*
 * Profiling aid: run one decode step like kf_decode_step, as a one-off CUDA
 * graph with an event record node on each side of every launch (launches in
 * order, without programmatic dependent launch).  ms_per_kind[i] and launches_per_kind[i]
 * (arrays of KF_KIND_COUNT, host) receive the summed device time and launch
 * count per kernel kind.  Synchronises.  The step's first kernel (row maps,
 * pending-token embeddings and noise features in one launch) is counted under
 * KF_KIND_EMBED, and the step's commit is taken by the token selection
 * (KF_KIND_HEAD_SELECT); KF_KIND_ROWMAP and KF_KIND_COMMIT stay at zero
 * launches.
 */
#define KF_KIND_ROWMAP 0
#define KF_KIND_EMBED 1
#define KF_KIND_NOISE_GEMM 2
#define KF_KIND_RMSNORM 3
#define KF_KIND_GEMM_QKV 4
#define KF_KIND_ROPE_KV 5
#define KF_KIND_ATTENTION 6
#define KF_KIND_ATTN_COMBINE 7
#define KF_KIND_GEMM_O 8
#define KF_KIND_GEMM_UP 9
#define KF_KIND_GEMM_DOWN 10
#define KF_KIND_HEAD_NORM 11
#define KF_KIND_GEMM_HEAD 12
#define KF_KIND_HEAD_SELECT 13
#define KF_KIND_COMMIT 14
#define KF_KIND_COUNT 15
int kf_profile_step(kf_ctx* ctx, int32_t B, int32_t k, const float* noise,
                    int32_t* out_tokens, float* ms_per_kind,
                    int32_t* launches_per_kind);

/* Release everything the context owns.  Accepts NULL. */
int kf_free(kf_ctx* ctx);

/* Message for the last failed call on ctx (or of the last failed kf_init
 * on this thread when ctx is NULL).  Never NULL. */
const char* kf_last_error(const kf_ctx* ctx);

#ifdef __cplusplus
}
#endif

#endif /* KFORCING_H */
