/*
 * kforcing_ops.h - single-kernel entry points of libkforcing.so, for
 * kernel-level parity tests and per-kernel timing.  Device pointers only;
 * work is enqueued on `stream` (cudaStream_t, NULL = legacy default).
 * Return KF_OK or a negative KF_E_* status (see kforcing.h).
 */
#ifndef KFORCING_OPS_H
#define KFORCING_OPS_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define KF_GEMM_TCGEN05 0   /* tcgen05 + TMEM tensor-core kernel, TMA fed   */
#define KF_GEMM_SIMT 1      /* CUDA-core kernel, fp32 FMA in ascending k    */
#define KF_GEMM_TCGEN05_PER_TILE 2 /* the tcgen05 kernel with one CTA per tile
                                      even past a wave of tiles            */
#define KF_GEMM_SKINNY 3    /* M <= 64: warp-level MMA, 16 columns per CTA,
                               K split over a cluster (the decode step at
                               small batch)                                */

/*
 * out[M][N] = A[M][K] . W[N][K]^T in fp32: the dense projections of the
 * backbone (Table 4: QKV, O, MLP) and the LM head are this contraction.
 * A, W: bf16, row-major, rows 16-byte aligned; K a multiple of 64 for
 * KF_GEMM_TCGEN05 and KF_GEMM_SKINNY (which also needs M <= 64), N a
 * multiple of 4.  out: fp32 row-major [M][N].  The first
 * call on a device allocates a 4-byte device error word for that device that
 * lives until process exit; each call clears it on `stream` before its
 * kernel runs, and the kernel ORs its error bits into it (a bounded
 * pipeline wait that ran out).  Asynchronous: kf_op_status(stream) reports
 * those errors.  Errors: KF_E_ARG (shapes / alignment), KF_E_CUDA.
 */
int kf_op_gemm_bf16(int32_t impl, int32_t M, int32_t N, int32_t K, const void* A, const void* W,
                    float* out, void* stream);

/*
 * The LM head and its noise -> token map for `rows` normalised head rows,
 * without writing logits to memory: l = x . w_head^T / tau with bf16
 * operands and fp32 accumulation on the tensor cores; per 32-id chunk the
 * maximum, sum of exp(l - max) and first argmax go to a record scratch
 * buffer; then per row the token for noise[row]:
 *   KF_MAP_ICDF:   the least id whose running softmax mass exceeds
 *                  noise[row] (Eq. 1 with App. B's strict '>', Eq. icdf);
 *   KF_MAP_ARGMAX: the lowest id of maximal logit (Alg. 1's arg max).
 * x: bf16 [rows][d], w_head: bf16 [V][d], both row-major with 16-byte
 * aligned rows, d a multiple of 64; noise: fp32 [rows] in [0,1);
 * tokens: int32 [rows].  All device pointers.  The record scratch
 * (rows x ceil(V/32) x 16 bytes) is allocated with cudaMalloc on first use
 * on each device and grown when a call needs more (growth first waits for
 * the whole device); it lives until process exit.  Host threads are
 * serialised around the buffer, but calls whose work overlaps on the GPU
 * (several streams) share it and race.  Asynchronous: the call clears the
 * device's op error word on `stream`; when a kernel of the call flags an
 * error (a bounded wait ran out, so records may be stale) every token is -1
 * and kf_op_status(stream) returns KF_E_DEVICE.
 * Errors: KF_E_ARG, KF_E_OOM, KF_E_CUDA.
 */
int kf_op_head_tokens(int32_t rows, int32_t V, int32_t d, const void* x, const void* w_head,
                      const float* noise, float tau, int32_t map_kind, int32_t* tokens,
                      void* stream);

/*
 * kf_op_head_tokens_noalloc: the same computation as kf_op_head_tokens, for
 * callers that must not allocate device memory, for instance code whose
 * device memory is fully owned by another allocator or budgeted up front,
 * or a loop that cannot afford the device-wide synchronisation cudaMalloc and
 * cudaFree may cause.  It calls no cudaMalloc, cudaFree or other allocating
 * routine.  The paper has no counterpart: this is a deployment variant.
 *
 * Scratch: the chunk records live in a fixed array inside the library's
 * device image, KF_NOALLOC_MAX_RECORDS records of 16 bytes (4 MiB) plus an
 * error word; every GPU that loads the library holds it until the process
 * exits.  A call needs rows * ceil(V/32) records; larger calls are rejected
 * with KF_E_CAPACITY (kf_last_error(NULL) says why) before anything runs.
 * The first call on each device, made with that device current, looks up the
 * array's device address (cudaGetSymbolAddress); make that first call before
 * any stream capture.  All calls share the one array: calls whose work
 * overlaps on the GPU (different streams, or other threads) race on it.
 * Its error word is also static and cleared at the start of each call; when
 * a kernel of the call flags an error every token is -1, and
 * kf_op_status(stream) reports it without allocating.
 * Arguments, layouts and the other errors are those of kf_op_head_tokens.
 */
#define KF_NOALLOC_MAX_RECORDS 262144
int kf_op_head_tokens_noalloc(int32_t rows, int32_t V, int32_t d, const void* x,
                              const void* w_head, const float* noise, float tau,
                              int32_t map_kind, int32_t* tokens, void* stream);

/*
 * Device errors of the entry points above on the current device: waits for
 * `stream`, then reads and clears the error word of the allocating entries
 * (the last kf_op_gemm_bf16 / kf_op_head_tokens call on this device) and the
 * static one of kf_op_head_tokens_noalloc (its last call).  Returns KF_OK,
 * KF_E_DEVICE when a kernel flagged an error (kf_last_error(NULL) gives the
 * bits), or KF_E_CUDA.  Allocates nothing.
 */
int kf_op_status(void* stream);

/*
 * Training-time attention of K-Forcing (App. C.2): SingleForward (blocks = 1)
 * or DoubleForward (blocks = 2) in one call, for B sequences and H heads of
 * head_dim 64.
 *   Token layout of a sequence (T = N + blocks * N * k tokens): context
 *   x_1..x_N at 0..N-1, then `blocks` blocks of N*k tokens, k per context
 *   position; token (t, a) of block b (t = 0..N-1, a = 0..k-1) at
 *   N + (b-1) N k + t k + a.  SingleForward's block 1 holds the noise
 *   tokens; DoubleForward's blocks hold the first-round predictions
 *   (Future-1) and the fresh noise (Future-2).
 *   Mask: a context row i sees context keys 0..i; a block-1 row (t, a) sees
 *   context 0..t and block-1 tokens (t, 0..a); a block-2 row (t, a) sees
 *   context 0..t, all k block-1 tokens of window t and block-2 tokens
 *   (t, 0..a) -- M_S and M_D of App. C.2.
 * q, kk, v: [B][T][H][64] bf16, device, 16-byte aligned.  Queries are the rows
 * [q_begin, q_end) of the layout (0..T for the whole mask; N + N k .. T for
 * Future-2 alone, reusing the other rows' keys).  out: [B][q_end - q_begin][H][64]
 * fp32, device, caller-owned.  Scale 1/sqrt(64), fp32 softmax, probabilities
 * rounded to bf16 for the P.V product.
 * dense: flags.  Without KF_TRAIN_ATTN_DENSE only the key tiles a query tile
 * can see are visited (the context prefix and its windows: O(k) pairs
 * relative to AR attention); with it every key tile, with the same mask (the
 * cost of a dense mask, for comparison).  The kernel runs on tcgen05 (S and
 * O in tensor memory, 128 query rows and 128-key tiles per step);
 * KF_TRAIN_ATTN_WARP_MMA selects the warp-level MMA kernel instead (64 query
 * rows, 64-key tiles), for comparison.
 * Errors: KF_E_ARG (sizes, ranges, alignment, unknown flags), KF_E_CUDA.
 * Asynchronous on `stream` (NULL: the default stream); a bounded wait that
 * ran out inside the tcgen05 kernel is reported by kf_op_status (KF_E_DEVICE).
 */
#define KF_TRAIN_ATTN_DENSE 1
#define KF_TRAIN_ATTN_WARP_MMA 2
int kf_op_train_attention(int32_t blocks, int32_t B, int32_t H, int32_t N, int32_t k,
                          int32_t q_begin, int32_t q_end, const void* q, const void* kk,
                          const void* v, float* out, int32_t dense, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* KFORCING_OPS_H */
