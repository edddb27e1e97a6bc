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

/*
 * out[M][N] = A[M][K] . W[N][K]^T in fp32: the dense projections of the
 * backbone (Table 4: QKV, O, MLP) and the LM head are this contraction.
 * A, W: bf16, row-major, rows 16-byte aligned; K a multiple of 64 for
 * KF_GEMM_TCGEN05.  out: fp32 row-major [M][N].  The first call allocates a
 * split-K workspace that lives until process exit.  Errors: KF_E_ARG
 * (shapes / alignment), KF_E_CUDA.
 */
int kf_op_gemm_bf16(int32_t impl, int32_t M, int32_t N, int32_t K, const void* A, const void* W,
                    float* out, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* KFORCING_OPS_H */
