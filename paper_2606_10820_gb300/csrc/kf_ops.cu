// Single-kernel entry points (include/kforcing_ops.h).
#include "../../include/kforcing_ops.h"
#include "kf_internal.cuh"

using namespace kf;

namespace {
void* g_ws = nullptr;
int* g_counters = nullptr;
int* g_err = nullptr;
constexpr size_t kWsBytes = (size_t)64 << 20;
constexpr int kCounters = 8192;
}  // namespace

extern "C" int kf_op_gemm_bf16(int32_t impl, int32_t M, int32_t N, int32_t K, const void* A,
                               const void* W, float* out, void* stream) {
  if (M <= 0 || N <= 0 || K <= 0 || !A || !W || !out) return KF_E_ARG;
  GemmDesc g{M, N, K, A, K, W, K, Epi{}};
  g.epi.kind = EPI_STORE_F32;
  g.epi.outf = out;
  g.epi.ldo = N;
  cudaStream_t s = (cudaStream_t)stream;
  if (impl == KF_GEMM_TCGEN05) {
    if (!tc_gemm_supported(g)) return KF_E_ARG;
    if (!g_ws) {
      if (cudaMalloc(&g_ws, kWsBytes) != cudaSuccess ||
          cudaMalloc(&g_counters, kCounters * sizeof(int)) != cudaSuccess ||
          cudaMalloc(&g_err, sizeof(int)) != cudaSuccess ||
          cudaMemset(g_counters, 0, kCounters * sizeof(int)) != cudaSuccess ||
          cudaMemset(g_err, 0, sizeof(int)) != cudaSuccess)
        return KF_E_CUDA;
    }
    if (launch_gemm_tc(g, g_ws, kWsBytes, g_counters, kCounters, g_err, s) != 0) return KF_E_CUDA;
  } else if (impl == KF_GEMM_SIMT) {
    launch_gemm_simt(true, g, s);
  } else {
    return KF_E_ARG;
  }
  return cudaGetLastError() == cudaSuccess ? KF_OK : KF_E_CUDA;
}
