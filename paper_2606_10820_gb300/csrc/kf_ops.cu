// Single-kernel entry points (include/kforcing_ops.h).
#include <mutex>
#include <string>

#include "../../include/kforcing_ops.h"
#include "kf_internal.cuh"

using namespace kf;

namespace {
int* g_err = nullptr;
HeadRec* g_rec = nullptr;
size_t g_rec_bytes = 0;

int ensure_err() {
  if (g_err) return KF_OK;
  if (cudaMalloc(&g_err, sizeof(int)) != cudaSuccess || cudaMemset(g_err, 0, sizeof(int)) != cudaSuccess)
    return KF_E_CUDA;
  return KF_OK;
}
}  // namespace

// the LM-head GEMM with the chunk-record epilogue, then the token select
static int head_tokens(int32_t rows, int32_t V, int32_t d, const void* x, const void* w_head,
                       const float* noise, float tau, int32_t map_kind, int32_t* tokens,
                       HeadRec* rec, int* err, cudaStream_t s) {
  const int nchunk = ceil_div(V, kChunk);
  GemmDesc g{rows, V, d, x, d, w_head, d, Epi{}};
  g.epi.kind = EPI_HEAD;
  g.epi.inv_tau = 1.0f / tau;
  g.epi.n_valid = V;
  g.epi.rec = rec;
  g.epi.nchunk = nchunk;
  if (!tc_gemm_supported(g)) return KF_E_ARG;
  if (launch_gemm_tc(g, err, s) != 0) return KF_E_CUDA;
  launch_head_select(true, rows, rec, nchunk, x, d, w_head, V, 1.0f / tau, map_kind, noise, tokens, 0, 0, s);
  return cudaGetLastError() == cudaSuccess ? KF_OK : KF_E_CUDA;
}

static bool head_args_ok(int32_t rows, int32_t V, int32_t d, const void* x, const void* w,
                         const float* noise, float tau, int32_t map_kind, const int32_t* tokens) {
  return rows > 0 && V > 0 && d > 0 && d % 64 == 0 && x && w && noise && tokens && tau > 0.f &&
         (map_kind == KF_MAP_ICDF || map_kind == KF_MAP_ARGMAX);
}

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
    if (ensure_err() != KF_OK) return KF_E_CUDA;
    if (launch_gemm_tc(g, g_err, s) != 0) return KF_E_CUDA;
  } else if (impl == KF_GEMM_SIMT) {
    launch_gemm_simt(true, g, s);
  } else {
    return KF_E_ARG;
  }
  return cudaGetLastError() == cudaSuccess ? KF_OK : KF_E_CUDA;
}

extern "C" int kf_op_head_tokens(int32_t rows, int32_t V, int32_t d, const void* x,
                                 const void* w_head, const float* noise, float tau,
                                 int32_t map_kind, int32_t* tokens, void* stream) {
  if (!head_args_ok(rows, V, d, x, w_head, noise, tau, map_kind, tokens)) return KF_E_ARG;
  if (ensure_err() != KF_OK) return KF_E_CUDA;
  const size_t need = (size_t)rows * ceil_div(V, kChunk) * sizeof(HeadRec);
  if (need > g_rec_bytes) {
    cudaStream_t s = (cudaStream_t)stream;
    if (g_rec) {
      cudaStreamSynchronize(s);   // a pending call may still read the old buffer
      cudaFree(g_rec);
      g_rec = nullptr;
      g_rec_bytes = 0;
    }
    if (cudaMalloc(&g_rec, need) != cudaSuccess) {
      cudaGetLastError();
      return KF_E_OOM;
    }
    g_rec_bytes = need;
  }
  return head_tokens(rows, V, d, x, w_head, noise, tau, map_kind, tokens, g_rec, g_err,
                     (cudaStream_t)stream);
}

// ------------------------------------------------- no-allocation variant
// Scratch for callers that cannot allocate device memory: a fixed array in
// the library's own device image.  Every device that loads the library holds
// it (4 MiB of records plus an error word) until the process exits.
static __device__ __align__(256) HeadRec g_noalloc_rec[KF_NOALLOC_MAX_RECORDS];
static __device__ __align__(256) int g_noalloc_err;

namespace {
constexpr int kMaxDevices = 64;
struct NoAllocScratch {
  HeadRec* rec = nullptr;
  int* err = nullptr;
};
NoAllocScratch g_noalloc[kMaxDevices];
std::mutex g_noalloc_mu;
}  // namespace

extern "C" int kf_op_head_tokens_noalloc(int32_t rows, int32_t V, int32_t d, const void* x,
                                         const void* w_head, const float* noise, float tau,
                                         int32_t map_kind, int32_t* tokens, void* stream) {
  if (!head_args_ok(rows, V, d, x, w_head, noise, tau, map_kind, tokens)) return KF_E_ARG;
  const size_t need = (size_t)rows * ceil_div(V, kChunk);
  if (need > (size_t)KF_NOALLOC_MAX_RECORDS) {
    set_global_error("kf_op_head_tokens_noalloc: rows * ceil(V/32) = " + std::to_string(need) +
                     " exceeds the static scratch of " + std::to_string(KF_NOALLOC_MAX_RECORDS) +
                     " records");
    return KF_E_CAPACITY;
  }
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return KF_E_CUDA;
  NoAllocScratch sc;
  {
    // first call on this device (which is current): look up the device
    // addresses of the static arrays; host code may not use their names
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!g_noalloc[dev].rec) {
      void* r = nullptr;
      void* e = nullptr;
      if (cudaGetSymbolAddress(&r, g_noalloc_rec) != cudaSuccess ||
          cudaGetSymbolAddress(&e, g_noalloc_err) != cudaSuccess) {
        cudaGetLastError();
        set_global_error("kf_op_head_tokens_noalloc: cudaGetSymbolAddress failed");
        return KF_E_CUDA;
      }
      g_noalloc[dev].rec = static_cast<HeadRec*>(r);
      g_noalloc[dev].err = static_cast<int*>(e);
    }
    sc = g_noalloc[dev];
  }
  cudaStream_t s = (cudaStream_t)stream;
  // the error word keeps the previous call's value: clear it (the records
  // need no clearing, every one this call reads it writes first)
  if (cudaMemsetAsync(sc.err, 0, sizeof(int), s) != cudaSuccess) return KF_E_CUDA;
  return head_tokens(rows, V, d, x, w_head, noise, tau, map_kind, tokens, sc.rec, sc.err, s);
}
