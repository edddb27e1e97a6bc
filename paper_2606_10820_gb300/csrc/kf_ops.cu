// Single-kernel entry points (include/kforcing_ops.h).
#include <mutex>
#include <string>

#include "../../include/kforcing_ops.h"
#include "kf_internal.cuh"

using namespace kf;

namespace {
// Scratch of the allocating entry points, per device: an error word (the
// kernels OR their error bits into it; kf_op_status reads and clears it)
// and the LM-head record buffer.  g_ops_mu guards both tables.
struct OpScratch {
  int* err = nullptr;
  HeadRec* rec = nullptr;
  size_t rec_bytes = 0;
};
OpScratch g_ops[kMaxDevices];
std::mutex g_ops_mu;

int current_device(int* dev) {
  if (cudaGetDevice(dev) != cudaSuccess || *dev < 0 || *dev >= kMaxDevices) {
    cudaGetLastError();
    return KF_E_CUDA;
  }
  return KF_OK;
}

// the current device's error word (allocated and zeroed on first use);
// call with g_ops_mu held
int ensure_err(int dev) {
  if (g_ops[dev].err) return KF_OK;
  int* e = nullptr;
  if (cudaMalloc(&e, sizeof(int)) != cudaSuccess || cudaMemset(e, 0, sizeof(int)) != cudaSuccess) {
    cudaGetLastError();
    if (e) cudaFree(e);
    return KF_E_CUDA;
  }
  g_ops[dev].err = e;
  return KF_OK;
}
}  // namespace

namespace kf {
// the calling thread's device's op error word, cleared on `s` (kf_op_status
// reads it); nullptr if it cannot be had
int* op_error_word(cudaStream_t s) {
  int dev = 0;
  if (current_device(&dev) != KF_OK) return nullptr;
  int* err = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_ops_mu);
    if (ensure_err(dev) != KF_OK) return nullptr;
    err = g_ops[dev].err;
  }
  if (cudaMemsetAsync(err, 0, sizeof(int), s) != cudaSuccess) return nullptr;
  return err;
}
}  // namespace kf

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
  launch_head_select(true, rows, rec, nchunk, x, d, w_head, V, 1.0f / tau, map_kind, noise, tokens, 0, 0,
                     err, StepCommit{}, s);
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
  if (impl == KF_GEMM_TCGEN05 || impl == KF_GEMM_TCGEN05_PER_TILE) {
    if (!tc_gemm_supported(g)) return KF_E_ARG;
    g_gemm_flags = impl == KF_GEMM_TCGEN05_PER_TILE ? kGemmNoPersist : 0;
    int dev = 0;
    if (current_device(&dev) != KF_OK) return KF_E_CUDA;
    int* err = nullptr;
    {
      std::lock_guard<std::mutex> lock(g_ops_mu);
      if (ensure_err(dev) != KF_OK) return KF_E_CUDA;
      err = g_ops[dev].err;
    }
    // each call starts with a clear error word (kf_op_status reads it)
    if (cudaMemsetAsync(err, 0, sizeof(int), s) != cudaSuccess) return KF_E_CUDA;
    if (launch_gemm_tc(g, err, s) != 0) return KF_E_CUDA;
  } else if (impl == KF_GEMM_SKINNY) {
    if (!skinny_gemm_supported(g)) return KF_E_ARG;
    int* err = op_error_word(s);
    if (!err) return KF_E_CUDA;
    if (launch_gemm_skinny(g, err, s) != 0) return KF_E_CUDA;
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
  int dev = 0;
  if (current_device(&dev) != KF_OK) return KF_E_CUDA;
  cudaStream_t s = (cudaStream_t)stream;
  const size_t need = (size_t)rows * ceil_div(V, kChunk) * sizeof(HeadRec);
  // The lock covers the buffer's growth and the launches that use it, so two
  // host threads never free a buffer the other is about to launch on.  Work
  // already enqueued on another stream may still read an old buffer: growth
  // waits for the whole device first.
  std::lock_guard<std::mutex> lock(g_ops_mu);
  if (ensure_err(dev) != KF_OK) return KF_E_CUDA;
  OpScratch& sc = g_ops[dev];
  if (need > sc.rec_bytes) {
    if (sc.rec) {
      if (cudaDeviceSynchronize() != cudaSuccess) return KF_E_CUDA;
      cudaFree(sc.rec);
      sc.rec = nullptr;
      sc.rec_bytes = 0;
    }
    if (cudaMalloc(&sc.rec, need) != cudaSuccess) {
      cudaGetLastError();
      sc.rec = nullptr;
      return KF_E_OOM;
    }
    sc.rec_bytes = need;
  }
  if (cudaMemsetAsync(sc.err, 0, sizeof(int), s) != cudaSuccess) return KF_E_CUDA;
  return head_tokens(rows, V, d, x, w_head, noise, tau, map_kind, tokens, sc.rec, sc.err, s);
}

// ------------------------------------------------- no-allocation variant
// Scratch for callers that cannot allocate device memory: a fixed array in
// the library's own device image.  Every device that loads the library holds
// it (4 MiB of records plus an error word) until the process exits.
static __device__ __align__(256) HeadRec g_noalloc_rec[KF_NOALLOC_MAX_RECORDS];
static __device__ __align__(256) int g_noalloc_err;

namespace {
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

// Reads and clears the error words of the op entry points on the current
// device after `stream` finishes: the allocating entries' word (if one of
// them has run on this device) and the no-allocation entry's static word.
// Allocates nothing.
extern "C" int kf_op_status(void* stream) {
  int dev = 0;
  if (current_device(&dev) != KF_OK) return KF_E_CUDA;
  if (cudaStreamSynchronize((cudaStream_t)stream) != cudaSuccess) {
    cudaGetLastError();
    set_global_error("kf_op_status: the stream reported a CUDA error");
    return KF_E_CUDA;
  }
  int bits = 0;
  int* err = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_ops_mu);
    err = g_ops[dev].err;
  }
  if (err) {
    int v = 0;
    if (cudaMemcpy(&v, err, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess ||
        cudaMemset(err, 0, sizeof(int)) != cudaSuccess)
      return KF_E_CUDA;
    bits |= v;
  }
  int v = 0;
  const int zero = 0;
  if (cudaMemcpyFromSymbol(&v, g_noalloc_err, sizeof(int)) != cudaSuccess ||
      cudaMemcpyToSymbol(g_noalloc_err, &zero, sizeof(int)) != cudaSuccess) {
    cudaGetLastError();
    return KF_E_CUDA;
  }
  bits |= v;
  if (bits) {
    set_global_error("kf_op_status: device error flags " + std::to_string(bits));
    return KF_E_DEVICE;
  }
  return KF_OK;
}
