// Internal declarations shared by the library's CUDA translation units.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>
#include <string>
#include <vector>

#include "../../include/kforcing.h"

namespace kf {

constexpr int kMaxHeadDim = 64;   // head_dim is 32 or 64
constexpr int kPage = 16;
constexpr int kChunk = 32;          // vocab ids per LM-head record
constexpr int kMaxGroupRows = 16;   // query rows per attention CTA

// device error bits (ORed into ctx->d_err)
constexpr int kErrBadToken = 1;
constexpr int kErrBadPage = 2;
constexpr int kErrTimeout = 4;
constexpr int kErrBadRow = 8;
constexpr int kErrInternal = 16;   // a launch invariant of the host plan did not hold

__host__ __device__ inline int ceil_div(int a, int b) { return (a + b - 1) / b; }

// One-time setup per device (function attributes, occupancy limits and SM
// counts belong to each device's context): per_device(pd, f) returns f()'s
// value for the current device, computed on the first call made with that
// device current.  Thread-safe; devices past kMaxDevices recompute each call.
constexpr int kMaxDevices = 64;
struct PerDevice {
  std::mutex mu;
  bool done[kMaxDevices] = {};
  long long val[kMaxDevices] = {};
};
template <typename F>
inline long long per_device(PerDevice& pd, F init) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    cudaGetLastError();
    return init();
  }
  std::lock_guard<std::mutex> lock(pd.mu);
  if (!pd.done[dev]) {
    pd.val[dev] = init();
    pd.done[dev] = true;
  }
  return pd.val[dev];
}
// the SM count of the current device
inline int device_sms() {
  static PerDevice pd;
  return (int)per_device(pd, [] {
    int dev = 0, n = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    return (long long)(n > 0 ? n : 1);
  });
}
// raise a kernel's dynamic shared-memory limit to `bytes` on the current
// device (once per device and size; thread-safe)
template <typename K>
inline void set_smem_attr(PerDevice& pd, K* kern, size_t bytes) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    cudaGetLastError();
    cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    return;
  }
  std::lock_guard<std::mutex> lock(pd.mu);
  if (pd.val[dev] < (long long)bytes) {
    cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    pd.val[dev] = (long long)bytes;
  }
}
__host__ __device__ inline int round_up(int a, int b) { return ceil_div(a, b) * b; }

// storage <-> fp32
__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(__nv_bfloat16 x) { return __bfloat162float(x); }
template <typename T> __device__ __forceinline__ T from_f(float x);
template <> __device__ __forceinline__ float from_f<float>(float x) { return x; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float x) {
  return __float2bfloat16_rn(x);
}

__device__ __forceinline__ float gelu_tanh(float x) {
  const float c = 0.7978845608028654f;  // sqrt(2/pi)
  return 0.5f * x * (1.0f + tanhf(c * (x + 0.044715f * x * x * x)));
}
// the same with the hardware tanh (tanh.approx.f32, absolute error about
// 5e-4): for bf16 outputs, whose rounding (2^-9 relative) is of that size
__device__ __forceinline__ float gelu_tanh_bf16(float x) {
  const float c = 0.7978845608028654f;
  float t;
  asm("tanh.approx.f32 %0, %1;" : "=f"(t) : "f"(c * (x + 0.044715f * x * x * x)));
  return 0.5f * x * (1.0f + t);
}
template <typename TA> __device__ __forceinline__ float gelu_for(float x) { return gelu_tanh(x); }
template <> __device__ __forceinline__ float gelu_for<__nv_bfloat16>(float x) { return gelu_tanh_bf16(x); }

// ---------------------------------------------------------------- GEMM epilogues
// Every GEMM computes D[M][N] = A[M][K] . W[N][K]^T with fp32 accumulation and
// hands each thread runs of 32 consecutive columns of one row to epi_run32.
enum EpiKind : int {
  EPI_STORE = 0,      // out[row][col] = D            (storage type TA)
  EPI_BIAS_GELU = 1,  // out[row][col] = gelu(D + bias[col])
  EPI_RESID = 2,      // x[row][col] += D             (fp32 residual stream)
  EPI_NOISE_OUT = 3,  // x[map[row]][col] = D + bias[col] (+ pos_emb[pos][col])
  EPI_HEAD = 4,       // per (row, 32-id chunk): max, sum exp(l - max), argmax of l = D/tau
  EPI_LOGITS = 5,     // outf[row][col] = D / tau     (fp32, col < n_valid)
  EPI_STORE_F32 = 6,  // outf[row][col] = D
  EPI_QKV = 7,        // RoPE on q, k; q -> q_out (fp32), k and v -> paged KV cache
};

struct HeadRec {   // one record per (head row, chunk of 32 vocab ids)
  float m;         // max of l over the chunk
  float s;         // sum over the chunk of exp(l - m), ascending id order
  int a;           // lowest id attaining m
  int pad;
};

__device__ __forceinline__ void st_ta4(float* p, float4 v);
__device__ __forceinline__ void st_ta4(__nv_bfloat16* p, float4 v);

struct Epi {
  int kind = EPI_STORE;
  void* out = nullptr;          // TA
  float* outf = nullptr;        // fp32 outputs
  int ldo = 0;
  const float* bias = nullptr;
  float* x = nullptr;           // residual stream
  int ldx = 0;
  const int32_t* row_map = nullptr;
  const int32_t* row_pos = nullptr;
  const float* pos_emb = nullptr;
  float inv_tau = 1.0f;
  int n_valid = 0;
  HeadRec* rec = nullptr;
  int nchunk = 0;
  // EPI_QKV
  float* q_out = nullptr;          // [rows][H][64]
  void* kv = nullptr;              // [L][n_pages][2][H][16][64]
  int layer = 0, n_pages = 0, H = 0, max_pages = 0, dsec = 0;
  const int32_t* row_seq = nullptr;
  const int32_t* page_table = nullptr;
  const float* cos_t = nullptr;    // [max_len][32] or NULL (no rotation)
  const float* sin_t = nullptr;
  int* d_err = nullptr;
  // fused RMSNorm (tensor-core path).  Producers of the residual stream
  // (EPI_RESID, EPI_NOISE_OUT) also write xb = bf16(x) and, per row, the sum
  // of squares of each 64-column slot of x into ss_out[row][nslot].  The
  // consumers (EPI_QKV, EPI_BIAS_GELU on the normed input) read ss_in and
  // scale each row of D by rsqrt(sum / d + eps) (the gains are folded into
  // their weights).
  void* xb_out = nullptr;
  float* ss_out = nullptr;
  const float* ss_in = nullptr;
  int nslot = 0;
  float inv_d = 0.f, eps = 0.f;
  // EPI_QKV in a decode step (rows_per_seq rows per sequence, row r at
  // position seq_len[r / rows_per_seq] + r % rows_per_seq): the skinny
  // kernel reads positions and pages before its dependency wait (seq_len
  // changes only at the step's commit), or NULL
  const int32_t* seq_len = nullptr;
  int rows_per_seq = 0;
};

// rsqrt(mean of squares + eps) of row `row` from its per-slot sums
__device__ __forceinline__ float row_rinv(const Epi& e, int row) {
  const float* p = e.ss_in + (size_t)row * e.nslot;
  float s = 0.f;
  for (int i = 0; i < e.nslot; ++i) s += p[i];
  return rsqrtf(s * e.inv_d + e.eps);
}

// EPI_QKV for one row at position pos whose KV page is `page` (-1: invalid,
// already flagged): lo = columns col0+gc .. +3 and hi = the same columns + 32
// of one 64-wide head block (col0 % 64 == 0, col0 < 3 * dsec, head_dim 64).
// Rotates the pairs (i, i + 32) of q and k at the row's position, with
// c4 / s4 = cos / sin of the angles gc .. gc + 3 at pos (read by the caller:
// cos_t / sin_t [pos][gc]), and stores q, k, v.
template <typename TA>
__device__ __forceinline__ void epi_qkv_rot(const Epi& e, int row, int pos, int page, int col0, int gc,
                                            float4 lo, float4 hi, float4 c4, float4 s4) {
  const int sec = col0 / e.dsec;                 // 0 q, 1 k, 2 v
  const int h = (col0 - sec * e.dsec) >> 6;
  float a[4] = {lo.x, lo.y, lo.z, lo.w}, b[4] = {hi.x, hi.y, hi.z, hi.w};
  if (sec < 2 && e.cos_t) {
    const float c[4] = {c4.x, c4.y, c4.z, c4.w}, sn[4] = {s4.x, s4.y, s4.z, s4.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float x1 = a[j], x2 = b[j];
      a[j] = x1 * c[j] - x2 * sn[j];
      b[j] = x2 * c[j] + x1 * sn[j];
    }
  }
  if (sec == 0) {
    float* q = e.q_out + ((size_t)row * e.H + h) * 64 + gc;
    *reinterpret_cast<float4*>(q) = make_float4(a[0], a[1], a[2], a[3]);
    *reinterpret_cast<float4*>(q + 32) = make_float4(b[0], b[1], b[2], b[3]);
    return;
  }
  if (page < 0) return;
  TA* dst = reinterpret_cast<TA*>(e.kv) +
            ((((size_t)e.layer * e.n_pages + page) * 2 + (sec - 1)) * e.H + h) * (kPage * 64) +
            (size_t)(pos % kPage) * 64 + gc;
  st_ta4(dst, make_float4(a[0], a[1], a[2], a[3]));
  st_ta4(dst + 32, make_float4(b[0], b[1], b[2], b[3]));
}

// the same, reading the angles' cos / sin itself
template <typename TA>
__device__ __forceinline__ void epi_qkv(const Epi& e, int row, int pos, int page, int col0, int gc,
                                        float4 lo, float4 hi) {
  float4 c4 = make_float4(1.f, 1.f, 1.f, 1.f), s4 = make_float4(0.f, 0.f, 0.f, 0.f);
  if (e.cos_t && col0 < 2 * e.dsec) {
    c4 = __ldg(reinterpret_cast<const float4*>(e.cos_t + (size_t)pos * 32 + gc));
    s4 = __ldg(reinterpret_cast<const float4*>(e.sin_t + (size_t)pos * 32 + gc));
  }
  epi_qkv_rot<TA>(e, row, pos, page, col0, gc, lo, hi, c4, s4);
}

template <typename TA>
__device__ __forceinline__ void epi_run32(const Epi& e, int row, int col0, const float* v, int N) {
  switch (e.kind) {
    case EPI_STORE: {
      TA* o = reinterpret_cast<TA*>(e.out) + (size_t)row * e.ldo + col0;
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (col0 + j < N) o[j] = from_f<TA>(v[j]);
      break;
    }
    case EPI_STORE_F32: {
      float* o = e.outf + (size_t)row * e.ldo + col0;
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (col0 + j < N) o[j] = v[j];
      break;
    }
    case EPI_BIAS_GELU: {
      TA* o = reinterpret_cast<TA*>(e.out) + (size_t)row * e.ldo + col0;
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (col0 + j < N) o[j] = from_f<TA>(gelu_tanh(v[j] + (e.bias ? e.bias[col0 + j] : 0.f)));
      break;
    }
    case EPI_RESID: {
      float* o = e.x + (size_t)row * e.ldx + col0;
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (col0 + j < N) o[j] += v[j];
      break;
    }
    case EPI_NOISE_OUT: {
      int xr = e.row_map[row];
      float* o = e.x + (size_t)xr * e.ldx + col0;
      const float* pe = e.pos_emb ? e.pos_emb + (size_t)e.row_pos[xr] * N + col0 : nullptr;
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (col0 + j < N) o[j] = v[j] + (e.bias ? e.bias[col0 + j] : 0.f) + (pe ? pe[j] : 0.f);
      break;
    }
    case EPI_HEAD: {
      // col0 is a multiple of 32: one record for ids col0 .. col0+31 (< n_valid)
      const int nv = e.n_valid - col0;
      if (nv <= 0) break;
      float m = -INFINITY;
      int a = col0;
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        float l = v[j] * e.inv_tau;
        if (j < nv && l > m) { m = l; a = col0 + j; }
      }
      float s = 0.f;
      if (sizeof(TA) == 2) {
        // bf16 path: the hardware 2^x on log2(e)-scaled differences (relative
        // error ~2^-22 per term)
        const float k2 = 1.4426950408889634f;
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          float t;
          asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(t) : "f"((v[j] * e.inv_tau - m) * k2));
          if (j < nv) s += t;
        }
      } else {
#pragma unroll
        for (int j = 0; j < 32; ++j)
          if (j < nv) s += expf(v[j] * e.inv_tau - m);
      }
      HeadRec r;
      r.m = m; r.s = s; r.a = a; r.pad = 0;
      e.rec[(size_t)row * e.nchunk + col0 / 32] = r;
      break;
    }
    case EPI_LOGITS: {
      float* o = e.outf + (size_t)row * e.ldo + col0;
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (col0 + j < e.n_valid) o[j] = v[j] * e.inv_tau;
      break;
    }
  }
}

// Four consecutive output columns of one row (col % 4 == 0), for epilogues
// whose lanes run along the columns of a row (coalesced vector stores).
// EPI_HEAD is not handled here (it reduces over a run of 32 columns:
// epi_run32).  Requires ldo, ldx and N to be multiples of 4.
__device__ __forceinline__ void st_ta4(float* p, float4 v) { *reinterpret_cast<float4*>(p) = v; }
__device__ __forceinline__ void st_ta4(__nv_bfloat16* p, float4 v) {
  __nv_bfloat162 a = __floats2bfloat162_rn(v.x, v.y), b = __floats2bfloat162_rn(v.z, v.w);
  uint2 u;
  u.x = *reinterpret_cast<uint32_t*>(&a);
  u.y = *reinterpret_cast<uint32_t*>(&b);
  *reinterpret_cast<uint2*>(p) = u;
}

// EPI_RESID with the residual x[row][col..+3] already loaded (xo): the
// callers fetch every residual of a batch of outputs before any store, so
// the loads are not serialised behind stores that might alias them
template <typename TA>
__device__ __forceinline__ float epi_resid4(const Epi& e, int row, int col, float4 v, float4 xo) {
  v = make_float4(xo.x + v.x, xo.y + v.y, xo.z + v.z, xo.w + v.w);
  *reinterpret_cast<float4*>(e.x + (size_t)row * e.ldx + col) = v;
  if (e.xb_out) st_ta4(reinterpret_cast<TA*>(e.xb_out) + (size_t)row * e.ldx + col, v);
  return v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
}

template <typename TA, int EPI>
__device__ __forceinline__ float epi_vec4(const Epi& e, int row, int col, float4 v, int N,
                                         bool add_bias = true) {
  if (col >= N) return 0.f;
  if (EPI == EPI_STORE) {
    st_ta4(reinterpret_cast<TA*>(e.out) + (size_t)row * e.ldo + col, v);
  } else if (EPI == EPI_STORE_F32) {
    *reinterpret_cast<float4*>(e.outf + (size_t)row * e.ldo + col) = v;
  } else if (EPI == EPI_BIAS_GELU) {
    if (e.bias && add_bias) {   // (false: the caller has added it)
      float4 b = __ldg(reinterpret_cast<const float4*>(e.bias + col));
      v.x += b.x; v.y += b.y; v.z += b.z; v.w += b.w;
    }
    v = make_float4(gelu_for<TA>(v.x), gelu_for<TA>(v.y), gelu_for<TA>(v.z), gelu_for<TA>(v.w));
    st_ta4(reinterpret_cast<TA*>(e.out) + (size_t)row * e.ldo + col, v);
  } else if (EPI == EPI_RESID || EPI == EPI_NOISE_OUT) {
    int xr = row;
    if (EPI == EPI_RESID) {
      float4 x = *reinterpret_cast<const float4*>(e.x + (size_t)row * e.ldx + col);
      v = make_float4(x.x + v.x, x.y + v.y, x.z + v.z, x.w + v.w);
    } else {
      xr = e.row_map[row];
      if (e.bias) {
        float4 b = __ldg(reinterpret_cast<const float4*>(e.bias + col));
        v.x += b.x; v.y += b.y; v.z += b.z; v.w += b.w;
      }
      if (e.pos_emb) {
        float4 q = __ldg(reinterpret_cast<const float4*>(e.pos_emb + (size_t)e.row_pos[xr] * N + col));
        v.x += q.x; v.y += q.y; v.z += q.z; v.w += q.w;
      }
    }
    *reinterpret_cast<float4*>(e.x + (size_t)xr * e.ldx + col) = v;
    if (e.xb_out) st_ta4(reinterpret_cast<TA*>(e.xb_out) + (size_t)xr * e.ldx + col, v);
    return v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  } else if (EPI == EPI_LOGITS) {
    float* o = e.outf + (size_t)row * e.ldo + col;
    const float t = e.inv_tau;
    if (col + 3 < e.n_valid) {
      o[0] = v.x * t; o[1] = v.y * t; o[2] = v.z * t; o[3] = v.w * t;
    } else {
      if (col < e.n_valid) o[0] = v.x * t;
      if (col + 1 < e.n_valid) o[1] = v.y * t;
      if (col + 2 < e.n_valid) o[2] = v.z * t;
    }
  }
  return 0.f;
}

__device__ __forceinline__ float4 scale4(float4 v, float r) {
  return make_float4(v.x * r, v.y * r, v.z * r, v.w * r);
}
__device__ __forceinline__ float4 add4(float4 a, float4 b) {
  return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
}

// ---------------------------------------------------------------- launches
// Programmatic dependent launch: every kernel of the step waits for its
// predecessor grid to complete and publish its writes (pdl_wait) before its
// first access to any buffer another kernel of the step reads or writes, and
// only then lets its successor launch.  So one kernel at a time runs ahead:
// the successor's CTAs become resident while this kernel works and load what
// does not depend on it (weights, the cached K/V pages below the committed
// length), then wait.  Triggering at kernel entry instead let four or five
// kernels' CTAs pile up on the SMs and slowed the running kernel about 2x
// (measured per phase with %globaltimer stamps at batch 1).  Every kernel
// waits unconditionally, so completion stays ordered along the chain;
// launched without the attribute both instructions are no-ops.
__device__ __forceinline__ void pdl_wait() {
  asm volatile("griddepcontrol.wait;\n\tgriddepcontrol.launch_dependents;" ::: "memory");
}

extern thread_local bool g_pdl;   // launch with the programmatic-serialization attribute
// tensor-core GEMM launch options for the launches made by this thread
constexpr int kGemmNoPersist = 1;  // one CTA per tile even past a wave of tiles
extern thread_local int g_gemm_flags;

template <typename... KArgs, typename... Args>
inline void kf_launch(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                      Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = g_pdl ? 1 : 0;
  cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

struct GemmDesc {
  int M, N, K;
  const void* A;   // [M][lda] storage TA
  int lda;
  const void* W;   // [N][ldw] storage TA
  int ldw;
  Epi epi;
  // weights of the next projection of the step: the tensor-core kernel's CTAs
  // prefetch them into L2 at their start (16-byte aligned), or NULL
  const void* l2_next = nullptr;
  size_t l2_bytes = 0;
};

// SIMT GEMM (any storage type; fp32 accumulation, k ascending per output)
void launch_gemm_simt(bool bf16, const GemmDesc& g, cudaStream_t s);

// tcgen05 GEMM (bf16 only).  Requires K % 64 == 0, 16-byte aligned rows,
// A rows readable up to round_up(M,128), W rows up to round_up(N,BN).
bool tc_gemm_supported(const GemmDesc& g);
int launch_gemm_tc(const GemmDesc& g, int* d_err, cudaStream_t s);

// Skinny projections (kf_gemm_skinny.cu): M <= 64 rows on warp-level MMA,
// weights staged before the dependency wait.  The fused RMSNorm scale comes
// from the A rows themselves (epi.ss_in set means "normed input"; it is not
// read), and residual producers must not ask for per-slot sums (ss_out NULL).
bool skinny_gemm_supported(const GemmDesc& g);
int launch_gemm_skinny(const GemmDesc& g, int* d_err, cudaStream_t s);

struct AttnArgs {
  const float* q;          // [R][H][hd] (rotated, unscaled)
  const void* kv;          // pool [L][n_pages][2][H][16][hd]
  int layer, n_pages, H, hd;
  const int32_t* page_table;  // [max_batch][max_pages]
  int max_pages;
  const int32_t* row_seq;  // [R]
  const int32_t* row_pos;  // [R]
  const int4* groups;      // {b, row0, nrows, 0} or NULL (uniform: group g = seq g)
  int uniform_rows;        // rows per sequence when groups == NULL
  void* out;               // [R][H*hd] TA
  float* part_o;           // [n_split][R][H][hd]
  float2* part_ml;         // [n_split][R][H]
  int R;
  int n_split;
  int keys_per_split;      // multiple of 64
  int* d_err;
  const int32_t* len = nullptr;  // decode: committed length per sequence (keys below it are
                                 // not written during the step), or NULL
  int pg_cap = 0;                // pages of one CTA's key range (set by the launcher)
  int* split_count = nullptr;    // [groups][H] zeroed counters: the warp-MMA kernel merges
                                 // its own splits (no k_attn_combine launch)
  int cluster_merge = 0;           // warp-MMA kernel, n_split > 1: the key splits of a
                                   // (group, head) form a thread-block cluster and merge
                                   // their partial softmaxes over distributed shared memory
  const int32_t* order = nullptr;  // uniform groups: group g is sequence order[g] (a
                                   // permutation, longest first: each head's longest CTAs
                                   // start first and the grid's last wave holds the
                                   // shortest), or NULL
};
// max_keys: the most keys any row of the launch can see (max_len bound)
void launch_attention(bool bf16, const AttnArgs& a, int n_groups, int max_keys, cudaStream_t s);
void launch_attn_combine(bool bf16, const AttnArgs& a, cudaStream_t s);
// decode attention on warp-level MMA (bf16 cache, head_dim 64, <= 16 rows per
// group; rows: the most rows of any group); -1 if the TMA map is refused
bool attention_mma_supported(bool bf16, int hd, int rows);
// *merged: the kernel merged its key splits itself (no k_attn_combine needed)
int launch_attention_mma(const AttnArgs& a, int n_groups, int rows, int max_keys, cudaStream_t s,
                         bool* merged);

// the op entry points' error word on the current device, cleared on s
// (read back by kf_op_status); nullptr on failure
int* op_error_word(cudaStream_t s);

// message for kf_last_error(NULL) (calls without a context)
void set_global_error(const std::string& msg);

// elementwise / bookkeeping kernels
// the first kernel of a decode step: the row maps, the embedding of the B*P
// pending rows (xb / ss: bf16 copy and per-64-column sums of squares for the
// fused RMSNorm, or NULL) and the features of n_noise noise values
void launch_step_prologue(bool bf16, int B, int P, int kz, const int32_t* d_len, const int32_t* pending,
                          int pend_stride, const void* tok_emb, const float* pos_emb, int V, int d,
                          float* x, void* xb, float* ss, int* d_err, int32_t* row_seq, int32_t* row_pos,
                          int32_t* noise_map, int32_t* head_map, int n_noise, const float* noise,
                          const float* freq, const float* tau_feat, float scale, void* feat,
                          cudaStream_t s);
void launch_embed_tokens(bool bf16, int R, const int32_t* row_tok, const void* tok_emb,
                         const float* pos_emb, const int32_t* row_pos, int V, int d, float* x,
                         void* xb, float* ss, int* d_err, cudaStream_t s);
void launch_scale_cols(float* w, const float* g, int rows_per_layer, int cols, size_t total,
                       cudaStream_t s);
void launch_rmsnorm(bool bf16, int R, const int32_t* row_map, const float* x, int d,
                    const float* g, float eps, void* out, cudaStream_t s);
void launch_rope_append(bool bf16, int R, const void* qkv, int d, int H, int hd,
                        const int32_t* row_seq,
                        const int32_t* row_pos, const float* cos_t, const float* sin_t, float* q,
                        void* kv, int layer, int n_pages, const int32_t* page_table, int max_pages,
                        int* d_err, cudaStream_t s);
// A decode step's commit, taken by the token selection: token b nout + j
// becomes pending id j of sequence b (pending[b pend_stride + j]) and len[b]
// grows by P.  pending == NULL: tokens only.
struct StepCommit {
  int32_t* pending = nullptr;
  int pend_stride = 0;
  int32_t* len = nullptr;
  int P = 0;
  int nout = 1;
};
// mtp_rows = B > 0: n_rows = B k blocks in head-major order, head j's weights
// at w_head + j head_stride (elements); 0: one block per row of head_in.
// err: the call's device error word (or NULL); when an earlier kernel set
// it, every token is -1
void launch_head_select(bool bf16, int n_rows, const HeadRec* rec, int nchunk, const void* head_in,
                        int d, const void* w_head, int V, float inv_tau, int map_kind,
                        const float* noise, int32_t* tokens, int mtp_rows, size_t head_stride,
                        const int* err, const StepCommit& cm, cudaStream_t s);

}  // namespace kf
