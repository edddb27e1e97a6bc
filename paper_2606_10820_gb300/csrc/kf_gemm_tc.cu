// bf16 GEMM on the 5th-generation tensor cores (tcgen05 + TMEM), fed by TMA.
//
//   D[M][N] = A[M][K] . W[N][K]^T, fp32 accumulation in tensor memory.
//
// One CTA computes a 128 x BN output tile (MMA M = 128, N = BN, K = 16 per
// instruction) over a range of 64-wide K blocks.  Warp roles (192 threads):
//   warp 0      TMA producer: A and W tiles (128B-swizzled, K-major) into a
//               ring of shared-memory stages, completion on mbarriers;
//   warp 1      allocates TMEM; one lane issues tcgen05.mma and commits each
//               stage back to the producer and the finished tile to the
//               epilogue;
//   warps 2..5  epilogue: tcgen05.ld 32 lanes x 32 columns per warp (one
//               output row's run of 32 columns per thread) -> epi_run32.
// When the output tiles cannot fill the SMs the K range is split over CTAs:
// each split writes an fp32 partial tile; the last CTA to arrive on the
// tile's counter sums the partials in split order (deterministic) and runs
// the epilogue, then re-arms the counter.
// Every mbarrier wait is bounded (about 2 s of %globaltimer); on expiry the
// kernel flags kErrTimeout, stops issuing work and exits after freeing TMEM.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <mutex>

#include "kf_internal.cuh"

namespace kf {

constexpr int kBM = 128;
constexpr int kBK = 64;                 // one 128-byte swizzle atom of bf16
constexpr int kThreads = 192;
constexpr unsigned long long kWaitNs = 2000000000ull;

struct TcArgs {
  int M, N, K;
  int kb_per_split;   // K blocks per split
  int splits;
  float* ws;          // [tiles][splits][128][BN] fp32 partials
  int* counters;      // [tiles]
  int* d_err;
  Epi epi;
};

// ------------------------------------------------------------ PTX helpers
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ unsigned long long globaltimer() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// bounded wait: false (and the error flag) after ~2 s
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, int* d_err) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = globaltimer();
  while (true) {
    for (int i = 0; i < 64; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (globaltimer() - t0 > kWaitNs) {
      atomicOr(d_err, kErrTimeout);
      return false;
    }
  }
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, uint32_t bar,
                                            int c0, int c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1)
      : "memory");
}

// shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups
// 1024 bytes apart (SBO), descriptor version 1 (tcgen05)
__device__ __forceinline__ uint64_t sdesc(uint32_t addr) {
  uint64_t d = 0;
  d |= (uint64_t)((addr >> 4) & 0x3FFF);
  d |= (uint64_t)1 << 16;                    // LBO (unused for swizzled K-major)
  d |= (uint64_t)(1024 >> 4) << 32;          // SBO
  d |= (uint64_t)1 << 46;                    // version
  d |= (uint64_t)2 << 61;                    // SWIZZLE_128B
  return d;
}

// instruction descriptor, kind::f16: D fp32, A and B bf16, both K-major
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) |
         ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void mma_bf16(uint32_t tmem_d, uint64_t a, uint64_t b, uint32_t idesc,
                                         uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
      : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float* v) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
        "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
        "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ void epi_bar() {
  asm volatile("bar.sync 1, 128;" ::: "memory");
}

// ------------------------------------------------------------ the kernel
template <int BN, int STAGES, int EPI>
__global__ void __launch_bounds__(kThreads, 1)
k_gemm_tc(const __grid_constant__ CUtensorMap map_a, const __grid_constant__ CUtensorMap map_w,
          TcArgs g) {
  constexpr uint32_t A_BYTES = kBM * kBK * 2;
  constexpr uint32_t B_BYTES = BN * kBK * 2;
  constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
  static_assert(4 * 32 * 36 * 4 <= STAGE_BYTES, "epilogue transpose blocks live in stage 0");
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // 1024-byte alignment for the 128B swizzle pattern
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
  // bars[0..S): full, bars[S..2S): empty, bars[2S]: accumulator ready
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 1);
  int* s_flag = reinterpret_cast<int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_tile = blockIdx.x, m_tile = blockIdx.y, split = blockIdx.z;
  const int n0 = n_tile * BN, m0 = m_tile * kBM;
  const int kb_total = g.K / kBK;
  const int kb0 = split * g.kb_per_split;
  const int kb1 = min(kb_total, kb0 + g.kb_per_split);
  const int nkb = kb1 - kb0;
  pdl_trigger();

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(smem_u32(&bars[s]), 1);
      mbar_init(smem_u32(&bars[STAGES + s]), 1);
    }
    mbar_init(smem_u32(&bars[2 * STAGES]), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_a)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_w)) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_slot)),
                 "r"(BN)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // Weights are constant during a step: the first stages' weight tiles
      // stream in while the predecessor kernel finishes; the activation tiles
      // it produces are loaded after pdl_wait.
      const int pre = min(nkb, STAGES);
      for (int i = 0; i < pre; ++i) {
        const uint32_t full = smem_u32(&bars[i]);
        mbar_expect_tx(full, STAGE_BYTES);
        tma_load_2d(smem_u32(smem + i * STAGE_BYTES) + A_BYTES, &map_w, full, (kb0 + i) * kBK, n0);
      }
      pdl_wait();
      for (int i = 0; i < pre; ++i)
        tma_load_2d(smem_u32(smem + i * STAGE_BYTES), &map_a, smem_u32(&bars[i]), (kb0 + i) * kBK, m0);
      for (int i = pre; i < nkb; ++i) {
        const int s = i % STAGES;
        const uint32_t ph = (i / STAGES) & 1;
        if (!mbar_wait(smem_u32(&bars[STAGES + s]), ph ^ 1, g.d_err)) break;
        const uint32_t full = smem_u32(&bars[s]);
        mbar_expect_tx(full, STAGE_BYTES);
        const uint32_t sa = smem_u32(smem + s * STAGE_BYTES);
        const int kc = (kb0 + i) * kBK;
        tma_load_2d(sa, &map_a, full, kc, m0);
        tma_load_2d(sa + A_BYTES, &map_w, full, kc, n0);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16(kBM, BN);
      bool ok = true;
      for (int i = 0; i < nkb; ++i) {
        const int s = i % STAGES;
        const uint32_t ph = (i / STAGES) & 1;
        if (!mbar_wait(smem_u32(&bars[s]), ph, g.d_err)) { ok = false; break; }
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t sa = smem_u32(smem + s * STAGE_BYTES);
        const uint32_t sb = sa + A_BYTES;
#pragma unroll
        for (int kk = 0; kk < kBK / 16; ++kk)
          mma_bf16(tmem, sdesc(sa + kk * 32), sdesc(sb + kk * 32), idesc,
                   (i > 0 || kk > 0) ? 1u : 0u);
        mma_commit(smem_u32(&bars[STAGES + s]));
      }
      if (ok) mma_commit(smem_u32(&bars[2 * STAGES]));
    }
  } else {
    // epilogue warps 2..5: TMEM lanes 32*(warp%4) .. +31
    const int quarter = warp & 3;
    const int et = threadIdx.x - 64;              // 0..127
    pdl_wait();
    // one waiter, result broadcast: every epilogue thread takes the same path
    if (et == 0) s_flag[1] = mbar_wait(smem_u32(&bars[2 * STAGES]), 0, g.d_err) ? 1 : 0;
    epi_bar();
    const bool ready = s_flag[1] != 0;
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t lane_addr = tmem + ((uint32_t)(quarter * 32) << 16);
    // Per epilogue warp a 32 x 36 fp32 block in the (now idle) pipeline
    // stage 0: tcgen05.ld gives a thread one row's 32 columns; re-read with
    // lane l on row (l / 8) + 4 i, columns 4 (l % 8) .. +3, every warp store
    // covers four 128-byte row segments.
    float* T = reinterpret_cast<float*>(smem) + quarter * (32 * 36);
    const int rbase = m0 + quarter * 32;
    const bool active = rbase < g.M;          // warp-uniform
    const int gr = lane >> 3, gc = (lane & 7) * 4;
    if (ready) {
      const int tile = m_tile * gridDim.x + n_tile;
      bool last = true;
      if (g.splits > 1) {
        // this split's partial tile, [128 rows][BN] fp32
        float* part = g.ws + ((size_t)tile * g.splits + split) * (kBM * BN) + (size_t)(quarter * 32) * BN;
        if (active) {
#pragma unroll 1
          for (int c = 0; c < BN; c += 32) {
            float v[32];
            tmem_ld32(lane_addr + c, v);
#pragma unroll
            for (int q = 0; q < 8; ++q)
              *reinterpret_cast<float4*>(T + lane * 36 + 4 * q) =
                  make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
            __syncwarp();
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              const int rr = gr + 4 * i;
              __stcg(reinterpret_cast<float4*>(part + (size_t)rr * BN + c + gc),
                     *reinterpret_cast<const float4*>(T + rr * 36 + gc));
            }
            __syncwarp();
          }
        }
        __threadfence();
        epi_bar();
        if (et == 0) {
          int old = atomicAdd(&g.counters[tile], 1);
          s_flag[0] = (old == g.splits - 1);
        }
        epi_bar();
        last = s_flag[0] != 0;
        if (last) {
          __threadfence();
          if (et == 0) g.counters[tile] = 0;   // re-arm for the next launch
        }
      }
      if (last && active) {
        const float* base = g.ws + (size_t)tile * g.splits * (kBM * BN) + (size_t)(quarter * 32) * BN;
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          float4 f[8];
          if (g.splits == 1) {
            float v[32];
            tmem_ld32(lane_addr + c, v);
            if (EPI == EPI_HEAD) {
              const int row = rbase + lane;
              if (row < g.M && n0 + c < g.N) epi_run32<__nv_bfloat16>(g.epi, row, n0 + c, v, g.N);
              continue;
            }
#pragma unroll
            for (int q = 0; q < 8; ++q)
              *reinterpret_cast<float4*>(T + lane * 36 + 4 * q) =
                  make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
            __syncwarp();
#pragma unroll
            for (int i = 0; i < 8; ++i) f[i] = *reinterpret_cast<const float4*>(T + (gr + 4 * i) * 36 + gc);
            __syncwarp();
          } else {
            // sum the partials in split order (deterministic)
#pragma unroll
            for (int i = 0; i < 8; ++i) f[i] = make_float4(0.f, 0.f, 0.f, 0.f);
            for (int sp = 0; sp < g.splits; ++sp) {
              const float* ps = base + (size_t)sp * (kBM * BN) + c + gc;
#pragma unroll
              for (int i = 0; i < 8; ++i) {
                float4 q = __ldcg(reinterpret_cast<const float4*>(ps + (size_t)(gr + 4 * i) * BN));
                f[i].x += q.x; f[i].y += q.y; f[i].z += q.z; f[i].w += q.w;
              }
            }
            if (EPI == EPI_HEAD) {
#pragma unroll
              for (int i = 0; i < 8; ++i) *reinterpret_cast<float4*>(T + (gr + 4 * i) * 36 + gc) = f[i];
              __syncwarp();
              float v[32];
#pragma unroll
              for (int q = 0; q < 8; ++q) {
                float4 t4 = *reinterpret_cast<const float4*>(T + lane * 36 + 4 * q);
                v[4 * q] = t4.x; v[4 * q + 1] = t4.y; v[4 * q + 2] = t4.z; v[4 * q + 3] = t4.w;
              }
              __syncwarp();
              const int row = rbase + lane;
              if (row < g.M && n0 + c < g.N) epi_run32<__nv_bfloat16>(g.epi, row, n0 + c, v, g.N);
              continue;
            }
          }
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const int row = rbase + gr + 4 * i;
            if (row < g.M) epi_vec4<__nv_bfloat16, EPI>(g.epi, row, n0 + c + gc, f[i], g.N);
          }
        }
      }
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  if (warp == 1)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(BN)
                 : "memory");
}

// ------------------------------------------------------------ host side
static PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
static std::once_flag g_encode_once;

static bool get_encode() {
  std::call_once(g_encode_once, [] {
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    cudaGetLastError();
  });
  return g_encode != nullptr;
}

static bool make_map(CUtensorMap* m, const void* ptr, int rows, int cols, int ld, int box_rows) {
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
  cuuint32_t box[2] = {(cuuint32_t)kBK, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims,
                        strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool tc_gemm_supported(const GemmDesc& g) {
  if (g.K % kBK || g.K == 0 || g.M <= 0 || g.N <= 0) return false;
  if ((g.lda * 2) % 16 || (g.ldw * 2) % 16) return false;
  if ((reinterpret_cast<uintptr_t>(g.A) & 15) || (reinterpret_cast<uintptr_t>(g.W) & 15)) return false;
  // the vector epilogue writes groups of 4 columns
  if (g.N % 4) return false;
  const int k = g.epi.kind;
  if ((k == EPI_STORE || k == EPI_STORE_F32 || k == EPI_BIAS_GELU) && g.epi.ldo % 4) return false;
  if ((k == EPI_RESID || k == EPI_NOISE_OUT) && g.epi.ldx % 4) return false;
  return get_encode();
}

template <int BN, int STAGES, int EPI>
static int launch_epi(const GemmDesc& g, void* ws, size_t ws_bytes, int* counters, int n_counters,
                     int* d_err, int num_sms, cudaStream_t s) {
  const int n_tiles = ceil_div(g.N, BN), m_tiles = ceil_div(g.M, kBM);
  const int tiles = n_tiles * m_tiles;
  const int kb_total = g.K / kBK;
  int splits = 1;
  if (tiles < num_sms) splits = std::min(std::max(1, num_sms / tiles), std::max(1, kb_total / 2));
  while (splits > 1 && ((size_t)tiles * splits * kBM * BN * 4 > ws_bytes || tiles > n_counters))
    --splits;
  int kbps = ceil_div(kb_total, splits);
  splits = ceil_div(kb_total, kbps);   // no empty splits
  CUtensorMap ma, mw;
  if (!make_map(&ma, g.A, g.M, g.K, g.lda, kBM) || !make_map(&mw, g.W, g.N, g.K, g.ldw, BN))
    return -1;
  TcArgs a;
  a.M = g.M; a.N = g.N; a.K = g.K; a.kb_per_split = kbps; a.splits = splits;
  a.ws = reinterpret_cast<float*>(ws); a.counters = counters; a.d_err = d_err; a.epi = g.epi;
  const size_t smem = (size_t)STAGES * (kBM * kBK * 2 + BN * kBK * 2) + 1024 + 256;
  static bool attr_set = false;
  if (!attr_set) {
    cudaFuncSetAttribute(k_gemm_tc<BN, STAGES, EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)smem);
    attr_set = true;
  }
  dim3 grid(n_tiles, m_tiles, splits);
  kf_launch(k_gemm_tc<BN, STAGES, EPI>, dim3(grid), dim3(kThreads), smem, s, ma, mw, a);
  return 0;
}

template <int BN, int STAGES>
static int launch_bn(const GemmDesc& g, void* ws, size_t ws_bytes, int* counters, int n_counters,
                     int* d_err, int num_sms, cudaStream_t s) {
  switch (g.epi.kind) {
    case EPI_STORE: return launch_epi<BN, STAGES, EPI_STORE>(g, ws, ws_bytes, counters, n_counters, d_err, num_sms, s);
    case EPI_BIAS_GELU: return launch_epi<BN, STAGES, EPI_BIAS_GELU>(g, ws, ws_bytes, counters, n_counters, d_err, num_sms, s);
    case EPI_RESID: return launch_epi<BN, STAGES, EPI_RESID>(g, ws, ws_bytes, counters, n_counters, d_err, num_sms, s);
    case EPI_NOISE_OUT: return launch_epi<BN, STAGES, EPI_NOISE_OUT>(g, ws, ws_bytes, counters, n_counters, d_err, num_sms, s);
    case EPI_HEAD: return launch_epi<BN, STAGES, EPI_HEAD>(g, ws, ws_bytes, counters, n_counters, d_err, num_sms, s);
    case EPI_LOGITS: return launch_epi<BN, STAGES, EPI_LOGITS>(g, ws, ws_bytes, counters, n_counters, d_err, num_sms, s);
    case EPI_STORE_F32: return launch_epi<BN, STAGES, EPI_STORE_F32>(g, ws, ws_bytes, counters, n_counters, d_err, num_sms, s);
  }
  return -1;
}

int launch_gemm_tc(const GemmDesc& g, void* ws, size_t ws_bytes, int* counters, int n_counters,
                   int* d_err, cudaStream_t s) {
  static int num_sms = 0;
  if (!num_sms) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&num_sms, cudaDevAttrMultiProcessorCount, dev);
  }
  // wide tiles when they already fill the SMs; otherwise narrow tiles (and
  // split-K) so that small-M projections still spread over every SM
  const int tiles128 = ceil_div(g.N, 128) * ceil_div(g.M, kBM);
  if (tiles128 >= num_sms)
    return launch_bn<128, 6>(g, ws, ws_bytes, counters, n_counters, d_err, num_sms, s);
  return launch_bn<64, 8>(g, ws, ws_bytes, counters, n_counters, d_err, num_sms, s);
}

}  // namespace kf
