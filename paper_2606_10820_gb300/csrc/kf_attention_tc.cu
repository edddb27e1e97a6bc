// Decode attention on the 5th-generation tensor cores (bf16 cache, head_dim
// 64).  One CTA (128 threads) per (row group of one sequence, head, key
// split); up to 16 query rows, padded to the MMA's N = 16.  Per tile of 128
// keys (8 pages):
//   S   = K . Q^T          tcgen05.mma M=128 (keys) x N=16 (rows) x K=64,
//                          fp32 in TMEM; thread t reads key t's 16 scores;
//   P   = exp(S/8 - m_t)   per row, masked causally (key <= row position),
//                          tile maximum m_t and sum l_t kept per row;
//   O_t = V^T . P^T        tcgen05.mma M=128 (64 head dims + 64 ignored
//                          rows) x N=16 x K=128 keys into the tile's own TMEM
//                          columns (V is transposed into a K-major tile).
// At the end each head dim d sums O_t[d][row] exp(m_t - M) over the tiles in
// order and divides by L = sum l_t exp(m_t - M): the exact softmax with no
// rescaling of running accumulators.  All shared-memory operands use the
// K-major 128-byte-swizzle layout of the tcgen05 GEMM; the threads write
// them and fence them into the async proxy before the MMA.
#include "kf_tc.cuh"

namespace kf {

constexpr int kTcKeys = 128;
constexpr int kTcRows = 16;
constexpr int kTcMaxTiles = 7;        // TMEM: 16 (S) + 7 x 16 (O_t) <= 128 columns
constexpr int kTcCols = 128;

// shared memory (bytes from a 1024-aligned base)
constexpr int OFF_VT = 0;       // V^T: 2 K-blocks (64 keys) x 64 dim rows x 128 B; each block's
                                // padding rows 64..127 (results ignored) read the next 8 KB
constexpr int OFF_K = 16384;    // K: 128 keys x 128 B
constexpr int OFF_Q = 32768;    // Q: 16 rows x 128 B
constexpr int OFF_P = 34816;    // P: 2 K-blocks x 16 rows x 128 B
constexpr int OFF_RED = 38912;  // [4 warps][16] maxima, then [4][16] sums
constexpr int OFF_ML = OFF_RED + 512;                      // m_t, then l_t: [kTcMaxTiles][16]
constexpr int OFF_POS = OFF_ML + 2 * kTcMaxTiles * 16 * 4;  // row positions [16]
constexpr int OFF_BAR = OFF_POS + 64;                      // 2 mbarriers, TMEM slot, flag
constexpr int kTcSmem = OFF_BAR + 64 + 1024;
// 4 CTAs per SM at most: TMEM holds 4 x 128 columns
constexpr int kTcSmemLaunch = 46 * 1024;
static_assert(kTcSmem <= kTcSmemLaunch, "attention smem");

// byte offset of (row, byte) in a K-major SW128 block of 128-byte rows
__device__ __forceinline__ uint32_t sw128(int row, int byte) {
  return (uint32_t)(row * 128 + ((((byte >> 4) ^ (row & 7))) << 4) + (byte & 15));
}

__device__ __forceinline__ void fence_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void cpa16(uint32_t dst, const void* src, int nbytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(nbytes)
               : "memory");
}

__global__ void __launch_bounds__(128) k_attention_tc(AttnArgs a) {
  pdl_trigger();
  pdl_wait();
  extern __shared__ __align__(1024) uint8_t smraw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smraw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + OFF_BAR);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2);
  int* flag = reinterpret_cast<int*>(tmem_slot + 1);
  float* red = reinterpret_cast<float*>(sm + OFF_RED);
  float* mt = reinterpret_cast<float*>(sm + OFF_ML);
  float* lt = mt + kTcMaxTiles * kTcRows;
  int* s_pos = reinterpret_cast<int*>(sm + OFF_POS);

  const int g = blockIdx.x, h = blockIdx.y, split = blockIdx.z;
  int b, row0, nr;
  if (a.groups) {
    int4 gg = a.groups[g];
    b = gg.x; row0 = gg.y; nr = gg.z;
  } else {
    b = g; row0 = g * a.uniform_rows; nr = a.uniform_rows;
  }
  const int n_keys = a.row_pos[row0 + nr - 1] + 1;
  const int k_begin = split * a.keys_per_split;
  const int k_end = min(n_keys, k_begin + a.keys_per_split);
  const int n_tiles = k_end > k_begin ? min(kTcMaxTiles, ceil_div(k_end - k_begin, kTcKeys)) : 0;
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;

  if (t == 0) {
    mbar_init(smem_u32(&bars[0]), 1);
    mbar_init(smem_u32(&bars[1]), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (t < kTcRows) s_pos[t] = (t < nr) ? a.row_pos[row0 + t] : -1;
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_slot)),
                 "r"(kTcCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  // Q rows -> bf16, K-major SW128 (thread: one row, 8 dims)
  {
    const int r = t >> 3, c = t & 7;
    uint4 pk = make_uint4(0u, 0u, 0u, 0u);
    if (r < nr) {
      const float* src = a.q + ((size_t)(row0 + r) * a.H + h) * 64 + c * 8;
      const float4 x0 = *reinterpret_cast<const float4*>(src);
      const float4 x1 = *reinterpret_cast<const float4*>(src + 4);
      __nv_bfloat162 p0 = __floats2bfloat162_rn(x0.x, x0.y), p1 = __floats2bfloat162_rn(x0.z, x0.w);
      __nv_bfloat162 p2 = __floats2bfloat162_rn(x1.x, x1.y), p3 = __floats2bfloat162_rn(x1.z, x1.w);
      pk.x = *reinterpret_cast<uint32_t*>(&p0); pk.y = *reinterpret_cast<uint32_t*>(&p1);
      pk.z = *reinterpret_cast<uint32_t*>(&p2); pk.w = *reinterpret_cast<uint32_t*>(&p3);
    }
    *reinterpret_cast<uint4*>(sm + OFF_Q + sw128(r, c * 16)) = pk;
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;

  const __nv_bfloat16* kv = reinterpret_cast<const __nv_bfloat16*>(a.kv);
  const size_t head_page = (size_t)kPage * 64;
  const size_t layer_base = (size_t)a.layer * a.n_pages * 2 * a.H * head_page;
  const uint32_t idesc = idesc_bf16(128, kTcRows);
  bool bad_page = false;
  bool ok = true;

  for (int it = 0; it < n_tiles && ok; ++it) {
    const int kt = k_begin + it * kTcKeys;
    // K: 128 keys x 8 chunks of 16 B, cp.async into the swizzled layout
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int idx = t + 128 * i, kl = idx >> 3, c = idx & 7, key = kt + kl;
      const __nv_bfloat16* src = kv;
      int nb = 0;
      if (key < k_end) {
        const int pi = key / kPage;
        const int page = pi < a.max_pages ? a.page_table[b * a.max_pages + pi] : -1;
        if (page >= 0 && page < a.n_pages) {
          src = kv + layer_base + (((size_t)page * 2) * a.H + h) * head_page +
                (size_t)(key % kPage) * 64 + c * 8;
          nb = 16;
        } else {
          bad_page = true;
        }
      }
      cpa16(smem_u32(sm + OFF_K + sw128(kl, c * 16)), src, nb);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
    // V: thread t loads key t's 64 dims and writes them transposed (V^T)
    {
      const int key = kt + t;
      uint4 v[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) v[i] = make_uint4(0u, 0u, 0u, 0u);
      if (key < k_end) {
        const int pi = key / kPage;
        const int page = pi < a.max_pages ? a.page_table[b * a.max_pages + pi] : -1;
        if (page >= 0 && page < a.n_pages) {
          const uint4* src = reinterpret_cast<const uint4*>(
              kv + layer_base + (((size_t)page * 2 + 1) * a.H + h) * head_page +
              (size_t)(key % kPage) * 64);
#pragma unroll
          for (int i = 0; i < 8; ++i) v[i] = src[i];
        }
      }
      uint8_t* blk = sm + OFF_VT + (t >> 6) * 8192;
      const int kb = (t & 63) * 2;
      const __nv_bfloat16* ve = reinterpret_cast<const __nv_bfloat16*>(v);
#pragma unroll
      for (int d = 0; d < 64; ++d) *reinterpret_cast<__nv_bfloat16*>(blk + sw128(d, kb)) = ve[d];
    }
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    fence_async_smem();
    __syncthreads();

    // S = K . Q^T
    if (t == 0) {
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)
        mma_bf16(tmem, sdesc(smem_u32(sm + OFF_K) + kk * 32), sdesc(smem_u32(sm + OFF_Q) + kk * 32),
                 idesc, kk > 0 ? 1u : 0u);
      mma_commit(smem_u32(&bars[0]));
      *flag = mbar_wait(smem_u32(&bars[0]), it & 1, a.d_err) ? 1 : 0;
    }
    __syncthreads();
    if (!*flag) { ok = false; break; }
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    float s[kTcRows];
    tmem_ld16(tmem + ((uint32_t)(warp * 32) << 16), s);
    const int key = kt + t;
#pragma unroll
    for (int r = 0; r < kTcRows; ++r)
      s[r] = (r < nr && key < k_end && key <= s_pos[r]) ? s[r] * 0.125f : -INFINITY;
    // tile maximum per row
#pragma unroll
    for (int r = 0; r < kTcRows; ++r) {
      float m = s[r];
      for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
      if (lane == 0) red[warp * kTcRows + r] = m;
    }
    __syncthreads();
    uint8_t* pblk = sm + OFF_P + (t >> 6) * 2048;
    const int pb = (t & 63) * 2;
#pragma unroll
    for (int r = 0; r < kTcRows; ++r) {
      const float tm = fmaxf(fmaxf(red[r], red[kTcRows + r]), fmaxf(red[2 * kTcRows + r], red[3 * kTcRows + r]));
      s[r] = (tm == -INFINITY) ? 0.f : expf(s[r] - tm);
      *reinterpret_cast<__nv_bfloat16*>(pblk + sw128(r, pb)) = __float2bfloat16_rn(s[r]);
    }
    // row sums of the probabilities as the PV product will see them (bf16)
#pragma unroll
    for (int r = 0; r < kTcRows; ++r) {
      float sum = __bfloat162float(__float2bfloat16_rn(s[r]));
      for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
      if (lane == 0) red[4 * kTcRows + warp * kTcRows + r] = sum;
    }
    fence_async_smem();
    __syncthreads();
    if (t < kTcRows) {
      mt[it * kTcRows + t] = fmaxf(fmaxf(red[t], red[kTcRows + t]), fmaxf(red[2 * kTcRows + t], red[3 * kTcRows + t]));
      const float* rs = red + 4 * kTcRows;
      lt[it * kTcRows + t] = (rs[t] + rs[kTcRows + t]) + (rs[2 * kTcRows + t] + rs[3 * kTcRows + t]);
    }
    // O_t = V^T . P^T into the tile's own TMEM columns
    if (t == 0) {
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const uint32_t dcol = tmem + kTcRows + kTcRows * it;
#pragma unroll
      for (int blk = 0; blk < 2; ++blk)
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
          mma_bf16(dcol, sdesc(smem_u32(sm + OFF_VT + blk * 8192) + kk * 32),
                   sdesc(smem_u32(sm + OFF_P + blk * 2048) + kk * 32), idesc,
                   (blk | kk) ? 1u : 0u);
      mma_commit(smem_u32(&bars[1]));
      *flag = mbar_wait(smem_u32(&bars[1]), it & 1, a.d_err) ? 1 : 0;
    }
    __syncthreads();   // the tile's buffers are free again
    if (!*flag) ok = false;
  }
  if (bad_page) atomicOr(a.d_err, kErrBadPage);

  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  if (ok && warp < 2) {
    // head dim d = t: combine the tiles in order
    const int d = t;
    float M[kTcRows], L[kTcRows], acc[kTcRows];
#pragma unroll
    for (int r = 0; r < kTcRows; ++r) {
      M[r] = -INFINITY;
      for (int i = 0; i < n_tiles; ++i) M[r] = fmaxf(M[r], mt[i * kTcRows + r]);
      L[r] = 0.f;
      acc[r] = 0.f;
    }
    for (int i = 0; i < n_tiles; ++i) {
      float o[kTcRows];
      tmem_ld16(tmem + ((uint32_t)(warp * 32) << 16) + kTcRows + kTcRows * i, o);
#pragma unroll
      for (int r = 0; r < kTcRows; ++r) {
        const float m = mt[i * kTcRows + r];
        const float wgt = (m == -INFINITY) ? 0.f : expf(m - M[r]);
        L[r] += lt[i * kTcRows + r] * wgt;
        acc[r] += o[r] * wgt;
      }
    }
#pragma unroll
    for (int r = 0; r < kTcRows; ++r) {
      if (r >= nr) continue;
      const int row = row0 + r;
      if (a.n_split == 1) {
        reinterpret_cast<__nv_bfloat16*>(a.out)[(size_t)row * a.H * 64 + h * 64 + d] =
            __float2bfloat16_rn(acc[r] / L[r]);
      } else {
        a.part_o[(((size_t)split * a.R + row) * a.H + h) * 64 + d] = acc[r];
        if (d == 0) a.part_ml[((size_t)split * a.R + row) * a.H + h] = make_float2(M[r], L[r]);
      }
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  if (warp == 0)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTcCols)
                 : "memory");
}

int attention_tc_max_keys() { return kTcMaxTiles * kTcKeys; }

void launch_attention_tc(const AttnArgs& a, int n_groups, cudaStream_t s) {
  if (n_groups == 0) return;
  static bool attr = false;
  if (!attr) {
    cudaFuncSetAttribute(k_attention_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, kTcSmemLaunch);
    attr = true;
  }
  kf_launch(k_attention_tc, dim3(n_groups, a.H, a.n_split), dim3(128), kTcSmemLaunch, s, a);
}

}  // namespace kf
