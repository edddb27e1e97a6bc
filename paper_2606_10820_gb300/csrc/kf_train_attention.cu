// Training-time attention of App. C.2 (SingleForward / DoubleForward) on
// warp-level bf16 MMA, visiting only the key tiles the mask opens.
//
// Token layout of one sequence (T tokens): context x_1..x_N at 0..N-1, then
// `blocks` blocks of N*k tokens, k per context position; token (t, a) of
// block b sits at N + (b-1) N k + t k + a.  A query row sees
//   context row i:          context keys 0..i;
//   block-1 row (t, a):     context 0..t, block-1 tokens (t, 0..a);
//   block-2 row (t, a):     context 0..t, block-1 tokens (t, 0..k-1),
//                           block-2 tokens (t, 0..a).
// SingleForward is blocks = 1 (block 1 = the noise tokens); DoubleForward is
// blocks = 2 (Future-1 predictions, Future-2 noise).
//
// A CTA (4 warps) takes 64 consecutive query rows of one (sequence, head),
// warp w owning rows 16w..16w+15 (FlashAttention-2 layout: no cross-warp
// merge).  The CTA walks three disjoint key ranges: the context prefix up to
// the largest context key any of its rows sees, and the block-1 / block-2
// windows of its rows' groups, in 64-key tiles (cp.async into swizzled shared
// memory, double-buffered) that all four warps read.  A warp skips a tile
// none of its rows sees; inside a tile every (row, key) pair is masked by
// the rule above, except in tiles of context keys every row of the warp sees.
// S = Q K^T and O += P V run on mma.sync m16n8k16 with P in registers and
// an online softmax per row.  The visited pairs grow like the mask (O(k) over
// AR attention) instead of the (N + N k)^2 of a dense mask; dense = 1 visits
// every key tile with the same per-element mask, the cost of passing the mask
// densely.
#include <cuda_bf16.h>

#include <algorithm>

#include "../../include/kforcing_ops.h"
#include "kf_internal.cuh"
#include "kf_mma.cuh"
#include "kf_tc.cuh"

namespace kf {
namespace {

using namespace mma;

constexpr int kTile = 64;      // keys per K/V tile
constexpr int kThr = 128;      // 4 warps, 16 query rows each
constexpr int kRows = 64;      // query rows per CTA

struct TrainAttnArgs {
  const __nv_bfloat16* q;      // [B][T][H][64]
  const __nv_bfloat16* k;
  const __nv_bfloat16* v;
  float* out;                  // [B][q_end - q_begin][H][64]
  int N, kw, blocks, T, H, q_begin, q_end, dense;
};

// the keys row qi sees: context keys <= ctx, and [w1lo, w1hi), [w2lo, w2hi)
struct RowVis {
  int ctx, w1lo, w1hi, w2lo, w2hi;
};

__device__ __forceinline__ RowVis row_vis(const TrainAttnArgs& a, int qi) {
  RowVis r{-1, 0, 0, 0, 0};
  if (qi < a.q_begin || qi >= a.q_end) return r;
  const int Nk = a.N * a.kw;
  if (qi < a.N) {
    r.ctx = qi;
    return r;
  }
  const int rel = qi - a.N;
  const int blk = rel / Nk;                 // 0: block 1, 1: block 2
  const int t = (rel - blk * Nk) / a.kw, pos = (rel - blk * Nk) - t * a.kw;
  r.ctx = t;
  r.w1lo = a.N + t * a.kw;
  r.w1hi = r.w1lo + (blk == 0 ? pos + 1 : a.kw);
  if (blk == 1) {
    r.w2lo = a.N + Nk + t * a.kw;
    r.w2hi = r.w2lo + pos + 1;
  }
  return r;
}

__device__ __forceinline__ bool sees(const RowVis& r, int key) {
  return key <= r.ctx || (key >= r.w1lo && key < r.w1hi) || (key >= r.w2lo && key < r.w2hi);
}

constexpr size_t smem_bytes() { return (size_t)kRows * kHD * 2 + 2 * 2 * (size_t)kTile * kHD * 2; }

}  // namespace

__global__ void __launch_bounds__(kThr, 3) k_train_attention(TrainAttnArgs a) {
  pdl_wait();
  extern __shared__ __align__(128) uint8_t sm[];
  __nv_bfloat16* Qs = reinterpret_cast<__nv_bfloat16*>(sm);       // [64][64] swizzled
  __nv_bfloat16* Ks = Qs + kRows * kHD;                           // [2][64][64] swizzled
  __nv_bfloat16* Vs = Ks + 2 * kTile * kHD;

  const int q0 = a.q_begin + blockIdx.x * kRows, h = blockIdx.y, b = blockIdx.z;
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const int g = lane >> 2, tq = lane & 3;
  const size_t seq = (size_t)b * a.T;
  const int qw = q0 + 16 * warp;                                  // this warp's 16 rows
  const RowVis v0 = row_vis(a, qw + g), v1 = row_vis(a, qw + g + 8);

  // key ranges of the CTA's 64 rows (every thread computes the same), and per
  // warp the context keys all its valid rows see and the last key any sees
  int rlo[3], rhi[3], nr = 0;
  int wcmin = 1 << 30, wmax = -1;
  {
    int cmax = -1, w1lo = 1 << 30, w1hi = 0, w2lo = 1 << 30, w2hi = 0;
    for (int i = 0; i < kRows; ++i) {
      const RowVis r = row_vis(a, q0 + i);
      cmax = max(cmax, r.ctx);
      if (r.w1hi > r.w1lo) { w1lo = min(w1lo, r.w1lo); w1hi = max(w1hi, r.w1hi); }
      if (r.w2hi > r.w2lo) { w2lo = min(w2lo, r.w2lo); w2hi = max(w2hi, r.w2hi); }
      if (i / 16 == warp && r.ctx >= 0) {
        wcmin = min(wcmin, r.ctx);
        wmax = max(wmax, max(r.ctx, max(r.w1hi, r.w2hi) - 1));
      }
    }
    if (a.dense) {
      rlo[0] = 0; rhi[0] = a.T; nr = 1;
    } else {
      if (cmax >= 0) { rlo[nr] = 0; rhi[nr] = cmax + 1; ++nr; }
      if (w1hi > w1lo) { rlo[nr] = w1lo; rhi[nr] = w1hi; ++nr; }
      if (w2hi > w2lo) { rlo[nr] = w2lo; rhi[nr] = w2hi; ++nr; }
    }
  }
  int n_tiles = 0;
  for (int i = 0; i < nr; ++i) n_tiles += ceil_div(rhi[i] - rlo[i], kTile);
  auto tile_at = [&](int j, int* lo, int* hi) {
    for (int i = 0; i < nr; ++i) {
      const int n = ceil_div(rhi[i] - rlo[i], kTile);
      if (j < n) { *lo = rlo[i] + j * kTile; *hi = rhi[i]; return; }
      j -= n;
    }
  };
  auto load_tile = [&](int j, int buf) {
    int kt = 0, kend = 0;
    tile_at(j, &kt, &kend);
    __nv_bfloat16* kd = Ks + (size_t)buf * kTile * kHD;
    __nv_bfloat16* vd = Vs + (size_t)buf * kTile * kHD;
#pragma unroll
    for (int q = 0; q < kTile * 8 / kThr; ++q) {
      const int idx = t + q * kThr;
      const int r = idx >> 3, c = idx & 7;
      const int key = kt + r;
      const bool in = key < kend;
      const size_t off = ((seq + (in ? key : 0)) * a.H + h) * kHD + c * 8;
      cp_async16(smem_addr(kd + swz(r, c)), a.k + off, in ? 16 : 0);
      cp_async16(smem_addr(vd + swz(r, c)), a.v + off, in ? 16 : 0);
    }
    cp_commit();
  };

  if (n_tiles > 0) load_tile(0, 0);
#pragma unroll
  for (int q = 0; q < kRows * 8 / kThr; ++q) {
    // the CTA's query rows (zero beyond q_end)
    const int idx = t + q * kThr;
    const int r = idx >> 3, c = idx & 7;
    const int qi = q0 + r;
    uint4 val = make_uint4(0, 0, 0, 0);
    if (qi < a.q_end) val = *reinterpret_cast<const uint4*>(a.q + ((seq + qi) * a.H + h) * kHD + c * 8);
    *reinterpret_cast<uint4*>(Qs + swz(r, c)) = val;
  }
  __syncthreads();
  // this warp's Q fragments, kept in registers for every tile
  uint32_t qa[4][4];
  {
    const uint32_t qbase = smem_addr(Qs);
    const int r = 16 * warp + (lane & 7) + 8 * ((lane >> 3) & 1);
#pragma unroll
    for (int ks = 0; ks < 4; ++ks) ldsm_x4(qbase + 2 * swz(r, 2 * ks + (lane >> 4)), qa[ks]);
  }
  // scores in base-2 units: log2(e) / sqrt(hd), applied to S in fp32
  const float sc = 1.4426950408889634f * rsqrtf((float)kHD);

  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  float o[8][4];
#pragma unroll
  for (int nd = 0; nd < 8; ++nd) o[nd][0] = o[nd][1] = o[nd][2] = o[nd][3] = 0.f;

  for (int it = 0; it < n_tiles; ++it) {
    const int buf = it & 1;
    if (it + 1 < n_tiles) {
      load_tile(it + 1, buf ^ 1);
      cp_wait<1>();
    } else {
      cp_wait<0>();
    }
    __syncthreads();
    int kt = 0, kend = 0;
    tile_at(it, &kt, &kend);
    // warp-uniform: skip a tile none of this warp's rows sees
    if (kt <= wmax) {
      const uint32_t kbase = smem_addr(Ks + (size_t)buf * kTile * kHD);
      const uint32_t vbase = smem_addr(Vs + (size_t)buf * kTile * kHD);
      // S = Q K^T: 16 rows x 64 keys (n-tile j = keys kt + 8j .. +7)
      float s[8][4];
#pragma unroll
      for (int j = 0; j < 8; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
#pragma unroll
        for (int p = 0; p < 2; ++p) {
          uint32_t kb[4];
          ldsm_x4(kbase + 2 * swz(8 * j + (lane & 7), 4 * p + (lane >> 3)), kb);
          mma16816(s[j], qa[2 * p], kb[0], kb[1]);
          mma16816(s[j], qa[2 * p + 1], kb[2], kb[3]);
        }
      }
      // mask; a tile of context keys every row of the warp sees needs none
      const bool open = kt + kTile - 1 < kend && kt + kTile - 1 <= wcmin && a.dense == 0;
      float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int key = kt + 8 * j + 2 * tq + e;
          const bool in = key < kend;
          s[j][e] = (open || (in && sees(v0, key))) ? s[j][e] * sc : -INFINITY;
          s[j][2 + e] = (open || (in && sees(v1, key))) ? s[j][2 + e] * sc : -INFINITY;
          mx0 = fmaxf(mx0, s[j][e]);
          mx1 = fmaxf(mx1, s[j][2 + e]);
        }
      }
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
      const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
      const float c0 = (mn0 == -INFINITY) ? 1.f : ex2(m0 - mn0);
      const float c1 = (mn1 == -INFINITY) ? 1.f : ex2(m1 - mn1);
      m0 = mn0;
      m1 = mn1;
      uint32_t pk[8][2];
      float ps0 = 0.f, ps1 = 0.f;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        pk[j][0] = (mn0 == -INFINITY) ? 0u : pack_bf16(ex2(s[j][0] - mn0), ex2(s[j][1] - mn0));
        pk[j][1] = (mn1 == -INFINITY) ? 0u : pack_bf16(ex2(s[j][2] - mn1), ex2(s[j][3] - mn1));
        const float2 f0 = unpack_bf16(pk[j][0]), f1 = unpack_bf16(pk[j][1]);
        ps0 += f0.x + f0.y;
        ps1 += f1.x + f1.y;
      }
      l0 = l0 * c0 + ps0;
      l1 = l1 * c1 + ps1;
#pragma unroll
      for (int nd = 0; nd < 8; ++nd) {
        o[nd][0] *= c0; o[nd][1] *= c0;
        o[nd][2] *= c1; o[nd][3] *= c1;
      }
      // O += P V: k-step kk = keys kt + 16kk .. +15
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        const uint32_t pa[4] = {pk[2 * kk][0], pk[2 * kk][1], pk[2 * kk + 1][0], pk[2 * kk + 1][1]};
        const int vr = 16 * kk + 8 * ((lane >> 3) & 1) + (lane & 7);
#pragma unroll
        for (int np = 0; np < 4; ++np) {
          uint32_t vb[4];
          ldsm_x4_t(vbase + 2 * swz(vr, 2 * np + (lane >> 4)), vb);
          mma16816(o[2 * np], pa, vb[0], vb[1]);
          mma16816(o[2 * np + 1], pa, vb[2], vb[3]);
        }
      }
    }
    __syncthreads();   // the buffer is refilled next iteration
  }

  // each warp owns its rows: normalise and store
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  const int qa0 = qw + g, qa1 = qw + g + 8;
  const size_t nq = (size_t)(a.q_end - a.q_begin);
  if (qa0 < a.q_end) {
    const float inv = 1.f / l0;
    float* dst = a.out + (((size_t)b * nq + (qa0 - a.q_begin)) * a.H + h) * kHD + 2 * tq;
#pragma unroll
    for (int nd = 0; nd < 8; ++nd)
      *reinterpret_cast<float2*>(dst + 8 * nd) = make_float2(o[nd][0] * inv, o[nd][1] * inv);
  }
  if (qa1 < a.q_end) {
    const float inv = 1.f / l1;
    float* dst = a.out + (((size_t)b * nq + (qa1 - a.q_begin)) * a.H + h) * kHD + 2 * tq;
#pragma unroll
    for (int nd = 0; nd < 8; ++nd)
      *reinterpret_cast<float2*>(dst + 8 * nd) = make_float2(o[nd][2] * inv, o[nd][3] * inv);
  }
}

// ------------------------------------------------------------------ tcgen05
// The same attention on the 5th-generation tensor cores.  A work item is 128
// query rows of one (sequence, head); its key ranges are walked in tiles of
// 128 keys (each range's tiles start at its first key; keys past the range's
// end are masked, so no key is counted twice).  The kernel is persistent:
// one CTA per SM takes items blockIdx.x, blockIdx.x + gridDim.x, ... (the
// query tiles with the most keys first), and its roles run ahead across
// items, so that the next item's copies and first products overlap this
// item's last softmax tile and output:
//   warp 0      TMA: an item's Q (once the previous item's last S product
//               has read the Q buffer), then its K and V tiles of
//               [128 keys][64] bf16 (128-byte swizzle) into a four-stage ring;
//   warp 1      one thread issues tcgen05.mma: S_j = Q K_j^T (M = 128 rows,
//               N = 128 keys, K = 64) into one of two TMEM buffers, and
//               O += P_j V_j (M = 128, N = 64, K = 128 keys; V is the
//               MN-major operand as loaded) into one TMEM accumulator, an
//               item's first P V overwriting it once the softmax has read
//               the previous item's O;
//   warps 2..9  two threads per query row (TMEM lane), each with half of
//               its keys and of its output (four threads measured 5 % slower:
//               the per-tile chain of waits and barriers, not the arithmetic,
//               bounds the softmax): mask S_j, share the row max with the
//               partner warp (the other half of the same rows) through shared
//               memory and a barrier of the pair, keep a reference max m and
//               their part of the sum l, and write P_j = exp2(S_j - m) as
//               bf16 into shared memory (K-major, swizzled: the A operand of
//               P V); every softmax thread arrives on the barrier that
//               releases P_j to the tensor cores.  m
//               is raised only when a tile's max exceeds it by more than 2^8
//               (P stays below 256); then O in TMEM and l are scaled to the
//               new m before P_j is released.  At the item's end O / l is
//               the row's output.
// Tiles are numbered across the CTA's items (g): S of tile g + 1 is computed
// while the softmax works on tile g, and P V of tile g is issued after it
// (an item's last P V right after its last S).
// Every wait is bounded; a wait that runs out sets the error word and ends
// the CTA's loops.
namespace {
constexpr int kTcRows = 128;
constexpr int kTcKeys = 128;
constexpr int kTcSplit = 2;                          // softmax threads per query row
constexpr int kTcSoftmax = 128 * kTcSplit;           // kTcSplit warps per TMEM lane quarter
constexpr int kTcThreads = 64 + kTcSoftmax;
constexpr int kTcPart = kTcKeys / kTcSplit;          // keys of a row per softmax thread
constexpr int kTcOut = kHD / kTcSplit;               // output dims of a row per softmax thread
constexpr uint32_t kTcTile = kTcRows * kHD * 2;       // 16 KB: Q, a K tile, a V tile
constexpr uint32_t kTcP = kTcRows * kTcKeys * 2;      // 32 KB: one P tile (two 64-key atoms)
// K/V ring stages: tile j's copies are issued while tile j - 1 is in the
// softmax and tile j - 2's V still feeds P V (two stages measured 2.0 us per
// tile, the copy latency on the critical path)
constexpr int kTcStages = 4;
// [Q][K stages][V stages][P 2], the barriers and shared scalars (256 B),
// then the row-max exchange [2 tiles][kTcSplit parts][128 rows] and the row
// sums [2 items][kTcSplit][128]
constexpr size_t tc_smem_bytes() {
  return 1024 + (1 + 2 * kTcStages) * (size_t)kTcTile + 2 * (size_t)kTcP + 256 + 4 * kTcSplit * 128 * 4;
}

// The key ranges an item's 128 query rows open (the union over its rows:
// the context prefix up to the largest context key, the block-1 and block-2
// windows; an empty one has lo == hi), the smallest context key every valid
// row sees, and the number of 128-key tiles.  Warp-collective: each lane
// takes four rows.
struct TileRanges {
  int lo[3], hi[3], cmin, n;
};

__device__ __forceinline__ TileRanges tile_ranges(const TrainAttnArgs& a, int q0, int lane) {
  int cmax = -1, cmin = 1 << 30, w1lo = 1 << 30, w1hi = 0, w2lo = 1 << 30, w2hi = 0;
#pragma unroll
  for (int i = 0; i < kTcRows / 32; ++i) {
    const RowVis v = row_vis(a, q0 + lane + 32 * i);
    if (v.ctx < 0) continue;
    cmax = max(cmax, v.ctx);
    cmin = min(cmin, v.ctx);
    if (v.w1hi > v.w1lo) { w1lo = min(w1lo, v.w1lo); w1hi = max(w1hi, v.w1hi); }
    if (v.w2hi > v.w2lo) { w2lo = min(w2lo, v.w2lo); w2hi = max(w2hi, v.w2hi); }
  }
  cmax = __reduce_max_sync(0xffffffffu, cmax);
  cmin = __reduce_min_sync(0xffffffffu, cmin);
  w1lo = __reduce_min_sync(0xffffffffu, w1lo);
  w1hi = __reduce_max_sync(0xffffffffu, w1hi);
  w2lo = __reduce_min_sync(0xffffffffu, w2lo);
  w2hi = __reduce_max_sync(0xffffffffu, w2hi);
  TileRanges r;
  if (a.dense) {
    r.lo[0] = 0; r.hi[0] = a.T;
    r.lo[1] = r.hi[1] = r.lo[2] = r.hi[2] = 0;
  } else {
    r.lo[0] = 0; r.hi[0] = cmax + 1;                              // 0 when no valid row
    r.lo[1] = w1lo; r.hi[1] = max(w1lo, w1hi);
    r.lo[2] = w2lo; r.hi[2] = max(w2lo, w2hi);
  }
  r.cmin = cmin;
  r.n = 0;
#pragma unroll
  for (int i = 0; i < 3; ++i) r.n += ceil_div(r.hi[i] - r.lo[i], kTcKeys);
  return r;
}

// The two softmax warps of a TMEM lane quarter hold the two parts of the same
// rows; they meet on named barrier 2 + quarter (64 threads), which also ORs
// a predicate over them: both get the same answer and leave a loop together.
__device__ __forceinline__ bool pair_bar_or(int quarter, bool pred) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.or.pred q, %2, 64, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"((uint32_t)pred), "r"(2 + quarter)
      : "memory");
  return r != 0;
}
__device__ __forceinline__ void pair_bar(int quarter) {
  asm volatile("bar.sync %0, 64;" ::"r"(2 + quarter) : "memory");
}

// three-way max, and packed pairs of fp32 (two lanes of one 64-bit register)
__device__ __forceinline__ float max3f(float x, float y, float z) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(x), "f"(y), "f"(z));
  return r;
}
__device__ __forceinline__ uint64_t f2(float x, float y) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(x), "f"(y));
  return r;
}
__device__ __forceinline__ float2 f2_split(uint64_t p) {
  float2 r;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(r.x), "=f"(r.y) : "l"(p));
  return r;
}
__device__ __forceinline__ uint64_t fma_f2(uint64_t x, uint64_t y, uint64_t z) {
  uint64_t r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(x), "l"(y), "l"(z));
  return r;
}
__device__ __forceinline__ uint64_t add_f2(uint64_t x, uint64_t y) {
  uint64_t r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(x), "l"(y));
  return r;
}

// first key and range end of tile j of an item (constant indices only: the
// ranges stay in registers)
__device__ __forceinline__ void tile_at(const TileRanges& r, int j, int* lo, int* hi) {
  *lo = 0; *hi = 0;
#pragma unroll
  for (int i = 0; i < 3; ++i) {
    const int n = ceil_div(r.hi[i] - r.lo[i], kTcKeys);
    if (j >= 0 && j < n) { *lo = r.lo[i] + j * kTcKeys; *hi = r.hi[i]; }
    j -= n;
  }
}
}  // namespace

__global__ void __launch_bounds__(kTcThreads, 1)
k_train_attention_tc(const __grid_constant__ CUtensorMap map_q, const __grid_constant__ CUtensorMap map_k,
                     const __grid_constant__ CUtensorMap map_v, TrainAttnArgs a, int n_batch, int* d_err) {
  extern __shared__ __align__(1024) uint8_t tsm_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(tsm_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sQ = smem_u32(sm);
  const uint32_t sK = sQ + kTcTile;                  // [kTcStages]
  const uint32_t sV = sK + kTcStages * kTcTile;      // [kTcStages]
  constexpr uint32_t kPOff = (1 + 2 * kTcStages) * kTcTile;
  uint8_t* Pp = sm + kPOff;                          // [2][2 atoms][128 rows][128 B]
  const uint32_t sP = smem_u32(Pp);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + kPOff + 2 * kTcP);
  uint64_t* q_full = bars;
  uint64_t* q_empty = bars + 1;                      // the item's last S product done
  uint64_t* kv_full = bars + 2;                      // [kTcStages]
  uint64_t* kv_empty = kv_full + kTcStages;          // [kTcStages]
  uint64_t* s_full = kv_empty + kTcStages;           // [2]
  uint64_t* p_full = s_full + 2;                     // [2]: P_g written (and S_g read)
  uint64_t* o_full = p_full + 2;                     // [2]
  uint64_t* o_free = o_full + 2;                     // the item's O read out
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(o_free + 1);
  int* s_cnt = reinterpret_cast<int*>(tmem_slot + 1);    // K/V tiles the MMA thread has taken
  int* s_qcnt = s_cnt + 1;                               // Q tiles the MMA thread has taken
  float* s_mx = reinterpret_cast<float*>(sm + kPOff + 2 * kTcP + 256);         // [2][kTcSplit][128]
  float* s_l = s_mx + 2 * kTcSplit * kTcRows;                                  // [2][kTcSplit][128]

  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  const int quarter = warp & 3;                 // softmax warps: TMEM lanes 32 quarter ..
  const int row = 32 * quarter + lane;          // this softmax thread's query row in the tile
  const int part = (warp - 2) >> 2;             // its keys kTcPart part .. and output dims kTcOut part ..
  const int n_qt = ceil_div(a.q_end - a.q_begin, kTcRows);
  const int n_hb = a.H * n_batch;
  const int n_items = n_qt * n_hb;
  // the CTA's i-th item: rounds of gridDim.x items, walked forwards in even
  // rounds and backwards in odd ones, so that each CTA's items add up to
  // about the same number of tiles; -1 past the last
  auto item_at = [&](int i) -> int {
    const int P = gridDim.x, c = blockIdx.x;
    const long long w = (long long)i * P + ((i & 1) ? P - 1 - c : c);
    return w < n_items ? (int)w : -1;
  };
  // item w: query tile n_qt - 1 - w / n_hb (the most keys first), then head
  // and sequence
  auto item = [&](int w, int* q0, int* h, int* b) {
    const int qt = w / n_hb, hb = w - qt * n_hb;
    *q0 = a.q_begin + (n_qt - 1 - qt) * kTcRows;
    *h = hb % a.H;
    *b = hb / a.H;
  };

  if (t == 0) {
    mbar_init(smem_u32(q_full), 1);
    mbar_init(smem_u32(q_empty), 1);
    for (int i = 0; i < kTcStages; ++i) {
      mbar_init(smem_u32(&kv_full[i]), 1);
      mbar_init(smem_u32(&kv_empty[i]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&s_full[i]), 1);
      mbar_init(smem_u32(&p_full[i]), kTcSoftmax);      // every softmax thread
      mbar_init(smem_u32(&o_full[i]), 1);
    }
    mbar_init(smem_u32(o_free), kTcSoftmax);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_q)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_k)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_v)) : "memory");
    s_cnt[0] = 0;
    s_qcnt[0] = 0;
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(512)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;
  pdl_wait();

  if (warp == 0) {
    bool ok = true;
    int g = 0, issued = 0, q_issued = 0, it = 0;
    for (int w = item_at(0); ok && w >= 0; w = item_at(++it)) {
      int q0, h, b;
      item(w, &q0, &h, &b);
      const TileRanges r = tile_ranges(a, q0, lane);
      if (lane == 0) {
        // the Q buffer is free once the previous item's last S product is done
        if (it > 0 && !mbar_wait(smem_u32(q_empty), (it - 1) & 1, d_err)) ok = false;
        if (ok) {
          mbar_expect_tx(smem_u32(q_full), kTcTile);
          tma_load_4d(sQ, &map_q, smem_u32(q_full), 0, h, q0, b);
          q_issued = it + 1;
        }
        for (int j = 0; ok && j < r.n; ++j, ++g) {
          const int st = g % kTcStages;
          if (g >= kTcStages && !mbar_wait(smem_u32(&kv_empty[st]), ((g / kTcStages) - 1) & 1, d_err)) {
            ok = false;
            break;
          }
          int kt, kend;
          tile_at(r, j, &kt, &kend);
          mbar_expect_tx(smem_u32(&kv_full[st]), 2 * kTcTile);
          tma_load_4d(sK + st * kTcTile, &map_k, smem_u32(&kv_full[st]), 0, h, kt, b);
          tma_load_4d(sV + st * kTcTile, &map_v, smem_u32(&kv_full[st]), 0, h, kt, b);
          issued = g + 1;
        }
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
    }
    if (lane == 0 && !ok) {
      // let the copies still in flight land before the CTA ends (bounded)
      for (int j = *(volatile int*)s_cnt; j < issued; ++j)
        mbar_wait(smem_u32(&kv_full[j % kTcStages]), (j / kTcStages) & 1, d_err);
      if (q_issued > *(volatile int*)s_qcnt) mbar_wait(smem_u32(q_full), (q_issued - 1) & 1, d_err);
    }
    __syncwarp();
  } else if (warp == 1) {
    constexpr uint32_t idesc_s = idesc_bf16(kTcRows, kTcKeys);
    constexpr uint32_t idesc_o = idesc_bf16(kTcRows, kHD) | (1u << 16);   // B (V) MN-major
    bool ok = true;
    int g = 0, it = 0, o_items = 0;
    int pv = -1;                  // the tile whose S is issued and whose P V is not
    bool pv_first = false;        // ... the first tile of its item
    // O += P_i V_i in TMEM columns 256 .. 319.  An item's first tile
    // overwrites O once the softmax has read the previous item's O out; the
    // softmax rescales O in place before it releases P_i when the row max
    // has grown.
    auto issue_pv = [&](int i, bool first) -> bool {
      if (first) {
        if (o_items > 0 && !mbar_wait(smem_u32(o_free), (o_items - 1) & 1, d_err)) return false;
        ++o_items;
      }
      const int st = i & 1;
      if (!mbar_wait(smem_u32(&p_full[st]), (i >> 1) & 1, d_err)) return false;
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const int kvs = i % kTcStages;
      const uint32_t pa = sP + st * kTcP, vb = sV + kvs * kTcTile;
#pragma unroll
      for (int kk = 0; kk < kTcKeys / 16; ++kk)
        mma_bf16(tmem + 256, sdesc(pa + (kk >> 2) * (kTcP / 2) + (kk & 3) * 32),
                 sdesc_mn(vb + kk * 16 * 128), idesc_o, (!first || kk > 0) ? 1u : 0u);
      mma_commit(smem_u32(&o_full[st]));
      mma_commit(smem_u32(&kv_empty[kvs]));
      return true;
    };
    for (int w = item_at(0); ok && w >= 0; w = item_at(++it)) {
      int q0, h, b;
      item(w, &q0, &h, &b);
      const TileRanges r = tile_ranges(a, q0, lane);
      if (lane == 0) {
        ok = mbar_wait(smem_u32(q_full), it & 1, d_err);
        if (ok) *(volatile int*)s_qcnt = it + 1;
        for (int j = 0; ok && j < r.n; ++j, ++g) {
          const int st = g & 1;
          if (!mbar_wait(smem_u32(&kv_full[g % kTcStages]), (g / kTcStages) & 1, d_err)) { ok = false; break; }
          *(volatile int*)s_cnt = g + 1;
          // S buffer st is free once the softmax has read S_{g-2}
          if (g >= 2 && !mbar_wait(smem_u32(&p_full[st]), ((g - 2) >> 1) & 1, d_err)) { ok = false; break; }
          asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
          const uint32_t kb = sK + (g % kTcStages) * kTcTile;
#pragma unroll
          for (int kk = 0; kk < kHD / 16; ++kk)
            mma_bf16(tmem + kTcKeys * st, sdesc(sQ + kk * 32), sdesc(kb + kk * 32), idesc_s, kk > 0 ? 1u : 0u);
          mma_commit(smem_u32(&s_full[st]));
          if (j == r.n - 1) mma_commit(smem_u32(q_empty));
          if (pv >= 0 && !issue_pv(pv, pv_first)) { ok = false; break; }
          pv = g;
          pv_first = j == 0;
          // the item's last P V follows at once: the softmax's read of O
          // does not wait for the next item's copies
          if (j == r.n - 1) {
            if (!issue_pv(pv, pv_first)) { ok = false; break; }
            pv = -1;
          }
        }
        if (ok && r.n == 0) mma_commit(smem_u32(q_empty));
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
    }
    if (lane == 0 && ok && pv >= 0) issue_pv(pv, pv_first);
    __syncwarp();
  } else {
    // softmax: kTcSplit threads per query row, `part` of its keys and output each
    static_assert(kTcPart % 32 == 0 && kTcPart <= 64 && (kTcOut == 16 || kTcOut == 32),
                  "32-column TMEM loads of S, one load of O per thread");
    const float sc = 1.4426950408889634f * rsqrtf((float)kHD);
    const uint32_t lane_base = (uint32_t)(32 * quarter) << 16;
    const int kb0 = kTcPart * part;               // first key of this thread's part of a tile
    constexpr float kRescale = 8.f;
    // this row's 16-byte chunks of P buffer 0 for keys kb0 .. kb0 + 31: atom
    // kb0 / 64, chunks (kb0 % 64) / 8 + q at position chunk ^ (row % 8)
    const uint32_t prow = sP + (kb0 >> 6) * (kTcP / 2) + row * 128;
    const int chunk0 = (kb0 & 63) >> 3;
    // this thread's output dims of the O accumulator in TMEM
    const uint32_t o_addr = tmem + lane_base + 256 + kTcOut * part;
    // A bounded wait that runs out marks the thread failed; the next
    // OR-barrier tells its partner warp, and both leave the loops (the other
    // pairs' waits then run out in turn).
    bool failed = false;
    auto wait_or_abort = [&](uint64_t* bar, uint32_t parity) {
      if (!mbar_wait(smem_u32(bar), parity, d_err)) failed = true;
    };
    bool ok = true;
    int g = 0, it = 0;
    for (int w = item_at(0); ok && w >= 0; w = item_at(++it)) {
      int q0, h, b;
      item(w, &q0, &h, &b);
      const TileRanges r = tile_ranges(a, q0, lane);
      const RowVis v = row_vis(a, q0 + row);
      // the visible keys kb0 + i (i < kTcPart) of a row as a bit mask: [lo, hi) relative to the tile
      auto range_bits = [&](int lo, int hi) -> unsigned long long {
        lo = max(lo - kb0, 0);
        hi = min(hi - kb0, kTcPart);
        if (hi <= lo) return 0ull;
        const unsigned long long up = hi >= 64 ? ~0ull : ((1ull << hi) - 1ull);
        return up & ~((1ull << lo) - 1ull);
      };
      // m: the row max the probabilities of the item's tiles so far are
      // taken against (raised only when a tile's max exceeds it by more than
      // 2^8, so P stays below 256); l: this thread's part of their sum
      float m = -INFINITY, l = 0.f;
      for (int j = 0; j < r.n; ++j, ++g) {
        const int st = g & 1;
        int kt, kend;
        tile_at(r, j, &kt, &kend);
        // visible keys of this part: the context prefix [0, ctx], the windows,
        // none past the range's end (each key belongs to one range's tiles)
        const int lim = min(kend - kt, kTcKeys);
        const bool open = !a.dense && kt + kTcKeys - 1 < kend && kt + kTcKeys - 1 <= r.cmin && v.ctx >= 0;
        unsigned long long vis = ~0ull;
        if (!open)
          vis = (range_bits(0, v.ctx - kt + 1) | range_bits(v.w1lo - kt, v.w1hi - kt) |
                 range_bits(v.w2lo - kt, v.w2hi - kt)) &
                range_bits(0, lim);
        wait_or_abort(&s_full[st], (g >> 1) & 1);
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        float sv[kTcPart];
#pragma unroll
        for (int c = 0; c < kTcPart / 32; ++c) tmem_ld32(tmem + lane_base + kTcKeys * st + kb0 + 32 * c, sv + 32 * c);
        // raw scores: sc > 0, so the max commutes with the scaling
        if (vis != ~0ull) {
#pragma unroll
          for (int e = 0; e < kTcPart; ++e) sv[e] = ((vis >> e) & 1ull) ? sv[e] : -INFINITY;
        }
        // four independent max chains, then combined
        float mq[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
        for (int e = 0; e < kTcPart; e += 8)
#pragma unroll
          for (int c = 0; c < 4; ++c) mq[c] = max3f(mq[c], sv[e + 2 * c], sv[e + 2 * c + 1]);
        float mx = fmaxf(fmaxf(mq[0], mq[1]), fmaxf(mq[2], mq[3]));
        // the row's max over its parts (the partner warp)
        s_mx[(st * kTcSplit + part) * kTcRows + row] = mx;
        if (pair_bar_or(quarter, failed)) { ok = false; break; }
        mx = s_mx[(st * kTcSplit) * kTcRows + row];
#pragma unroll
        for (int q = 1; q < kTcSplit; ++q) mx = fmaxf(mx, s_mx[(st * kTcSplit + q) * kTcRows + row]);
        // A new reference max when this tile's exceeds it by more than 2^8: O
        // and l so far are scaled to it (O once the previous tile's P V has
        // landed; nothing is accumulated before a finite max).  The TMEM
        // load and store are warp-wide: a warp rescales when any of its rows
        // needs it, the others by 1.
        const bool raise = mx * sc > m + kRescale;
        const float f = (raise && m != -INFINITY) ? ex2(m - mx * sc) : 1.f;
        if (__any_sync(0xffffffffu, f != 1.f)) {
          wait_or_abort(&o_full[(g - 1) & 1], ((g - 1) >> 1) & 1);
          asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
          float rr[kTcOut];
          tmem_ld32(o_addr, rr);
#pragma unroll
          for (int d = 0; d < kTcOut; ++d) rr[d] *= f;
          tmem_st32(o_addr, rr);
        }
        if (raise) {
          l *= f;
          m = mx * sc;
        }
        const float mn = m;
        // P = exp2(S sc - mn) rounded to bf16 (ex2(-inf) = 0 for masked keys),
        // the sum of the rounded values
        const uint32_t pbase = prow + st * kTcP;
        const float nmn = mn == -INFINITY ? 0.f : -mn;
        const uint64_t sc2 = f2(sc, sc), nmn2 = f2(nmn, nmn);
        uint64_t ps2[4] = {f2(0.f, 0.f), f2(0.f, 0.f), f2(0.f, 0.f), f2(0.f, 0.f)};   // independent sums
#pragma unroll
        for (int q = 0; q < kTcPart / 8; ++q) {
          uint32_t pk[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int e = 8 * q + 2 * u;
            const float2 arg = f2_split(fma_f2(f2(sv[e], sv[e + 1]), sc2, nmn2));
            pk[u] = pack_bf16(ex2(arg.x), ex2(arg.y));
            const float2 pf = unpack_bf16(pk[u]);
            ps2[u] = add_f2(ps2[u], f2(pf.x, pf.y));
          }
          const uint32_t addr = pbase + (((chunk0 + q) ^ (row & 7)) << 4);
          asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(pk[0]), "r"(pk[1]), "r"(pk[2]),
                       "r"(pk[3])
                       : "memory");
        }
        const float2 ps = f2_split(add_f2(add_f2(ps2[0], ps2[1]), add_f2(ps2[2], ps2[3])));
        l += ps.x + ps.y;
        // S_g read, P_g written: to the tensor cores (async proxy); every
        // softmax thread arrives
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0];" ::"r"(smem_u32(&p_full[st])) : "memory");
      }
      if (!ok) break;
      float o[kTcOut];
#pragma unroll
      for (int d = 0; d < kTcOut; ++d) o[d] = 0.f;
      if (r.n > 0) {
        // the item's last P V completes the accumulator; once every softmax
        // thread has read it, the next item's first P V may overwrite it
        wait_or_abort(&o_full[(g - 1) & 1], ((g - 1) >> 1) & 1);
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        tmem_ld32(o_addr, o);
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        if (pair_bar_or(quarter, failed)) { ok = false; break; }
        asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0];" ::"r"(smem_u32(o_free)) : "memory");
      }
      // the row's sum over its parts, in a fixed order (one buffer per item
      // parity: a thread writes the next item's sums only after the pair
      // barrier below, which its partner passes after reading this item's)
      float* sl = s_l + (it & 1) * kTcSplit * kTcRows;
      sl[part * kTcRows + row] = l;
      pair_bar(quarter);
      float lt = 0.f;
#pragma unroll
      for (int q = 0; q < kTcSplit; ++q) lt += sl[q * kTcRows + row];
      const int qi = q0 + row;
      if (qi < a.q_end && lt > 0.f) {
        const float inv = 1.f / lt;
        float* dst =
            a.out + (((size_t)b * (a.q_end - a.q_begin) + (qi - a.q_begin)) * a.H + h) * kHD + kTcOut * part;
#pragma unroll
        for (int d = 0; d < kTcOut; d += 4)
          *reinterpret_cast<float4*>(dst + d) = make_float4(o[d] * inv, o[d + 1] * inv, o[d + 2] * inv, o[d + 3] * inv);
      }
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  if (warp == 1)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(512) : "memory");
}

}  // namespace kf

using namespace kf;

extern "C" int kf_op_train_attention(int32_t blocks, int32_t B, int32_t H, int32_t N, int32_t k,
                                     int32_t q_begin, int32_t q_end, const void* q, const void* kk,
                                     const void* v, float* out, int32_t dense, void* stream) {
  if ((blocks != 1 && blocks != 2) || B < 1 || H < 1 || N < 1 || k < 1 || !q || !kk || !v || !out)
    return KF_E_ARG;
  const long long T = (long long)N + (long long)blocks * N * k;
  if (T > (1 << 30) / 64 || q_begin < 0 || q_end > T || q_begin >= q_end) return KF_E_ARG;
  if ((reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(kk) | reinterpret_cast<uintptr_t>(v) |
       reinterpret_cast<uintptr_t>(out)) & 15)
    return KF_E_ARG;
  if (dense & ~(KF_TRAIN_ATTN_DENSE | KF_TRAIN_ATTN_WARP_MMA)) return KF_E_ARG;
  TrainAttnArgs a{static_cast<const __nv_bfloat16*>(q), static_cast<const __nv_bfloat16*>(kk),
                  static_cast<const __nv_bfloat16*>(v), out, N, k, blocks, (int)T, H, q_begin, q_end,
                  (dense & KF_TRAIN_ATTN_DENSE) ? 1 : 0};
  cudaStream_t s = (cudaStream_t)stream;
  if (dense & KF_TRAIN_ATTN_WARP_MMA) {
    static PerDevice attr;
    set_smem_attr(attr, k_train_attention, smem_bytes());
    const dim3 grid(ceil_div(q_end - q_begin, kRows), H, B);
    kf_launch(k_train_attention, grid, dim3(kThr), smem_bytes(), s, a);
    return cudaGetLastError() == cudaSuccess ? KF_OK : KF_E_CUDA;
  }
  // q, kk, v as [B][T][H][64] with the head one coordinate: boxes of one
  // head's 128 consecutive tokens (rows past T read as zero)
  const uint64_t dims[4] = {64, (uint64_t)H, (uint64_t)T, (uint64_t)B};
  const uint64_t strides[3] = {128, (uint64_t)H * 128, (uint64_t)T * H * 128};
  const uint32_t box[4] = {64, 1, kTcRows, 1};
  CUtensorMap mq, mk, mv;
  if (!encode_map_bf16(&mq, q, 4, dims, strides, box) || !encode_map_bf16(&mk, kk, 4, dims, strides, box) ||
      !encode_map_bf16(&mv, v, 4, dims, strides, box))
    return KF_E_CUDA;
  int* err = op_error_word(s);
  if (!err) return KF_E_CUDA;
  static PerDevice attr_tc;
  set_smem_attr(attr_tc, k_train_attention_tc, tc_smem_bytes());
  // persistent: one CTA per SM over the (query tile, head, sequence) items
  const long long items = (long long)ceil_div(q_end - q_begin, kTcRows) * H * B;
  if (items > (1ll << 30)) return KF_E_ARG;
  const dim3 grid((unsigned)std::min<long long>(items, device_sms()));
  kf_launch(k_train_attention_tc, grid, dim3(kTcThreads), tc_smem_bytes(), s, mq, mk, mv, a, (int)B, err);
  return cudaGetLastError() == cudaSuccess ? KF_OK : KF_E_CUDA;
}
