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
  pdl_trigger();
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
  TrainAttnArgs a{static_cast<const __nv_bfloat16*>(q), static_cast<const __nv_bfloat16*>(kk),
                  static_cast<const __nv_bfloat16*>(v), out, N, k, blocks, (int)T, H, q_begin, q_end,
                  dense ? 1 : 0};
  static PerDevice attr;
  set_smem_attr(attr, k_train_attention, smem_bytes());
  const dim3 grid(ceil_div(q_end - q_begin, kRows), H, B);
  kf_launch(k_train_attention, grid, dim3(kThr), smem_bytes(), (cudaStream_t)stream, a);
  return cudaGetLastError() == cudaSuccess ? KF_OK : KF_E_CUDA;
}
