// Decode attention on warp-level tensor-core MMA (mma.sync m16n8k16, bf16
// operands, fp32 accumulation) for the bf16 cache with head_dim 64: up to 16
// query rows of one sequence and one head per CTA against every cached key
// at or before each row's position (the fully causal mask of Sec. 3.3 /
// Alg. 1).
//
// Per CTA (4 warps), keys in tiles of 128 (8 pages).  Each page of K and of
// V for the CTA's head is 16 contiguous 128-byte rows of the cache; one TMA
// copy per page and operand lands it 128-byte swizzled (16-byte chunk c of
// row r at chunk c ^ (r % 8)), so ldmatrix reads are conflict-free, and one
// mbarrier per buffer counts the bytes.  NBUF = 2: a ring of two buffers,
// the next tile in flight while one is reduced (3 CTAs per SM); NBUF = 1:
// one buffer refilled after each tile, 6 CTAs per SM overlapping each
// other's loads.  Warp w owns keys
// 32w .. 32w+31 of every tile and keeps its own online softmax over them
// (FlashAttention-2 style):
//   S = Q K^T      16 rows x 32 keys, 16 MMAs (Q zero-padded to 16 rows)
//   P = exp(S - m) in registers; the S accumulator layout is the A-operand
//                  layout of the next MMA, so P never leaves the registers
//   O += P V       16 rows x 64 dims, 16 MMAs (V through ldmatrix.trans)
// Only tiles that reach past the first row's position are masked.  The four
// warps' (m, l, O) are merged once at the end in a fixed order
// (deterministic); with n_split > 1 each CTA covers one key range and
// k_attn_combine merges the partial softmaxes in split order.
//
// Decode attention reads every cached K/V byte once and is bound by HBM; at
// 1..16 query rows a tcgen05 MMA (M >= 64, accumulators in tensor memory)
// would need a TMEM round trip for the softmax of every tile, while these
// register-resident fragments keep the per-tile work to about 40
// instructions per warp besides the MMAs.
#include <cuda_bf16.h>

#include <algorithm>

#include "kf_mma.cuh"
#include "kf_tc.cuh"

namespace kf {
namespace {

using namespace mma;

constexpr int kTile = 128;     // keys per K/V tile
constexpr int kThr = 128;      // 4 warps x 32 keys of each tile
constexpr int kQRows = 16;     // MMA M: query rows of the group, zero-padded
constexpr int kPageBytes = kPage * kHD * 2;                  // one page of K (or V) of one head
constexpr int kTileBytes = kTile * kHD * 2;                  // 16 KB

// [NBUF K tiles][NBUF V tiles][Q 16 x 64][NBUF mbarriers][flag][page ids], from a
// 1024-byte aligned base (the swizzle pattern repeats every 8 rows)
constexpr size_t smem_bytes(int nbuf, int pg_cap) {
  return 1024 + (size_t)2 * nbuf * kTileBytes + (size_t)kQRows * kHD * 2 + 8 * nbuf + 8 + 4 * pg_cap;
}

}  // namespace

// the split merge of one (group, head), by thread t: row t / 8, dims
// 8 (t % 8) .. +7
__device__ __forceinline__ void merge_splits(const float* part_o, const float2* part_ml, __nv_bfloat16* out,
                                          int n_split, int R, int H, int row0, int nr, int h, int t) {
  const int r = t >> 3, d0 = (t & 7) * 8;
  if (r < nr) {
    // one pass in split order, four splits' loads in flight at a time;
    // the running maximum M rescales the sums when it grows
    const int row = row0 + r;
    float M = -INFINITY, L = 0.f, acc[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) acc[q] = 0.f;
    for (int sp0 = 0; sp0 < n_split; sp0 += 4) {
      float2 ml[4];
      float4 u0[4], u1[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        if (sp0 + j < n_split) {
          const size_t u = ((size_t)(sp0 + j) * R + row) * H + h;
          ml[j] = __ldcg(part_ml + u);
          const float4* po = reinterpret_cast<const float4*>(part_o + u * kHD + d0);
          u0[j] = __ldcg(po);
          u1[j] = __ldcg(po + 1);
        } else {
          ml[j] = make_float2(-INFINITY, 0.f);
        }
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        if (ml[j].x == -INFINITY) continue;        // an empty split
        const float Mn = fmaxf(M, ml[j].x);
        const float cs = (M == -INFINITY) ? 0.f : expf(M - Mn);
        const float w = expf(ml[j].x - Mn);
        M = Mn;
        L = L * cs + ml[j].y * w;
        acc[0] = acc[0] * cs + u0[j].x * w; acc[1] = acc[1] * cs + u0[j].y * w;
        acc[2] = acc[2] * cs + u0[j].z * w; acc[3] = acc[3] * cs + u0[j].w * w;
        acc[4] = acc[4] * cs + u1[j].x * w; acc[5] = acc[5] * cs + u1[j].y * w;
        acc[6] = acc[6] * cs + u1[j].z * w; acc[7] = acc[7] * cs + u1[j].w * w;
      }
    }
    const float inv = 1.f / L;
    uint4 pk;
    pk.x = pack_bf16(acc[0] * inv, acc[1] * inv);
    pk.y = pack_bf16(acc[2] * inv, acc[3] * inv);
    pk.z = pack_bf16(acc[4] * inv, acc[5] * inv);
    pk.w = pack_bf16(acc[6] * inv, acc[7] * inv);
    *reinterpret_cast<uint4*>(out + (size_t)row * H * kHD + h * kHD + d0) = pk;
  }
}

// NBUF = 1: one tile buffer, refilled after each tile; NBUF = 2: two tile buffers.  TWO:
// groups of more than 8 rows (rows 8..15 of the MMA carry data).  Decode
// CTAs (a.len set, one group per sequence): the pages wholly before the
// sequence's committed length were written by earlier steps and the page
// table by the host before the step, so the page ids and the copies of those
// pages are issued before waiting for the kernel that appends this step's
// keys; the other pages and Q are loaded after the wait.
template <int NBUF, bool TWO>
__global__ void __launch_bounds__(kThr, NBUF == 1 ? (TWO ? 5 : 6) : 3)
k_attention_mma(const __grid_constant__ CUtensorMap map_kv, AttnArgs a) {
  extern __shared__ __align__(1024) uint8_t sm_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(sm_raw) + 1023) & ~uintptr_t(1023));
  __nv_bfloat16* Ks = reinterpret_cast<__nv_bfloat16*>(sm);   // [NBUF][128][64] swizzled
  __nv_bfloat16* Vs = Ks + NBUF * kTile * kHD;                // [NBUF][128][64] swizzled
  __nv_bfloat16* Qs = Vs + NBUF * kTile * kHD;                // [16][64] swizzled
  uint64_t* bars = reinterpret_cast<uint64_t*>(Qs + kQRows * kHD);
  int* s_pg = reinterpret_cast<int*>(bars + NBUF) + 2;       // [a.pg_cap] (NBUF = 2), after a flag

  const int gi = blockIdx.x, h = blockIdx.y, split = blockIdx.z;
  const bool early = a.len != nullptr && a.groups == nullptr;
  int b, row0, nr, n_keys, stable;
  if (early) {
    b = a.order ? __ldg(a.order + gi) : gi;
    row0 = b * a.uniform_rows; nr = a.uniform_rows;
    stable = a.len[b];                       // committed length: positions row_pos of the step
    n_keys = stable + nr;
  } else {
    pdl_wait();
    if (a.groups) {
      const int4 gg = a.groups[gi];
      b = gg.x; row0 = gg.y; nr = gg.z;
    } else {
      b = a.order ? __ldg(a.order + gi) : gi;
      row0 = b * a.uniform_rows; nr = a.uniform_rows;
    }
    n_keys = a.row_pos[row0 + nr - 1] + 1;
    stable = 0;
  }
  const int k_begin = split * a.keys_per_split;
  const int k_end = min(n_keys, k_begin + a.keys_per_split);
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const int g = lane >> 2, tq = lane & 3;     // MMA fragment row group / column pair

  const int n_tiles = k_end > k_begin ? ceil_div(k_end - k_begin, kTile) : 0;
  const int pg0 = k_begin / kPage;            // k_begin is a multiple of the page size
  int n_pg = 0;
  if constexpr (NBUF > 1) {
    // the page ids of the keys [k_begin, k_end)
    n_pg = k_end > k_begin ? ceil_div(k_end, kPage) - pg0 : 0;
    if (n_pg > a.pg_cap) {
      if (t == 0) atomicOr(a.d_err, kErrInternal);
      n_pg = a.pg_cap;
    }
    for (int i = t; i < n_pg; i += kThr)
      s_pg[i] = pg0 + i < a.max_pages ? __ldg(a.page_table + (size_t)b * a.max_pages + pg0 + i) : -1;
  }
  // V rows of pages that are not copied (past the last key) stay finite: the
  // masked keys' probabilities are 0 and 0 * V must be 0
  for (int i = t; i < NBUF * kTile * kHD / 8; i += kThr)
    reinterpret_cast<uint4*>(Vs)[i] = make_uint4(0u, 0u, 0u, 0u);
  if (t == 0) {
    for (int i = 0; i < NBUF; ++i) mbar_init(smem_u32(&bars[i]), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");   // zeros before the copies
  __syncthreads();

  // One buffer: lane i of warp 0 holds the page id of page i of the tile at
  // pf_kt, read one tile ahead so that its latency overlaps the compute of
  // the tile before (the page table does not change during the step)
  int pf_page = -1, pf_kt = -1;
  auto page_id = [&](int kq) -> int {
    const int pi = kq / kPage;
    return kq < k_end && pi < a.max_pages ? __ldg(a.page_table + (size_t)b * a.max_pages + pi) : -1;
  };
  // Copies of the pages of the tile at kt whose first key lies in
  // [key_lo, key_hi) (multiples of the page size) into buffer buf, by lanes
  // 0..7 of warp 0 (one page each).  The bytes are added to the buffer's
  // mbarrier; `arrive` completes its single arrival (the last part of a tile).
  auto issue = [&](int kt, int buf, int key_lo, int key_hi, bool arrive) {
    if (warp != 0) return;
    const int kq = kt + lane * kPage;         // first key of this lane's page
    int page = -1;
    bool go = false;
    if constexpr (NBUF == 1) {
      if (lane < kTile / kPage && pf_kt != kt) {
        pf_page = page_id(kq);
        pf_kt = kt;
      }
    }
    if (lane < kTile / kPage && kq < k_end && kq >= key_lo && kq < key_hi) {
      const int pi = kq / kPage;
      if constexpr (NBUF == 1)
        page = pf_page;
      else
        page = pi - pg0 < n_pg ? s_pg[pi - pg0] : -1;
      go = page >= 0 && page < a.n_pages;
      if (!go) atomicOr(a.d_err, kErrBadPage);
    }
    const unsigned m = __ballot_sync(0xffffffffu, go);
    const uint32_t bar = smem_u32(&bars[buf]);
    if (lane == 0) {
      const uint32_t bytes = (uint32_t)__popc(m) * 2u * kPageBytes;
      if (arrive)
        mbar_expect_tx(bar, bytes);
      else if (bytes)
        asm volatile("mbarrier.expect_tx.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
    }
    __syncwarp();
    if (go) {
      const int row = (page * 2 * a.H + h) * kPage;   // K rows; V rows follow H pages later
      const uint32_t off = (uint32_t)(buf * kTileBytes + lane * kPageBytes);
      // each K/V byte is read once per step: evict first
      const uint64_t pol = l2_evict_first_policy();
      tma_load_2d_hint(smem_u32(Ks) + off, &map_kv, bar, 0, row, pol);
      tma_load_2d_hint(smem_u32(Vs) + off, &map_kv, bar, 0, row + a.H * kPage, pol);
    }
    if constexpr (NBUF == 1) {
      // the next tile's page ids, consumed at its issue after this tile's compute
      if (arrive && lane < kTile / kPage && kt + kTile < k_end) {
        pf_page = page_id(kt + kTile + lane * kPage);
        pf_kt = kt + kTile;
      }
    }
  };

  // the first tiles: pages wholly below the committed length now, the rest
  // after the wait
  {
    const int pre = min(NBUF, n_tiles);
    const int cut = early ? (stable / kPage) * kPage : k_begin;   // first page not yet stable
    if (early) {
      for (int i = 0; i < pre; ++i) {
        const int kt = k_begin + i * kTile;
        issue(kt, i, kt, min(cut, kt + kTile), false);
      }
      pdl_wait();
    }
    for (int i = 0; i < pre; ++i) {
      const int kt = k_begin + i * kTile;
      issue(kt, i, max(kt, cut), kt + kTile, true);
    }
  }
  const int pos0 = g < nr ? a.row_pos[row0 + g] : -1;          // rows g and g + 8
  const int pos1 = g + 8 < nr ? a.row_pos[row0 + g + 8] : -1;
  {
    // Q rows scaled by log2(e) / sqrt(hd) (scores in base-2 units for ex2)
    // as bf16; rows >= nr are zero
    const float scale = 1.4426950408889634f * rsqrtf((float)kHD);
    const int r = t >> 3, c = t & 7;
    float4 v0 = make_float4(0.f, 0.f, 0.f, 0.f), v1 = v0;
    if (r < nr) {
      const float* qp = a.q + ((size_t)(row0 + r) * a.H + h) * kHD + c * 8;
      v0 = *reinterpret_cast<const float4*>(qp);
      v1 = *reinterpret_cast<const float4*>(qp + 4);
    }
    uint4 pk;
    pk.x = pack_bf16(v0.x * scale, v0.y * scale);
    pk.y = pack_bf16(v0.z * scale, v0.w * scale);
    pk.z = pack_bf16(v1.x * scale, v1.y * scale);
    pk.w = pack_bf16(v1.z * scale, v1.w * scale);
    *reinterpret_cast<uint4*>(Qs + swz(r, c)) = pk;
  }

  float m0 = -INFINITY, m1 = -INFINITY;   // running max of rows g, g + 8 (quad-uniform)
  float l0 = 0.f, l1 = 0.f;               // this thread's share of the running sums
  float o[8][4];
#pragma unroll
  for (int nd = 0; nd < 8; ++nd) o[nd][0] = o[nd][1] = o[nd][2] = o[nd][3] = 0.f;
  const int kw = warp * 32;               // this warp's keys within a tile
  const uint32_t qbase = smem_addr(Qs);
  // keys every row of the group sees: those at or before the first row's position
  const int full_end = min(k_end, nr > 0 ? a.row_pos[row0] + 1 : 0);
  __syncthreads();                        // Q

  for (int it = 0; it < n_tiles; ++it) {
    const int kt = k_begin + it * kTile;
    const int buf = it % NBUF;
    mbar_wait(smem_u32(&bars[buf]), (uint32_t)(it / NBUF) & 1u, a.d_err);
    const uint32_t kbase = smem_addr(Ks + (size_t)buf * kTile * kHD);
    const uint32_t vbase = smem_addr(Vs + (size_t)buf * kTile * kHD);

    // S = Q K^T over this warp's 32 keys: n-tile j = keys kw + 8j .. +7
    float s[4][4];
#pragma unroll
    for (int j = 0; j < 4; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
#pragma unroll
    for (int p = 0; p < 2; ++p) {            // head dims 32p .. 32p+31 (two k-steps)
      uint32_t qa0[4], qa1[4];
      {
        const int r = (lane & 7) + 8 * ((lane >> 3) & 1);
        ldsm_x4(qbase + 2 * swz(r, 4 * p + (lane >> 4)), qa0);
        ldsm_x4(qbase + 2 * swz(r, 4 * p + 2 + (lane >> 4)), qa1);
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        uint32_t kb[4];
        ldsm_x4(kbase + 2 * swz(kw + 8 * j + (lane & 7), 4 * p + (lane >> 3)), kb);
        mma16816(s[j], qa0, kb[0], kb[1]);
        mma16816(s[j], qa1, kb[2], kb[3]);
      }
    }

    // causal mask (tiles past the first row's position only) and online
    // softmax (per warp)
    if (kt + kTile > full_end) {
      const int key0 = kt + kw + 2 * tq;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int key = key0 + 8 * j + e;
          if (!(key < k_end && key <= pos0)) s[j][e] = -INFINITY;
          if (TWO && !(key < k_end && key <= pos1)) s[j][2 + e] = -INFINITY;
        }
      }
    }
    float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      mx0 = fmaxf(mx0, fmaxf(s[j][0], s[j][1]));
      if (TWO) mx1 = fmaxf(mx1, fmaxf(s[j][2], s[j][3]));
    }
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    if (TWO) {
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
    }
    const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
    const float c0 = (mn0 == -INFINITY) ? 1.f : ex2(m0 - mn0);
    const float c1 = (!TWO || mn1 == -INFINITY) ? 1.f : ex2(m1 - mn1);
    m0 = mn0;
    m1 = mn1;
    // probabilities as bf16 pairs (the MMA A operand); the sums use the
    // rounded values so numerator and denominator match
    uint32_t pk[4][2];
    float ps0 = 0.f, ps1 = 0.f;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      pk[j][0] = (mn0 == -INFINITY) ? 0u : pack_bf16(ex2(s[j][0] - mn0), ex2(s[j][1] - mn0));
      const float2 f0 = unpack_bf16(pk[j][0]);
      ps0 += f0.x + f0.y;
      pk[j][1] = 0u;
      if (TWO) {
        pk[j][1] = (mn1 == -INFINITY) ? 0u : pack_bf16(ex2(s[j][2] - mn1), ex2(s[j][3] - mn1));
        const float2 f1 = unpack_bf16(pk[j][1]);
        ps1 += f1.x + f1.y;
      }
    }
    l0 = l0 * c0 + ps0;
    l1 = l1 * c1 + ps1;
#pragma unroll
    for (int nd = 0; nd < 8; ++nd) {
      o[nd][0] *= c0; o[nd][1] *= c0;
      if (TWO) { o[nd][2] *= c1; o[nd][3] *= c1; }
    }

    // O += P V: k-step kk = keys kw + 16kk .. +15; V fragments by ldmatrix.trans
#pragma unroll
    for (int kk = 0; kk < 2; ++kk) {
      const uint32_t pa[4] = {pk[2 * kk][0], pk[2 * kk][1], pk[2 * kk + 1][0], pk[2 * kk + 1][1]};
      const int vr = kw + 16 * kk + 8 * ((lane >> 3) & 1) + (lane & 7);
#pragma unroll
      for (int np = 0; np < 4; ++np) {       // head dims 16np .. 16np+15
        uint32_t vb[4];
        ldsm_x4_t(vbase + 2 * swz(vr, 2 * np + (lane >> 4)), vb);
        mma16816(o[2 * np], pa, vb[0], vb[1]);
        mma16816(o[2 * np + 1], pa, vb[2], vb[3]);
      }
    }
    __syncthreads();   // buffer buf is free: tile it + NBUF goes there
    if (it + NBUF < n_tiles) {
      const int kn = kt + NBUF * kTile;
      issue(kn, buf, kn, kn + kTile, true);
    }
  }

  // merge the four warps (fixed order): per warp m, l and O of the 16 rows
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  float* Ow = reinterpret_cast<float*>(Ks);              // [4][16][64], K/V buffers are free
  float2* ML = reinterpret_cast<float2*>(Ow + 4 * kQRows * kHD);   // [4][16]
#pragma unroll
  for (int nd = 0; nd < 8; ++nd) {
    *reinterpret_cast<float2*>(Ow + ((size_t)warp * kQRows + g) * kHD + 8 * nd + 2 * tq) =
        make_float2(o[nd][0], o[nd][1]);
    *reinterpret_cast<float2*>(Ow + ((size_t)warp * kQRows + g + 8) * kHD + 8 * nd + 2 * tq) =
        make_float2(o[nd][2], o[nd][3]);
  }
  if (tq == 0) {
    ML[warp * kQRows + g] = make_float2(m0, l0);
    ML[warp * kQRows + g + 8] = make_float2(m1, l1);
  }
  __syncthreads();
  {
    const int r = t >> 3, d0 = (t & 7) * 8;    // 16 rows x 64 dims, 8 per thread
    if (r < nr) {
      float M = -INFINITY;
#pragma unroll
      for (int w = 0; w < 4; ++w) M = fmaxf(M, ML[w * kQRows + r].x);
      float wt[4], L = 0.f;
#pragma unroll
      for (int w = 0; w < 4; ++w) {
        const float2 ml = ML[w * kQRows + r];
        wt[w] = (ml.x == -INFINITY) ? 0.f : ex2(ml.x - M);
        L += ml.y * wt[w];
      }
      float acc[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) acc[q] = 0.f;
#pragma unroll
      for (int w = 0; w < 4; ++w) {
        const float4* src = reinterpret_cast<const float4*>(Ow + ((size_t)w * kQRows + r) * kHD + d0);
        const float4 u0 = src[0], u1 = src[1];
        acc[0] += u0.x * wt[w]; acc[1] += u0.y * wt[w]; acc[2] += u0.z * wt[w]; acc[3] += u0.w * wt[w];
        acc[4] += u1.x * wt[w]; acc[5] += u1.y * wt[w]; acc[6] += u1.z * wt[w]; acc[7] += u1.w * wt[w];
      }
      const int row = row0 + r;
      if (a.cluster_merge) {
        // this split's partial (base-2 units) for the cluster merge below;
        // past the 4-warp merge's buffers (Ow and ML end 16.5 KB in)
        float* Ps = reinterpret_cast<float*>(sm + 17408);          // [16][64]
        float2* MLs = reinterpret_cast<float2*>(Ps + kQRows * kHD);  // [16]
        *reinterpret_cast<float4*>(Ps + r * kHD + d0) = make_float4(acc[0], acc[1], acc[2], acc[3]);
        *reinterpret_cast<float4*>(Ps + r * kHD + d0 + 4) = make_float4(acc[4], acc[5], acc[6], acc[7]);
        if (d0 == 0) MLs[r] = make_float2(M, L);
      } else if (a.n_split == 1) {
        const float inv = 1.f / L;
        uint4 pk;
        pk.x = pack_bf16(acc[0] * inv, acc[1] * inv);
        pk.y = pack_bf16(acc[2] * inv, acc[3] * inv);
        pk.z = pack_bf16(acc[4] * inv, acc[5] * inv);
        pk.w = pack_bf16(acc[6] * inv, acc[7] * inv);
        *reinterpret_cast<uint4*>(reinterpret_cast<__nv_bfloat16*>(a.out) + (size_t)row * a.H * kHD +
                                  h * kHD + d0) = pk;
      } else {
        float* po = a.part_o + (((size_t)split * a.R + row) * a.H + h) * kHD + d0;
#pragma unroll
        for (int q = 0; q < 8; q += 4)
          *reinterpret_cast<float4*>(po + q) = make_float4(acc[q], acc[q + 1], acc[q + 2], acc[q + 3]);
        // the combine works in natural-log units
        if (d0 == 0) a.part_ml[((size_t)split * a.R + row) * a.H + h] = make_float2(M * 0.6931471805599453f, L);
      }
    }
  }
  if (a.cluster_merge) {
    // The key splits of this (group, head) are one cluster (rank = split):
    // after the barrier CTA q merges rows q, q + n_split, ... reading every
    // split's partial from its shared memory in split order; the second
    // barrier keeps each CTA's partial alive until all have read it.
    cluster_sync();
    const int r = t >> 3, d0 = (t & 7) * 8;
    if (r < nr && r % a.n_split == split) {
      const float* Ps = reinterpret_cast<const float*>(sm + 17408);
      const float2* MLs = reinterpret_cast<const float2*>(Ps + kQRows * kHD);
      float M = -INFINITY, L = 0.f, acc[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) acc[q] = 0.f;
      for (int sp = 0; sp < a.n_split; ++sp) {
        const float2 ml = ld_dsmem2(smem_u32(MLs + r), (uint32_t)sp);
        if (ml.x == -INFINITY) continue;            // no visible key in this split
        const float4 u0 = ld_dsmem4(smem_u32(Ps + r * kHD + d0), (uint32_t)sp);
        const float4 u1 = ld_dsmem4(smem_u32(Ps + r * kHD + d0 + 4), (uint32_t)sp);
        const float Mn = fmaxf(M, ml.x);
        const float cs = (M == -INFINITY) ? 0.f : ex2(M - Mn);
        const float w = ex2(ml.x - Mn);
        M = Mn;
        L = L * cs + ml.y * w;
        acc[0] = acc[0] * cs + u0.x * w; acc[1] = acc[1] * cs + u0.y * w;
        acc[2] = acc[2] * cs + u0.z * w; acc[3] = acc[3] * cs + u0.w * w;
        acc[4] = acc[4] * cs + u1.x * w; acc[5] = acc[5] * cs + u1.y * w;
        acc[6] = acc[6] * cs + u1.z * w; acc[7] = acc[7] * cs + u1.w * w;
      }
      const float inv = 1.f / L;
      uint4 pk;
      pk.x = pack_bf16(acc[0] * inv, acc[1] * inv);
      pk.y = pack_bf16(acc[2] * inv, acc[3] * inv);
      pk.z = pack_bf16(acc[4] * inv, acc[5] * inv);
      pk.w = pack_bf16(acc[6] * inv, acc[7] * inv);
      *reinterpret_cast<uint4*>(reinterpret_cast<__nv_bfloat16*>(a.out) + (size_t)(row0 + r) * a.H * kHD +
                                h * kHD + d0) = pk;
    }
    cluster_sync();
    return;
  }
  if constexpr (NBUF > 1) {
    // the last split CTA of this (group, head) to finish merges the
    // partials in split order (the same result whichever CTA it is) and
    // re-arms the counter for the next launch
    if (a.split_count == nullptr) return;
    int* s_last = s_pg - 2;
    __threadfence();
    __syncthreads();
    int* cnt = a.split_count + (size_t)gi * a.H + h;
    if (t == 0) *s_last = atomicAdd(cnt, 1) == a.n_split - 1;
    __syncthreads();
    if (*s_last) {
      __threadfence();
      merge_splits(a.part_o, a.part_ml, reinterpret_cast<__nv_bfloat16*>(a.out), a.n_split, a.R, a.H, row0,
                   nr, h, t);
      if (t == 0) *cnt = 0;
    }
  }
}

template <int NBUF, bool TWO>
static int launch_nb(const CUtensorMap& map, const AttnArgs& a, int n_groups, cudaStream_t s) {
  static PerDevice attr;
  const size_t smem = smem_bytes(NBUF, a.pg_cap);
  set_smem_attr(attr, k_attention_mma<NBUF, TWO>, smem);
  if (!a.cluster_merge) {
    kf_launch(k_attention_mma<NBUF, TWO>, dim3(n_groups, a.H, a.n_split), dim3(kThr), smem, s, map, a);
    return 0;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(n_groups, a.H, a.n_split);
  cfg.blockDim = dim3(kThr);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[2];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = 1;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = a.n_split;
  at[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = g_pdl ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, k_attention_mma<NBUF, TWO>, map, a) == cudaSuccess ? 0 : -1;
}

bool attention_mma_supported(bool bf16, int hd, int rows) { return bf16 && hd == kHD && rows <= kQRows; }

int launch_attention_mma(const AttnArgs& a0, int n_groups, int rows, int max_keys, cudaStream_t s,
                         bool* merged) {
  *merged = false;
  if (n_groups == 0) return 0;
  AttnArgs a = a0;
  const int keys = std::min(a.keys_per_split, max_keys);   // the most keys of one CTA
  const int num_sms = device_sms();
  const bool two = rows > 8;
  const long ctas = (long)n_groups * a.H * a.n_split;
  // two buffers (3 CTAs per SM) only while the CTAs fit in one wave of
  // them; otherwise one buffer (6 per SM, 5 with 16-row groups; a CTA of
  // several tiles refills it after each), twice the CTAs in flight.
  // Measured on OWT-shaped decode at k = 4: batch 128 401k -> 423k, batch
  // 256 481k -> 493k tokens/s; batch 32 (384 CTAs) 239k with two buffers,
  // 209k with one
  const bool one = keys <= kTile || ctas > 3L * num_sms;
  // the key splits of each (group, head) run as one cluster (at most 4
  // CTAs) and merge in the kernel
  a.split_count = nullptr;
  a.cluster_merge = a.n_split > 1 && a.n_split <= 8 ? 1 : 0;
  if (a.n_split > 8) return -1;
  *merged = a.cluster_merge != 0;
  a.pg_cap = one ? 0 : ceil_div(keys, kPage);   // staged page ids (two-buffer CTAs)
  // this layer's K/V pages as rows of 64 bf16: ((page * 2 + kv) * H + head) * 16 + key
  const size_t layer_elems = (size_t)a.n_pages * 2 * a.H * kPage * kHD;
  CUtensorMap map;
  if (!encode_rows_map_bf16(&map, static_cast<const __nv_bfloat16*>(a.kv) + (size_t)a.layer * layer_elems,
                            (uint64_t)a.n_pages * 2 * a.H * kPage, kHD, kPage))
    return -1;
  if (one) return two ? launch_nb<1, true>(map, a, n_groups, s) : launch_nb<1, false>(map, a, n_groups, s);
  return two ? launch_nb<2, true>(map, a, n_groups, s) : launch_nb<2, false>(map, a, n_groups, s);
}

}  // namespace kf
