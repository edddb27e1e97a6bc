// Decode attention on warp-level tensor-core MMA (mma.sync m16n8k16, bf16
// operands, fp32 accumulation) for the bf16 cache with head_dim 64: up to 16
// query rows of one sequence and one head per CTA against every cached key
// at or before each row's position (the fully causal mask of Sec. 3.3 /
// Alg. 1).
//
// Per CTA (4 warps), keys in tiles of 128 streamed into shared memory with
// 16-byte cp.async (double-buffered when the CTA sees more than one tile);
// rows are XOR-swizzled in 16-byte chunks so ldmatrix reads are
// conflict-free without padding.  Warp w owns keys 32w .. 32w+31 of every
// tile and keeps its own online softmax over them (FlashAttention-2 style):
//   S = Q K^T      16 rows x 32 keys, 16 MMAs (Q zero-padded to 16 rows)
//   P = exp(S - m) in registers; the S accumulator layout is the A-operand
//                  layout of the next MMA, so P never leaves the registers
//   O += P V       16 rows x 64 dims, 16 MMAs (V through ldmatrix.trans)
// The four warps' (m, l, O) are merged once at the end in a fixed order
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

#include "kf_internal.cuh"
#include "kf_mma.cuh"

namespace kf {
namespace {

using namespace mma;

constexpr int kTile = 128;     // keys per K/V tile
constexpr int kThr = 128;      // 4 warps x 32 keys of each tile
constexpr int kQRows = 16;     // MMA M: query rows of the group, zero-padded

constexpr size_t smem_bytes(int nbuf) {
  return (size_t)kQRows * kHD * 2 + (size_t)nbuf * 2 * kTile * kHD * 2;
}

}  // namespace

// NBUF = 1: CTAs of at most one key tile; NBUF = 2: double-buffered tiles.
// Single-tile decode CTAs (a.len set, one group per sequence): the keys before the
// sequence's committed length were written by earlier steps and the page
// table by the host before the step, so the copies of those keys are issued
// before waiting for the kernel that appends this step's keys; the new keys
// and Q are loaded after the wait.
template <int NBUF>
__global__ void __launch_bounds__(kThr, NBUF == 1 ? 6 : 3) k_attention_mma(AttnArgs a) {
  pdl_trigger();
  extern __shared__ __align__(128) uint8_t sm[];
  __nv_bfloat16* Qs = reinterpret_cast<__nv_bfloat16*>(sm);   // [16][64] swizzled
  __nv_bfloat16* Ks = Qs + kQRows * kHD;                      // [NBUF][128][64] swizzled
  __nv_bfloat16* Vs = Ks + NBUF * kTile * kHD;                // [NBUF][128][64] swizzled

  const int gi = blockIdx.x, h = blockIdx.y, split = blockIdx.z;
  // (single-tile CTAs only: with several tiles the double buffer hides the
  // first tile's latency already)
  const bool early = NBUF == 1 && a.len != nullptr && a.groups == nullptr;
  int b, row0, nr, n_keys, stable;
  if (early) {
    b = gi; row0 = gi * a.uniform_rows; nr = a.uniform_rows;
    stable = a.len[b];                       // committed length: positions row_pos of the step
    n_keys = stable + nr;
  } else {
    pdl_wait();
    if (a.groups) {
      const int4 gg = a.groups[gi];
      b = gg.x; row0 = gg.y; nr = gg.z;
    } else {
      b = gi; row0 = gi * a.uniform_rows; nr = a.uniform_rows;
    }
    n_keys = a.row_pos[row0 + nr - 1] + 1;
    stable = 0;
  }
  const int k_begin = split * a.keys_per_split;
  const int k_end = min(n_keys, k_begin + a.keys_per_split);
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const int g = lane >> 2, tq = lane & 3;     // MMA fragment row group / column pair

  const __nv_bfloat16* kv = reinterpret_cast<const __nv_bfloat16*>(a.kv);
  const size_t head_page = (size_t)kPage * kHD;
  const size_t layer_base = (size_t)a.layer * a.n_pages * 2 * a.H * head_page;
  bool bad_page = false;

  // cp.async of the keys [key_lo, key_hi) of the tile starting at kt into
  // buffer buf (keys >= k_end are zero-filled).  kt is a multiple of the page
  // size: thread t copies chunk t % 8 of keys kt + t / 8 + 16 q, i.e. one key
  // of page kt / 16 + q for q = 0..7; the page ids are all fetched before the
  // first copy is issued.
  auto load_tile = [&](int kt, int buf, int key_lo, int key_hi) {
    __nv_bfloat16* kd = Ks + (size_t)buf * kTile * kHD;
    __nv_bfloat16* vd = Vs + (size_t)buf * kTile * kHD;
    constexpr int NQ = kTile * 8 / kThr;
    static_assert(kThr / 8 == kPage, "one page per copy round");
    int pg[NQ];
#pragma unroll
    for (int q = 0; q < NQ; ++q) {
      const int pi = kt / kPage + q;
      const int kq = kt + q * kPage;        // first key of the page
      pg[q] = (kq < k_end && kq + kPage > key_lo && kq < key_hi && pi < a.max_pages)
                  ? __ldg(a.page_table + b * a.max_pages + pi) : -1;
    }
#pragma unroll
    for (int q = 0; q < NQ; ++q) {
      const int idx = t + q * kThr;
      const int j = idx >> 3, c = idx & 7;
      const int key = kt + j;
      if (key < key_lo || key >= key_hi) continue;
      const __nv_bfloat16* src = kv;
      int nbytes = 0;
      if (key < k_end) {
        const int page = pg[q];
        if (page >= 0 && page < a.n_pages) {
          src = kv + layer_base + (((size_t)page * 2) * a.H + h) * head_page + (size_t)(key % kPage) * kHD + c * 8;
          nbytes = 16;
        } else {
          bad_page = true;
        }
      }
      cp_async16(smem_addr(kd + swz(j, c)), src, nbytes);
      cp_async16(smem_addr(vd + swz(j, c)), src + (nbytes ? a.H * head_page : 0), nbytes);
    }
    cp_commit();
  };

  int n_tiles = k_end > k_begin ? ceil_div(k_end - k_begin, kTile) : 0;
  if (NBUF == 1 && n_tiles > 1) {
    // the single-buffer variant is launched only for CTAs of at most one tile
    if (t == 0) atomicOr(a.d_err, kErrInternal);
    n_tiles = 1;
  }
  if (n_tiles > 0) {
    // first tile: its stable keys now, the rest after the wait
    const int split_key = early ? max(k_begin, min(stable, k_begin + kTile)) : k_begin;
    if (split_key > k_begin) load_tile(k_begin, 0, k_begin, split_key);
    if (early) pdl_wait();
    load_tile(k_begin, 0, split_key, k_begin + kTile);
  } else if (early) {
    pdl_wait();
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
  const bool two = nr > 8;                // rows 8..15 exist (else zero padding)
  const uint32_t qbase = smem_addr(Qs);

  for (int it = 0; it < n_tiles; ++it) {
    const int kt = k_begin + it * kTile;
    const int buf = (NBUF == 2) ? (it & 1) : 0;
    if (NBUF == 2 && it + 1 < n_tiles) {
      load_tile(kt + kTile, buf ^ 1, kt + kTile, kt + 2 * kTile);
      cp_wait<1>();
    } else {
      cp_wait<0>();
    }
    __syncthreads();
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

    // causal mask and online softmax (per warp)
    const int key0 = kt + kw + 2 * tq;
    float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int key = key0 + 8 * j + e;
        if (!(key < k_end && key <= pos0)) s[j][e] = -INFINITY;
        if (!(key < k_end && key <= pos1)) s[j][2 + e] = -INFINITY;
        mx0 = fmaxf(mx0, s[j][e]);
        mx1 = fmaxf(mx1, s[j][2 + e]);
      }
    }
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    if (two) {
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
    }
    const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
    const float c0 = (mn0 == -INFINITY) ? 1.f : ex2(m0 - mn0);
    const float c1 = (mn1 == -INFINITY) ? 1.f : ex2(m1 - mn1);
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
      if (two) {
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
      o[nd][2] *= c1; o[nd][3] *= c1;
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
    __syncthreads();   // the buffer is refilled next iteration
  }
  if (bad_page) atomicOr(a.d_err, kErrBadPage);

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
      if (a.n_split == 1) {
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
}

template <int NBUF>
static void launch_nb(const AttnArgs& a, int n_groups, cudaStream_t s) {
  const size_t smem = smem_bytes(NBUF);
  static bool attr = false;
  if (!attr) {
    cudaFuncSetAttribute(k_attention_mma<NBUF>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    attr = true;
  }
  kf_launch(k_attention_mma<NBUF>, dim3(n_groups, a.H, a.n_split), dim3(kThr), smem, s, a);
}

bool attention_mma_supported(bool bf16, int hd, int rows) { return bf16 && hd == kHD && rows <= kQRows; }

void launch_attention_mma(const AttnArgs& a, int n_groups, int max_keys, cudaStream_t s) {
  if (n_groups == 0) return;
  // one K/V buffer when no CTA sees more than one tile of keys
  if (std::min(a.keys_per_split, max_keys) <= kTile) launch_nb<1>(a, n_groups, s);
  else launch_nb<2>(a, n_groups, s);
}

}  // namespace kf
