// Decode attention over the paged KV cache: up to 16 query rows of one
// sequence and one head per CTA against every cached key at or before each
// row's position (the fully causal mask of Sec. 3.3 / Alg. 1: pending rows
// and noise slots see the cache, earlier pending rows and earlier slots).
//
// Per CTA (128 threads), keys in tiles of 128 (8 pages):
//   - K and V tiles stream into shared memory with 16-byte cp.async,
//     double-buffered so the next tile loads while this one is computed;
//   - scores: thread t owns key t and all R query rows (register-blocked);
//   - online softmax per row (fp32), probabilities written transposed
//     (P[key][row]) so the PV product broadcasts them;
//   - PV: warp w accumulates keys 32w..32w+31 of every tile for all R rows,
//     lanes along the head dims; the four warp partials are summed once at
//     the end in a fixed order.
// With n_split > 1 each CTA covers one key range and k_attn_combine merges
// the partial softmaxes in split order.
#include <algorithm>
#include <cstring>

#include "kf_internal.cuh"

namespace kf {

constexpr int kKeyTile = 128;
constexpr int kAttnThreads = 128;

template <typename TA> struct KvPad;
template <> struct KvPad<float> { static constexpr int V = 4; };
template <> struct KvPad<__nv_bfloat16> { static constexpr int V = 8; };

__device__ __forceinline__ void load8(const float* p, float* o) {
  float4 a = *reinterpret_cast<const float4*>(p);
  float4 b = *reinterpret_cast<const float4*>(p + 4);
  o[0] = a.x; o[1] = a.y; o[2] = a.z; o[3] = a.w; o[4] = b.x; o[5] = b.y; o[6] = b.z; o[7] = b.w;
}
__device__ __forceinline__ void load8(const __nv_bfloat16* p, float* o) {
  uint4 v = *reinterpret_cast<const uint4*>(p);
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float2 f = __bfloat1622float2(h[i]);
    o[2 * i] = f.x;
    o[2 * i + 1] = f.y;
  }
}
// DPL consecutive values at p (DPL = 1 or 2)
template <int DPL>
__device__ __forceinline__ void loadd(const float* p, float* o) {
  if (DPL == 2) { float2 f = *reinterpret_cast<const float2*>(p); o[0] = f.x; o[1] = f.y; }
  else o[0] = p[0];
}
template <int DPL>
__device__ __forceinline__ void loadd(const __nv_bfloat16* p, float* o) {
  if (DPL == 2) {
    float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(p));
    o[0] = f.x; o[1] = f.y;
  } else {
    o[0] = __bfloat162float(p[0]);
  }
}

// packed fp32 FMA (two lanes per instruction; each lane rounds like fmaf)
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) {
  unsigned long long A, B, C, D;
  memcpy(&A, &a, 8); memcpy(&B, &b, 8); memcpy(&C, &c, 8);
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(D) : "l"(A), "l"(B), "l"(C));
  float2 d;
  memcpy(&d, &D, 8);
  return d;
}
__device__ __forceinline__ void load8p(const float* p, float2* o) {
  float4 a = *reinterpret_cast<const float4*>(p);
  float4 b = *reinterpret_cast<const float4*>(p + 4);
  o[0] = make_float2(a.x, a.y); o[1] = make_float2(a.z, a.w);
  o[2] = make_float2(b.x, b.y); o[3] = make_float2(b.z, b.w);
}
__device__ __forceinline__ void load8p(const __nv_bfloat16* p, float2* o) {
  uint4 v = *reinterpret_cast<const uint4*>(p);
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
  for (int i = 0; i < 4; ++i) o[i] = __bfloat1622float2(h[i]);
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, int src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
               "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

template <typename TA, int HD>
struct AttnSmem {
  static constexpr int KP = HD + KvPad<TA>::V;      // padded K row (conflict-free 16B reads)
  static constexpr size_t k_tile = (size_t)kKeyTile * KP * sizeof(TA);
  static constexpr size_t v_tile = (size_t)kKeyTile * HD * sizeof(TA);
  static size_t bytes(int R, int nbuf) {
    size_t b = 0;
    b += (size_t)R * HD * 4;              // Q
    b += nbuf * (k_tile + v_tile);        // K, V (double-buffered when a CTA has > 1 tile)
    b += (size_t)kKeyTile * R * 4;        // P^T
    b += 2 * 4 * (size_t)R * 4;           // warp max / sum
    return b;
  }
};

template <typename TA, int HD, int R, int NBUF>
__global__ void __launch_bounds__(kAttnThreads) k_attention(AttnArgs a) {
  pdl_wait();
  using S = AttnSmem<TA, HD>;
  constexpr int KP = S::KP;
  constexpr int DPL = HD / 32;          // head dims per lane in the PV product
  constexpr int CPR = HD * (int)sizeof(TA) / 16;   // 16-byte chunks per key row
  extern __shared__ __align__(16) uint8_t sm[];
  float* Qs = reinterpret_cast<float*>(sm);
  TA* Kt = reinterpret_cast<TA*>(sm + (size_t)R * HD * 4);
  TA* Vt = reinterpret_cast<TA*>(reinterpret_cast<uint8_t*>(Kt) + NBUF * S::k_tile);
  float* Ps = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(Vt) + NBUF * S::v_tile);
  float* red_m = Ps + kKeyTile * R;
  float* red_s = red_m + 4 * R;

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
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;

  int pos[R];
#pragma unroll
  for (int r = 0; r < R; ++r) pos[r] = (r < nr) ? a.row_pos[row0 + r] : -1;

  const TA* kv = reinterpret_cast<const TA*>(a.kv);
  const size_t head_page = (size_t)kPage * HD;
  const size_t layer_base = (size_t)a.layer * a.n_pages * 2 * a.H * head_page;
  bool bad_page = false;

  // issue the cp.async loads of the tile starting at key kt into buffer buf
  auto load_tile = [&](int kt, int buf) {
    TA* kd = Kt + (size_t)buf * kKeyTile * KP;
    TA* vd = Vt + (size_t)buf * kKeyTile * HD;
    for (int idx = t; idx < kKeyTile * CPR; idx += kAttnThreads) {
      const int j = idx / CPR, c = idx - j * CPR;
      const int key = kt + j;
      const TA* src = kv;
      int nbytes = 0;
      if (key < k_end) {
        const int pi = key / kPage;
        const int page = pi < a.max_pages ? a.page_table[b * a.max_pages + pi] : -1;
        if (page >= 0 && page < a.n_pages) {
          src = kv + layer_base + (((size_t)page * 2) * a.H + h) * head_page +
                (size_t)(key % kPage) * HD + c * (16 / sizeof(TA));
          nbytes = 16;
        } else {
          bad_page = true;
        }
      }
      cp_async16(static_cast<uint32_t>(__cvta_generic_to_shared(kd + (size_t)j * KP + c * (16 / sizeof(TA)))),
                 src, nbytes);
      cp_async16(static_cast<uint32_t>(__cvta_generic_to_shared(vd + (size_t)j * HD + c * (16 / sizeof(TA)))),
                 src + (nbytes ? a.H * head_page : 0), nbytes);
    }
    cp_commit();
  };

  // running max / sum per row; the PV accumulators hold row pairs (r, r+1)
  // of head dims lane*DPL + q, so a packed FMA updates both rows at once
  constexpr int RP = (R + 1) / 2;
  float m_run[R], l_run[R];
  float2 acc2[RP][DPL];
#pragma unroll
  for (int r = 0; r < R; ++r) {
    m_run[r] = -INFINITY;
    l_run[r] = 0.f;
  }
#pragma unroll
  for (int rp = 0; rp < RP; ++rp)
#pragma unroll
    for (int q = 0; q < DPL; ++q) acc2[rp][q] = make_float2(0.f, 0.f);

  const int n_tiles = k_end > k_begin ? ceil_div(k_end - k_begin, kKeyTile) : 0;
  if (n_tiles > 0) load_tile(k_begin, 0);   // first K/V tile in flight while Q loads
  const float scale = rsqrtf((float)HD);
  for (int i = t * 4; i < R * HD; i += kAttnThreads * 4) {
    const int r = i / HD, dd = i % HD;
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    if (r < nr) v = *reinterpret_cast<const float4*>(a.q + ((size_t)(row0 + r) * a.H + h) * HD + dd);
    *reinterpret_cast<float4*>(Qs + i) = make_float4(v.x * scale, v.y * scale, v.z * scale, v.w * scale);
  }
  __syncthreads();   // Q visible

  for (int it = 0; it < n_tiles; ++it) {
    const int kt = k_begin + it * kKeyTile;
    const int buf = (NBUF == 2) ? (it & 1) : 0;
    if (NBUF == 2 && it + 1 < n_tiles) {
      load_tile(kt + kKeyTile, buf ^ 1);
      cp_wait<1>();
    } else {
      if (NBUF == 1 && it > 0) load_tile(kt, 0);
      cp_wait<0>();
    }
    __syncthreads();
    const TA* kb = Kt + (size_t)buf * kKeyTile * KP;
    const TA* vb = Vt + (size_t)buf * kKeyTile * HD;

    // scores: thread t <-> key kt + t, all R rows; packed FMAs accumulate
    // the even and odd head dims separately, summed at the end
    float2 s2[R];
#pragma unroll
    for (int r = 0; r < R; ++r) s2[r] = make_float2(0.f, 0.f);
#pragma unroll 2
    for (int d0 = 0; d0 < HD; d0 += 8) {
      float2 k2[4];
      load8p(kb + (size_t)t * KP + d0, k2);
#pragma unroll
      for (int r = 0; r < R; ++r) {
        float2 q2[4];
        load8p(Qs + r * HD + d0, q2);
#pragma unroll
        for (int i = 0; i < 4; ++i) s2[r] = ffma2(q2[i], k2[i], s2[r]);
      }
    }
    float s[R];
#pragma unroll
    for (int r = 0; r < R; ++r) s[r] = s2[r].x + s2[r].y;
    const int key = kt + t;
#pragma unroll
    for (int r = 0; r < R; ++r)
      if (!(key < k_end && key <= pos[r])) s[r] = -INFINITY;

    // tile max per row
#pragma unroll
    for (int r = 0; r < R; ++r) {
      float m = s[r];
      for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
      if (lane == 0) red_m[warp * R + r] = m;
    }
    __syncthreads();
    float corr[R];
#pragma unroll
    for (int r = 0; r < R; ++r) {
      float tm = fmaxf(fmaxf(red_m[r], red_m[R + r]), fmaxf(red_m[2 * R + r], red_m[3 * R + r]));
      float mn = fmaxf(m_run[r], tm);
      float p = (mn == -INFINITY) ? 0.f : expf(s[r] - mn);
      corr[r] = (mn == -INFINITY) ? 1.f : expf(m_run[r] - mn);
      m_run[r] = mn;
      s[r] = p;
    }
    // P^T[key][row]
    if (R % 4 == 0) {
#pragma unroll
      for (int r = 0; r < R; r += 4)
        *reinterpret_cast<float4*>(Ps + t * R + r) = make_float4(s[r], s[r + 1], s[r + 2], s[r + 3]);
    } else {
#pragma unroll
      for (int r = 0; r < R; ++r) Ps[t * R + r] = s[r];
    }
#pragma unroll
    for (int r = 0; r < R; ++r) {
      float sum = s[r];
      for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
      if (lane == 0) red_s[warp * R + r] = sum;
    }
    __syncthreads();
#pragma unroll
    for (int r = 0; r < R; ++r) {
      float ts = (red_s[r] + red_s[R + r]) + (red_s[2 * R + r] + red_s[3 * R + r]);
      l_run[r] = l_run[r] * corr[r] + ts;
    }
#pragma unroll
    for (int rp = 0; rp < RP; ++rp) {
      const float c0 = corr[2 * rp], c1 = (2 * rp + 1 < R) ? corr[2 * rp + 1] : 1.f;
#pragma unroll
      for (int q = 0; q < DPL; ++q) {
        acc2[rp][q].x *= c0;
        acc2[rp][q].y *= c1;
      }
    }
    // PV over this warp's 32 keys of the tile; packed FMAs over row pairs
#pragma unroll 4
    for (int jj = 0; jj < 32; ++jj) {
      const int j = warp * 32 + jj;
      float v[DPL];
      loadd<DPL>(vb + (size_t)j * HD + lane * DPL, v);
      const float* pj = Ps + j * R;
      if (R == 1) {
#pragma unroll
        for (int q = 0; q < DPL; ++q) acc2[0][q].x = fmaf(pj[0], v[q], acc2[0][q].x);
      } else {
#pragma unroll
        for (int rp = 0; rp < RP; ++rp) {
          const float2 p2 = *reinterpret_cast<const float2*>(pj + 2 * rp);
#pragma unroll
          for (int q = 0; q < DPL; ++q) acc2[rp][q] = ffma2(p2, make_float2(v[q], v[q]), acc2[rp][q]);
        }
      }
    }
    __syncthreads();   // buffers are refilled next iteration
  }
  if (bad_page) atomicOr(a.d_err, kErrBadPage);

  // sum the four warps' partial outputs (fixed order), then normalise
  float* Ored = reinterpret_cast<float*>(Kt);      // [4][R][HD], K/V buffers are free
#pragma unroll
  for (int rp = 0; rp < RP; ++rp)
#pragma unroll
    for (int q = 0; q < DPL; ++q) {
      Ored[((size_t)warp * R + 2 * rp) * HD + lane * DPL + q] = acc2[rp][q].x;
      if (2 * rp + 1 < R) Ored[((size_t)warp * R + 2 * rp + 1) * HD + lane * DPL + q] = acc2[rp][q].y;
    }
  __syncthreads();
  for (int i = t; i < R * HD; i += kAttnThreads) {
    const int r = i / HD, dd = i - r * HD;
    if (r >= nr) continue;
    float o = (Ored[i] + Ored[R * HD + i]) + (Ored[2 * R * HD + i] + Ored[3 * R * HD + i]);
    float l = 0.f, m = -INFINITY;
#pragma unroll
    for (int rr = 0; rr < R; ++rr)
      if (rr == r) { l = l_run[rr]; m = m_run[rr]; }
    const int row = row0 + r;
    if (a.n_split == 1) {
      TA* out = reinterpret_cast<TA*>(a.out) + (size_t)row * a.H * HD + h * HD + dd;
      *out = from_f<TA>(o / l);
    } else {
      a.part_o[(((size_t)split * a.R + row) * a.H + h) * HD + dd] = o;
      if (dd == 0) a.part_ml[((size_t)split * a.R + row) * a.H + h] = make_float2(m, l);
    }
  }
}

// merge the split partial softmaxes of one (row, head), splits in order
template <typename TA>
__global__ void k_attn_combine(AttnArgs a) {
  pdl_wait();
  const int row = blockIdx.x, h = blockIdx.y, dd = threadIdx.x;
  float M = -INFINITY;
  for (int s = 0; s < a.n_split; ++s) M = fmaxf(M, a.part_ml[((size_t)s * a.R + row) * a.H + h].x);
  float L = 0.f, O = 0.f;
  for (int s = 0; s < a.n_split; ++s) {
    float2 ml = a.part_ml[((size_t)s * a.R + row) * a.H + h];
    float w = (ml.x == -INFINITY) ? 0.f : expf(ml.x - M);
    L += ml.y * w;
    O += a.part_o[(((size_t)s * a.R + row) * a.H + h) * a.hd + dd] * w;
  }
  TA* o = reinterpret_cast<TA*>(a.out) + (size_t)row * a.H * a.hd + h * a.hd + dd;
  *o = from_f<TA>(O / L);
}

template <typename TA, int HD, int R, int NBUF>
static void launch_rb(const AttnArgs& a, int n_groups, cudaStream_t s) {
  const size_t smem = AttnSmem<TA, HD>::bytes(R, NBUF);
  static PerDevice attr;
  set_smem_attr(attr, k_attention<TA, HD, R, NBUF>, smem);
  dim3 grid(n_groups, a.H, a.n_split);
  kf_launch(k_attention<TA, HD, R, NBUF>, grid, dim3(kAttnThreads), smem, s, a);
}

template <typename TA, int HD, int R>
static void launch_r(const AttnArgs& a, int n_groups, int max_keys, cudaStream_t s) {
  // one K/V buffer when no CTA sees more than one tile of keys
  if (std::min(a.keys_per_split, max_keys) <= kKeyTile) launch_rb<TA, HD, R, 1>(a, n_groups, s);
  else launch_rb<TA, HD, R, 2>(a, n_groups, s);
}

template <typename TA, int HD>
static void launch_hd(const AttnArgs& a, int n_groups, int rows, int max_keys, cudaStream_t s) {
  if (rows <= 1) launch_r<TA, HD, 1>(a, n_groups, max_keys, s);
  else if (rows <= 2) launch_r<TA, HD, 2>(a, n_groups, max_keys, s);
  else if (rows <= 4) launch_r<TA, HD, 4>(a, n_groups, max_keys, s);
  else if (rows <= 8) launch_r<TA, HD, 8>(a, n_groups, max_keys, s);
  else launch_r<TA, HD, 16>(a, n_groups, max_keys, s);
}

void launch_attention(bool bf16, const AttnArgs& a, int n_groups, int max_keys, cudaStream_t s) {
  if (n_groups == 0) return;
  // rows per group: uniform in decode, at most 16 in prefill groups
  const int rows = a.groups ? kMaxGroupRows : a.uniform_rows;
  if (a.hd == 64) {
    if (bf16) launch_hd<__nv_bfloat16, 64>(a, n_groups, rows, max_keys, s);
    else launch_hd<float, 64>(a, n_groups, rows, max_keys, s);
  } else {
    if (bf16) launch_hd<__nv_bfloat16, 32>(a, n_groups, rows, max_keys, s);
    else launch_hd<float, 32>(a, n_groups, rows, max_keys, s);
  }
}

void launch_attn_combine(bool bf16, const AttnArgs& a, cudaStream_t s) {
  if (a.R == 0 || a.n_split <= 1) return;
  dim3 grid(a.R, a.H);
  if (bf16) kf_launch(k_attn_combine<__nv_bfloat16>, dim3(grid), dim3(a.hd), 0, s, a);
  else kf_launch(k_attn_combine<float>, dim3(grid), dim3(a.hd), 0, s, a);
}

}  // namespace kf
