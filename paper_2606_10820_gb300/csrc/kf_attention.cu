// Decode attention over the paged KV cache: up to 16 query rows of one
// sequence and one head per CTA against every cached key at or before each
// row's position (the fully causal mask of Sec. 3.3 / Alg. 1: pending rows
// and noise slots see the cache, earlier pending rows and earlier slots).
// fp32 scores and online softmax; keys staged through shared memory with
// 16-byte loads, 64 keys (4 pages) per tile.  With n_split > 1 each CTA
// covers one key range and a combine kernel merges the partial softmaxes
// in split order.
#include "kf_internal.cuh"

namespace kf {

template <typename T> struct Vec;
template <> struct Vec<float> { static constexpr int N = 4; using V = float4; };
template <> struct Vec<__nv_bfloat16> { static constexpr int N = 8; using V = uint4; };

__device__ __forceinline__ void unpack(const float4& v, float* o) {
  o[0] = v.x; o[1] = v.y; o[2] = v.z; o[3] = v.w;
}
__device__ __forceinline__ void unpack(const uint4& v, float* o) {
  const __nv_bfloat162* p = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float2 f = __bfloat1622float2(p[i]);
    o[2 * i] = f.x;
    o[2 * i + 1] = f.y;
  }
}

constexpr int kKeyTile = 64;

template <typename TA, int HD>
__global__ void __launch_bounds__(128) k_attention(AttnArgs a) {
  constexpr int PD = HD / 8;   // output dims per thread in the PV product
  using VT = typename Vec<TA>::V;
  constexpr int VN = Vec<TA>::N;
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

  __shared__ float Qs[kMaxGroupRows][HD];
  __shared__ float Ks[kKeyTile][HD + 1];
  __shared__ __align__(16) float Vs[kKeyTile][HD];
  __shared__ float Ps[kMaxGroupRows][kKeyTile];
  __shared__ float s_m[kMaxGroupRows], s_l[kMaxGroupRows], s_corr[kMaxGroupRows];
  __shared__ int s_pos[kMaxGroupRows];

  const int t = threadIdx.x;
  const float scale = rsqrtf((float)HD);
  for (int i = t; i < kMaxGroupRows * HD; i += 128) {
    int r = i / HD, dd = i % HD;
    Qs[r][dd] = (r < nr) ? a.q[((size_t)(row0 + r) * a.H + h) * HD + dd] * scale : 0.f;
  }
  if (t < kMaxGroupRows) {
    s_m[t] = -INFINITY;
    s_l[t] = 0.f;
    s_corr[t] = 1.f;
    s_pos[t] = (t < nr) ? a.row_pos[row0 + t] : -1;
  }
  const int pr = t >> 3, pd = (t & 7) * PD;
  float acc[PD];
#pragma unroll
  for (int q = 0; q < PD; ++q) acc[q] = 0.f;
  __syncthreads();

  const TA* kv = reinterpret_cast<const TA*>(a.kv);
  const size_t head_page = (size_t)kPage * HD;
  const size_t layer_base = (size_t)a.layer * a.n_pages * 2 * a.H * head_page;
  bool bad_page = false;

  for (int kt = k_begin; kt < k_end; kt += kKeyTile) {
    for (int e = t * VN; e < kKeyTile * HD; e += 128 * VN) {
      int j = e / HD, dd = e % HD;
      int key = kt + j;
      float kf[VN], vf[VN];
      int page = -1;
      if (key < k_end) {
        int pi = key / kPage;
        page = pi < a.max_pages ? a.page_table[b * a.max_pages + pi] : -1;
        if (page < 0 || page >= a.n_pages) { bad_page = true; page = -1; }
      }
      if (page >= 0) {
        const TA* kp = kv + layer_base + (((size_t)page * 2) * a.H + h) * head_page +
                       (size_t)(key % kPage) * HD + dd;
        const TA* vp = kp + (size_t)a.H * head_page;
        unpack(*reinterpret_cast<const VT*>(kp), kf);
        unpack(*reinterpret_cast<const VT*>(vp), vf);
      } else {
#pragma unroll
        for (int q = 0; q < VN; ++q) { kf[q] = 0.f; vf[q] = 0.f; }
      }
#pragma unroll
      for (int q = 0; q < VN; ++q) { Ks[j][dd + q] = kf[q]; Vs[j][dd + q] = vf[q]; }
    }
    __syncthreads();
    {  // scores for 8 rows x 1 key per thread
      const int j = t & (kKeyTile - 1), rb = (t >> 6) * 8;
      float sc[8];
#pragma unroll
      for (int r = 0; r < 8; ++r) sc[r] = 0.f;
#pragma unroll 8
      for (int dd = 0; dd < HD; ++dd) {
        float kv_ = Ks[j][dd];
#pragma unroll
        for (int r = 0; r < 8; ++r) sc[r] += Qs[rb + r][dd] * kv_;
      }
      const int key = kt + j;
#pragma unroll
      for (int r = 0; r < 8; ++r) {
        bool ok = (rb + r < nr) && key < k_end && key <= s_pos[rb + r];
        Ps[rb + r][j] = ok ? sc[r] : -INFINITY;
      }
    }
    __syncthreads();
    {  // online softmax, 4 rows per warp
      const int w = t >> 5, lane = t & 31;
#pragma unroll
      for (int rr = 0; rr < 4; ++rr) {
        const int r = w * 4 + rr;
        float x0 = Ps[r][lane], x1 = Ps[r][lane + 32];
        float mx = fmaxf(x0, x1);
        for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        const float m_old = s_m[r];
        const float m_new = fmaxf(m_old, mx);
        float p0 = 0.f, p1 = 0.f, corr = 1.f;
        if (m_new != -INFINITY) {
          p0 = expf(x0 - m_new);
          p1 = expf(x1 - m_new);
          corr = expf(m_old - m_new);
        }
        float sum = p0 + p1;
        for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
        Ps[r][lane] = p0;
        Ps[r][lane + 32] = p1;
        __syncwarp();
        if (lane == 0) {
          s_l[r] = s_l[r] * corr + sum;
          s_m[r] = m_new;
          s_corr[r] = corr;
        }
      }
    }
    __syncthreads();
    {  // O = O * corr + P V
      const float c = s_corr[pr];
#pragma unroll
      for (int q = 0; q < PD; ++q) acc[q] *= c;
      for (int j = 0; j < kKeyTile; ++j) {
        const float p = Ps[pr][j];
#pragma unroll
        for (int q4 = 0; q4 < PD; q4 += 4) {
          const float4 v = *reinterpret_cast<const float4*>(&Vs[j][pd + q4]);
          acc[q4] += p * v.x; acc[q4 + 1] += p * v.y; acc[q4 + 2] += p * v.z; acc[q4 + 3] += p * v.w;
        }
      }
    }
    __syncthreads();
  }
  if (bad_page) atomicOr(a.d_err, kErrBadPage);
  if (pr < nr) {
    const int row = row0 + pr;
    if (a.n_split == 1) {
      const float inv = 1.f / s_l[pr];
      TA* o = reinterpret_cast<TA*>(a.out) + (size_t)row * a.H * HD + h * HD + pd;
#pragma unroll
      for (int q = 0; q < PD; ++q) o[q] = from_f<TA>(acc[q] * inv);
    } else {
      float* o = a.part_o + (((size_t)split * a.R + row) * a.H + h) * HD + pd;
#pragma unroll
      for (int q = 0; q < PD; ++q) o[q] = acc[q];
      if ((t & 7) == 0) a.part_ml[((size_t)split * a.R + row) * a.H + h] = make_float2(s_m[pr], s_l[pr]);
    }
  }
}

// merge the split partial softmaxes of one (row, head), splits in order
template <typename TA>
__global__ void k_attn_combine(AttnArgs a) {
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

void launch_attention(bool bf16, const AttnArgs& a, int n_groups, cudaStream_t s) {
  if (n_groups == 0) return;
  dim3 grid(n_groups, a.H, a.n_split);
  if (a.hd == 64) {
    if (bf16) k_attention<__nv_bfloat16, 64><<<grid, 128, 0, s>>>(a);
    else k_attention<float, 64><<<grid, 128, 0, s>>>(a);
  } else {
    if (bf16) k_attention<__nv_bfloat16, 32><<<grid, 128, 0, s>>>(a);
    else k_attention<float, 32><<<grid, 128, 0, s>>>(a);
  }
}

void launch_attn_combine(bool bf16, const AttnArgs& a, cudaStream_t s) {
  if (a.R == 0 || a.n_split <= 1) return;
  dim3 grid(a.R, a.H);
  if (bf16) k_attn_combine<__nv_bfloat16><<<grid, a.hd, 0, s>>>(a);
  else k_attn_combine<float><<<grid, a.hd, 0, s>>>(a);
}

}  // namespace kf
