// Row bookkeeping, embeddings, noise features, RMSNorm, RoPE + KV append,
// the LM head's noise -> token selection, and the step commit.
#include <algorithm>

#include <type_traits>

#include "kf_internal.cuh"

namespace kf {

// ------------------------------------------------------------ embeddings
// x[r] = E[tok] (+ pos_row).  With the fused RMSNorm (xb != NULL) the row is
// also written as bf16 into xb and the sum of squares of each of its
// 64-column slots into ss[r][d/64] (warp partials over 32 columns, then the
// pair of a slot added in order).  A thread loads its (at most kEmbedPer)
// columns of the embedding row before the dependency wait, all loads in
// flight at once (a no-op wait where the caller has already waited).
constexpr int kEmbedThreads = 128;
constexpr int kEmbedPer = 8;           // d <= 1024 kept in registers

template <typename TA>
__device__ void embed_row(int r, int tok, const float* __restrict__ pos_row, const TA* __restrict__ emb,
                          int V, int d, float* x, TA* xb, float* ss, int* d_err) {
  __shared__ float part[128];          // d <= 4096
  const bool good = tok >= 0 && tok < V;
  const TA* e = emb + (size_t)(good ? tok : 0) * d;
  const int lane = threadIdx.x & 31;
  const bool held = d <= kEmbedPer * kEmbedThreads;
  float v[kEmbedPer];
#pragma unroll
  for (int j = 0; j < kEmbedPer; ++j) {
    const int c = threadIdx.x + j * kEmbedThreads;
    v[j] = held && good && c < d ? to_f(e[c]) : 0.f;
  }
  pdl_wait();
  if (!good && threadIdx.x == 0) atomicOr(d_err, kErrBadToken);
  float* o = x + (size_t)r * d;
  for (int c0 = threadIdx.x - lane, j = 0; c0 < d; c0 += kEmbedThreads, ++j) {
    const int c = c0 + lane;
    float w = 0.f;
    if (c < d) {
      float base = 0.f;
      if (held) {
#pragma unroll
        for (int q = 0; q < kEmbedPer; ++q)
          if (q == j) base = v[q];
      } else {
        base = good ? to_f(e[c]) : 0.f;
      }
      w = good ? base + (pos_row ? pos_row[c] : 0.f) : 0.f;
      o[c] = w;
      if (xb) xb[(size_t)r * d + c] = from_f<TA>(w);
    }
    if (ss) {
      float q = w * w;
      for (int k = 16; k > 0; k >>= 1) q += __shfl_xor_sync(0xffffffffu, q, k);
      if (lane == 0) part[c0 / 32] = q;
    }
  }
  if (ss) {
    __syncthreads();
    for (int sl = threadIdx.x; sl < d / 64; sl += kEmbedThreads)
      ss[(size_t)r * (d / 64) + sl] = part[2 * sl] + part[2 * sl + 1];
  }
}

// the row tokens and positions are copied from the host before the launch
template <typename TA>
__global__ void __launch_bounds__(kEmbedThreads)
k_embed_tokens(const int32_t* __restrict__ row_tok, const TA* __restrict__ emb,
               const float* __restrict__ pos_emb, const int32_t* __restrict__ row_pos,
               int V, int d, float* x, TA* xb, float* ss, int* d_err) {
  int r = blockIdx.x;
  embed_row<TA>(r, row_tok[r], pos_emb ? pos_emb + (size_t)row_pos[r] * d : nullptr, emb, V, d, x,
                xb, ss, d_err);
}

void launch_embed_tokens(bool bf16, int R, const int32_t* row_tok, const void* tok_emb,
                         const float* pos_emb, const int32_t* row_pos, int V, int d, float* x,
                         void* xb, float* ss, int* d_err, cudaStream_t s) {
  if (R == 0) return;
  if (bf16)
    kf_launch(k_embed_tokens<__nv_bfloat16>, dim3(R), dim3(kEmbedThreads), 0, s, row_tok,
              (const __nv_bfloat16*)tok_emb, pos_emb, row_pos, V, d, x, (__nv_bfloat16*)xb, ss,
              d_err);
  else
    kf_launch(k_embed_tokens<float>, dim3(R), dim3(kEmbedThreads), 0, s, row_tok, (const float*)tok_emb,
              pos_emb, row_pos, V, d, x, (float*)xb, ss, d_err);
}

// --------------------------------------------------------- step prologue
// The first kernel of a decode step runs three independent jobs, one per
// block range, so that no kernel boundary separates them:
//  - blocks [0, B*P): the embedding of pending token i of sequence b into
//    row b*S + i at position c_b + i (Alg. 1 row layout: P pending tokens at
//    c_b .. c_b+P-1, then kz noise slots at c_b+P .. c_b+P+kz-1, S = P + kz);
//  - the next map_blocks blocks: the row maps (sequence and position of each
//    row, the noise rows that NoiseEnc writes, the rows the LM head reads);
//  - the rest: the noise features of the n_noise noise values (Table 4:
//    sinusoidal encodings of z and of tau, summed; [cos | sin] halves,
//    freq[t] = exp(-ln(1e4) t / (d/2)), the argument (scale * z) * freq[t]
//    formed in fp32 in that order (the oracle's arithmetic), its cosine
//    and sine from sincosf; tau's encoding is the same for every row and is
//    formed once per context).
// Every block first waits for the previous step: its commit wrote the
// lengths and the pending ids.  The wait also releases the step's later
// kernels, which may then read the lengths before their own waits (they
// change only at a commit).
template <typename TA>
__global__ void __launch_bounds__(kEmbedThreads)
k_step_prologue(int B, int P, int kz, int map_blocks, const int32_t* __restrict__ len,
                const int32_t* __restrict__ pending, int pend_stride, const TA* __restrict__ emb,
                const float* __restrict__ pos_emb, int V, int d, float* x, TA* xb, float* ss,
                int* d_err, int32_t* row_seq, int32_t* row_pos, int32_t* noise_map, int32_t* head_map,
                int n_noise, const float* __restrict__ noise, const float* __restrict__ freq,
                const float* __restrict__ tau_feat, float scale, TA* __restrict__ feat) {
  pdl_wait();
  const int S = P + kz;
  int blk = blockIdx.x;
  if (blk < B * P) {
    const int b = blk / P, i = blk - b * P;
    const int pos = len[b] + i;
    embed_row<TA>(b * S + i, pending[b * pend_stride + i],
                  pos_emb ? pos_emb + (size_t)pos * d : nullptr, emb, V, d, x, xb, ss, d_err);
    return;
  }
  blk -= B * P;
  if (blk < map_blocks) {
    const int r = blk * kEmbedThreads + threadIdx.x;
    if (r < B * S) {
      const int b = r / S, i = r - b * S;
      row_seq[r] = b;
      row_pos[r] = len[b] + i;
    }
    if (kz > 0 && r < B * kz) {
      const int b = r / kz, j = r - b * kz;
      noise_map[r] = b * S + P + j;
      head_map[r] = b * S + P + j;
    }
    if (kz == 0 && r < B) head_map[r] = r * S + P - 1;
    return;
  }
  blk -= map_blocks;
  const int half = d / 2;
  const int idx = blk * kEmbedThreads + threadIdx.x;
  if (idx >= n_noise * half) return;
  const int r = idx / half, t = idx - r * half;
  const float ang = __fmul_rn(__fmul_rn(scale, noise[r]), freq[t]);
  float sz, cz;
  sincosf(ang, &sz, &cz);
  feat[(size_t)r * d + t] = from_f<TA>(cz + tau_feat[t]);
  feat[(size_t)r * d + half + t] = from_f<TA>(sz + tau_feat[half + t]);
}

void launch_step_prologue(bool bf16, int B, int P, int kz, const int32_t* d_len, const int32_t* pending,
                          int pend_stride, const void* tok_emb, const float* pos_emb, int V, int d,
                          float* x, void* xb, float* ss, int* d_err, int32_t* row_seq, int32_t* row_pos,
                          int32_t* noise_map, int32_t* head_map, int n_noise, const float* noise,
                          const float* freq, const float* tau_feat, float scale, void* feat,
                          cudaStream_t s) {
  const int map_blocks = ceil_div(B * (P + kz), kEmbedThreads);
  const int noise_blocks = ceil_div(n_noise * (d / 2), kEmbedThreads);
  const dim3 grid(B * P + map_blocks + noise_blocks);
  if (grid.x == 0) return;
  if (bf16)
    kf_launch(k_step_prologue<__nv_bfloat16>, grid, dim3(kEmbedThreads), 0, s, B, P, kz, map_blocks,
              d_len, pending, pend_stride, (const __nv_bfloat16*)tok_emb, pos_emb, V, d, x,
              (__nv_bfloat16*)xb, ss, d_err, row_seq, row_pos, noise_map, head_map, n_noise, noise,
              freq, tau_feat, scale, (__nv_bfloat16*)feat);
  else
    kf_launch(k_step_prologue<float>, grid, dim3(kEmbedThreads), 0, s, B, P, kz, map_blocks, d_len,
              pending, pend_stride, (const float*)tok_emb, pos_emb, V, d, x, (float*)xb, ss, d_err,
              row_seq, row_pos, noise_map, head_map, n_noise, noise, freq, tau_feat, scale,
              (float*)feat);
}

// w[r][c] *= g[(r / rows_per_layer) * cols + c]: folds RMSNorm gains into the
// columns of the projection that consumes the normed rows
__global__ void k_scale_cols(float* __restrict__ w, const float* __restrict__ g, int rows_per_layer,
                             int cols, size_t total) {
  size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  size_t stride = (size_t)gridDim.x * blockDim.x;
  for (; i < total; i += stride) {
    const size_t r = i / cols;
    const int c = (int)(i - r * cols);
    w[i] *= g[(r / rows_per_layer) * cols + c];
  }
}

void launch_scale_cols(float* w, const float* g, int rows_per_layer, int cols, size_t total,
                       cudaStream_t s) {
  if (total == 0) return;
  int blocks = (int)std::min<size_t>((total + 255) / 256, 65535);
  k_scale_cols<<<blocks, 256, 0, s>>>(w, g, rows_per_layer, cols, total);
}

// --------------------------------------------------------------- RMSNorm
// out[r] = x[src] / sqrt(mean(x[src]^2) + eps) * g   (Table 4 pre-norm)
constexpr int kNormThreads = 128;
constexpr int kNormPer = 8;            // d <= 1024 kept in registers
template <typename TA>
__global__ void __launch_bounds__(kNormThreads)
k_rmsnorm(const int32_t* __restrict__ row_map, const float* __restrict__ x, int d,
          const float* __restrict__ g, float eps, TA* __restrict__ out) {
  const bool held = d <= kNormPer * kNormThreads;
  float gv[kNormPer], xv[kNormPer];
#pragma unroll
  for (int j = 0; j < kNormPer; ++j) {     // the gains before the dependency
    const int c = threadIdx.x + j * kNormThreads;
    gv[j] = held && c < d ? g[c] : 0.f;
  }
  pdl_wait();
  int r = blockIdx.x;
  int src = row_map ? row_map[r] : r;
  const float* xr = x + (size_t)src * d;
  float ss = 0.f;
  if (held) {
#pragma unroll
    for (int j = 0; j < kNormPer; ++j) {
      const int c = threadIdx.x + j * kNormThreads;
      xv[j] = c < d ? xr[c] : 0.f;
    }
#pragma unroll
    for (int j = 0; j < kNormPer; ++j) ss += xv[j] * xv[j];
  } else {
    for (int c = threadIdx.x; c < d; c += kNormThreads) ss += xr[c] * xr[c];
  }
  __shared__ float red[32];
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  if (threadIdx.x < 32) {
    float v = threadIdx.x < (kNormThreads >> 5) ? red[threadIdx.x] : 0.f;
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (threadIdx.x == 0) red[0] = v;
  }
  __syncthreads();
  float inv = rsqrtf(red[0] / (float)d + eps);
  TA* o = out + (size_t)r * d;
  if (held) {
#pragma unroll
    for (int j = 0; j < kNormPer; ++j) {
      const int c = threadIdx.x + j * kNormThreads;
      if (c < d) o[c] = from_f<TA>(xv[j] * inv * gv[j]);
    }
  } else {
    for (int c = threadIdx.x; c < d; c += kNormThreads) o[c] = from_f<TA>(xr[c] * inv * g[c]);
  }
}

void launch_rmsnorm(bool bf16, int R, const int32_t* row_map, const float* x, int d,
                    const float* g, float eps, void* out, cudaStream_t s) {
  if (R == 0) return;
  if (bf16)
    kf_launch(k_rmsnorm<__nv_bfloat16>, dim3(R), dim3(kNormThreads), 0, s, row_map, x, d, g, eps, (__nv_bfloat16*)out);
  else
    kf_launch(k_rmsnorm<float>, dim3(R), dim3(kNormThreads), 0, s, row_map, x, d, g, eps, (float*)out);
}

// ------------------------------------------------------ RoPE + KV append
// Rotate q and k of every row at its position (pairs (i, i+hd/2)), keep the
// rotated q (fp32) for attention and write k, v of ALL rows (pending and
// noise) into the paged cache.  Noise rows' entries sit at positions the
// next step overwrites with committed tokens (Alg. 1 discards C_z).
// KV pool layout: [layer][page][K|V][head][16 slots][hd].
template <typename TA, int HD>
__global__ void k_rope_append(const TA* __restrict__ qkv, int d, int H,
                              const int32_t* __restrict__ row_seq, const int32_t* __restrict__ row_pos,
                              const float* __restrict__ cos_t, const float* __restrict__ sin_t,
                              float* __restrict__ q, TA* __restrict__ kv, int layer, int n_pages,
                              const int32_t* __restrict__ page_table, int max_pages, int* d_err) {
  pdl_wait();
  constexpr int HALF = HD / 2;
  int r = blockIdx.x;
  int h = threadIdx.x / HALF, i = threadIdx.x % HALF;
  if (h >= H) return;
  int b = row_seq[r], pos = row_pos[r];
  const TA* src = qkv + (size_t)r * 3 * d + h * HD;
  float q1 = to_f(src[i]), q2 = to_f(src[i + HALF]);
  float k1 = to_f(src[d + i]), k2 = to_f(src[d + i + HALF]);
  float v1 = to_f(src[2 * d + i]), v2 = to_f(src[2 * d + i + HALF]);
  if (cos_t) {
    float c = cos_t[pos * HALF + i], sn = sin_t[pos * HALF + i];
    float a1 = q1 * c - q2 * sn, a2 = q2 * c + q1 * sn;
    q1 = a1; q2 = a2;
    float b1 = k1 * c - k2 * sn, b2 = k2 * c + k1 * sn;
    k1 = b1; k2 = b2;
  }
  float* qo = q + ((size_t)r * H + h) * HD;
  qo[i] = q1;
  qo[i + HALF] = q2;
  int pi = pos / kPage;
  int page = (pi < max_pages) ? page_table[b * max_pages + pi] : -1;
  if (page < 0 || page >= n_pages) {
    if (i == 0) atomicOr(d_err, kErrBadPage);
    return;
  }
  size_t base = ((((size_t)layer * n_pages + page) * 2) * H + h) * (kPage * HD) +
                (size_t)(pos % kPage) * HD;
  size_t vofs = (size_t)H * kPage * HD;
  kv[base + i] = from_f<TA>(k1);
  kv[base + i + HALF] = from_f<TA>(k2);
  kv[base + vofs + i] = from_f<TA>(v1);
  kv[base + vofs + i + HALF] = from_f<TA>(v2);
}

template <int HD>
static void rope_append_hd(bool bf16, int R, const void* qkv, int d, int H, const int32_t* row_seq,
                           const int32_t* row_pos, const float* cos_t, const float* sin_t, float* q,
                           void* kv, int layer, int n_pages, const int32_t* page_table,
                           int max_pages, int* d_err, cudaStream_t s) {
  int threads = H * (HD / 2);
  if (bf16)
    kf_launch(k_rope_append<__nv_bfloat16, HD>, dim3(R), dim3(threads), 0, s, (const __nv_bfloat16*)qkv, d, H,
        row_seq, row_pos, cos_t, sin_t, q, (__nv_bfloat16*)kv, layer, n_pages, page_table,
        max_pages, d_err);
  else
    kf_launch(k_rope_append<float, HD>, dim3(R), dim3(threads), 0, s, (const float*)qkv, d, H, row_seq, row_pos,
        cos_t, sin_t, q, (float*)kv, layer, n_pages, page_table, max_pages, d_err);
}

void launch_rope_append(bool bf16, int R, const void* qkv, int d, int H, int hd,
                        const int32_t* row_seq, const int32_t* row_pos, const float* cos_t,
                        const float* sin_t, float* q, void* kv, int layer, int n_pages,
                        const int32_t* page_table, int max_pages, int* d_err, cudaStream_t s) {
  if (R == 0) return;
  if (hd == 64)
    rope_append_hd<64>(bf16, R, qkv, d, H, row_seq, row_pos, cos_t, sin_t, q, kv, layer, n_pages,
                       page_table, max_pages, d_err, s);
  else
    rope_append_hd<32>(bf16, R, qkv, d, H, row_seq, row_pos, cos_t, sin_t, q, kv, layer, n_pages,
                       page_table, max_pages, d_err, s);
}

// ------------------------------------------------- noise -> token select
// Combines the per-chunk records of one head row (l = logits / tau):
//   M = max_c m_c,  S = sum_c s_c exp(m_c - M)        (chunks in id order)
// ICDF (Eq. 1, App. B strict '>'): T = z S; the first chunk c* whose running
// sum exceeds T; its 32 logits are recomputed and the first id whose running
// sum (from the chunk start, T' = T - sum before c*) exceeds T' is the token.
// If rounding leaves no crossing, the largest id with exp(l - M) > 0 wins.
// ARGMAX: the lowest id attaining M.
constexpr int kSelThreads = 256;

__device__ __forceinline__ void ld_vec(const float* p, float* o) {
  float4 a = *reinterpret_cast<const float4*>(p);
  o[0] = a.x; o[1] = a.y; o[2] = a.z; o[3] = a.w;
}
__device__ __forceinline__ void ld_vec(const __nv_bfloat16* p, float* o) {
  uint4 v = *reinterpret_cast<const uint4*>(p);
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float2 f = __bfloat1622float2(h[i]);
    o[2 * i] = f.x;
    o[2 * i + 1] = f.y;
  }
}

// exp(m - M) in the precision of the inverse-CDF sums
template <typename Acc> __device__ __forceinline__ Acc chunk_scale(float m, float M);
template <> __device__ __forceinline__ float chunk_scale<float>(float m, float M) { return expf(m - M); }
template <> __device__ __forceinline__ double chunk_scale<double>(float m, float M) {
  return exp((double)m - (double)M);
}

// Token zrow = b nout + j is written to tokens and, in a decode step, the
// step's commit (C <- [C; C_x], App. C.1 fixed stride) is taken here: it
// becomes pending token j of sequence b, and sequence b's block j = 0 adds the
// P newly cached tokens to its length.  Every kernel that reads the lengths or
// the pending ids in this step has completed (the dependency wait), and the
// next step's first kernel reads them only after its own wait.
__device__ __forceinline__ void emit_token(int32_t* tokens, int zrow, int tok, const StepCommit& cm) {
  tokens[zrow] = tok;
  if (cm.pending) {
    const int b = zrow / cm.nout, j = zrow - b * cm.nout;
    cm.pending[(size_t)b * cm.pend_stride + j] = tok;
    if (j == 0) cm.len[b] += cm.P;
  }
}

template <typename TA>
__global__ void __launch_bounds__(kSelThreads)
k_head_select(const HeadRec* __restrict__ rec_all, int nchunk, const TA* __restrict__ head_in, int d,
              const TA* __restrict__ w_head_all, int V, float inv_tau, int map_kind,
              const float* __restrict__ noise, int32_t* __restrict__ tokens, int mtp_rows,
              size_t head_stride, const int* __restrict__ err, StepCommit cm) {
  pdl_wait();
  // one block per mapped row; MTP (mtp_rows = B > 0): block j B + b is head j
  // of sequence b (records in that order), hidden row b, weights w_head + j
  // head_stride, noise and token index b k + j
  const int row = blockIdx.x;
  int hrow = row, zrow = row;
  const TA* w_head = w_head_all;
  if (mtp_rows > 0) {
    const int b = row % mtp_rows, j = row / mtp_rows, kk = gridDim.x / mtp_rows;
    hrow = b;
    zrow = b * kk + j;
    w_head = w_head_all + (size_t)j * head_stride;
  }
  // an earlier kernel of the call flagged an error (e.g. a bounded wait ran
  // out, so the records may be stale): token -1 instead of a stale choice.
  // Every earlier kernel has completed (pdl_wait), so all threads read the
  // same value.
  if (err && *err) {
    if (threadIdx.x == 0) emit_token(tokens, zrow, -1, cm);
    return;
  }
  // the inverse-CDF sums: fp32 for the bf16 model (its logits carry bf16
  // rounding far above fp32's); fp64 for the fp32 model, so its decision is
  // limited by its fp32 logits and not by ~5e4 fp32 additions
  using Acc = typename std::conditional<sizeof(TA) == 4, double, float>::type;
  const HeadRec* rec = rec_all + (size_t)row * nchunk;
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  __shared__ float s_red[kSelThreads / 32];
  __shared__ Acc s_acc[kSelThreads / 32];
  __shared__ int s_redi[kSelThreads / 32];
  __shared__ float s_M;
  __shared__ Acc s_T;
  __shared__ int s_chunk;
  __shared__ Acc s_before;

  // contiguous chunk range per thread keeps id order inside each partial sum
  const int per = ceil_div(nchunk, kSelThreads);
  const int c0 = min(nchunk, t * per), c1 = min(nchunk, c0 + per);

  // 1) M and (for argmax) the lowest id attaining it; the thread's records
  //    stay in registers for step 2 when they fit
  constexpr int kKeep = 8;
  const bool keep = c1 - c0 <= kKeep;
  float km[kKeep], ks[kKeep];
  float m = -INFINITY;
  int am = 0x7fffffff;
#pragma unroll
  for (int i = 0; i < kKeep; ++i) {
    km[i] = -INFINITY;
    ks[i] = 0.f;
    if (keep && c0 + i < c1) {
      const HeadRec r = rec[c0 + i];
      km[i] = r.m;
      ks[i] = r.s;
      if (r.m > m) { m = r.m; am = r.a; }
    }
  }
  if (!keep) {
    for (int c = c0; c < c1; ++c) {
      HeadRec r = rec[c];
      if (r.m > m) { m = r.m; am = r.a; }
    }
  }
  for (int o = 16; o > 0; o >>= 1) {
    float m2 = __shfl_xor_sync(0xffffffffu, m, o);
    int a2 = __shfl_xor_sync(0xffffffffu, am, o);
    if (m2 > m || (m2 == m && a2 < am)) { m = m2; am = a2; }
  }
  if (lane == 0) { s_red[warp] = m; s_redi[warp] = am; }
  __syncthreads();
  if (t == 0) {
    float M = s_red[0];
    int A = s_redi[0];
    for (int w = 1; w < kSelThreads / 32; ++w)
      if (s_red[w] > M || (s_red[w] == M && s_redi[w] < A)) { M = s_red[w]; A = s_redi[w]; }
    s_M = M;
    s_redi[0] = A;
  }
  __syncthreads();
  if (map_kind == KF_MAP_ARGMAX) {
    if (t == 0) emit_token(tokens, zrow, s_redi[0], cm);
    return;
  }
  const float M = s_M;

  // 2) per-thread partial sums (id order inside each range), then a
  //    fixed-order block scan over the threads: lanes by shuffles, warps by
  //    their totals.  The scan's last element is the total S, so T = z S
  //    is crossed for every z < 1.
  Acc part = 0;
  if (keep) {
#pragma unroll
    for (int i = 0; i < kKeep; ++i)
      if (c0 + i < c1) part += (Acc)ks[i] * chunk_scale<Acc>(km[i], M);
  } else {
    for (int c = c0; c < c1; ++c) {
      HeadRec r = rec[c];
      part += (Acc)r.s * chunk_scale<Acc>(r.m, M);
    }
  }
  Acc inc = part;
  for (int o = 1; o < 32; o <<= 1) {
    const Acc y = __shfl_up_sync(0xffffffffu, inc, o);
    if (lane >= o) inc += y;
  }
  Acc lane_excl = __shfl_up_sync(0xffffffffu, inc, 1);
  if (lane == 0) lane_excl = 0;
  if (lane == 31) s_acc[warp] = inc;
  __syncthreads();
  __shared__ Acc s_wexcl[kSelThreads / 32 + 1];
  if (t == 0) {
    Acc run = 0;
    for (int w = 0; w < kSelThreads / 32; ++w) {
      s_wexcl[w] = run;
      run += s_acc[w];
    }
    s_wexcl[kSelThreads / 32] = run;     // S
    s_T = (Acc)noise[zrow] * run;
    s_redi[2] = kSelThreads;             // first crossing thread (none yet)
  }
  __syncthreads();
  const Acc T = s_T;
  const Acc excl = s_wexcl[warp] + lane_excl, incl = s_wexcl[warp] + inc;
  {
    const unsigned cross = __ballot_sync(0xffffffffu, incl > T);
    if (lane == 0 && cross) atomicMin(&s_redi[2], warp * 32 + __ffs(cross) - 1);
  }
  __syncthreads();
  if (t == s_redi[2]) {
    // the crossing range: walk its chunks in id order from its exclusive prefix
    Acc acc = excl;
    int cstar = c1 - 1;
    Acc before = acc;
    for (int c = c0; c < c1; ++c) {
      HeadRec r = rec[c];
      const Acc sc = (Acc)r.s * chunk_scale<Acc>(r.m, M);
      // the range's own order can round differently from its partial sum:
      // its last chunk takes the crossing then
      if (acc + sc > T || c == c1 - 1) { cstar = c; before = acc; break; }
      acc += sc;
    }
    s_chunk = cstar;
    s_before = before;
    s_redi[1] = 0;
  }
  if (t == 0 && s_redi[2] >= kSelThreads) {
    // no crossing at all (z near 1): the last chunk with mass, last id in it
    int cstar = nchunk - 1;
    while (cstar > 0 && !(rec[cstar].s * expf(rec[cstar].m - M) > 0.f)) --cstar;
    s_chunk = cstar;
    s_before = 0;
    s_redi[1] = 1;
  }
  __syncthreads();

  // 3) recompute chunk c*'s 32 logits (each warp 4 ids, lanes along d with
  //    16-byte loads), then warp 0 locates the token in id order
  __shared__ float s_logit[kChunk];
  const int cstar = s_chunk;
  {
    // the warp's NQ ids side by side, so their weight loads are in flight together
    const TA* hr = head_in + (size_t)hrow * d;
    constexpr int VEC = 16 / sizeof(TA);
    constexpr int NQ = kChunk / (kSelThreads / 32);
    const int jj0 = warp * NQ;
    float acc[NQ];
#pragma unroll
    for (int q = 0; q < NQ; ++q) acc[q] = 0.f;
    for (int c0 = lane * VEC; c0 < d; c0 += 32 * VEC) {
      float hv[VEC];
      ld_vec(hr + c0, hv);
#pragma unroll
      for (int q = 0; q < NQ; ++q) {
        const int v = cstar * kChunk + jj0 + q;
        if (v < V) {
          float wv[VEC];
          ld_vec(w_head + (size_t)v * d + c0, wv);
#pragma unroll
          for (int i = 0; i < VEC; ++i) acc[q] = fmaf(hv[i], wv[i], acc[q]);
        }
      }
    }
#pragma unroll
    for (int q = 0; q < NQ; ++q) {
      float a = acc[q];
      for (int o = 16; o > 0; o >>= 1) a += __shfl_xor_sync(0xffffffffu, a, o);
      const int v = cstar * kChunk + jj0 + q;
      if (lane == 0) s_logit[jj0 + q] = (v < V) ? a * inv_tau : -INFINITY;
    }
  }
  __syncthreads();
  if (warp != 0) return;
  const int v = cstar * kChunk + lane;
  const float l = s_logit[lane];
  const Acc e = (v < V) ? chunk_scale<Acc>(l, M) : (Acc)0;
  // inclusive prefix over lanes in id order
  Acc pre = e;
  for (int o = 1; o < 32; o <<= 1) {
    Acc y = __shfl_up_sync(0xffffffffu, pre, o);
    if (lane >= o) pre += y;
  }
  const Acc Tp = s_T - s_before;
  const bool fallback = s_redi[1] != 0;
  unsigned hit = __ballot_sync(0xffffffffu, !fallback && (v < V) && (pre > Tp));
  unsigned pos = __ballot_sync(0xffffffffu, (v < V) && (e > (Acc)0));
  if (lane == 0) {
    int tok;
    if (hit) tok = cstar * kChunk + (__ffs(hit) - 1);
    else if (pos) tok = cstar * kChunk + (31 - __clz(pos));
    else tok = min(V - 1, cstar * kChunk + 31);
    emit_token(tokens, zrow, tok, cm);
  }
}

void launch_head_select(bool bf16, int n_rows, const HeadRec* rec, int nchunk, const void* head_in,
                        int d, const void* w_head, int V, float inv_tau, int map_kind,
                        const float* noise, int32_t* tokens, int mtp_rows, size_t head_stride,
                        const int* err, const StepCommit& cm, cudaStream_t s) {
  if (n_rows == 0) return;
  if (bf16)
    kf_launch(k_head_select<__nv_bfloat16>, dim3(n_rows), dim3(kSelThreads), 0, s, rec, nchunk,
        (const __nv_bfloat16*)head_in, d, (const __nv_bfloat16*)w_head, V, inv_tau, map_kind,
        noise, tokens, mtp_rows, head_stride, err, cm);
  else
    kf_launch(k_head_select<float>, dim3(n_rows), dim3(kSelThreads), 0, s, rec, nchunk, (const float*)head_in, d,
        (const float*)w_head, V, inv_tau, map_kind, noise, tokens, mtp_rows, head_stride, err, cm);
}

}  // namespace kf

namespace kf {

// fp32 -> storage type (round to nearest even for bf16)
template <typename T>
__global__ void k_convert(const float* __restrict__ src, T* __restrict__ dst, size_t n) {
  pdl_wait();
  size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  size_t stride = (size_t)gridDim.x * blockDim.x;
  for (; i < n; i += stride) dst[i] = from_f<T>(src[i]);
}

void launch_convert_f32(bool bf16, const float* src, void* dst, size_t n, cudaStream_t s) {
  if (n == 0) return;
  int blocks = (int)std::min<size_t>((n + 255) / 256, 65535);
  if (bf16) kf_launch(k_convert<__nv_bfloat16>, dim3(blocks), dim3(256), 0, s, src, (__nv_bfloat16*)dst, n);
  else kf_launch(k_convert<float>, dim3(blocks), dim3(256), 0, s, src, (float*)dst, n);
}

}  // namespace kf
