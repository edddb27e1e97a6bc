// Skinny projections: D[M][N] = A[M][K] . W[N][K]^T for M <= 64 rows, with
// the fused epilogues of the tcgen05 GEMM (kf_gemm_tc.cu).
//
// A decode step at small batch feeds batch x (P + k) rows through every
// projection (Alg. 1): 8 rows for one sequence at k = 4, 64 for eight.  Each
// weight element is then used by at most 64 rows, 2 M flops per 2 bytes, far
// below the tensor cores' ridge, and each kernel of the step is a few
// microseconds of dependent latency: the dependency on the previous kernel,
// the A load, the products, the stores.  A 128-row tcgen05 tile spends its
// fixed MMA time whatever the rows, so these kernels take another shape:
//  - a CTA owns 16 output columns (weight rows) over a K range.  Its weight
//    boxes are TMA-loaded at entry, before griddepcontrol.wait: with
//    programmatic dependent launch the CTA is resident while the previous
//    kernel still runs (CTAs stay under ~64 KB of shared memory so they fit
//    beside it), and its weights arrive before the dependency resolves;
//  - after the wait it loads its A rows (one 64-wide K atom per TMA box) and
//    multiplies on warp-level MMA (m16n8k16: 16 weight rows x 8 A rows),
//    the K range split over the warps and summed in shared memory in warp
//    order;
//  - where A and W of the whole K exceed the budget, K is split over a
//    cluster of 2..8 CTAs.  After a cluster barrier CTA q sums rows q, q+S,
//    ... of the S partials over distributed shared memory in split order
//    (deterministic, no workspace) and runs the epilogue on them.
// Fused RMSNorm (QKV, MLP-up on the normed input): the CTA takes each A row's
// sum of squares from the bf16 row it holds (summed over the cluster's K
// ranges) and scales its outputs by rsqrt(sum / d + eps); the gains are folded
// into the weights as on the tcgen05 path.  Residual producers therefore write
// x and bf16(x) only: in a step that runs these kernels nothing reads per-slot
// sums of squares.
// EPI_QKV: a CTA's 16 weight rows are columns j0 .. j0+7 of one 64-wide head
// block and the 8 columns 32 further on, so the MMA hands each thread both
// members of a RoPE pair (accumulator rows g and g + 8).
// Waits on the TMA barriers are bounded (about 2 s); on expiry the kernel
// flags kErrTimeout and stores nothing.
#include <cuda.h>

#include "kf_mma.cuh"
#include "kf_tc.cuh"

namespace kf {

constexpr int kSkThreads = 256;
constexpr int kSkWarps = kSkThreads / 32;
constexpr int kSkNW = 16;                 // weight rows (output columns) per CTA
constexpr int kSkMaxRows = 64;
constexpr int kSkAtom = 64;               // K columns per TMA box (128 bytes of bf16)
constexpr int kSkWBox = kSkNW * 128;      // bytes of one atom of the CTA's weights
constexpr int kSkBudget = 64 * 1024;      // A + W bytes per CTA before K is split

bool encode_kmajor_bf16(CUtensorMap* m, const void* ptr, int rows, int cols, int ld, int box_rows);

struct SkArgs {
  int M, N, K;
  int kc;         // K columns per CTA (a multiple of 64)
  int splits;     // CTAs per cluster, one K range each
  int m_pad;      // M rounded up to 8: rows of an A box
  int norm;       // scale output rows by the RMSNorm of their A rows
  const char* l2_next;   // the next projection's weights, prefetched into L2 (or NULL)
  unsigned long long l2_bytes;
  int* d_err;
  Epi epi;
};

__device__ __forceinline__ float ld_dsmem1(uint32_t local_addr, uint32_t rank) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(local_addr), "r"(rank));
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(remote) : "memory");
  return v;
}

// value of this CTA's partial at float offset `off`, summed over the
// cluster's splits in split order
__device__ __forceinline__ float split_sum(const float* base, int off, int S) {
  if (S == 1) return base[off];
  const uint32_t a = smem_u32(base + off);
  float v = 0.f;
  for (int s = 0; s < S; ++s) v += ld_dsmem1(a, (uint32_t)s);
  return v;
}

// per-thread epilogue elements: QKV 8 RoPE pairs per row, others 16 columns
// per row; a CTA holds at most 64 rows, so at most 2 (QKV) or 4 per thread
constexpr int kSkMaxE = 4;

template <int EPI>
__global__ void __launch_bounds__(kSkThreads)
k_gemm_skinny(const __grid_constant__ CUtensorMap map_a, const __grid_constant__ CUtensorMap map_w, SkArgs g) {
  extern __shared__ __align__(1024) uint8_t sk_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(sk_raw) + 1023) & ~uintptr_t(1023));
  const int natoms = g.kc / kSkAtom;
  const uint32_t a_atom = (uint32_t)g.m_pad * 128;
  uint8_t* sw = smem;                                   // [atom][16 rows][128 B], swizzled
  uint8_t* sa = smem + natoms * kSkWBox;                // [atom][m_pad rows][128 B], swizzled
  float* red = reinterpret_cast<float*>(sa + natoms * a_atom);   // [warp][16][8]
  float* P = red + kSkWarps * 128;                      // [row][16] this CTA's partial
  float* ssq = P + kSkMaxRows * 16;                     // [row] partial sums of squares
  float* rinv = ssq + kSkMaxRows;                       // [row] RMSNorm scales
  uint64_t* bars = reinterpret_cast<uint64_t*>(rinv + kSkMaxRows);   // [0] W, [1] A
  int* flag = reinterpret_cast<int*>(bars + 2);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int S = g.splits;
  const int split = blockIdx.x;       // the cluster spans x: the CTA's rank
  const int blk = blockIdx.y;
  const int k0 = split * g.kc;
  const Epi& e = g.epi;

  // first weight row of the CTA's box(es): QKV two 8-row boxes 32 apart
  const int hb = blk >> 2, j0 = (blk & 3) * 8;
  const int w0 = EPI == EPI_QKV ? hb * 64 + j0 : blk * kSkNW;
  const uint32_t bw = smem_u32(&bars[0]), ba = smem_u32(&bars[1]);

  if (tid == 0) {
    mbar_init(bw, 1);
    mbar_init(ba, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_a)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_w)) : "memory");
    // both barriers armed before any copy is issued
    mbar_expect_tx(bw, (uint32_t)natoms * kSkWBox);
    mbar_expect_tx(ba, (uint32_t)natoms * a_atom);
  }
  __syncthreads();
  // Copies are issued by lane 0 of every warp (atoms w, w + 8, ...): one
  // thread issues them one after another.
  if (lane == 0) {
    // weights do not change during a step: load them before the dependency
    for (int a = warp; a < natoms; a += kSkWarps) {
      const uint32_t dst = smem_u32(sw + a * kSkWBox);
      if (EPI == EPI_QKV) {
        tma_load_2d(dst, &map_w, bw, k0 + a * kSkAtom, w0);
        tma_load_2d(dst + 1024, &map_w, bw, k0 + a * kSkAtom, w0 + 32);
      } else {
        tma_load_2d(dst, &map_w, bw, k0 + a * kSkAtom, w0);
      }
    }
    if (warp == kSkWarps - 1 && g.l2_next) {
      // this CTA's share of the next projection's weights (256-byte slices,
      // one prefetch each of at most 1 MiB)
      const unsigned long long nct = (unsigned long long)gridDim.x * gridDim.y;
      const unsigned long long cta = (unsigned long long)blockIdx.y * gridDim.x + blockIdx.x;
      const unsigned long long per = ((g.l2_bytes + nct - 1) / nct + 255) & ~255ull;
      for (unsigned long long o = cta * per; o < min(g.l2_bytes, (cta + 1) * per); o += (1u << 20)) {
        const unsigned long long n = min(min((unsigned long long)(1u << 20), (cta + 1) * per - o), g.l2_bytes - o);
        prefetch_l2(g.l2_next + o, (uint32_t)(n & ~15ull));
      }
    }
  }
  // epilogue data that is constant during the step, before the dependency
  const int nr = split < g.M ? (g.M - split + S - 1) / S : 0;   // rows split, split + S, ... (< M)
  const int per_row = EPI == EPI_QKV ? 8 : kSkNW;
  const int ne = nr * per_row;
  float pbias[kSkMaxE];
#pragma unroll
  for (int j = 0; j < kSkMaxE; ++j) {
    const int i = tid + j * kSkThreads;
    const int n = w0 + (i & 15);
    pbias[j] = ((EPI == EPI_BIAS_GELU || EPI == EPI_NOISE_OUT) && e.bias && i < ne && n < g.N) ? __ldg(e.bias + n) : 0.f;
  }
  float px[kSkMaxE], pc[kSkMaxE], psn[kSkMaxE];
  int pidx[kSkMaxE];
#pragma unroll
  for (int j = 0; j < kSkMaxE; ++j) { px[j] = 0.f; pc[j] = 1.f; psn[j] = 0.f; pidx[j] = -1; }
  // EPI_QKV: the RoPE angles and the KV slot of each element's row, from the
  // row's position and sequence
  auto qkv_meta = [&](int j, int i, int pos, int seq) {
    const int gc = j0 + (i & 7);
    const int sec = (hb * 64 + gc) / e.dsec;
    if (sec < 2 && e.cos_t) {
      pc[j] = __ldg(e.cos_t + (size_t)pos * 32 + gc);
      psn[j] = __ldg(e.sin_t + (size_t)pos * 32 + gc);
    }
    if (sec == 0) {
      pidx[j] = 0;
    } else {
      const int pg = pos / kPage;
      const int page = pg < e.max_pages ? __ldg(e.page_table + (size_t)seq * e.max_pages + pg) : -1;
      if (page < 0 || page >= e.n_pages) {
        atomicOr(e.d_err, kErrBadPage);
        pidx[j] = -1;
      } else {
        pidx[j] = page * kPage + pos % kPage;   // page slot
      }
    }
  };
  const bool early_meta = EPI == EPI_QKV && e.seq_len != nullptr;
  if (early_meta) {
    // decode: lengths and the page table are fixed for the whole step
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int i = tid + j * kSkThreads;
      if (i >= ne) continue;
      const int m = split + (i / per_row) * S;
      const int seq = m / e.rows_per_seq;
      qkv_meta(j, i, __ldg(e.seq_len + seq) + m % e.rows_per_seq, seq);
    }
  }
  pdl_wait();
  if (lane == 0)
    for (int a = warp; a < natoms; a += kSkWarps)
      tma_load_2d(smem_u32(sa + a * a_atom), &map_a, ba, k0 + a * kSkAtom, 0);
  // the epilogue's per-row data and residuals while A is in flight
#pragma unroll
  for (int j = 0; j < kSkMaxE; ++j) {
    const int i = tid + j * kSkThreads;
    if (i >= ne) continue;
    const int m = split + (i / per_row) * S;
    if (EPI == EPI_QKV) {
      if (!early_meta && j < 2) qkv_meta(j, i, __ldg(e.row_pos + m), __ldg(e.row_seq + m));
    } else if (EPI == EPI_RESID) {
      const int n = w0 + (i & 15);
      if (n < g.N) px[j] = e.x[(size_t)m * e.ldx + n];
    } else if (EPI == EPI_NOISE_OUT) {
      const int n = w0 + (i & 15);
      const int xr = __ldg(e.row_map + m);
      pidx[j] = xr;
      if (e.pos_emb && n < g.N) px[j] = __ldg(e.pos_emb + (size_t)__ldg(e.row_pos + xr) * g.N + n);
    }
  }
  if (tid == 0) flag[0] = (mbar_wait(bw, 0, g.d_err) && mbar_wait(ba, 0, g.d_err)) ? 1 : 0;
  __syncthreads();
  const bool ok = flag[0] != 0;

  if (ok && g.norm && g.m_pad <= 8) {
    // sum of squares of each A row over this CTA's K range: warp w takes row
    // w, lane l the l-th 4-byte word of the row in every atom
    const int m = warp;
    float sq = 0.f;
    for (int a = 0; a < natoms; ++a) {
      const float2 f = mma::unpack_bf16(*reinterpret_cast<const uint32_t*>(sa + a * a_atom + m * 128 + lane * 4));
      sq += f.x * f.x + f.y * f.y;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
    if (lane == 0) {
      ssq[m] = sq;
      if (S == 1) rinv[m] = rsqrtf(sq * e.inv_d + e.eps);
    }
  } else if (ok && g.norm) {
    // the same with tpr consecutive lanes per row, each summing wpt of the 32
    // words of the row in every atom; lane (row m, part t) starts at word
    // t * wpt + m, so the 32 lanes of a warp read 32 different banks
    const int tpr = g.m_pad <= 16 ? 16 : g.m_pad <= 32 ? 8 : 4;
    const int wpt = 32 / tpr;
    const int m = tid / tpr, t = tid % tpr;
    float sq = 0.f;
    if (m < g.m_pad) {
      for (int a = 0; a < natoms; ++a) {
        const uint8_t* row = sa + a * a_atom + m * 128;
        for (int w = 0; w < wpt; ++w) {
          const uint32_t u = *reinterpret_cast<const uint32_t*>(row + ((t * wpt + w + m) & 31) * 4);
          const float2 f = mma::unpack_bf16(u);
          sq += f.x * f.x + f.y * f.y;
        }
      }
    }
    for (int o = tpr / 2; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
    if (m < g.m_pad && t == 0) {
      ssq[m] = sq;
      if (S == 1) rinv[m] = rsqrtf(sq * e.inv_d + e.eps);
    }
  }

  // products: n-block nbi (A rows 8 nbi .. +7), K steps of part `part`
  const int nb = g.m_pad >> 3;
  const int kw = max(1, kSkWarps / nb);
  if (ok && warp < nb * kw) {
    const int nbi = warp / kw, part = warp % kw;
    const int nsteps = g.kc / 16;
    const int per = (nsteps + kw - 1) / kw;
    const int j1 = min(nsteps, (part + 1) * per);
    const int wrow = (lane & 7) + ((lane >> 3) & 1) * 8, wch = lane >> 4;
    const int xrow = nbi * 8 + (lane & 7), xch = (lane >> 3) & 1;
    const uint32_t swb = smem_u32(sw) + wrow * 128, sab = smem_u32(sa) + xrow * 128;
    // two accumulators over alternate K steps (two independent MMA chains),
    // added at the end
    float acc[4] = {0.f, 0.f, 0.f, 0.f}, acc2[4] = {0.f, 0.f, 0.f, 0.f};
    int j = part * per;
    for (; j + 1 < j1; j += 2) {
      uint32_t af[4], bf[2], af2[4], bf2[2];
      const int a = j >> 2, kk = j & 3, a2 = (j + 1) >> 2, kk2 = (j + 1) & 3;
      mma::ldsm_x4(swb + a * kSkWBox + (((kk * 2 + wch) ^ (wrow & 7)) << 4), af);
      mma::ldsm_x2(sab + a * a_atom + (((kk * 2 + xch) ^ (xrow & 7)) << 4), bf);
      mma::ldsm_x4(swb + a2 * kSkWBox + (((kk2 * 2 + wch) ^ (wrow & 7)) << 4), af2);
      mma::ldsm_x2(sab + a2 * a_atom + (((kk2 * 2 + xch) ^ (xrow & 7)) << 4), bf2);
      mma::mma16816(acc, af, bf[0], bf[1]);
      mma::mma16816(acc2, af2, bf2[0], bf2[1]);
    }
    if (j < j1) {
      uint32_t af[4], bf[2];
      const int a = j >> 2, kk = j & 3;
      mma::ldsm_x4(swb + a * kSkWBox + (((kk * 2 + wch) ^ (wrow & 7)) << 4), af);
      mma::ldsm_x2(sab + a * a_atom + (((kk * 2 + xch) ^ (xrow & 7)) << 4), bf);
      mma::mma16816(acc, af, bf[0], bf[1]);
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) acc[q] += acc2[q];
    const int gq = lane >> 2, t2 = (lane & 3) * 2;
    float* r = red + warp * 128;
    r[gq * 8 + t2] = acc[0];
    r[gq * 8 + t2 + 1] = acc[1];
    r[(gq + 8) * 8 + t2] = acc[2];
    r[(gq + 8) * 8 + t2 + 1] = acc[3];
  }
  __syncthreads();
  // this CTA's partial P[row][col], the warps' K parts summed in order
  for (int i = tid; i < g.m_pad * kSkNW; i += kSkThreads) {
    const int m = i >> 4, c = i & 15;
    const int nbi = m >> 3, xc = m & 7;
    float v = 0.f;
    for (int p = 0; p < kw; ++p) v += red[(nbi * kw + p) * 128 + c * 8 + xc];
    P[i] = v;
  }
  if (S > 1) {
    cluster_sync();
    if (ok && g.norm && tid < nr) {
      const int m = split + tid * S;
      rinv[m] = rsqrtf(split_sum(ssq, m, S) * e.inv_d + e.eps);
    }
  }
  __syncthreads();

  // this thread's outputs summed over the splits (QKV: both members of a
  // RoPE pair), then the peers may leave once every CTA has read (the
  // cluster barrier's arrive here, its wait after the stores)
  float va[kSkMaxE], vb[kSkMaxE];
#pragma unroll
  for (int j = 0; j < kSkMaxE; ++j) {
    const int i = tid + j * kSkThreads;
    va[j] = vb[j] = 0.f;
    if (!ok || i >= ne) continue;
    const int m = split + (i / per_row) * S;
    if (EPI == EPI_QKV) {
      va[j] = split_sum(P, m * 16 + (i & 7), S);
      vb[j] = split_sum(P, m * 16 + (i & 7) + 8, S);
    } else if (w0 + (i & 15) < g.N) {
      va[j] = split_sum(P, m * 16 + (i & 15), S);
    }
  }
  if (S > 1) cluster_arrive();

  if (ok) {
#pragma unroll
    for (int j = 0; j < kSkMaxE; ++j) {
      const int i = tid + j * kSkThreads;
      if (i >= ne) continue;
      const int m = split + (i / per_row) * S;
      if (EPI == EPI_QKV) {
        const int pi = i & 7;
        float a = va[j], b = vb[j];
        if (g.norm) { a *= rinv[m]; b *= rinv[m]; }
        const int gc = j0 + pi;
        const int col = hb * 64 + gc;
        const int sec = col / e.dsec;                 // 0 q, 1 k, 2 v
        const int h = (col - sec * e.dsec) >> 6;
        const float x1 = a, x2 = b;                   // (cos, sin) = (1, 0) for v
        a = x1 * pc[j] - x2 * psn[j];
        b = x2 * pc[j] + x1 * psn[j];
        if (sec == 0) {
          float* q = e.q_out + ((size_t)m * e.H + h) * 64 + gc;
          q[0] = a;
          q[32] = b;
        } else if (pidx[j] >= 0) {
          const int page = pidx[j] / kPage, slot = pidx[j] % kPage;
          __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(e.kv) +
                               ((((size_t)e.layer * e.n_pages + page) * 2 + (sec - 1)) * e.H + h) * (kPage * 64) +
                               (size_t)slot * 64 + gc;
          dst[0] = __float2bfloat16_rn(a);
          dst[32] = __float2bfloat16_rn(b);
        }
      } else {
        const int c = i & 15;
        const int n = w0 + c;
        if (n >= g.N) continue;
        float v = va[j];
        if (EPI == EPI_STORE_F32) {
          e.outf[(size_t)m * e.ldo + n] = v;
        } else if (EPI == EPI_STORE) {
          reinterpret_cast<__nv_bfloat16*>(e.out)[(size_t)m * e.ldo + n] = __float2bfloat16_rn(v);
        } else if (EPI == EPI_BIAS_GELU) {
          if (g.norm) v *= rinv[m];
          v += pbias[j];
          reinterpret_cast<__nv_bfloat16*>(e.out)[(size_t)m * e.ldo + n] = __float2bfloat16_rn(gelu_tanh_bf16(v));
        } else if (EPI == EPI_RESID) {
          const float xv = px[j] + v;
          e.x[(size_t)m * e.ldx + n] = xv;
          if (e.xb_out) reinterpret_cast<__nv_bfloat16*>(e.xb_out)[(size_t)m * e.ldx + n] = __float2bfloat16_rn(xv);
        } else if (EPI == EPI_NOISE_OUT) {
          const int xr = pidx[j];
          v = v + pbias[j] + px[j];
          e.x[(size_t)xr * e.ldx + n] = v;
          if (e.xb_out) reinterpret_cast<__nv_bfloat16*>(e.xb_out)[(size_t)xr * e.ldx + n] = __float2bfloat16_rn(v);
        }
      }
    }
  }
  // no CTA leaves while a peer may still read its partial
  if (S > 1) cluster_wait();
}

// ------------------------------------------------------------ host side
bool skinny_gemm_supported(const GemmDesc& g) {
  if (g.M < 1 || g.M > kSkMaxRows || g.N <= 0 || g.K <= 0 || g.K % kSkAtom) return false;
  if ((g.lda * 2) % 16 || (g.ldw * 2) % 16) return false;
  if ((reinterpret_cast<uintptr_t>(g.A) & 15) || (reinterpret_cast<uintptr_t>(g.W) & 15)) return false;
  switch (g.epi.kind) {
    case EPI_QKV:
      return g.N % 64 == 0 && g.epi.dsec > 0 && g.epi.dsec % 64 == 0;
    case EPI_RESID:
    case EPI_NOISE_OUT:
      return g.epi.ss_out == nullptr;   // no per-slot sums: see the file comment
    case EPI_BIAS_GELU:
    case EPI_STORE:
    case EPI_STORE_F32:
      return true;
    default:
      return false;
  }
}

// K split: the fewest K ranges (a power of two up to 8 dividing the K atoms)
// whose A and W boxes fit the per-CTA budget
static void skinny_plan(const GemmDesc& g, int* splits, int* kc, int* m_pad) {
  *m_pad = round_up(g.M, 8);
  const int kb = g.K / kSkAtom;
  int s = 1;
  while (s < 8 && kb % (2 * s) == 0 && (size_t)(g.K / s) * 2 * (kSkNW + *m_pad) > (size_t)kSkBudget) s *= 2;
  *splits = s;
  *kc = g.K / s;
}

static size_t skinny_smem(int kc, int m_pad) {
  const int natoms = kc / kSkAtom;
  return (size_t)natoms * kSkWBox + (size_t)natoms * m_pad * 128 +
         (size_t)(kSkWarps * 128 + kSkMaxRows * 16 + 2 * kSkMaxRows) * 4 + 64 + 1024;
}

template <int EPI>
static int launch_skinny_epi(const GemmDesc& g, int* d_err, cudaStream_t s) {
  int splits, kc, m_pad;
  skinny_plan(g, &splits, &kc, &m_pad);
  const size_t smem = skinny_smem(kc, m_pad);
  if (smem > 200 * 1024) return -1;
  static PerDevice attr;
  set_smem_attr(attr, k_gemm_skinny<EPI>, smem);
  CUtensorMap ma, mw;
  if (!encode_kmajor_bf16(&ma, g.A, g.M, g.K, g.lda, m_pad) ||
      !encode_kmajor_bf16(&mw, g.W, g.N, g.K, g.ldw, EPI == EPI_QKV ? 8 : kSkNW))
    return -1;
  SkArgs a;
  a.M = g.M; a.N = g.N; a.K = g.K; a.kc = kc; a.splits = splits; a.m_pad = m_pad;
  a.norm = (EPI == EPI_QKV || EPI == EPI_BIAS_GELU) && g.epi.ss_in ? 1 : 0;
  const bool pf = g.l2_next && g.l2_bytes >= 16 && !(reinterpret_cast<uintptr_t>(g.l2_next) & 15);
  a.l2_next = pf ? static_cast<const char*>(g.l2_next) : nullptr;
  a.l2_bytes = pf ? (g.l2_bytes & ~(size_t)15) : 0;
  a.d_err = d_err;
  a.epi = g.epi;
  const int nblk = EPI == EPI_QKV ? g.N / kSkNW : ceil_div(g.N, kSkNW);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(splits, nblk, 1);
  cfg.blockDim = dim3(kSkThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[2];
  int na = 0;
  if (splits > 1) {
    at[na].id = cudaLaunchAttributeClusterDimension;
    at[na].val.clusterDim.x = splits;
    at[na].val.clusterDim.y = 1;
    at[na].val.clusterDim.z = 1;
    ++na;
  }
  if (g_pdl) {
    at[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  cfg.attrs = at;
  cfg.numAttrs = na;
  return cudaLaunchKernelEx(&cfg, k_gemm_skinny<EPI>, ma, mw, a) == cudaSuccess ? 0 : -1;
}

int launch_gemm_skinny(const GemmDesc& g, int* d_err, cudaStream_t s) {
  switch (g.epi.kind) {
    case EPI_QKV: return launch_skinny_epi<EPI_QKV>(g, d_err, s);
    case EPI_RESID: return launch_skinny_epi<EPI_RESID>(g, d_err, s);
    case EPI_BIAS_GELU: return launch_skinny_epi<EPI_BIAS_GELU>(g, d_err, s);
    case EPI_NOISE_OUT: return launch_skinny_epi<EPI_NOISE_OUT>(g, d_err, s);
    case EPI_STORE: return launch_skinny_epi<EPI_STORE>(g, d_err, s);
    case EPI_STORE_F32: return launch_skinny_epi<EPI_STORE_F32>(g, d_err, s);
  }
  return -1;
}

}  // namespace kf
