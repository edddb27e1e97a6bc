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
//   warps 2..9  epilogue: warp w reads TMEM lanes 32 (w % 4) .. +31 (its 32
//               rows); the two warps of a lane quarter take alternate
//               64-column blocks of the tile (or, with a single block,
//               alternate halves of its rows).  While the mainloop runs they
//               fetch the per-row data of the tile (RMSNorm scales, positions,
//               KV pages) into shared memory.
// When the output tiles cannot fill the SMs the K range is split over a
// thread-block cluster of up to 8 CTAs (one per split): each keeps its fp32
// partial tile in its own shared memory and, after a cluster barrier, CTA q
// sums rows q, q+S, ... over distributed shared memory in split order
// (deterministic) and runs the epilogue on them.
// With programmatic dependent launch the producer streams the first stages'
// weight tiles before waiting for the kernel that writes the activations.
// Every mbarrier wait is bounded (about 2 s of %globaltimer); on expiry the
// kernel flags kErrTimeout, stops issuing work and exits after freeing TMEM.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <mutex>

#include "kf_tc.cuh"

namespace kf {

constexpr int kBM = 128;
constexpr int kBK = 64;                 // one 128-byte swizzle atom of bf16

constexpr int kEpiWarps = 8;
constexpr int kThreads = 64 + 32 * kEpiWarps;
constexpr int kPersistWarps = 2 + kEpiWarps + 1;   // + a second TMA producer

// TMEM columns to allocate for n accumulator columns: a power of two >= 32
__host__ __device__ constexpr int tmem_alloc_cols(int n) { return n <= 32 ? 32 : n <= 64 ? 64 : n <= 128 ? 128 : n <= 256 ? 256 : 512; }

// per-row data of a tile, fetched by the epilogue warps during the mainloop
struct EpiMeta {
  float rinv[kBM];   // fused RMSNorm scale of the A row
  int pos[kBM];      // EPI_QKV: position of the row
  int aux[kBM];      // EPI_QKV: KV page of the row (-1 if invalid)
};

struct TcArgs {
  int M, N, K;
  int kb_per_split;   // K blocks per split
  int splits;
  uint32_t a_box;     // bytes of one A box: its rows (min(128, M rounded up to 8)) x 128
  const char* l2_next;   // the next projection's weights, prefetched into L2 (or NULL)
  unsigned long long l2_bytes;
  int* d_err;
  Epi epi;
};

__device__ __forceinline__ void epi_bar() {
  asm volatile("bar.sync 1, %0;" ::"n"(32 * kEpiWarps) : "memory");
}

// the per-row data of tile row et (row m0 + et): RMSNorm scale of the A row
// (EPI_QKV, EPI_BIAS_GELU with ss_in), position and KV page (EPI_QKV; an
// out-of-range page is flagged and stored as -1)
template <int EPI>
__device__ __forceinline__ void fill_meta(EpiMeta* meta, const TcArgs& g, int m0, int et) {
  const int row = m0 + et;
  const bool in = row < g.M;
  if ((EPI == EPI_QKV || EPI == EPI_BIAS_GELU) && g.epi.ss_in) meta->rinv[et] = in ? row_rinv(g.epi, row) : 0.f;
  if (EPI == EPI_QKV) {
    int pos = 0, page = -1;
    if (in) {
      pos = __ldg(g.epi.row_pos + row);
      const int pi = pos / kPage;
      page = pi < g.epi.max_pages
                 ? __ldg(g.epi.page_table + (size_t)__ldg(g.epi.row_seq + row) * g.epi.max_pages + pi)
                 : -1;
      if (page < 0 || page >= g.epi.n_pages) {
        page = -1;
        atomicOr(g.epi.d_err, kErrBadPage);
      }
    }
    meta->pos[et] = pos;
    meta->aux[et] = page;
  }
}

// The vector epilogue of one 128 x BN accumulator tile (one warp's share):
// per 64-column block a 32 x 68 fp32 staging block T.  tcgen05.ld gives a
// thread one row's columns; the block is re-read with lane l on row
// (l / 8) + 4 i, columns 4 (l % 8) .. +3 (and + 32), so every warp store
// covers four 128-byte row segments.  quarter: the warp's TMEM lane quarter;
// ch: which of the quarter's two warps (alternate 64-column blocks, or
// alternate halves of the rows when the tile has one block).
template <int BN, int EPI>
struct EpiRows {
  static constexpr int NB = BN / 64;                  // 64-column blocks
  static constexpr int NI = NB >= 2 ? 8 : 4;          // row groups per warp
  static constexpr bool kAny = EPI == EPI_QKV || EPI == EPI_RESID;
  // per row group of one block: QKV the RoPE cos / sin at the row's
  // position, RESID the residual x (columns gc and gc + 32)
  float4 a[kAny ? NI : 1], b[kAny ? NI : 1];
};

// the first 64-column block of this warp (NB >= 2: block ch, else block 0)
template <int BN>
__device__ __forceinline__ int epi_first_block(int ch) { return BN / 64 >= 2 ? ch : 0; }

// Issue the global loads of the per-row data of block bb (all row groups at
// once, so their latencies overlap); EPI_QKV reads meta->pos.
template <int BN, int EPI>
__device__ __forceinline__ void epi_rows_load(EpiRows<BN, EPI>& r, const TcArgs& g, const EpiMeta* meta, int m0,
                                              int n0, int quarter, int ch, int lane, int bb) {
  using R = EpiRows<BN, EPI>;
  const int ibase = R::NB >= 2 ? 0 : ch * 4;
  const int gr = lane >> 3, gc = (lane & 7) * 4;
  const int c = bb * 64;
  if (EPI == EPI_QKV) {
    if (g.epi.cos_t && n0 + c < 2 * g.epi.dsec) {         // q and k rotate
#pragma unroll
      for (int ii = 0; ii < R::NI; ++ii) {
        const int pos = meta->pos[quarter * 32 + gr + 4 * (ibase + ii)];
        r.a[ii] = __ldg(reinterpret_cast<const float4*>(g.epi.cos_t + (size_t)pos * 32 + gc));
        r.b[ii] = __ldg(reinterpret_cast<const float4*>(g.epi.sin_t + (size_t)pos * 32 + gc));
      }
    }
  } else if (EPI == EPI_RESID) {
#pragma unroll
    for (int ii = 0; ii < R::NI; ++ii) {
      const int row = m0 + quarter * 32 + gr + 4 * (ibase + ii);
      const float* xp = g.epi.x + (size_t)row * g.epi.ldx + n0 + c + gc;
      const bool okr = row < g.M && n0 + c + gc < g.N;
      r.a[ii] = okr ? *reinterpret_cast<const float4*>(xp) : make_float4(0.f, 0.f, 0.f, 0.f);
      r.b[ii] = (okr && n0 + c + 32 + gc < g.N) ? *reinterpret_cast<const float4*>(xp + 32)
                                                : make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }
}

// r holds the per-row data of the warp's first block on entry (epi_rows_load
// with epi_first_block, issued before the accumulator wait)
template <int BN, int EPI>
__device__ __forceinline__ void epi_vec_tile(const TcArgs& g, const EpiMeta* meta, float* __restrict__ T,
                                             uint32_t lane_addr,
                                             int m0, int n0, int quarter, int ch, int lane, EpiRows<BN, EPI>& r) {
  using R = EpiRows<BN, EPI>;
  constexpr int NB = R::NB, NI = R::NI;
  const int b0 = epi_first_block<BN>(ch);
  const int ibase = NB >= 2 ? 0 : ch * 4;
  const int gr = lane >> 3, gc = (lane & 7) * 4;
#pragma unroll 1
  for (int bb = b0; bb < NB; bb += (NB >= 2 ? 2 : 1)) {
    const int c = bb * 64;
    if (n0 + c >= g.N) break;                  // past the last column (warp-uniform)
    if (bb != b0) epi_rows_load<BN, EPI>(r, g, meta, m0, n0, quarter, ch, lane, bb);
#pragma unroll
    for (int h2 = 0; h2 < 2; ++h2) {
      float v[32];
      tmem_ld32(lane_addr + c + 32 * h2, v);
#pragma unroll
      for (int q = 0; q < 8; ++q)
        *reinterpret_cast<float4*>(T + lane * 68 + 32 * h2 + 4 * q) =
            make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
    }
    __syncwarp();
    float4 bias_lo = make_float4(0.f, 0.f, 0.f, 0.f), bias_hi = bias_lo;
    if (EPI == EPI_BIAS_GELU && g.epi.bias) {
      bias_lo = __ldg(reinterpret_cast<const float4*>(g.epi.bias + n0 + c + gc));
      if (n0 + c + 32 + gc < g.N) bias_hi = __ldg(reinterpret_cast<const float4*>(g.epi.bias + n0 + c + 32 + gc));
    }
#pragma unroll
    for (int ii = 0; ii < NI; ++ii) {
      const int rl = quarter * 32 + gr + 4 * (ibase + ii);   // row within the tile
      const int row = m0 + rl;
      const bool ok = row < g.M;                 // uniform over 8 lanes
      float4 lo = *reinterpret_cast<const float4*>(T + (rl - quarter * 32) * 68 + gc);
      float4 hi = *reinterpret_cast<const float4*>(T + (rl - quarter * 32) * 68 + 32 + gc);
      if ((EPI == EPI_QKV || EPI == EPI_BIAS_GELU) && ok && g.epi.ss_in) {
        const float ri = meta->rinv[rl];        // fused RMSNorm of the A rows
        lo = scale4(lo, ri);
        hi = scale4(hi, ri);
      }
      float sq = 0.f;
      if (ok) {
        if (EPI == EPI_QKV) {
          epi_qkv_rot<__nv_bfloat16>(g.epi, row, meta->pos[rl], meta->aux[rl], n0 + c, gc, lo, hi, r.a[ii], r.b[ii]);
        } else if (EPI == EPI_RESID) {
          if (n0 + c + gc < g.N) sq = epi_resid4<__nv_bfloat16>(g.epi, row, n0 + c + gc, lo, r.a[ii]);
          if (n0 + c + 32 + gc < g.N)
            sq += epi_resid4<__nv_bfloat16>(g.epi, row, n0 + c + 32 + gc, hi, r.b[ii]);
        } else if (EPI == EPI_BIAS_GELU) {
          sq = epi_vec4<__nv_bfloat16, EPI>(g.epi, row, n0 + c + gc, add4(lo, bias_lo), g.N, false) +
               epi_vec4<__nv_bfloat16, EPI>(g.epi, row, n0 + c + 32 + gc, add4(hi, bias_hi), g.N, false);
        } else {
          sq = epi_vec4<__nv_bfloat16, EPI>(g.epi, row, n0 + c + gc, lo, g.N) +
               epi_vec4<__nv_bfloat16, EPI>(g.epi, row, n0 + c + 32 + gc, hi, g.N);
        }
      }
      if ((EPI == EPI_RESID || EPI == EPI_NOISE_OUT) && g.epi.ss_out) {
        // the 8 lanes of this row hold its 64-column slot: fixed-order butterfly
        sq += __shfl_xor_sync(0xffffffffu, sq, 1);
        sq += __shfl_xor_sync(0xffffffffu, sq, 2);
        sq += __shfl_xor_sync(0xffffffffu, sq, 4);
        if (ok && (lane & 7) == 0) {
          const int xr = (EPI == EPI_NOISE_OUT) ? g.epi.row_map[row] : row;
          g.epi.ss_out[(size_t)xr * g.epi.nslot + (n0 + c) / 64] = sq;
        }
      }
    }
    __syncwarp();
  }
}

// ------------------------------------------------------------ the kernel
// MT: 128-row M tiles per CTA, each with its own TMEM accumulator (2 only for
// the LM-head records, which need no per-row data); AT: 64-wide K atoms per
// pipeline stage, so that one mbarrier wait and one commit cover 4 * MT * AT
// MMAs
template <int BN, int STAGES, int EPI, int MT, int AT>
__global__ void __launch_bounds__(kThreads, 1)
k_gemm_tc(const __grid_constant__ CUtensorMap map_a, const __grid_constant__ CUtensorMap map_w,
          TcArgs g) {
  constexpr uint32_t A_ATOM = kBM * kBK * 2;            // one 128 x 64 A box
  constexpr uint32_t B_ATOM = BN * kBK * 2;             // one BN x 64 W box
  constexpr uint32_t A_BYTES = AT * MT * A_ATOM;        // [atom][M tile] A boxes
  constexpr uint32_t STAGE_BYTES = AT * (MT * A_ATOM + B_ATOM);   // [A boxes][W atoms]
  constexpr int TMEM_COLS = tmem_alloc_cols(MT * BN);
  static_assert(MT * BN <= 512 && BN % 16 == 0 && BN <= 256, "a 128 x BN MMA and its accumulators");
  static_assert(MT == 1 || EPI == EPI_HEAD, "two M tiles per CTA only for the LM-head records");
  static_assert(kEpiWarps * 32 * 68 * 4 <= STAGES * STAGE_BYTES &&
                    kBM * (BN + 4) * 4 <= STAGES * STAGE_BYTES,
                "epilogue blocks and split partials live in the idle pipeline stages");
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // 1024-byte alignment for the 128B swizzle pattern
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
  // bars[0..S): full, bars[S..2S): empty, bars[2S]: accumulator ready
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 1);
  int* s_flag = reinterpret_cast<int*>(tmem_slot + 1);
  EpiMeta* meta = reinterpret_cast<EpiMeta*>(smem + STAGES * STAGE_BYTES + 256);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_tile = blockIdx.x, m_tile = blockIdx.y, split = blockIdx.z;
  const int n0 = n_tile * BN, m0 = m_tile * kBM * MT;
  const int kb_total = g.K / kBK;
  const int kb0 = split * g.kb_per_split;
  const int kb1 = min(kb_total, kb0 + g.kb_per_split);
  const int nkb = kb1 - kb0;                  // K atoms of this split
  const int nst = (nkb + AT - 1) / AT;        // pipeline stages (the last may be short)

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
                 "r"(TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;

  // Producers: warp 0 and, for stages of several boxes, the last epilogue
  // warps (idle until the accumulator is ready) each issue their share of a
  // stage's TMA boxes.  One thread issues about one copy per 250 ns whatever
  // its size, so copies from one thread cap the operand stream; warps issue
  // side by side.  Box j of a stage: K atom j / (MT + 1); A box (M half
  // j % (MT + 1)) or, for the last one, the W box.  Warp 0 arms each stage's
  // barrier.  Weights are constant during a step: the first stages' W boxes
  // stream in while the predecessor kernel finishes; the A boxes it produces
  // are loaded after pdl_wait.
  constexpr int NBOX = AT * (MT + 1);
  constexpr int NPW = NBOX < 4 ? NBOX : 4;
  const int pw = warp == 0 ? 0 : (warp > kThreads / 32 - NPW ? kThreads / 32 - warp : -1);
  if (pw >= 0) {
    if (lane == 0) {
      const int pre = min(nst, STAGES);
      if (pw == 0 && g.l2_next) {
        // this CTA's share of the next projection's weights, into L2 for the
        // kernel after this one (256-byte slices, one prefetch each of at
        // most 1 MiB)
        const unsigned long long nct = (unsigned long long)gridDim.x * gridDim.y * gridDim.z;
        const unsigned long long cta = ((unsigned long long)blockIdx.z * gridDim.y + blockIdx.y) * gridDim.x + blockIdx.x;
        const unsigned long long per = ((g.l2_bytes + nct - 1) / nct + 255) & ~255ull;
        for (unsigned long long o = cta * per; o < min(g.l2_bytes, (cta + 1) * per); o += (1u << 20)) {
          const unsigned long long n = min(min((unsigned long long)(1u << 20), (cta + 1) * per - o), g.l2_bytes - o);
          prefetch_l2(g.l2_next + o, (uint32_t)(n & ~15ull));
        }
      }
      // the boxes of stage i that this warp issues: W (w = true) or A boxes
      auto issue = [&](int i, uint32_t sa, uint32_t full, bool w_boxes) {
        const int na = min(AT, nkb - i * AT);
        for (int j = pw; j < na * (MT + 1); j += NPW) {
          const int a = j / (MT + 1), r = j % (MT + 1);
          const int kc = (kb0 + i * AT + a) * kBK;
          if (r == MT && w_boxes) tma_load_2d(sa + A_BYTES + a * B_ATOM, &map_w, full, kc, n0);
          if (r < MT && !w_boxes) tma_load_2d(sa + (a * MT + r) * A_ATOM, &map_a, full, kc, m0 + r * kBM);
        }
      };
      for (int i = 0; i < pre; ++i) {
        const uint32_t full = smem_u32(&bars[i]);
        if (pw == 0) mbar_expect_tx(full, min(AT, nkb - i * AT) * (MT * g.a_box + B_ATOM));
        issue(i, smem_u32(smem + i * STAGE_BYTES), full, true);
      }
      pdl_wait();
      for (int i = 0; i < pre; ++i) issue(i, smem_u32(smem + i * STAGE_BYTES), smem_u32(&bars[i]), false);
      for (int i = pre; i < nst; ++i) {
        const int s = i % STAGES;
        const uint32_t ph = (i / STAGES) & 1;
        if (!mbar_wait(smem_u32(&bars[STAGES + s]), ph ^ 1, g.d_err)) break;
        const uint32_t full = smem_u32(&bars[s]);
        if (pw == 0) mbar_expect_tx(full, min(AT, nkb - i * AT) * (MT * g.a_box + B_ATOM));
        const uint32_t sa = smem_u32(smem + s * STAGE_BYTES);
        issue(i, sa, full, true);
        issue(i, sa, full, false);
      }
    }
    __syncwarp();
  }
  if (warp == 0) {
    // producer only
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16(kBM, BN);
      bool ok = true;
      for (int i = 0; i < nst; ++i) {
        const int s = i % STAGES;
        const uint32_t ph = (i / STAGES) & 1;
        if (!mbar_wait(smem_u32(&bars[s]), ph, g.d_err)) { ok = false; break; }
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t sa = smem_u32(smem + s * STAGE_BYTES);
        const uint32_t sb = sa + A_BYTES;
        const int na = min(AT, nkb - i * AT);
#pragma unroll
        for (int a = 0; a < AT; ++a) {
          if (a < na) {
#pragma unroll
            for (int kk = 0; kk < kBK / 16; ++kk)
#pragma unroll
              for (int mh = 0; mh < MT; ++mh)
                mma_bf16(tmem + mh * BN, sdesc(sa + (a * MT + mh) * A_ATOM + kk * 32),
                         sdesc(sb + a * B_ATOM + kk * 32), idesc, (i > 0 || a > 0 || kk > 0) ? 1u : 0u);
          }
        }
        mma_commit(smem_u32(&bars[STAGES + s]));
      }
      if (ok) mma_commit(smem_u32(&bars[2 * STAGES]));
    }
  } else {
    const int quarter = warp & 3;                 // TMEM lanes 32*quarter .. +31
    const int ch = (warp - 2) >> 2;               // which warp of the quarter
    const int et = threadIdx.x - 64;              // 0 .. 32*kEpiWarps-1
    pdl_wait();
    // the tile's per-row data, while the mainloop runs
    if (et < kBM) fill_meta<EPI>(meta, g, m0, et);
    const int rbase = m0 + quarter * 32;
    const bool active = rbase < g.M;          // warp-uniform
    // the per-row data of the warp's first block, before the accumulator is
    // ready (QKV: after the positions above are published)
    EpiRows<BN, EPI> rows;
    const bool vec = EPI != EPI_HEAD && g.splits == 1 && active;
    if (EPI == EPI_QKV) epi_bar();
    if (vec) epi_rows_load<BN, EPI>(rows, g, meta, m0, n0, quarter, ch, lane, epi_first_block<BN>(ch));
    // one waiter, result broadcast: every epilogue thread takes the same path
    if (et == 0) s_flag[1] = mbar_wait(smem_u32(&bars[2 * STAGES]), 0, g.d_err) ? 1 : 0;
    epi_bar();
    const bool ready = s_flag[1] != 0;
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t lane_addr = tmem + ((uint32_t)(quarter * 32) << 16);
    if (ready && active) {
      if (g.splits > 1) {
        // this split's partial: rows of the tile in the CTA's own shared
        // memory (pitch BN + 4), reduced across the cluster below; the two
        // warps of a quarter write alternate halves of the columns
        float* P = reinterpret_cast<float*>(smem) + (size_t)(quarter * 32 + lane) * (BN + 4);
#pragma unroll 1
        for (int c = ch * (BN / 2); c < (ch + 1) * (BN / 2); c += 32) {
          float v[32];
          tmem_ld32(lane_addr + c, v);
#pragma unroll
          for (int q = 0; q < 8; ++q)
            *reinterpret_cast<float4*>(P + c + 4 * q) =
                make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
        }
      } else if (EPI == EPI_HEAD) {
        // row mode: a thread reduces its row's 32-id chunks; with two M
        // tiles the warps of a quarter take one accumulator each, else
        // alternate halves of the tile's columns
        const int row = rbase + (MT == 2 ? ch * kBM : 0) + lane;
        const int c0 = MT == 2 ? 0 : ch * (BN / 2), c1 = MT == 2 ? BN : (ch + 1) * (BN / 2);
        const uint32_t acc_addr = lane_addr + (MT == 2 ? ch * BN : 0);
#pragma unroll 1
        for (int c = c0; c < c1; c += 32) {
          float v[32];
          tmem_ld32(acc_addr + c, v);
          if (row < g.M && n0 + c < g.N) epi_run32<__nv_bfloat16>(g.epi, row, n0 + c, v, g.N);
        }
      } else {
        // per epilogue warp a 32 x 68 fp32 block in the idle pipeline stages
        epi_vec_tile<BN, EPI>(g, meta, reinterpret_cast<float*>(smem) + (warp - 2) * (32 * 68), lane_addr, m0, n0,
                              quarter, ch, lane, rows);
      }
    }
  }
  if (g.splits > 1) {
    // split-K across the cluster (one CTA per split): partials wait in each
    // CTA's shared memory; CTA q then reduces rows q, q + S, ... of the tile
    // over DSMEM, adding the splits in order (deterministic), and runs the
    // epilogue on them.  Every thread of every CTA takes both barriers.
    cluster_sync();
    if (EPI == EPI_QKV && warp >= 2) {
      // QKV: RoPE rotates columns (i, i + 32) of each 64-wide head block, so a
      // thread takes four columns of the block's first half and the same
      // four of its second half
      constexpr int GQ = BN / 8;                   // (block, 4-column group) pairs per row
      const int S = g.splits;
      const int q = (int)cluster_rank();
      const int et = threadIdx.x - 64;
      const int items = ((kBM - q + S - 1) / S) * GQ;
      const uint32_t pbase = smem_u32(smem);
      for (int idx = et; idx < items; idx += 32 * kEpiWarps) {
        const int rr = q + S * (idx / GQ);
        const int pr = idx % GQ;
        const int blk = (pr / 8) * 64, g4 = (pr % 8) * 4;
        const int row = m0 + rr;
        if (row >= g.M || n0 + blk >= g.N) continue;
        float4 lo = make_float4(0.f, 0.f, 0.f, 0.f), hi = lo;
        const uint32_t off = (uint32_t)((rr * (BN + 4) + blk + g4) * 4);
        for (int sp = 0; sp < S; ++sp) {
          const float4 a = ld_dsmem4(pbase + off, (uint32_t)sp);
          const float4 b = ld_dsmem4(pbase + off + 32 * 4, (uint32_t)sp);
          lo.x += a.x; lo.y += a.y; lo.z += a.z; lo.w += a.w;
          hi.x += b.x; hi.y += b.y; hi.z += b.z; hi.w += b.w;
        }
        if (g.epi.ss_in) {
          lo = scale4(lo, meta->rinv[rr]);
          hi = scale4(hi, meta->rinv[rr]);
        }
        epi_qkv<__nv_bfloat16>(g.epi, row, meta->pos[rr], meta->aux[rr], n0 + blk, g4, lo, hi);
      }
    } else if (warp >= 2) {
      // this CTA's rows q, q + S, ...: each thread takes U groups of four
      // columns at a time and issues all their DSMEM loads before the
      // epilogue stores, so the latencies overlap
      constexpr int U = 4;
      constexpr int GROUPS = BN / 4;               // float4 groups per row
      const int S = g.splits;
      const int q = (int)cluster_rank();
      const int et = threadIdx.x - 64;
      const int rows_mine = (kBM - q + S - 1) / S;
      const int items = rows_mine * GROUPS;
      const uint32_t pbase = smem_u32(smem);
      // warp-uniform trip count (the butterflies below need every lane)
      for (int it0 = et - (et & 31); it0 < items; it0 += 32 * kEpiWarps * U) {
        float4 acc[U];
        int row[U], gcol[U];
        bool ok[U];
        uint32_t off[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
          const int idx = it0 + (et & 31) + u * 32 * kEpiWarps;
          const int rr = q + S * (idx / GROUPS);
          gcol[u] = (idx % GROUPS) * 4;
          row[u] = m0 + rr;
          ok[u] = idx < items && row[u] < g.M;
          off[u] = (uint32_t)((rr * (BN + 4) + gcol[u]) * 4);
          acc[u] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
        float4 xo[EPI == EPI_RESID ? U : 1];
        if (EPI == EPI_RESID) {
#pragma unroll
          for (int u = 0; u < U; ++u)
            xo[u] = (ok[u] && n0 + gcol[u] < g.N) ? *reinterpret_cast<const float4*>(g.epi.x + (size_t)row[u] * g.epi.ldx + n0 + gcol[u])
                          : make_float4(0.f, 0.f, 0.f, 0.f);
        }
        for (int sp = 0; sp < S; ++sp) {
#pragma unroll
          for (int u = 0; u < U; ++u) {
            if (ok[u]) {
              const float4 v = ld_dsmem4(pbase + off[u], (uint32_t)sp);
              acc[u].x += v.x; acc[u].y += v.y; acc[u].z += v.z; acc[u].w += v.w;
            }
          }
        }
        if (EPI != EPI_HEAD && EPI != EPI_QKV) {   // the LM-head records never split; QKV above
#pragma unroll
          for (int u = 0; u < U; ++u) {
            if (EPI == EPI_BIAS_GELU && ok[u] && g.epi.ss_in) acc[u] = scale4(acc[u], meta->rinv[row[u] - m0]);
            float sq = 0.f;
            if (EPI == EPI_RESID) {
              if (ok[u] && n0 + gcol[u] < g.N) sq = epi_resid4<__nv_bfloat16>(g.epi, row[u], n0 + gcol[u], acc[u], xo[u]);
            } else {
              sq = ok[u] ? epi_vec4<__nv_bfloat16, EPI>(g.epi, row[u], n0 + gcol[u], acc[u], g.N) : 0.f;
            }
            if ((EPI == EPI_RESID || EPI == EPI_NOISE_OUT) && g.epi.ss_out) {
              // 16 consecutive lanes hold one row's 64-column slot
              sq += __shfl_xor_sync(0xffffffffu, sq, 1);
              sq += __shfl_xor_sync(0xffffffffu, sq, 2);
              sq += __shfl_xor_sync(0xffffffffu, sq, 4);
              sq += __shfl_xor_sync(0xffffffffu, sq, 8);
              if (ok[u] && (et & 15) == 0) {
                const int xr = (EPI == EPI_NOISE_OUT) ? g.epi.row_map[row[u]] : row[u];
                g.epi.ss_out[(size_t)xr * g.epi.nslot + (n0 + gcol[u]) / 64] = sq;
              }
            }
          }
        }
      }
    }
    cluster_sync();
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  if (warp == 1)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TMEM_COLS)
                 : "memory");
}

// ------------------------------------------------------------ persistent tiles
// For products of more than one wave of tiles: one CTA per SM takes tiles
// blockIdx.x, blockIdx.x + gridDim.x, ... in M-tile-major order (neighbouring
// CTAs share an A row block in L2).  The producer streams one 64-wide K atom
// of A and W per pipeline stage through the whole tile sequence; two TMEM
// accumulators (2 BN columns) let the MMA warp run tile i+1's mainloop while
// the epilogue warps drain tile i from the other one, so each CTA's tiles
// cost about one mainloop each instead of a mainloop plus an epilogue.  The
// epilogue stages through its own shared memory (the ring stays busy).
template <int BN, int STAGES, int EPI>
__global__ void __launch_bounds__(kPersistWarps * 32, 1)
k_gemm_tc_persist(const __grid_constant__ CUtensorMap map_a, const __grid_constant__ CUtensorMap map_w,
                  TcArgs g) {
  constexpr uint32_t A_ATOM = kBM * kBK * 2;
  constexpr uint32_t B_ATOM = BN * kBK * 2;
  constexpr uint32_t STAGE_BYTES = A_ATOM + B_ATOM;
  constexpr uint32_t STG_BYTES = kEpiWarps * 32 * 68 * 4;
  constexpr int TMEM_COLS = tmem_alloc_cols(2 * BN);
  // tile order: M-tile-major (neighbouring CTAs share an A row block), or
  // for the LM-head records N-tile-major (the M tiles of one weight tile run
  // side by side, so each weight tile is read from HBM once)
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  float* stg = reinterpret_cast<float*>(smem + STAGES * STAGE_BYTES);
  EpiMeta* meta = reinterpret_cast<EpiMeta*>(smem + STAGES * STAGE_BYTES + STG_BYTES);
  uint64_t* bars = reinterpret_cast<uint64_t*>(meta + 1);
  // bars[0..S): full, [S..2S): empty, [2S..2S+2): accumulator full, [2S+2..2S+4): accumulator empty
  uint64_t* full = bars;
  uint64_t* empty = bars + STAGES;
  uint64_t* accf = bars + 2 * STAGES;
  uint64_t* acce = accf + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acce + 2);
  int* s_flag = reinterpret_cast<int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_tiles = ceil_div(g.N, BN), m_tiles = ceil_div(g.M, kBM), tiles = n_tiles * m_tiles;
  auto tile_m0 = [&](int t) { return (EPI == EPI_HEAD ? t % m_tiles : t / n_tiles) * kBM; };
  auto tile_n0 = [&](int t) { return (EPI == EPI_HEAD ? t / m_tiles : t % n_tiles) * BN; };
  const int nkb = g.K / kBK;
  if (threadIdx.x == 0) {
    for (int i = 0; i < STAGES; ++i) {
      mbar_init(smem_u32(&full[i]), 1);
      mbar_init(smem_u32(&empty[i]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&accf[i]), 1);
      mbar_init(smem_u32(&acce[i]), 1);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_a)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_w)) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;

  if (warp == 0 || warp == kPersistWarps - 1) {
    // two producers issue side by side (one thread issues about one TMA copy
    // per 250 ns): warp 0 arms each stage's barrier and loads its A box, the
    // last warp loads its W box.  The first tile's W boxes stream in while the
    // predecessor kernel finishes.
    if (lane == 0) {
      const bool wp = warp != 0;
      uint32_t stage = 0;
      bool first = true;
      for (int t = blockIdx.x; t < tiles; t += gridDim.x) {
        const int m0 = tile_m0(t), n0 = tile_n0(t);
        int i0 = 0;
        if (first) {
          const int pre = min(nkb, STAGES);
          for (int i = 0; i < pre; ++i) {
            if (!wp) mbar_expect_tx(smem_u32(&full[i]), g.a_box + B_ATOM);
            else tma_load_2d(smem_u32(smem + i * STAGE_BYTES) + A_ATOM, &map_w, smem_u32(&full[i]), i * kBK, n0);
          }
          if (!wp) {
            pdl_wait();
            for (int i = 0; i < pre; ++i)
              tma_load_2d(smem_u32(smem + i * STAGE_BYTES), &map_a, smem_u32(&full[i]), i * kBK, m0);
          }
          i0 = pre;
          first = false;
        }
        bool live = true;
        for (int i = i0; i < nkb; ++i) {
          const uint32_t sc = stage + i, s = sc % STAGES;
          if (!mbar_wait(smem_u32(&empty[s]), ((sc / STAGES) & 1) ^ 1, g.d_err)) {
            live = false;
            break;
          }
          const uint32_t fb = smem_u32(&full[s]);
          const uint32_t sa = smem_u32(smem + s * STAGE_BYTES);
          if (!wp) {
            mbar_expect_tx(fb, g.a_box + B_ATOM);
            tma_load_2d(sa, &map_a, fb, i * kBK, m0);
          } else {
            tma_load_2d(sa + A_ATOM, &map_w, fb, i * kBK, n0);
          }
        }
        if (!live) break;
        stage += nkb;
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16(kBM, BN);
      uint32_t stage = 0, ti = 0;
      bool ok = true;   // a timed-out wait ends this CTA's tiles
      for (int t = blockIdx.x; ok && t < tiles; t += gridDim.x, ++ti) {
        const uint32_t buf = ti & 1;
        if (!mbar_wait(smem_u32(&acce[buf]), ((ti >> 1) & 1) ^ 1, g.d_err)) break;
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t d = tmem + buf * BN;
        for (int i = 0; i < nkb; ++i, ++stage) {
          const uint32_t s = stage % STAGES;
          if (!mbar_wait(smem_u32(&full[s]), (stage / STAGES) & 1, g.d_err)) {
            ok = false;
            break;
          }
          asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
          const uint32_t sa = smem_u32(smem + s * STAGE_BYTES);
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk)
            mma_bf16(d, sdesc(sa + kk * 32), sdesc(sa + A_ATOM + kk * 32), idesc, (i > 0 || kk > 0) ? 1u : 0u);
          mma_commit(smem_u32(&empty[s]));
        }
        if (ok) mma_commit(smem_u32(&accf[buf]));
      }
    }
  } else {
    const int quarter = warp & 3;
    const int ch = (warp - 2) >> 2;
    const int et = threadIdx.x - 64;
    pdl_wait();
    uint32_t ti = 0;   // epilogue warps 2 .. kEpiWarps + 1
    for (int t = blockIdx.x; t < tiles; t += gridDim.x, ++ti) {
      const uint32_t buf = ti & 1;
      const int m0 = tile_m0(t), n0 = tile_n0(t);
      // the tile's per-row data while its mainloop runs
      if (et < kBM) fill_meta<EPI>(meta, g, m0, et);
      // the first block's per-row data before the accumulator is ready
      const bool active = m0 + quarter * 32 < g.M;   // warp-uniform
      EpiRows<BN, EPI> rows;
      if (EPI == EPI_QKV) epi_bar();
      if (active) epi_rows_load<BN, EPI>(rows, g, meta, m0, n0, quarter, ch, lane, epi_first_block<BN>(ch));
      if (et == 0) s_flag[0] = mbar_wait(smem_u32(&accf[buf]), (ti >> 1) & 1, g.d_err) ? 1 : 0;
      epi_bar();
      if (!s_flag[0]) break;   // timed out: the MMA warp has stopped too
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const uint32_t lane_addr = tmem + buf * BN + ((uint32_t)(quarter * 32) << 16);
      if (EPI == EPI_HEAD) {
        // row mode: a thread reduces its row's 32-id chunks, the two warps of
        // a quarter alternate halves of the tile's columns
        const int r = m0 + quarter * 32 + lane;
#pragma unroll 1
        for (int c = ch * (BN / 2); c < (ch + 1) * (BN / 2); c += 32) {
          float v[32];
          tmem_ld32(lane_addr + c, v);
          if (r < g.M && n0 + c < g.N) epi_run32<__nv_bfloat16>(g.epi, r, n0 + c, v, g.N);
        }
      } else if (active) {
        epi_vec_tile<BN, EPI>(g, meta, stg + (warp - 2) * (32 * 68), lane_addr, m0, n0, quarter, ch, lane, rows);
      }
      // every warp has read the accumulator: the MMA warp may refill it
      asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
      epi_bar();
      if (et == 0)
        asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0];" ::"r"(smem_u32(&acce[buf])) : "memory");
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  if (warp == 1)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TMEM_COLS)
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

// a K-major bf16 operand [rows][cols] (row pitch ld) read in boxes of 64
// columns x box_rows rows, 128-byte swizzle (the skinny projections)
bool encode_kmajor_bf16(CUtensorMap* m, const void* ptr, int rows, int cols, int ld, int box_rows) {
  return get_encode() && make_map(m, ptr, rows, cols, ld, box_rows);
}

bool encode_rows_map_bf16(CUtensorMap* m, const void* base, uint64_t rows, int cols, int box_rows) {
  if (!get_encode() || (reinterpret_cast<uintptr_t>(base) & 15) || (cols * 2) % 16) return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  cuuint32_t box[2] = {(cuuint32_t)cols, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  return g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
                  estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_map_bf16(CUtensorMap* m, const void* base, int rank, const uint64_t* dims, const uint64_t* strides,
                     const uint32_t* box) {
  if (!get_encode() || rank < 1 || rank > 5 || (reinterpret_cast<uintptr_t>(base) & 15) || box[0] * 2 > 128)
    return false;
  cuuint64_t d[5], st[4];
  cuuint32_t bx[5], es[5];
  for (int i = 0; i < rank; ++i) {
    d[i] = dims[i];
    bx[i] = box[i];
    es[i] = 1;
    if (i > 0) {
      if (strides[i - 1] % 16) return false;
      st[i - 1] = strides[i - 1];
    }
  }
  return g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(base), d, st, bx, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool tc_gemm_supported(const GemmDesc& g) {
  if (g.K % kBK || g.K == 0 || g.M <= 0 || g.N <= 0) return false;
  if ((g.lda * 2) % 16 || (g.ldw * 2) % 16) return false;
  if ((reinterpret_cast<uintptr_t>(g.A) & 15) || (reinterpret_cast<uintptr_t>(g.W) & 15)) return false;
  // the vector epilogues write groups of 4 columns (the LM-head records reduce
  // runs of 32 columns per row and take any N)
  const int k = g.epi.kind;
  if (k != EPI_HEAD && g.N % 4) return false;
  if ((k == EPI_STORE || k == EPI_STORE_F32 || k == EPI_BIAS_GELU) && g.epi.ldo % 4) return false;
  if ((k == EPI_RESID || k == EPI_NOISE_OUT) && g.epi.ldx % 4) return false;
  if (k == EPI_QKV && (g.N % 64 || g.epi.dsec % 64)) return false;
  return get_encode();
}

template <int BN, int STAGES, int EPI, int MT = 1, int AT = 2>
static int launch_epi(const GemmDesc& g, int* d_err, int num_sms, cudaStream_t s) {
  const int n_tiles = ceil_div(g.N, BN), m_tiles = ceil_div(g.M, kBM * MT);
  const int tiles = n_tiles * m_tiles;
  const int kb_total = g.K / kBK;
  // split K over a cluster of up to 8 CTAs when the tiles alone leave SMs
  // idle: the largest power of two that keeps one wave and two K blocks per
  // split (odd cluster sizes measured slower)
  // (QKV only within one M tile: at 256 rows its 2-way split measured slower)
  int splits = 1;
  if (EPI != EPI_HEAD && (EPI != EPI_QKV || m_tiles == 1))
    while (splits < 8 && tiles * splits * 2 <= num_sms && kb_total >= splits * 4) splits *= 2;
  int kbps = ceil_div(kb_total, splits);
  splits = ceil_div(kb_total, kbps);   // no empty splits
  const size_t smem = (size_t)STAGES * AT * (MT * kBM * kBK * 2 + BN * kBK * 2) + 1024 + 256 + sizeof(EpiMeta);
  static PerDevice attr, cluster;
  set_smem_attr(attr, k_gemm_tc<BN, STAGES, EPI, MT, AT>, smem);
  // the largest cluster of these CTAs that fits on one GPC of this device
  const int max_cluster = (int)per_device(cluster, [&] {
    for (int cs = 8; cs > 1; --cs) {
      cudaLaunchConfig_t q = {};
      q.gridDim = dim3(1, 1, cs);
      q.blockDim = dim3(kThreads);
      q.dynamicSmemBytes = smem;
      cudaLaunchAttribute ca;
      ca.id = cudaLaunchAttributeClusterDimension;
      ca.val.clusterDim.x = 1; ca.val.clusterDim.y = 1; ca.val.clusterDim.z = cs;
      q.attrs = &ca;
      q.numAttrs = 1;
      int n = 0;
      if (cudaOccupancyMaxActiveClusters(&n, k_gemm_tc<BN, STAGES, EPI, MT, AT>, &q) == cudaSuccess && n > 0)
        return (long long)cs;
      cudaGetLastError();
    }
    return 1ll;
  });
  if (splits > max_cluster) {
    splits = max_cluster;
    kbps = ceil_div(kb_total, splits);
    splits = ceil_div(kb_total, kbps);
  }
  // A boxes cover only the rows a tile can hold: at M <= 128 the 128-row MMA
  // reads the rows past the box from stale shared memory, and those rows of
  // the accumulator (all >= M) are never stored
  const int a_rows = MT == 1 ? std::min(kBM, round_up(g.M, 8)) : kBM;
  CUtensorMap ma, mw;
  if (!make_map(&ma, g.A, g.M, g.K, g.lda, a_rows) || !make_map(&mw, g.W, g.N, g.K, g.ldw, BN))
    return -1;
  TcArgs a;
  a.M = g.M; a.N = g.N; a.K = g.K; a.kb_per_split = kbps; a.splits = splits;
  a.a_box = (uint32_t)a_rows * kBK * 2;
  const bool pf = g.l2_next && g.l2_bytes >= 16 && !(reinterpret_cast<uintptr_t>(g.l2_next) & 15);
  a.l2_next = pf ? static_cast<const char*>(g.l2_next) : nullptr;
  a.l2_bytes = pf ? (g.l2_bytes & ~(size_t)15) : 0;
  a.d_err = d_err; a.epi = g.epi;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(n_tiles, m_tiles, splits);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[2];
  int na = 0;
  if (splits > 1) {
    at[na].id = cudaLaunchAttributeClusterDimension;
    at[na].val.clusterDim.x = 1;
    at[na].val.clusterDim.y = 1;
    at[na].val.clusterDim.z = splits;
    ++na;
  }
  if (g_pdl) {
    at[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  cfg.attrs = at;
  cfg.numAttrs = na;
  return cudaLaunchKernelEx(&cfg, k_gemm_tc<BN, STAGES, EPI, MT, AT>, ma, mw, a) == cudaSuccess ? 0 : -1;
}

template <int BN, int STAGES, int EPI>
static int launch_persist_epi(const GemmDesc& g, int* d_err, int num_sms, cudaStream_t s) {
  const int tiles = ceil_div(g.N, BN) * ceil_div(g.M, kBM);
  const size_t smem = (size_t)STAGES * (kBM * kBK * 2 + BN * kBK * 2) + kEpiWarps * 32 * 68 * 4 +
                      sizeof(EpiMeta) + 1024 + 128;
  static PerDevice attr;
  set_smem_attr(attr, k_gemm_tc_persist<BN, STAGES, EPI>, smem);
  const int a_rows = std::min(kBM, round_up(g.M, 8));
  CUtensorMap ma, mw;
  if (!make_map(&ma, g.A, g.M, g.K, g.lda, a_rows) || !make_map(&mw, g.W, g.N, g.K, g.ldw, BN)) return -1;
  TcArgs a;
  a.M = g.M; a.N = g.N; a.K = g.K; a.kb_per_split = g.K / kBK; a.splits = 1;
  a.a_box = (uint32_t)a_rows * kBK * 2;
  a.l2_next = nullptr; a.l2_bytes = 0;
  a.d_err = d_err; a.epi = g.epi;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(std::min(tiles, num_sms));
  cfg.blockDim = dim3(kPersistWarps * 32);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = g_pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, k_gemm_tc_persist<BN, STAGES, EPI>, ma, mw, a) == cudaSuccess ? 0 : -1;
}

template <int BN, int STAGES>
static int launch_persist(const GemmDesc& g, int* d_err, int num_sms, cudaStream_t s) {
  switch (g.epi.kind) {
    case EPI_STORE: return launch_persist_epi<BN, STAGES, EPI_STORE>(g, d_err, num_sms, s);
    case EPI_BIAS_GELU: return launch_persist_epi<BN, STAGES, EPI_BIAS_GELU>(g, d_err, num_sms, s);
    case EPI_RESID: return launch_persist_epi<BN, STAGES, EPI_RESID>(g, d_err, num_sms, s);
    case EPI_NOISE_OUT: return launch_persist_epi<BN, STAGES, EPI_NOISE_OUT>(g, d_err, num_sms, s);
    case EPI_LOGITS: return launch_persist_epi<BN, STAGES, EPI_LOGITS>(g, d_err, num_sms, s);
    case EPI_STORE_F32: return launch_persist_epi<BN, STAGES, EPI_STORE_F32>(g, d_err, num_sms, s);
    case EPI_QKV: return launch_persist_epi<BN, STAGES, EPI_QKV>(g, d_err, num_sms, s);
    case EPI_HEAD: return launch_persist_epi<BN, STAGES, EPI_HEAD>(g, d_err, num_sms, s);
  }
  return -1;
}

template <int BN, int STAGES, int AT>
static int launch_bn(const GemmDesc& g, int* d_err, int num_sms, cudaStream_t s) {
  switch (g.epi.kind) {
    case EPI_STORE: return launch_epi<BN, STAGES, EPI_STORE, 1, AT>(g, d_err, num_sms, s);
    case EPI_BIAS_GELU: return launch_epi<BN, STAGES, EPI_BIAS_GELU, 1, AT>(g, d_err, num_sms, s);
    case EPI_RESID: return launch_epi<BN, STAGES, EPI_RESID, 1, AT>(g, d_err, num_sms, s);
    case EPI_NOISE_OUT: return launch_epi<BN, STAGES, EPI_NOISE_OUT, 1, AT>(g, d_err, num_sms, s);
    case EPI_LOGITS: return launch_epi<BN, STAGES, EPI_LOGITS, 1, AT>(g, d_err, num_sms, s);
    case EPI_STORE_F32: return launch_epi<BN, STAGES, EPI_STORE_F32, 1, AT>(g, d_err, num_sms, s);
    case EPI_QKV: return launch_epi<BN, STAGES, EPI_QKV, 1, AT>(g, d_err, num_sms, s);
  }
  return -1;
}

int launch_gemm_tc(const GemmDesc& g, int* d_err, cudaStream_t s) {
  const int num_sms = device_sms();
  // LM-head records: 256-wide tiles; above 128 rows both M tiles of a row
  // pair in one CTA (each weight tile is streamed from HBM once per 256 rows)
  if (g.epi.kind == EPI_HEAD) {
    // above one M tile, more than a wave of 128 x 256 tiles: a persistent
    // loop, the M tiles of each weight tile side by side (the weights are read
    // from HBM once) and each tile's records overlapping the next tile's
    // mainloop
    if (g.M > kBM && !(g_gemm_flags & kGemmNoPersist) && ceil_div(g.N, 256) * ceil_div(g.M, kBM) > num_sms)
      return launch_persist<256, 3>(g, d_err, num_sms, s);
    if (g.M > kBM) return launch_epi<256, 3, EPI_HEAD, 2, 1>(g, d_err, num_sms, s);
    // one M tile, more than a wave of 256-wide tiles (the OWT-shaped vocab:
    // 197 tiles on 152 SMs left a second wave of 45): a persistent loop over
    // 128-wide tiles keeps every SM streaming weights to the end (batch 1,
    // k = 4: 309.5 -> 303.8 us per call)
    if (!(g_gemm_flags & kGemmNoPersist) && ceil_div(g.N, 256) > num_sms)
      return launch_persist_epi<128, 4, EPI_HEAD>(g, d_err, num_sms, s);
    return launch_epi<256, 2, EPI_HEAD, 1, 2>(g, d_err, num_sms, s);
  }
  // the narrowest tile that covers the product in one wave, else 256-wide
  // tiles: a tcgen05.mma re-reads its whole 128-row A operand from shared
  // memory for every BN columns, so wider tiles move fewer operand bytes per
  // flop, while narrower ones spread a small product over more SMs
  const int m_tiles = ceil_div(g.M, kBM);
  // A deep K that is split over a cluster anyway: 128-wide tiles halve the
  // K atoms each CTA streams (LM1B-shaped MLP-down, 512 x 768 x 3072: split-K
  // 4 over 24 tiles instead of 2 over 48, 9% faster; the O projection with
  // K = 768 is faster as it is)
  const bool deep_split = g.K >= 2048 && g.epi.kind != EPI_QKV &&
                          ceil_div(g.N, 64) * m_tiles * 4 > num_sms &&      // 64-wide: split 2 at most
                          ceil_div(g.N, 128) * m_tiles * 4 <= num_sms;      // 128-wide: split 4
  if (deep_split) return launch_bn<128, 3, 2>(g, d_err, num_sms, s);
  if (ceil_div(g.N, 64) * m_tiles <= num_sms) return launch_bn<64, 4, 2>(g, d_err, num_sms, s);
  if (ceil_div(g.N, 128) * m_tiles <= num_sms) return launch_bn<128, 3, 2>(g, d_err, num_sms, s);
  // More than a wave of 256-wide tiles: a persistent loop whose epilogues
  // overlap the next tile's mainloop (OWT-shaped batch 512, k = 4: QKV 35.1 ->
  // 30.1 us, MLP-up 38.2 -> 30.7 us per layer).  Within one wave a CTA per
  // tile keeps a fourth pipeline stage and has nothing to overlap.  The
  // LM-head records keep their kernel, which streams each weight tile once
  // per 256 rows.
  // One wave of 256-wide tiles that leaves SMs idle, where 192-wide tiles
  // still fit one wave: the narrower tiles (the OWT-shaped O projection and
  // MLP-down at 4096 rows: 128 CTAs of 128 x 192 instead of 96 of 128 x 256;
  // each streams 17 % fewer bytes per CTA).  (Persistent 128-wide tiles for
  // those two, 192 tiles on 152 SMs, were 1.3-1.6x slower: a 128 x 128 tile
  // streams twice the A bytes per flop, and the stream is the limit.)
  if (ceil_div(g.N, 256) * m_tiles <= num_sms && ceil_div(g.N, 192) * m_tiles <= num_sms &&
      ceil_div(g.N, 192) > ceil_div(g.N, 256))
    return launch_bn<192, 5, 1>(g, d_err, num_sms, s);
  if (g.epi.kind != EPI_HEAD && !(g_gemm_flags & kGemmNoPersist) && ceil_div(g.N, 256) * m_tiles > num_sms)
    return launch_persist<256, 3>(g, d_err, num_sms, s);
  return launch_bn<256, 4, 1>(g, d_err, num_sms, s);
}

}  // namespace kf
