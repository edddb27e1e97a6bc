// SIMT GEMM D[M][N] = A[M][K] . W[N][K]^T with fp32 FMA accumulation in
// ascending k for every output.  Used for the fp32 model (exact-token parity
// mode) and as the independent GPU check of the tcgen05 GEMM.  A block
// computes 32 rows x 128 columns; warp w owns columns w*32..w*32+31 and lane
// l owns row l, so each thread ends with one row's run of 32 consecutive
// columns, the unit the epilogues work on.
#include "kf_internal.cuh"

namespace kf {

template <typename TA>
__global__ void __launch_bounds__(128) k_gemm_simt(GemmDesc g) {
  pdl_wait();
  __shared__ float As[32][33];          // [row][k]
  __shared__ __align__(16) float Ws[32][132];  // [k][col]
  const int row0 = blockIdx.y * 32, col0 = blockIdx.x * 128;
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const TA* A = reinterpret_cast<const TA*>(g.A);
  const TA* W = reinterpret_cast<const TA*>(g.W);
  float acc[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) acc[j] = 0.f;

  for (int k0 = 0; k0 < g.K; k0 += 32) {
    for (int i = t; i < 32 * 32; i += 128) {
      int r = i >> 5, kk = i & 31;
      int gr = row0 + r, gk = k0 + kk;
      As[r][kk] = (gr < g.M && gk < g.K) ? to_f(A[(size_t)gr * g.lda + gk]) : 0.f;
    }
    for (int i = t; i < 128 * 32; i += 128) {
      int c = i >> 5, kk = i & 31;
      int gc = col0 + c, gk = k0 + kk;
      Ws[kk][c] = (gc < g.N && gk < g.K) ? to_f(W[(size_t)gc * g.ldw + gk]) : 0.f;
    }
    __syncthreads();
#pragma unroll 4
    for (int kk = 0; kk < 32; ++kk) {
      const float a = As[lane][kk];
      const float4* wp = reinterpret_cast<const float4*>(&Ws[kk][warp * 32]);
#pragma unroll
      for (int j4 = 0; j4 < 8; ++j4) {
        float4 w = wp[j4];
        acc[4 * j4 + 0] = fmaf(a, w.x, acc[4 * j4 + 0]);
        acc[4 * j4 + 1] = fmaf(a, w.y, acc[4 * j4 + 1]);
        acc[4 * j4 + 2] = fmaf(a, w.z, acc[4 * j4 + 2]);
        acc[4 * j4 + 3] = fmaf(a, w.w, acc[4 * j4 + 3]);
      }
    }
    __syncthreads();
  }
  const int row = row0 + lane, c0 = col0 + warp * 32;
  if (row < g.M && c0 < g.N) epi_run32<TA>(g.epi, row, c0, acc, g.N);
}

void launch_gemm_simt(bool bf16, const GemmDesc& g, cudaStream_t s) {
  if (g.M == 0 || g.N == 0) return;
  dim3 grid(ceil_div(g.N, 128), ceil_div(g.M, 32));
  if (bf16) kf_launch(k_gemm_simt<__nv_bfloat16>, dim3(grid), dim3(128), 0, s, g);
  else kf_launch(k_gemm_simt<float>, dim3(grid), dim3(128), 0, s, g);
}

}  // namespace kf
