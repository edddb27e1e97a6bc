// tcgen05 GEMM (placeholder until the kernel lands).
#include "kf_internal.cuh"

namespace kf {
bool tc_gemm_supported(const GemmDesc&) { return false; }
int launch_gemm_tc(const GemmDesc&, void*, size_t, int*, int, int*, cudaStream_t) { return -1; }
}  // namespace kf
