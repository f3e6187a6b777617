#include "tasq_internal.cuh"
namespace tasq {
cudaError_t launch_gemm_tc(const GemmArgs&, int, cudaStream_t, const char** why) {
    *why = "not built yet";
    return cudaSuccess;
}
}  // namespace tasq
