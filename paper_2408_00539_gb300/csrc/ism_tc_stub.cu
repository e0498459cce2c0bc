// Backward on tensor cores is not built yet: the CUDA-core backward runs.
#include "ism_internal.cuh"
namespace ism {
bool tc_bwd_available() { return false; }
cudaError_t launch_tc_bwd(const AttnArgs&, int64_t, cudaStream_t) { return cudaErrorNotSupported; }
}  // namespace ism
