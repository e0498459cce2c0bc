#include "ism_internal.cuh"
namespace ism {
bool tc_available() { return false; }
cudaError_t launch_tc_fwd(const AttnArgs&, int64_t, cudaStream_t) { return cudaErrorNotSupported; }
cudaError_t launch_tc_bwd(const AttnArgs&, int64_t, cudaStream_t) { return cudaErrorNotSupported; }
}
