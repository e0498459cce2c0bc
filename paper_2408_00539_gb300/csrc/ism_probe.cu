// Bounded-wait probe: waits on an mbarrier that nothing ever signals, gives
// up after `spin_limit` polls, records the timeout in the status word and
// returns.  Exercises the same wait helper the pipelined kernels use.
#include "ism_internal.cuh"
#include "ptx.cuh"

namespace ism {
namespace {

__global__ void timeout_probe_kernel(uint32_t spin_limit, uint32_t* status) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    ptx::mbar_init(&bar, 1);
    ptx::fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    // phase 0 never completes: no thread arrives
    if (!ptx::mbar_wait(&bar, 0, spin_limit)) atomicOr(status, kStatusTimeout);
  }
  __syncthreads();
}

}  // namespace

cudaError_t launch_timeout_probe(uint32_t spin_limit, uint32_t* status, cudaStream_t st) {
  timeout_probe_kernel<<<1, 32, 0, st>>>(spin_limit, status);
  return cudaGetLastError();
}

}  // namespace ism
