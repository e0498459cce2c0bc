// Forward entry point that allocates nothing, for callers that cannot call
// cudaMalloc where they run attention (inference servers whose device memory
// is carved into their own pools once at start-up and may not grow, or hosts
// that drive the GPU only through the plain C interface, with no device
// allocator of their own).  The forward's scratch (per-token key
// bounds, tile descriptors and the work order) lives in a fixed-size array in
// device memory that this library owns for the lifetime of the process.
#include <cstdio>
#include <mutex>
#include <string>
#include <vector>

#include "ism_internal.cuh"

namespace {

constexpr size_t kNoAllocScratchBytes = size_t(4) << 20;  // 4 MiB per device

// The scratch itself.  Every GPU that loads the library holds one copy until
// the process exits.  In host code this name is only a host-side stand-in:
// the device address comes from cudaGetSymbolAddress below.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_mu;
std::vector<void*> g_addr;  // device address of the scratch, per device

// Looked up once per device, with that device current.
ism_status_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    ism::set_error((std::string("cudaGetDevice: ") + cudaGetErrorString(e)).c_str());
    return ISM_ERR_CUDA;
  }
  std::lock_guard<std::mutex> lk(g_mu);
  if ((int)g_addr.size() <= dev) g_addr.resize(dev + 1, nullptr);
  if (!g_addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || p == nullptr) {
      ism::set_error((std::string("cudaGetSymbolAddress(no-alloc scratch): ") + cudaGetErrorString(e)).c_str());
      return ISM_ERR_CUDA;
    }
    g_addr[dev] = p;
  }
  *out = g_addr[dev];
  return ISM_OK;
}

}  // namespace

extern "C" {

size_t ism_attn_fwd_noalloc_max_workspace(void) { return kNoAllocScratchBytes; }

ism_status_t ism_attn_fwd_noalloc(const ism_segments_t* segs, const ism_attn_shape_t* shape, const void* q,
                                  const void* k, const void* v, void* o, float* lse, ism_stream_t stream) {
  size_t need = 0;
  ism_status_t r = ism_attn_fwd_workspace_size(segs, shape, &need);
  if (r != ISM_OK) return r;  // the argument error is already described by ism_last_error()
  if (need > kNoAllocScratchBytes) {
    char msg[160];
    snprintf(msg, sizeof(msg), "this batch needs %zu bytes of scratch; the fixed no-alloc scratch holds %zu",
             need, kNoAllocScratchBytes);
    ism::set_error(msg);
    return ISM_ERR_WORKSPACE;
  }
  void* scratch = nullptr;
  r = scratch_address(&scratch);
  if (r != ISM_OK) return r;
  // Nothing in the scratch has to start at zero: the forward's layout holds
  // only the per-token key bounds, tile descriptors and work lists, and its
  // metadata pass writes every entry the attention kernel then reads.  (The
  // backward's layout also carries work counters; a forward that ever gains
  // such state must clear it here before the launch.)
  return ism_attn_fwd(segs, shape, q, k, v, o, lse, scratch, kNoAllocScratchBytes, stream);
}

}  // extern "C"
