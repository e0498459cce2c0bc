// e4m3 (fp8) tensor-core building block check (sm_103a, kind::f8f6f4): one
// tile product in each operand layout the e4m3 forward (fwd_pair_kernel with
// e4m3 operands, ism_fwd2_tc.cu) uses.
#include "ism_tc_common.cuh"

namespace ism {
namespace tc {
namespace {

// Byte offset of element (r, c) of a [128 x 128] 8-bit tile with 128-byte
// rows in the 128-byte swizzled layout: 16-byte chunk index XOR (row mod 8).
__host__ __device__ constexpr uint32_t swz8_offset(int r, int c) {
  return (uint32_t)r * 128u + ((((uint32_t)c >> 4) ^ ((uint32_t)r & 7u)) << 4) + ((uint32_t)c & 15u);
}

// One 128x128x128 e4m3 tile product with fp32 result (diagnostic of the
// operand layouts the e4m3 forward uses).  a [128, 128] e4m3 row-major (M x K).
//   mode 0: b is N x K (K-major), c = a * b^T
//   mode 1: b is K x N (MN-major), c = a * b
//   mode 2: as mode 1 with a in tensor memory (four e4m3 a column)
__global__ void __launch_bounds__(128, 1)
    mma_tile_e4m3_kernel(const uint8_t* A, const uint8_t* B, float* C, int mode, uint32_t* status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sa = smem;
  uint8_t* sb = smem + 16384;
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + 32768);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bar + 1);
  const int warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) {
    ptx::mbar_init(bar, 1);
    ptx::fence_mbar_init();
  }
  if (warp == 0) {
    ptx::tmem_alloc(tslot, 256);
    ptx::tmem_relinquish();
  }
  for (int i = threadIdx.x; i < 128 * 128; i += blockDim.x) {
    const int r = i >> 7, c = i & 127;
    sa[swz8_offset(r, c)] = A[i];
    sb[swz8_offset(r, c)] = B[i];  // row r of b: an N row (mode 0) or a K row (modes 1, 2)
  }
  ptx::fence_proxy_async_smem();
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tslot;
  const uint32_t lane_addr = (uint32_t)(warp * 32) << 16;
  if (mode == 2) {
    // row r of a into lane r, columns [128, 160): bytes k = 4 c .. 4 c + 3 of column c
    const int r = threadIdx.x;
    uint32_t v[32];
    for (int c = 0; c < 32; ++c) v[c] = *reinterpret_cast<const uint32_t*>(A + r * 128 + 4 * c);
    ptx::tmem_st32(tmem + lane_addr + 128, v);
    ptx::tmem_st_wait();
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
  }
  bool ok = true;
  if (warp == 0) {
    const uint32_t b_mn = mode == 0 ? 0u : 1u;
    const uint32_t idesc = ptx::idesc_e4m3_f32(128, 128, 0, b_mn);
    const uint64_t ad = ptx::smem_desc(ptx::smem_u32(sa), 16u, 1024u, ptx::kSwizzle128B);
    const uint64_t bd = ptx::smem_desc(ptx::smem_u32(sb), 16u, 1024u, ptx::kSwizzle128B);
    if (mode == 0)
      ptx::mma4_e4m3_ss_warp<2, 2>(tmem, ad, bd, idesc, 0u);
    else if (mode == 1)
      ptx::mma4_e4m3_ss_warp<2, 256>(tmem, ad, bd, idesc, 0u);
    else
      ptx::mma4_e4m3_ts_warp<8, 256>(tmem, tmem + 128, bd, idesc, 0u);
    ptx::mma_commit_warp(bar);
    ok = wait_warp(bar, 0, status);
  }
  __syncthreads();
  ptx::tc_fence_after();
  for (int c = 0; c < 4; ++c) {
    uint32_t v[32];
    ptx::tmem_ld32(tmem + lane_addr + c * 32, v);
    ptx::tmem_ld_wait();
    ptx::reg_fence(v);
    for (int i = 0; i < 32; ++i) C[threadIdx.x * 128 + c * 32 + i] = ok ? __uint_as_float(v[i]) : 0.f;
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, 256);
  }
}

}  // namespace

cudaError_t launch_mma_tile_e4m3(const void* a, const void* b, float* c, int mode, uint32_t* status, cudaStream_t st) {
  const uint32_t smem = 32768 + 64 + 1024;
  cudaError_t e = cudaFuncSetAttribute(mma_tile_e4m3_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  mma_tile_e4m3_kernel<<<1, 128, smem, st>>>(static_cast<const uint8_t*>(a), static_cast<const uint8_t*>(b), c, mode,
                                             status);
  return cudaGetLastError();
}

}  // namespace tc
}  // namespace ism
