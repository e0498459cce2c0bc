// CUDA-core attention under the ISM mask: the fp32 path (and the fallback
// for head sizes the tensor-core kernels do not take).  fp32 arithmetic with
// natural-base exponentials throughout.
//
// Forward (Eq. e_ISM with softmax): one warp per query row, lanes over keys
// for the scores and over head dimensions for the output accumulator, online
// softmax over chunks of 32 keys restricted to the row's visible range
// [0, kv_end[row]).  Backward: the standard softmax-attention gradients with
// dQ accumulated per query row and dK/dV per key row (each key row walks the
// query rows that see it: those from the first row whose kv_end exceeds the
// key, to the end of the sequence, since kv_end is non-decreasing).
#include "ism_internal.cuh"

namespace ism {
namespace {

constexpr int kRowsPerTile = 128;  // must equal the tile size used for the work lists
constexpr int kWarps = 8;

__device__ __forceinline__ float ld(const float* p) { return *p; }
__device__ __forceinline__ float ld(const __nv_bfloat16* p) { return __bfloat162float(*p); }
__device__ __forceinline__ void st(float* p, float x) { *p = x; }
__device__ __forceinline__ void st(__nv_bfloat16* p, float x) { *p = __float2bfloat16_rn(x); }

__device__ __forceinline__ float warp_max(float x) {
  for (int o = 16; o > 0; o >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, o));
  return x;
}
__device__ __forceinline__ float warp_sum(float x) {
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

template <typename T, int D>
__device__ __forceinline__ float dot_row(const float* __restrict__ a_smem, const T* __restrict__ b) {
  float acc = 0.f;
#pragma unroll 8
  for (int d = 0; d < D; ++d) acc = fmaf(a_smem[d], ld(b + d), acc);
  return acc;
}

// grid: Hq * nq blocks; block: kWarps warps.  Block b handles query head
// b % Hq of the q-tile at rank b / Hq in q_order (most expensive first).
template <typename T, int D>
__global__ void __launch_bounds__(kWarps * 32) simt_fwd_kernel(AttnArgs a) {
  __shared__ float qs[kWarps][D];
  const int h = blockIdx.x % a.hq;
  const Tile w = a.qtiles[a.q_order[blockIdx.x / a.hq]];
  const int g = h / (a.hq / a.hkv);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const T* Q = (const T*)a.q;
  const T* K = (const T*)a.k;
  const T* V = (const T*)a.v;
  T* O = (T*)a.out;
  const int64_t qstride = (int64_t)a.hq * D, kstride = (int64_t)a.hkv * D;
  for (int r = warp; r < kRowsPerTile; r += kWarps) {
    const int row = w.tile * kRowsPerTile + r;
    if (row >= w.q_len) break;
    const int64_t qrow = (int64_t)w.q_base + row;
    __syncwarp();
    for (int d = lane; d < D; d += 32) qs[warp][d] = ld(Q + qrow * qstride + (int64_t)h * D + d);
    __syncwarp();
    const int ke = a.kv_end[w.kv_base + row];
    // K / V row of key p (through the page table for a paged cache)
    auto kvrow = [&](int p) -> int64_t {
      return a.pages.table ? paged_row(a.pages, w.k_base, p) : (int64_t)w.k_base + p;
    };
    float m = -INFINITY, l = 0.f;
    float acc[D / 32];
#pragma unroll
    for (int i = 0; i < D / 32; ++i) acc[i] = 0.f;
    for (int kb = 0; kb < ke; kb += 32) {
      const int key = kb + lane;
      float s = -INFINITY;
      if (key < ke) s = a.scale * dot_row<T, D>(qs[warp], K + kvrow(key) * kstride + (int64_t)g * D);
      const float mc = warp_max(s);
      const float mn = fmaxf(m, mc);
      const float alpha = (m == -INFINITY) ? 0.f : expf(m - mn);
      const float p = (key < ke) ? expf(s - mn) : 0.f;
      l = l * alpha + warp_sum(p);
#pragma unroll
      for (int i = 0; i < D / 32; ++i) acc[i] *= alpha;
      const int nk = min(32, ke - kb);
      for (int t = 0; t < nk; ++t) {
        const float pt = __shfl_sync(0xffffffffu, p, t);
        const T* vrow = V + kvrow(kb + t) * kstride + (int64_t)g * D;
#pragma unroll
        for (int i = 0; i < D / 32; ++i) acc[i] = fmaf(pt, ld(vrow + lane + 32 * i), acc[i]);
      }
      m = mn;
    }
    const float inv = 1.f / l;
#pragma unroll
    for (int i = 0; i < D / 32; ++i) st(O + qrow * qstride + (int64_t)h * D + lane + 32 * i, acc[i] * inv);
    if (a.lse && lane == 0) a.lse[(int64_t)h * a.q_rows + qrow] = m + logf(l);
  }
}

// Delta = rowsum(dO * O) per (row, head); grid-stride over rows*heads, one warp each.
template <typename T, int D>
__global__ void simt_delta_kernel(AttnArgs a) {
  const int lane = threadIdx.x & 31;
  const int64_t n = a.q_rows * a.hq;
  const T* O = (const T*)a.o;
  const T* dO = (const T*)a.dout;
  for (int64_t i = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; i < n;
       i += ((int64_t)gridDim.x * blockDim.x) >> 5) {
    const int64_t row = i / a.hq;
    const int h = (int)(i % a.hq);
    const int64_t off = (row * a.hq + h) * D;
    float acc = 0.f;
    for (int d = lane; d < D; d += 32) acc = fmaf(ld(O + off + d), ld(dO + off + d), acc);
    acc = warp_sum(acc);
    if (lane == 0) a.delta[(int64_t)h * a.q_rows + row] = acc;
  }
}

// dQ: same grid as the forward.
template <typename T, int D>
__global__ void __launch_bounds__(kWarps * 32) simt_dq_kernel(AttnArgs a) {
  __shared__ float qs[kWarps][D];
  __shared__ float dos[kWarps][D];
  const int h = blockIdx.x % a.hq;
  const Tile w = a.qtiles[a.q_order[blockIdx.x / a.hq]];
  const int g = h / (a.hq / a.hkv);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const T* Q = (const T*)a.q;
  const T* K = (const T*)a.k;
  const T* V = (const T*)a.v;
  const T* dO = (const T*)a.dout;
  T* dQ = (T*)a.dq;
  const int64_t qstride = (int64_t)a.hq * D, kstride = (int64_t)a.hkv * D;
  for (int r = warp; r < kRowsPerTile; r += kWarps) {
    const int row = w.tile * kRowsPerTile + r;
    if (row >= w.q_len) break;
    const int64_t qrow = (int64_t)w.q_base + row;
    __syncwarp();
    for (int d = lane; d < D; d += 32) {
      qs[warp][d] = ld(Q + qrow * qstride + (int64_t)h * D + d);
      dos[warp][d] = ld(dO + qrow * qstride + (int64_t)h * D + d);
    }
    __syncwarp();
    const int ke = a.kv_end[w.kv_base + row];
    const float lse = a.lse_in[(int64_t)h * a.q_rows + qrow];
    const float dl = a.delta[(int64_t)h * a.q_rows + qrow];
    float acc[D / 32];
#pragma unroll
    for (int i = 0; i < D / 32; ++i) acc[i] = 0.f;
    for (int kb = 0; kb < ke; kb += 32) {
      const int key = kb + lane;
      float ds = 0.f;
      if (key < ke) {
        const int64_t koff = ((int64_t)w.k_base + key) * kstride + (int64_t)g * D;
        const float p = expf(a.scale * dot_row<T, D>(qs[warp], K + koff) - lse);
        const float dp = dot_row<T, D>(dos[warp], V + koff);
        ds = p * (dp - dl);
      }
      const int nk = min(32, ke - kb);
      for (int t = 0; t < nk; ++t) {
        const float dst = __shfl_sync(0xffffffffu, ds, t);
        const T* krow = K + ((int64_t)w.k_base + kb + t) * kstride + (int64_t)g * D;
#pragma unroll
        for (int i = 0; i < D / 32; ++i) acc[i] = fmaf(dst, ld(krow + lane + 32 * i), acc[i]);
      }
    }
#pragma unroll
    for (int i = 0; i < D / 32; ++i) st(dQ + qrow * qstride + (int64_t)h * D + lane + 32 * i, a.scale * acc[i]);
  }
}

// dK/dV: Hkv * nk blocks (KV head fastest); one warp per key row; walks the query heads of the
// group and the query rows that see the key.
template <typename T, int D>
__global__ void __launch_bounds__(kWarps * 32) simt_dkdv_kernel(AttnArgs a) {
  __shared__ float ks[kWarps][D];
  __shared__ float vs[kWarps][D];
  const int g = blockIdx.x % a.hkv;
  const Tile w = a.ktiles[a.k_order[blockIdx.x / a.hkv]];
  const int group = a.hq / a.hkv;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const T* Q = (const T*)a.q;
  const T* K = (const T*)a.k;
  const T* V = (const T*)a.v;
  const T* dO = (const T*)a.dout;
  T* dK = (T*)a.dk;
  T* dV = (T*)a.dv;
  const int64_t qstride = (int64_t)a.hq * D, kstride = (int64_t)a.hkv * D;
  for (int r = warp; r < kRowsPerTile; r += kWarps) {
    const int key = w.tile * kRowsPerTile + r;
    if (key >= w.k_len) break;
    const int64_t krow = (int64_t)w.k_base + key;
    __syncwarp();
    for (int d = lane; d < D; d += 32) {
      ks[warp][d] = ld(K + krow * kstride + (int64_t)g * D + d);
      vs[warp][d] = ld(V + krow * kstride + (int64_t)g * D + d);
    }
    __syncwarp();
    // first query row whose bound exceeds this key
    int lo = 0, hi = w.q_len;
    const int32_t* ke = a.kv_end + w.kv_base;
    while (lo < hi) { int mid = (lo + hi) >> 1; if (ke[mid] > key) hi = mid; else lo = mid + 1; }
    const int j0 = lo;
    float accK[D / 32], accV[D / 32];
#pragma unroll
    for (int i = 0; i < D / 32; ++i) { accK[i] = 0.f; accV[i] = 0.f; }
    for (int hh = 0; hh < group; ++hh) {
      const int h = g * group + hh;
      for (int jb = j0; jb < w.q_len; jb += 32) {
        const int j = jb + lane;
        float p = 0.f, ds = 0.f;
        if (j < w.q_len) {
          const int64_t qrow = (int64_t)w.q_base + j;
          const int64_t qoff = qrow * qstride + (int64_t)h * D;
          const float lse = a.lse_in[(int64_t)h * a.q_rows + qrow];
          p = expf(a.scale * dot_row<T, D>(ks[warp], Q + qoff) - lse);
          const float dp = dot_row<T, D>(vs[warp], dO + qoff);
          ds = p * (dp - a.delta[(int64_t)h * a.q_rows + qrow]);
        }
        const int nj = min(32, w.q_len - jb);
        for (int t = 0; t < nj; ++t) {
          const float pt = __shfl_sync(0xffffffffu, p, t);
          const float dst = __shfl_sync(0xffffffffu, ds, t);
          const int64_t qoff = ((int64_t)w.q_base + jb + t) * qstride + (int64_t)h * D;
#pragma unroll
          for (int i = 0; i < D / 32; ++i) {
            accV[i] = fmaf(pt, ld(dO + qoff + lane + 32 * i), accV[i]);
            accK[i] = fmaf(dst, ld(Q + qoff + lane + 32 * i), accK[i]);
          }
        }
      }
    }
#pragma unroll
    for (int i = 0; i < D / 32; ++i) {
      st(dK + krow * kstride + (int64_t)g * D + lane + 32 * i, a.scale * accK[i]);
      st(dV + krow * kstride + (int64_t)g * D + lane + 32 * i, accV[i]);
    }
  }
}

template <typename T, int D>
cudaError_t fwd_impl(const AttnArgs& a, cudaStream_t st) {
  if (a.nq == 0) return cudaSuccess;
  simt_fwd_kernel<T, D><<<(unsigned)(a.nq * a.hq), kWarps * 32, 0, st>>>(a);
  return cudaGetLastError();
}

template <typename T, int D>
cudaError_t bwd_impl(const AttnArgs& a, cudaStream_t st) {
  if (a.q_rows == 0) return cudaSuccess;
  int64_t warps = a.q_rows * a.hq;
  int grid = (int)((warps * 32 + 255) / 256);
  if (grid > 152 * 32) grid = 152 * 32;
  timer_begin(ISM_KERNEL_BWD_PRE, st);
  simt_delta_kernel<T, D><<<grid, 256, 0, st>>>(a);
  timer_end(ISM_KERNEL_BWD_PRE, st);
  count_launch();
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (a.nq) {
    timer_begin(ISM_KERNEL_BWD_DQ, st);
    simt_dq_kernel<T, D><<<(unsigned)(a.nq * a.hq), kWarps * 32, 0, st>>>(a);
    timer_end(ISM_KERNEL_BWD_DQ, st);
    count_launch();
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  if (a.nk) {
    timer_begin(ISM_KERNEL_BWD_DKDV, st);
    simt_dkdv_kernel<T, D><<<(unsigned)(a.nk * a.hkv), kWarps * 32, 0, st>>>(a);
    timer_end(ISM_KERNEL_BWD_DKDV, st);
    count_launch();
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace

cudaError_t launch_simt_fwd(const AttnArgs& a, cudaStream_t st) {
  if (a.dtype == ISM_FP32) return a.d == 64 ? fwd_impl<float, 64>(a, st) : fwd_impl<float, 128>(a, st);
  return a.d == 64 ? fwd_impl<__nv_bfloat16, 64>(a, st) : fwd_impl<__nv_bfloat16, 128>(a, st);
}

cudaError_t launch_simt_bwd(const AttnArgs& a, cudaStream_t st) {
  if (a.dtype == ISM_FP32) return a.d == 64 ? bwd_impl<float, 64>(a, st) : bwd_impl<float, 128>(a, st);
  return a.d == 64 ? bwd_impl<__nv_bfloat16, 64>(a, st) : bwd_impl<__nv_bfloat16, 128>(a, st);
}

}  // namespace ism
