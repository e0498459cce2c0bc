// Rotary position encoding of the one-pass (training) path.  Positional
// encoding lies outside the paper's attention operation (Section 2.1 leaves
// it out); models that take up ISM (Section 2.3) rotate queries and keys by
// their positions first.  In a packed batch the positions restart at every
// sequence: token t of sequence b sits at position t - cu_seqlens[b].
//
// rope_rows_kernel turns each pair (x_k, x_{k+D/2}) of every query and key
// head row by the angle of the row's position (tables of cosines and sines,
// [rows, D/2] fp32) into separate output tensors, in fp32 with one rounding
// to the storage type.  With sin_sign = -1 it applies the transposed
// rotation (the rotation by the opposite angle), which takes the gradients of
// rotated queries and keys back to the unrotated inputs; that form runs in
// place on dQ and dK after the CUDA-core backward (the tensor-core backward
// applies it in its dQ / dK epilogues instead).
#include "ism_internal.cuh"

namespace ism {
namespace {

// Sequence of token t: the last b with cu_seqlens[b] <= t (zero-length
// sequences share their offset with the next one).
__device__ __forceinline__ int seq_of(const int32_t* __restrict__ cu, int num_seqs, int64_t t) {
  int lo = 0, hi = num_seqs;  // cu[lo] <= t < cu[hi]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if ((int64_t)__ldg(cu + mid) <= t) lo = mid; else hi = mid;
  }
  return lo;
}

template <typename E>
struct Vec;  // 16 bytes of E as fp32 values
template <>
struct Vec<__nv_bfloat16> {
  static constexpr int N = 8;
  __device__ static void load(const __nv_bfloat16* p, float (&x)[8]) {
    const uint4 u = *reinterpret_cast<const uint4*>(p);
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float2 f = __bfloat1622float2(h[e]);
      x[2 * e] = f.x;
      x[2 * e + 1] = f.y;
    }
  }
  __device__ static void store(__nv_bfloat16* p, const float (&x)[8]) {
    uint4 u;
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&u);
#pragma unroll
    for (int e = 0; e < 4; ++e) h[e] = __floats2bfloat162_rn(x[2 * e], x[2 * e + 1]);
    *reinterpret_cast<uint4*>(p) = u;
  }
};
template <>
struct Vec<float> {
  static constexpr int N = 4;
  __device__ static void load(const float* p, float (&x)[4]) {
    const float4 f = *reinterpret_cast<const float4*>(p);
    x[0] = f.x; x[1] = f.y; x[2] = f.z; x[3] = f.w;
  }
  __device__ static void store(float* p, const float (&x)[4]) {
    *reinterpret_cast<float4*>(p) = make_float4(x[0], x[1], x[2], x[3]);
  }
};

// One thread per 16-byte unit of the first half of one head row (query heads
// first, then key heads) and its partner unit in the second half.
template <typename E>
__global__ void __launch_bounds__(256) rope_rows_kernel(const int32_t* __restrict__ cu_seqlens, int num_seqs,
                                                        int64_t T, int hq, int hkv, int d, const E* q_src,
                                                        const E* k_src, E* q_dst, E* k_dst,
                                                        const float* __restrict__ cos_t,
                                                        const float* __restrict__ sin_t, float sin_sign) {
  constexpr int N = Vec<E>::N;
  const int half = d / 2;
  const int units = half / N;
  const int per_row = (hq + hkv) * units;
  const int64_t total = T * per_row;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t t = i / per_row;
    const int r = (int)(i % per_row);
    const int head = r / units;
    const int k0 = (r % units) * N;
    const int64_t pos = t - __ldg(cu_seqlens + seq_of(cu_seqlens, num_seqs, t));
    const E* src;
    E* dst;
    if (head < hq) {
      src = q_src + (t * hq + head) * d;
      dst = q_dst + (t * hq + head) * d;
    } else {
      src = k_src + (t * hkv + (head - hq)) * d;
      dst = k_dst + (t * hkv + (head - hq)) * d;
    }
    float lo[N], hi[N], c[N], s[N];
    Vec<E>::load(src + k0, lo);
    Vec<E>::load(src + half + k0, hi);
    const float4* cp = reinterpret_cast<const float4*>(cos_t + pos * half + k0);
    const float4* sp = reinterpret_cast<const float4*>(sin_t + pos * half + k0);
#pragma unroll
    for (int v = 0; v < N / 4; ++v) {
      const float4 cv = __ldg(cp + v), sv = __ldg(sp + v);
      c[4 * v] = cv.x; c[4 * v + 1] = cv.y; c[4 * v + 2] = cv.z; c[4 * v + 3] = cv.w;
      s[4 * v] = sv.x * sin_sign; s[4 * v + 1] = sv.y * sin_sign;
      s[4 * v + 2] = sv.z * sin_sign; s[4 * v + 3] = sv.w * sin_sign;
    }
    float ol[N], oh[N];
#pragma unroll
    for (int e = 0; e < N; ++e) {
      ol[e] = lo[e] * c[e] - hi[e] * s[e];
      oh[e] = hi[e] * c[e] + lo[e] * s[e];
    }
    Vec<E>::store(dst + k0, ol);
    Vec<E>::store(dst + half + k0, oh);
  }
}

}  // namespace

cudaError_t launch_rope_rows(const int32_t* cu_seqlens, int num_seqs, int64_t T, int hq, int hkv, int d, int dtype,
                             const void* q_src, const void* k_src, void* q_dst, void* k_dst, const float* cos_t,
                             const float* sin_t, float sin_sign, cudaStream_t st) {
  const int elems = dtype == ISM_BF16 ? 8 : 4;
  const int64_t total = T * (hq + hkv) * (d / 2 / elems);
  if (total == 0) return cudaSuccess;
  int64_t grid = (total + 255) / 256;
  const int64_t cap = (int64_t)sm_count() * 16;
  if (grid > cap) grid = cap;
  if (dtype == ISM_BF16) {
    rope_rows_kernel<__nv_bfloat16><<<(unsigned)grid, 256, 0, st>>>(
        cu_seqlens, num_seqs, T, hq, hkv, d, static_cast<const __nv_bfloat16*>(q_src),
        static_cast<const __nv_bfloat16*>(k_src), static_cast<__nv_bfloat16*>(q_dst),
        static_cast<__nv_bfloat16*>(k_dst), cos_t, sin_t, sin_sign);
  } else {
    rope_rows_kernel<float><<<(unsigned)grid, 256, 0, st>>>(cu_seqlens, num_seqs, T, hq, hkv, d,
                                                            static_cast<const float*>(q_src),
                                                            static_cast<const float*>(k_src),
                                                            static_cast<float*>(q_dst), static_cast<float*>(k_dst),
                                                            cos_t, sin_t, sin_sign);
  }
  return cudaGetLastError();
}

}  // namespace ism
