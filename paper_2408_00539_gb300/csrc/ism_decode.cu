// Single-token append (decode step of an answer token, Section 2.3: the new
// token reuses the cached keys/values [C_h; C_q] and sees all of them plus
// itself).  Bandwidth-bound: every K/V byte of the cache is read once.
// Split-KV: each CTA streams one chunk of one (sequence, KV head) cache and
// serves all query heads of that KV head's group; a second kernel merges the
// per-chunk softmax partials.  Scores are kept in base 2 (q pre-scaled by
// scale * log2 e).
#include "ism_internal.cuh"

namespace ism {
namespace {

constexpr int kDecWarps = 4;
constexpr int kKeysPerIter = 8;

template <int N>
struct BfVec;
template <>
struct BfVec<4> { using T = uint2; };
template <>
struct BfVec<2> { using T = uint32_t; };

template <int DPL>
__device__ __forceinline__ void load_bf16(const __nv_bfloat16* p, float (&x)[DPL]) {
  typename BfVec<DPL>::T raw = *reinterpret_cast<const typename BfVec<DPL>::T*>(p);
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&raw);
#pragma unroll
  for (int i = 0; i < DPL / 2; ++i) {
    float2 f = __bfloat1622float2(h[i]);
    x[2 * i] = f.x;
    x[2 * i + 1] = f.y;
  }
}

// grid (splits, Hkv, B); block kDecWarps warps.  Lane l owns head dims
// [l*DPL, l*DPL + DPL).
template <int D, int G>
__global__ void __launch_bounds__(kDecWarps * 32) decode_split_kernel(DecodeArgs a) {
  constexpr int DPL = D / 32;
  const int split = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int hq = a.hq;
  const int kv_len = a.c_snap[b] + 1;
  const int k0 = split * a.chunk;
  const int k1 = min(kv_len, k0 + a.chunk);
  const float qscale = a.scale * 1.4426950408889634f;

  const __nv_bfloat16* Q = (const __nv_bfloat16*)a.q;
  const __nv_bfloat16* Kc = (const __nv_bfloat16*)a.k_cache;
  const __nv_bfloat16* Vc = (const __nv_bfloat16*)a.v_cache;
  const int64_t kstride = (int64_t)a.hkv * D;

  float q[G][DPL];
#pragma unroll
  for (int h = 0; h < G; ++h) {
    load_bf16<DPL>(Q + ((int64_t)b * hq + g * G + h) * D + lane * DPL, q[h]);
#pragma unroll
    for (int i = 0; i < DPL; ++i) q[h][i] *= qscale;
  }
  float m[G], l[G], o[G][DPL];
#pragma unroll
  for (int h = 0; h < G; ++h) {
    m[h] = -INFINITY;
    l[h] = 0.f;
#pragma unroll
    for (int i = 0; i < DPL; ++i) o[h][i] = 0.f;
  }

  const __nv_bfloat16* kbase = Kc + (int64_t)b * a.cap * kstride + (int64_t)g * D + lane * DPL;
  const __nv_bfloat16* vbase = Vc + (int64_t)b * a.cap * kstride + (int64_t)g * D + lane * DPL;
  for (int kb = k0 + warp * kKeysPerIter; kb < k1; kb += kDecWarps * kKeysPerIter) {
    float s[G][kKeysPerIter];
#pragma unroll
    for (int t = 0; t < kKeysPerIter; ++t) {
      float kx[DPL];
      const int key = kb + t;
      if (key < k1) {
        load_bf16<DPL>(kbase + (int64_t)key * kstride, kx);
      } else {
#pragma unroll
        for (int i = 0; i < DPL; ++i) kx[i] = 0.f;
      }
#pragma unroll
      for (int h = 0; h < G; ++h) {
        float acc = 0.f;
#pragma unroll
        for (int i = 0; i < DPL; ++i) acc = fmaf(q[h][i], kx[i], acc);
        s[h][t] = acc;
      }
    }
#pragma unroll
    for (int h = 0; h < G; ++h)
#pragma unroll
      for (int t = 0; t < kKeysPerIter; ++t) {
        float x = s[h][t];
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) x += __shfl_xor_sync(0xffffffffu, x, off);
        s[h][t] = (kb + t < k1) ? x : -INFINITY;
      }
    float p[G][kKeysPerIter];
#pragma unroll
    for (int h = 0; h < G; ++h) {
      float mx = m[h];
#pragma unroll
      for (int t = 0; t < kKeysPerIter; ++t) mx = fmaxf(mx, s[h][t]);
      const float alpha = exp2f(m[h] - mx);  // m = -inf on the first batch: alpha = 0
      float sum = 0.f;
#pragma unroll
      for (int t = 0; t < kKeysPerIter; ++t) { p[h][t] = exp2f(s[h][t] - mx); sum += p[h][t]; }
      l[h] = l[h] * alpha + sum;
      m[h] = mx;
#pragma unroll
      for (int i = 0; i < DPL; ++i) o[h][i] *= alpha;
    }
#pragma unroll
    for (int t = 0; t < kKeysPerIter; ++t) {
      const int key = kb + t;
      if (key >= k1) break;
      float vx[DPL];
      load_bf16<DPL>(vbase + (int64_t)key * kstride, vx);
#pragma unroll
      for (int h = 0; h < G; ++h)
#pragma unroll
        for (int i = 0; i < DPL; ++i) o[h][i] = fmaf(p[h][t], vx[i], o[h][i]);
    }
  }

  // merge the warps of this CTA
  __shared__ float sm_m[kDecWarps][G], sm_l[kDecWarps][G];
  __shared__ float sm_o[kDecWarps][G][D];
  if (lane == 0) {
#pragma unroll
    for (int h = 0; h < G; ++h) { sm_m[warp][h] = m[h]; sm_l[warp][h] = l[h]; }
  }
#pragma unroll
  for (int h = 0; h < G; ++h)
#pragma unroll
    for (int i = 0; i < DPL; ++i) sm_o[warp][h][lane * DPL + i] = o[h][i];
  __syncthreads();
  for (int idx = threadIdx.x; idx < G * D; idx += blockDim.x) {
    const int h = idx / D, d = idx % D;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < kDecWarps; ++w) M = fmaxf(M, sm_m[w][h]);
    float acc = 0.f, lsum = 0.f;
    if (M != -INFINITY) {
#pragma unroll
      for (int w = 0; w < kDecWarps; ++w) {
        const float f = exp2f(sm_m[w][h] - M);
        acc = fmaf(sm_o[w][h][d], f, acc);
        lsum = fmaf(sm_l[w][h], f, lsum);
      }
    }
    const int64_t pidx = ((int64_t)b * hq + g * G + h) * a.splits + split;
    a.part_o[pidx * D + d] = acc;
    if (d == 0) { a.part_ml[pidx * 2] = M; a.part_ml[pidx * 2 + 1] = lsum; }
  }
}

// grid B*Hq, block D threads.
template <int D>
__global__ void decode_combine_kernel(DecodeArgs a) {
  const int bh = blockIdx.x;
  const int d = threadIdx.x;
  const float* pml = a.part_ml + (int64_t)bh * a.splits * 2;
  float M = -INFINITY;
  for (int s = 0; s < a.splits; ++s) M = fmaxf(M, pml[2 * s]);
  float acc = 0.f, L = 0.f;
  for (int s = 0; s < a.splits; ++s) {
    const float ms = pml[2 * s];
    if (ms == -INFINITY) continue;
    const float f = exp2f(ms - M);
    acc = fmaf(a.part_o[((int64_t)bh * a.splits + s) * D + d], f, acc);
    L = fmaf(pml[2 * s + 1], f, L);
  }
  ((__nv_bfloat16*)a.out)[(int64_t)bh * D + d] = __float2bfloat16_rn(acc / L);
  if (a.lse && d == 0) {
    const int b = bh / a.hq, h = bh % a.hq;
    a.lse[(int64_t)h * a.batch + b] = (M + log2f(L)) * 0.6931471805599453f;
  }
}

template <int D, int G>
cudaError_t run(const DecodeArgs& a, cudaStream_t st) {
  dim3 grid(a.splits, a.hkv, a.batch);
  decode_split_kernel<D, G><<<grid, kDecWarps * 32, 0, st>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  decode_combine_kernel<D><<<a.batch * a.hq, D, 0, st>>>(a);
  return cudaGetLastError();
}

template <int D>
cudaError_t run_d(const DecodeArgs& a, cudaStream_t st) {
  switch (a.hq / a.hkv) {
    case 1: return run<D, 1>(a, st);
    case 2: return run<D, 2>(a, st);
    case 4: return run<D, 4>(a, st);
    case 8: return run<D, 8>(a, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

cudaError_t launch_decode(const DecodeArgs& a, cudaStream_t st) {
  if (a.batch == 0) return cudaSuccess;
  return a.d == 64 ? run_d<64>(a, st) : run_d<128>(a, st);
}

}  // namespace ism
