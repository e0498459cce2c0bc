// Single-token append (decode step of an answer token, Section 2.3: the new
// token reuses the cached keys/values [C_h; C_q] and sees all of them plus
// itself).  Bandwidth-bound: every K/V byte of the cache is read once.
// Split-KV: each CTA streams one chunk of one (sequence, KV head) cache and
// serves all query heads of that KV head's group; a second kernel merges the
// per-chunk softmax partials.  Scores are kept in base 2 (q pre-scaled by
// scale * log2 e).
#include <cstdlib>
#include <type_traits>

#include <cuda_fp16.h>

#include "ism_internal.cuh"
#include "ism_tc_common.cuh"

namespace ism {
namespace {

constexpr int kDecWarps = 4;

template <int N>
struct BfVec;
template <>
struct BfVec<4> { using T = uint2; };
template <>
struct BfVec<2> { using T = uint32_t; };

// e4m3 elements: DPL bytes a lane
template <int N>
struct F8Vec;
template <>
struct F8Vec<4> { using T = uint32_t; };
template <>
struct F8Vec<2> { using T = uint16_t; };

template <int DPL>
__device__ __forceinline__ void unpack_e4m3(const typename F8Vec<DPL>::T& raw, float (&x)[DPL]) {
  const uint16_t* pairs = reinterpret_cast<const uint16_t*>(&raw);
#pragma unroll
  for (int i = 0; i < DPL / 2; ++i) {
    uint32_t h2;  // two halves, the lower from the lower byte
    asm("cvt.rn.f16x2.e4m3x2 %0, %1;" : "=r"(h2) : "h"(pairs[i]));
    const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&h2));
    x[2 * i] = f.x;
    x[2 * i + 1] = f.y;
  }
}

template <int DPL>
__device__ __forceinline__ void unpack_bf16(const typename BfVec<DPL>::T& raw, float (&x)[DPL]) {
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&raw);
#pragma unroll
  for (int i = 0; i < DPL / 2; ++i) {
    float2 f = __bfloat1622float2(h[i]);
    x[2 * i] = f.x;
    x[2 * i + 1] = f.y;
  }
}

// grid (splits, Hkv, B); block kDecWarps warps.  Lane l owns head dims
// [l*DPL, l*DPL + DPL) for the dot products and the output accumulator.
// A batch covers KPI = 32 / G keys, so the G x KPI partial dot products of a
// lane are 32 values: a butterfly reduce-scatter (31 shuffles) leaves lane l
// with the full score of (head l / KPI, key l % KPI); the softmax of a head
// then runs across its KPI lanes, and the probabilities are broadcast back
// for O += P V.
// kE4M3: e4m3 query and caches (one byte an element), dequantised by
// qk_descale in the scores and v_descale in the output.
template <int D, int G, bool kE4M3 = false>
__global__ void __launch_bounds__(kDecWarps * 32) decode_split_kernel(DecodeArgs a) {
  constexpr int DPL = D / 32;
  constexpr int KPI = 32 / G;  // keys per batch
  const int split = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int hq = a.hq;
  const int kv_len = a.c_snap[b] + 1;
  const int k0 = split * a.chunk;
  const int k1 = min(kv_len, k0 + a.chunk);
  const float qscale = a.scale * 1.4426950408889634f * (kE4M3 ? a.qk_descale : 1.f);
  using Raw = typename std::conditional<kE4M3, typename F8Vec<DPL>::T, typename BfVec<DPL>::T>::type;
  using Elem = typename std::conditional<kE4M3, uint8_t, __nv_bfloat16>::type;
  auto unpack = [](const Raw& raw, float (&x)[DPL]) {
    if constexpr (kE4M3)
      unpack_e4m3<DPL>(raw, x);
    else
      unpack_bf16<DPL>(raw, x);
  };

  const Elem* Q = (const Elem*)a.q;
  const Elem* Kc = (const Elem*)a.k_cache;
  const Elem* Vc = (const Elem*)a.v_cache;
  const int64_t kstride = (int64_t)a.hkv * D;

  // G is the group size padded to a power of two: heads h >= grp are zero and not written
  const int grp = a.group;
  float q[G][DPL];
#pragma unroll
  for (int h = 0; h < G; ++h) {
    if (h < grp) {
      unpack(*reinterpret_cast<const Raw*>(Q + ((int64_t)b * hq + g * grp + h) * D + lane * DPL), q[h]);
    } else {
#pragma unroll
      for (int i = 0; i < DPL; ++i) q[h][i] = 0.f;
    }
#pragma unroll
    for (int i = 0; i < DPL; ++i) q[h][i] *= qscale;
  }
  // running max and sum of this lane's head (uniform across the head's KPI lanes)
  const int my_h = lane / KPI, my_t = lane % KPI;
  float m = -INFINITY, l = 0.f;
  float o[G][DPL];
#pragma unroll
  for (int h = 0; h < G; ++h)
#pragma unroll
    for (int i = 0; i < DPL; ++i) o[h][i] = 0.f;

  const Elem* kbase = Kc + (int64_t)g * D + lane * DPL;
  const Elem* vbase = Vc + (int64_t)g * D + lane * DPL;
  for (int kb = k0 + warp * KPI; kb < k1; kb += kDecWarps * KPI) {
    // every K and V row load of the batch is issued before any use; rows past
    // the chunk re-read its last key and get probability 0
    Raw kraw[KPI], vraw[KPI];
#pragma unroll
    for (int t = 0; t < KPI; ++t) {
      const int key = min(kb + t, k1 - 1);
      const int64_t row = a.pages.table ? paged_row(a.pages, b, key) : (int64_t)b * a.cap + key;
      kraw[t] = *reinterpret_cast<const Raw*>(kbase + row * kstride);
      vraw[t] = *reinterpret_cast<const Raw*>(vbase + row * kstride);
    }
    float v[32];  // v[h * KPI + t]: this lane's partial dot product
#pragma unroll
    for (int t = 0; t < KPI; ++t) {
      float kx[DPL];
      unpack(kraw[t], kx);
#pragma unroll
      for (int h = 0; h < G; ++h) {
        float acc = 0.f;
#pragma unroll
        for (int i = 0; i < DPL; ++i) acc = fmaf(q[h][i], kx[i], acc);
        v[h * KPI + t] = acc;
      }
    }
    // butterfly reduce-scatter: after the step with offset sh a lane keeps the
    // half of its values selected by lane bit sh, plus the partner's partial sums
#pragma unroll
    for (int sh = 16; sh >= 1; sh >>= 1) {
      const bool hi = (lane & sh) != 0;
#pragma unroll
      for (int i = 0; i < sh; ++i) {
        const float send = hi ? v[i] : v[sh + i];
        const float keep = hi ? v[sh + i] : v[i];
        v[i] = keep + __shfl_xor_sync(0xffffffffu, send, sh);
      }
    }
    // lane holds the score of (my_h, my_t); softmax across the head's KPI lanes
    const float sc = (kb + my_t < k1) ? v[0] : -INFINITY;
    float mx = sc;
#pragma unroll
    for (int off = KPI / 2; off >= 1; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
    const float m_new = fmaxf(m, mx);  // finite: key kb is inside the chunk
    const float p = exp2f(sc - m_new);
    float ps = p;
#pragma unroll
    for (int off = KPI / 2; off >= 1; off >>= 1) ps += __shfl_xor_sync(0xffffffffu, ps, off);
    const float alpha = exp2f(m - m_new);  // 0 on the first batch (m = -inf)
    l = l * alpha + ps;
    m = m_new;
#pragma unroll
    for (int h = 0; h < G; ++h) {
      const float ah = __shfl_sync(0xffffffffu, alpha, h * KPI);
#pragma unroll
      for (int i = 0; i < DPL; ++i) o[h][i] *= ah;
    }
#pragma unroll
    for (int t = 0; t < KPI; ++t) {
      float vx[DPL];
      unpack(vraw[t], vx);
#pragma unroll
      for (int h = 0; h < G; ++h) {
        const float pht = __shfl_sync(0xffffffffu, p, h * KPI + t);
#pragma unroll
        for (int i = 0; i < DPL; ++i) o[h][i] = fmaf(pht, vx[i], o[h][i]);
      }
    }
  }

  // merge the warps of this CTA
  __shared__ float sm_m[kDecWarps][G], sm_l[kDecWarps][G];
  __shared__ float sm_o[kDecWarps][G][D];
  if (my_t == 0) {
    sm_m[warp][my_h] = m;
    sm_l[warp][my_h] = l;
  }
#pragma unroll
  for (int h = 0; h < G; ++h)
#pragma unroll
    for (int i = 0; i < DPL; ++i) sm_o[warp][h][lane * DPL + i] = o[h][i];
  __syncthreads();
  for (int idx = threadIdx.x; idx < grp * D; idx += blockDim.x) {
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
    const int64_t pidx = ((int64_t)b * hq + g * grp + h) * a.splits + split;
    a.part_o[pidx * D + d] = kE4M3 ? acc * a.v_descale : acc;
    if (d == 0) { a.part_ml[pidx * 2] = M; a.part_ml[pidx * 2 + 1] = lsum; }
  }
}

// TMA-pipelined variant for head_dim 128 and at least two query heads per KV
// head: warp 4 streams K and V tiles of the chunk into a shared-memory ring
// with TMA; warps 0-3 each take a quarter of a tile (batches of 32 / G keys,
// the same butterfly softmax as above) reading the rows from shared memory.
// Tile rows and ring depth: a warp's share of a tile (kTile / 4 rows) must
// hold whole batches of 32 / G keys.  A 2-stage ring of 64-key tiles (about
// 70 KB of shared memory) lets three CTAs share an SM; measured on the 8 x 16K
// cache it beats 3 or 4 stages and 32-key tiles.
// With e4m3 caches a row is 128 bytes (one box of 128 columns), a K or V
// tile half the bf16 size.
template <int G, bool kE4M3 = false> struct TmaCfg {
  static constexpr int kTile = 64;
  static constexpr int kStages = 2;
  static constexpr uint32_t kHalf = kTile * 128;                    // kTile rows x 128 bytes
  static constexpr uint32_t kKV = (kE4M3 ? 1 : 2) * kHalf;          // one K (or V) tile
  static constexpr uint32_t kStageBytes = 2 * kKV;                  // K and V
};

template <int G, bool kE4M3 = false>
__global__ void __launch_bounds__(160) decode_tma_kernel(const __grid_constant__ CUtensorMap tmK,
                                                        const __grid_constant__ CUtensorMap tmV, DecodeArgs a) {
  using Cfg = TmaCfg<G, kE4M3>;
  constexpr int kTmaTile = Cfg::kTile, kTmaStages = Cfg::kStages;
  constexpr uint32_t kTmaHalf = Cfg::kHalf, kTmaKV = Cfg::kKV, kTmaStageBytes = Cfg::kStageBytes;
  constexpr int D = 128, DPL = 4, KPI = 32 / G, RPW = kTmaTile / 4, NB = RPW / KPI;  // batches per warp per tile
  static_assert(NB >= 1 && RPW % KPI == 0, "a warp's rows must hold whole batches");
  extern __shared__ __align__(128) uint8_t dsm[];
  uint64_t* full = reinterpret_cast<uint64_t*>(dsm + kTmaStages * kTmaStageBytes);
  uint64_t* empty = full + kTmaStages;
  float* sm_m = reinterpret_cast<float*>(empty + kTmaStages);  // [4][G]
  float* sm_l = sm_m + 4 * G;                                   // [4][G]
  float* sm_o = sm_l + 4 * G;                                   // [4][G][D]
  const int split = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int kv_len = a.c_snap[b] + 1;
  const int k0 = split * a.chunk;
  const int k1 = min(kv_len, k0 + a.chunk);
  const int ntiles = k1 > k0 ? (k1 - k0 + kTmaTile - 1) / kTmaTile : 0;
  const int32_t row0 = (int32_t)((int64_t)b * a.cap + k0);
  if (threadIdx.x == 0) {
    for (int s = 0; s < kTmaStages; ++s) {
      ptx::mbar_init(&full[s], 1);
      ptx::mbar_init(&empty[s], 4);
    }
    ptx::fence_mbar_init();
  }
  __syncthreads();
  if (warp == 4) {
    if (lane == 0) {
      int issued = 0;
      for (int t = 0; t < ntiles; ++t) {
        const int s = t % kTmaStages;
        if (t >= kTmaStages && !tc::wait(&empty[s], (uint32_t)(t / kTmaStages - 1) & 1, a.status)) break;
        issued = t + 1;
        uint8_t* st = dsm + s * kTmaStageBytes;
        // a page holds whole tiles: page_size is a multiple of 128, tiles start at multiples of 64
        const int32_t y = a.pages.table ? (int32_t)paged_row(a.pages, b, (int64_t)k0 + t * kTmaTile)
                                        : row0 + t * kTmaTile;
        ptx::mbar_expect_tx(&full[s], kTmaStageBytes);
        ptx::tma_load_2d(st, &tmK, &full[s], g * D, y);
        ptx::tma_load_2d(st + kTmaKV, &tmV, &full[s], g * D, y);
        if (!kE4M3) {  // bf16 rows: the second 64 columns
          ptx::tma_load_2d(st + kTmaHalf, &tmK, &full[s], g * D + 64, y);
          ptx::tma_load_2d(st + kTmaKV + kTmaHalf, &tmV, &full[s], g * D + 64, y);
        }
      }
      // every issued copy completes before the CTA exits
      for (int t = issued - kTmaStages > 0 ? issued - kTmaStages : 0; t < issued; ++t)
        tc::wait(&full[t % kTmaStages], (uint32_t)(t / kTmaStages) & 1, a.status);
    }
  } else {
    const float qscale = a.scale * 1.4426950408889634f * (kE4M3 ? a.qk_descale : 1.f);
    // this lane's DPL elements of a row (bf16: 8 bytes in half lane / 16; e4m3: 4 bytes)
    auto row_at = [&](const uint8_t* base, float (&x)[DPL]) {
      if constexpr (kE4M3)
        unpack_e4m3<DPL>(*reinterpret_cast<const uint32_t*>(base + lane * 4), x);
      else
        unpack_bf16<DPL>(*reinterpret_cast<const uint2*>(base + (lane >> 4) * kTmaHalf + (lane & 15) * 8), x);
    };
    const uint8_t* Q = static_cast<const uint8_t*>(a.q);
    const int64_t qrow_bytes = (int64_t)D * (kE4M3 ? 1 : 2);
    float q[G][DPL];
#pragma unroll
    for (int h = 0; h < G; ++h) {
      if (h < a.group) {
        const uint8_t* qr = Q + ((int64_t)b * a.hq + g * a.group + h) * qrow_bytes + lane * DPL * (kE4M3 ? 1 : 2);
        if constexpr (kE4M3)
          unpack_e4m3<DPL>(*reinterpret_cast<const uint32_t*>(qr), q[h]);
        else
          unpack_bf16<DPL>(*reinterpret_cast<const uint2*>(qr), q[h]);
      } else {
#pragma unroll
        for (int i = 0; i < DPL; ++i) q[h][i] = 0.f;
      }
#pragma unroll
      for (int i = 0; i < DPL; ++i) q[h][i] *= qscale;
    }
    const int my_h = lane / KPI, my_t = lane % KPI;
    float m = -INFINITY, l = 0.f;
    float o[G][DPL];
#pragma unroll
    for (int h = 0; h < G; ++h)
#pragma unroll
      for (int i = 0; i < DPL; ++i) o[h][i] = 0.f;
    for (int t = 0; t < ntiles; ++t) {
      const int s = t % kTmaStages;
      if (!tc::wait(&full[s], (uint32_t)(t / kTmaStages) & 1, a.status)) break;
      const uint8_t* st = dsm + s * kTmaStageBytes;
#pragma unroll
      for (int nb = 0; nb < NB; ++nb) {
        const int r0 = warp * RPW + nb * KPI;          // first row of the batch in the tile
        const int kb = k0 + t * kTmaTile + r0;         // its key index
        float v[32];
#pragma unroll
        for (int tt = 0; tt < KPI; ++tt) {
          float kx[DPL];
          row_at(st + (uint32_t)(r0 + tt) * 128, kx);
#pragma unroll
          for (int h = 0; h < G; ++h) {
            float acc = 0.f;
#pragma unroll
            for (int i = 0; i < DPL; ++i) acc = fmaf(q[h][i], kx[i], acc);
            v[h * KPI + tt] = acc;
          }
        }
#pragma unroll
        for (int o2 = 16; o2 >= 1; o2 >>= 1) {
          const bool hi = (lane & o2) != 0;
#pragma unroll
          for (int i = 0; i < o2; ++i) {
            const float send = hi ? v[i] : v[o2 + i];
            const float keep = hi ? v[o2 + i] : v[i];
            v[i] = keep + __shfl_xor_sync(0xffffffffu, send, o2);
          }
        }
        const float sc = (kb + my_t < k1) ? v[0] : -INFINITY;
        float mx = sc;
#pragma unroll
        for (int off = KPI / 2; off >= 1; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
        if (mx == -INFINITY) continue;  // the whole batch lies past the chunk (uniform per head group)
        const float m_new = fmaxf(m, mx);
        const float p = exp2f(sc - m_new);
        float ps = p;
#pragma unroll
        for (int off = KPI / 2; off >= 1; off >>= 1) ps += __shfl_xor_sync(0xffffffffu, ps, off);
        const float alpha = exp2f(m - m_new);
        l = l * alpha + ps;
        m = m_new;
#pragma unroll
        for (int h = 0; h < G; ++h) {
          const float ah = __shfl_sync(0xffffffffu, alpha, h * KPI);
#pragma unroll
          for (int i = 0; i < DPL; ++i) o[h][i] *= ah;
        }
#pragma unroll
        for (int tt = 0; tt < KPI; ++tt) {
          float vx[DPL];
          row_at(st + kTmaKV + (uint32_t)(r0 + tt) * 128, vx);
#pragma unroll
          for (int h = 0; h < G; ++h) {
            const float pht = __shfl_sync(0xffffffffu, p, h * KPI + tt);
#pragma unroll
            for (int i = 0; i < DPL; ++i) o[h][i] = fmaf(pht, vx[i], o[h][i]);
          }
        }
      }
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(&empty[s]);
    }
    if (my_t == 0) {
      sm_m[warp * G + my_h] = m;
      sm_l[warp * G + my_h] = l;
    }
#pragma unroll
    for (int h = 0; h < G; ++h)
#pragma unroll
      for (int i = 0; i < DPL; ++i) sm_o[(warp * G + h) * D + lane * DPL + i] = o[h][i];
  }
  __syncthreads();
  for (int idx = threadIdx.x; idx < a.group * D; idx += blockDim.x) {
    const int h = idx / D, d = idx % D;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < 4; ++w) M = fmaxf(M, sm_m[w * G + h]);
    float acc = 0.f, lsum = 0.f;
    if (M != -INFINITY) {
#pragma unroll
      for (int w = 0; w < 4; ++w) {
        const float f = exp2f(sm_m[w * G + h] - M);
        acc = fmaf(sm_o[(w * G + h) * D + d], f, acc);
        lsum = fmaf(sm_l[w * G + h], f, lsum);
      }
    }
    const int64_t pidx = ((int64_t)b * a.hq + g * a.group + h) * a.splits + split;
    a.part_o[pidx * D + d] = kE4M3 ? acc * a.v_descale : acc;
    if (d == 0) { a.part_ml[pidx * 2] = M; a.part_ml[pidx * 2 + 1] = lsum; }
  }
}

// grid B*Hq, block D threads.  Launched as a programmatic dependent of the
// split kernel: it may start while that kernel runs and waits for it (and
// its memory) before reading the partials.
template <int D>
__global__ void decode_combine_kernel(DecodeArgs a) {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int bh = blockIdx.x;
  const int d = threadIdx.x;
  const float* pml = a.part_ml + (int64_t)bh * a.splits * 2;
  // splits in chunks of eight with every load of a chunk issued before any
  // use (a split count below eight is one chunk); a split without keys (max
  // -inf) has weight 0 and its partial O, never written, is replaced by 0
  const float* po = a.part_o + (int64_t)bh * a.splits * D + d;
  float M = -INFINITY;
  for (int s0 = 0; s0 < a.splits; s0 += 8) {
    float ms[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) ms[u] = s0 + u < a.splits ? pml[2 * (s0 + u)] : -INFINITY;
#pragma unroll
    for (int u = 0; u < 8; ++u) M = fmaxf(M, ms[u]);
  }
  float acc = 0.f, L = 0.f;
  for (int s0 = 0; s0 < a.splits; s0 += 8) {
    float ms[8], ls[8], v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const bool in = s0 + u < a.splits;
      ms[u] = in ? pml[2 * (s0 + u)] : -INFINITY;
      ls[u] = in ? pml[2 * (s0 + u) + 1] : 0.f;
      v[u] = in ? po[(int64_t)(s0 + u) * D] : 0.f;
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const bool live = ms[u] != -INFINITY;
      const float f = live ? exp2f(ms[u] - M) : 0.f;
      acc = fmaf(live ? v[u] : 0.f, f, acc);
      L = fmaf(live ? ls[u] : 0.f, f, L);
    }
  }
  ((__nv_bfloat16*)a.out)[(int64_t)bh * D + d] = __float2bfloat16_rn(acc / L);
  const int b = bh / a.hq, h = bh % a.hq;
  if (a.lse && d == 0) a.lse[(int64_t)h * a.batch + b] = (M + log2f(L)) * 0.6931471805599453f;
  // the attention of this step has read the cache lengths: advance them
  if (a.cache_len && h == 0 && d == 0) a.cache_len[b] = a.c_snap[b] + 1;
}

// The combine as a programmatic dependent launch of the kernel before it.
template <int D>
cudaError_t launch_combine(const DecodeArgs& a, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(a.batch * a.hq));
  cfg.blockDim = dim3(D);
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, decode_combine_kernel<D>, a);
}

template <int D, int G>
cudaError_t run(const DecodeArgs& a, cudaStream_t st) {
  dim3 grid(a.splits, a.hkv, a.batch);
  cudaError_t e;
  // the TMA kernel needs at least two heads per KV head (batches of 32 / G keys)
  if (a.dtype == ISM_E4M3 && !(a.tma && G >= 2)) {
    if (D != 128) return cudaErrorInvalidValue;
    decode_split_kernel<D, G, true><<<grid, kDecWarps * 32, 0, st>>>(a);
  } else if (a.dtype == ISM_E4M3) {
    using Cfg = TmaCfg<G >= 2 ? G : 2, true>;
    CUtensorMap tk, tv;
    const uint64_t rows = (uint64_t)a.kv_rows;
    if ((e = tc::make_tmap_e4m3_plain(&tk, a.k_cache, (uint64_t)a.hkv * D, rows, Cfg::kTile)) != cudaSuccess) return e;
    if ((e = tc::make_tmap_e4m3_plain(&tv, a.v_cache, (uint64_t)a.hkv * D, rows, Cfg::kTile)) != cudaSuccess) return e;
    const int smem = Cfg::kStages * Cfg::kStageBytes + 2 * Cfg::kStages * 8 + (8 * G + 4 * G * D) * 4;
    if ((e = cudaFuncSetAttribute(decode_tma_kernel<G >= 2 ? G : 2, true>,
                                  cudaFuncAttributeMaxDynamicSharedMemorySize, smem)) != cudaSuccess)
      return e;
    decode_tma_kernel<G >= 2 ? G : 2, true><<<grid, 160, smem, st>>>(tk, tv, a);
  } else if (a.tma && G >= 2) {
    using Cfg = TmaCfg<G >= 2 ? G : 2>;
    CUtensorMap tk, tv;
    const uint64_t rows = (uint64_t)a.kv_rows;
    if ((e = tc::make_tmap_bf16_plain(&tk, a.k_cache, (uint64_t)a.hkv * D, rows, Cfg::kTile)) != cudaSuccess) return e;
    if ((e = tc::make_tmap_bf16_plain(&tv, a.v_cache, (uint64_t)a.hkv * D, rows, Cfg::kTile)) != cudaSuccess) return e;
    const int smem = Cfg::kStages * Cfg::kStageBytes + 2 * Cfg::kStages * 8 + (8 * G + 4 * G * D) * 4;
    if ((e = cudaFuncSetAttribute(decode_tma_kernel<G >= 2 ? G : 2>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  smem)) !=
        cudaSuccess)
      return e;
    decode_tma_kernel<G >= 2 ? G : 2><<<grid, 160, smem, st>>>(tk, tv, a);
  } else {
    decode_split_kernel<D, G><<<grid, kDecWarps * 32, 0, st>>>(a);
  }
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  return launch_combine<D>(a, st);
}

// the kernels take the group size padded to a power of two (a batch of 32 / G keys)
template <int D>
cudaError_t run_d(const DecodeArgs& a, cudaStream_t st) {
  const int grp = a.group;
  if (grp <= 1) return run<D, 1>(a, st);
  if (grp <= 2) return run<D, 2>(a, st);
  if (grp <= 4) return run<D, 4>(a, st);
  if (grp <= 8) return run<D, 8>(a, st);
  if (grp <= 16) return run<D, 16>(a, st);
  return cudaErrorInvalidValue;
}

}  // namespace

cudaError_t launch_decode(const DecodeArgs& a, cudaStream_t st) {
  if (a.batch == 0) return cudaSuccess;
  if (a.tc) {
    cudaError_t e = tc::launch_decode_tc(a, st);
    if (e != cudaSuccess) return e;
    return launch_combine<128>(a, st);
  }
  return a.d == 64 ? run_d<64>(a, st) : run_d<128>(a, st);
}

}  // namespace ism
