// Shared pieces of the sm_103a tensor-core kernels: tile geometry, TMA
// tensor maps, bounded waits with a wall-clock limit, and the 128B-swizzled
// shared-memory layout the TMA writes and tcgen05.mma reads.
#pragma once

#include <cuda.h>

#include "ism_internal.cuh"
#include "ptx.cuh"

namespace ism {
namespace tc {

constexpr int kD = 128;                       // head dim handled by the tensor-core kernels
constexpr int kRows = 128;                    // rows of a Q / K / V / P tile
constexpr uint32_t kHalfBytes = 128u * 128u;  // one 64-column half of a tile: 128 rows x 128 B
constexpr uint32_t kTileBytes = 2u * kHalfBytes;

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// A device-side wait gives up after this long (ns of %globaltimer).
constexpr uint64_t kWaitLimitNs = 2000000000ull;

__device__ __forceinline__ uint64_t globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Bounded mbarrier wait; on giving up records the timeout in the status word.
__device__ __forceinline__ bool wait(uint64_t* bar, uint32_t parity, uint32_t* status) {
  if (ptx::mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer();
  while (true) {
#pragma unroll 1
    for (int i = 0; i < 64; ++i)
      if (ptx::mbar_try_wait(bar, parity)) return true;
    if (globaltimer() - t0 > kWaitLimitNs) {
      atomicOr(status, kStatusTimeout);
      return false;
    }
  }
}

// Bounded wait of a whole (converged) warp: lane 0 polls the phase with the
// non-blocking test and the warp stays converged.  (A blocking try_wait by
// one lane while the other lanes wait at a warp barrier wakes up late.)
__device__ __forceinline__ bool wait_warp(uint64_t* bar, uint32_t parity, uint32_t* status) {
  if (ptx::mbar_test_warp(bar, parity)) return true;
  const uint64_t t0 = globaltimer();
  while (true) {
#pragma unroll 1
    for (int i = 0; i < 64; ++i)
      if (ptx::mbar_test_warp(bar, parity)) return true;
    if (__shfl_sync(0xffffffffu, (globaltimer() - t0 > kWaitLimitNs) ? 1 : 0, 0)) {
      if ((threadIdx.x & 31) == 0) atomicOr(status, kStatusTimeout);
      return false;
    }
  }
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Packed two-lane fp32 arithmetic (fma/add/mul .rn.f32x2, sm_100 and later):
// one instruction for two independent values, same rounding as the scalar forms.
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) {
  float2 d;
  asm("{\n .reg .b64 ra, rb, rc, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n mov.b64 rc, {%6, %7};\n"
      " fma.rn.f32x2 rd, ra, rb, rc;\n mov.b64 {%0, %1}, rd;\n}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  return d;
}
__device__ __forceinline__ float2 add2(float2 a, float2 b) {
  float2 d;
  asm("{\n .reg .b64 ra, rb, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n"
      " add.rn.f32x2 rd, ra, rb;\n mov.b64 {%0, %1}, rd;\n}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}
__device__ __forceinline__ float2 mul2(float2 a, float2 b) {
  float2 d;
  asm("{\n .reg .b64 ra, rb, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n"
      " mul.rn.f32x2 rd, ra, rb;\n mov.b64 {%0, %1}, rd;\n}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}
// Four values as e4m3 (round to nearest, saturating), x0 in the lowest byte.
__device__ __forceinline__ uint32_t pack_e4m3x4(float x0, float x1, float x2, float x3) {
  uint32_t r;
  asm("{\n .reg .b16 lo, hi;\n cvt.rn.satfinite.e4m3x2.f32 lo, %2, %1;\n cvt.rn.satfinite.e4m3x2.f32 hi, %4, %3;\n"
      " mov.b32 %0, {lo, hi};\n}"
      : "=r"(r)
      : "f"(x0), "f"(x1), "f"(x2), "f"(x3));
  return r;
}

// Store of a 32-column slice of 32 consecutive rows held one row per lane
// (thread = TMEM lane): w holds this lane's 32 bf16 values as 16 packed
// pairs.  Stored as they are, each 16-byte store instruction of the warp
// would write 32 different rows; instead the lanes of each group of four
// (rows 4m .. 4m + 3) exchange their 16-byte pieces, a 4 x 4 transpose in two
// xor-shuffle rounds, after which lane 4m + i holds piece i of the group's
// four rows, and each store instruction writes 8 rows of 64 contiguous
// bytes.  Every lane of the warp must call it (full-warp shuffles).
// group_row: the slice's first column in row 4m, the first row of this
// lane's group; rs: the row stride in elements; n_rows: how many of the
// group's rows exist (rows 4m + j with j >= n_rows are not stored).
__device__ __forceinline__ void store_slice32(uint32_t (&w)[16], __nv_bfloat16* group_row, int64_t rs, int n_rows) {
  const int lane = (int)(threadIdx.x & 31), li = lane & 3;
#pragma unroll
  for (int d = 2; d >= 1; d >>= 1) {
    const bool upper = (lane & d) != 0;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      if (k & d) continue;
      // pieces k and k + d: the lower lane of the pair keeps k and receives
      // the upper lane's k (into k + d); the upper keeps k + d and receives
      // the lower lane's k + d (into k)
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const uint32_t out = upper ? w[4 * k + c] : w[4 * (k | d) + c];
        const uint32_t in = __shfl_xor_sync(0xffffffffu, out, d);
        if (upper)
          w[4 * k + c] = in;
        else
          w[4 * (k | d) + c] = in;
      }
    }
  }
#pragma unroll
  for (int j = 0; j < 4; ++j)
    if (j < n_rows)
      *reinterpret_cast<uint4*>(group_row + j * rs + 8 * li) =
          make_uint4(w[4 * j], w[4 * j + 1], w[4 * j + 2], w[4 * j + 3]);
}

// 32 fp32 accumulator columns (bit patterns) scaled by f, as 16 bf16 pairs.
__device__ __forceinline__ void pack_scaled32(const uint32_t (&v)[32], float f, uint32_t (&w)[16]) {
#pragma unroll
  for (int k = 0; k < 16; ++k) w[k] = pack_bf16(__uint_as_float(v[2 * k]) * f, __uint_as_float(v[2 * k + 1]) * f);
}

// Gradient of a rotary-encoded head row (the rotation of the one-pass path
// pairs column k with k + 64).  rope_row<N> loads the cosines and sines of N
// pairs of a row's position (all loads issued before any use, so their
// latency is paid once; callers issue them well before the values are
// needed).  rope_back_pack: lo holds columns k0..k0+31 and hi columns
// k0+64..k0+95 of the gradient of the ROTATED row (fp32 bit patterns);
// after scaling by f, each pair (g_k, g_{k+64}) goes back through the
// transposed rotation, x_k = g_k c + g_{k+64} s and
// x_{k+64} = g_{k+64} c - g_k s, packed as bf16 pairs into wl (columns
// k0..) and wh (columns k0+64..) for store_slice32.  c and s point into
// register arrays at offsets fixed at compile time (the loops are unrolled).
template <int N>
__device__ __forceinline__ void rope_row(const float* __restrict__ cs, const float* __restrict__ sn, float* c,
                                         float* s) {
  static_assert(N % 4 == 0, "whole float4 loads");
#pragma unroll
  for (int i = 0; i < N / 4; ++i) {
    const float4 cv = __ldg(reinterpret_cast<const float4*>(cs) + i);
    const float4 sv = __ldg(reinterpret_cast<const float4*>(sn) + i);
    c[4 * i] = cv.x; c[4 * i + 1] = cv.y; c[4 * i + 2] = cv.z; c[4 * i + 3] = cv.w;
    s[4 * i] = sv.x; s[4 * i + 1] = sv.y; s[4 * i + 2] = sv.z; s[4 * i + 3] = sv.w;
  }
}
__device__ __forceinline__ void rope_back_pack(const uint32_t (&lo)[32], const uint32_t (&hi)[32], float f,
                                               const float* c, const float* s, uint32_t (&wl)[16],
                                               uint32_t (&wh)[16]) {
#pragma unroll
  for (int k = 0; k < 16; ++k) {
    float xl[2], xh[2];
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const int j = 2 * k + e;
      const float gl = __uint_as_float(lo[j]) * f, gh = __uint_as_float(hi[j]) * f;
      xl[e] = gl * c[j] + gh * s[j];
      xh[e] = gh * c[j] - gl * s[j];
    }
    wl[k] = pack_bf16(xl[0], xl[1]);
    wh[k] = pack_bf16(xh[0], xh[1]);
  }
}

// Work item i of a list of n_tiles x n_heads items whose tiles come in cost
// order (most expensive first).  The tiles are taken in four buckets of a
// quarter of the list each, and inside a bucket head by head: the CTAs that
// run at the same time then work on one head of neighbouring tiles, which
// stream the same operand tiles (K / V in the forward, Q / dO in dK/dV) in
// the same order, so those reads mostly hit L2.  Taking the heads of a tile
// one after the other instead spreads the CTAs over all heads, which with
// one query head per KV head leaves almost no operand tile shared.
// With bucketed == false the order is the plain one (the heads of a tile
// one after the other), which keeps the cost order exact: the statically
// scheduled kernels take it whenever the heads of a tile already share
// operands (two or more query heads per KV head).
__device__ __forceinline__ void bucket_item(int64_t i, int64_t n_tiles, int n_heads, int64_t& tile_pos, int& head,
                                            bool bucketed = true) {
  if (!bucketed) {
    tile_pos = i / n_heads;
    head = (int)(i % n_heads);
    return;
  }
  const int64_t bt = (n_tiles + 3) / 4;
  const int64_t per_bucket = bt * n_heads;
  const int64_t b = i / per_bucket;
  const int64_t w = i - b * per_bucket;
  const int64_t t0 = b * bt;
  const int64_t nb = n_tiles - t0 < bt ? n_tiles - t0 : bt;
  head = (int)(w / nb);
  tile_pos = t0 + w % nb;
}

// Byte offset of element (r, c) of a [128 x 128] bf16 tile in the layout a
// 128B-swizzled TMA box of 64 columns x 128 rows produces (two such boxes,
// one per 64-column half): 16-byte chunk index XOR (row mod 8).
__host__ __device__ __forceinline__ uint32_t swz_offset(uint32_t r, uint32_t c) {
  return (c >> 6) * kHalfBytes + r * 128u + ((((c & 63u) >> 3) ^ (r & 7u)) << 4) + (c & 7u) * 2u;
}

// Descriptor of k-step kk (16 elements of K) of a K-major tile (rows = M or
// N, 128 K columns in two 64-column swizzled halves).
__device__ __forceinline__ uint64_t desc_kmajor(uint32_t tile_saddr, int kk) {
  return ptx::smem_desc(tile_saddr + (uint32_t)(kk >> 2) * kHalfBytes + (uint32_t)(kk & 3) * 32u, 16u, 1024u,
                        ptx::kSwizzle128B);
}

// Descriptor of k-step kk (16 rows of K) of an MN-major tile stored as
// [128 K rows x 128 N columns] (two 64-column swizzled halves): 8-row groups
// are 1024 B apart (stride offset), the halves 16 KB apart (leading offset).
__device__ __forceinline__ uint64_t desc_mnmajor(uint32_t tile_saddr, int kk) {
  return ptx::smem_desc(tile_saddr + (uint32_t)kk * 2048u, kHalfBytes, 1024u, ptx::kSwizzle128B);
}

// 8-interleaved MN-major tile, no swizzle: element (mn, k) of a
// [128 MN x 128 K] operand at byte ((mn / 8) * 128 + k) * 16 + (mn % 8) * 2,
// i.e. 16-byte units of 8 consecutive MN elements, K-consecutive units
// adjacent.  A core matrix (8 MN x 8 K) is 128 contiguous bytes; the next
// 8 K rows are 128 bytes on (leading offset), the next 8 MN columns 2048
// bytes on (stride offset).  k-step kk (16 K rows) starts 256 bytes on.
constexpr uint32_t kIlvUnitRow = 128 * 16;  // bytes between MN groups of 8
__host__ __device__ constexpr uint32_t ilv_offset(int mn, int k) {
  return (uint32_t)(mn >> 3) * kIlvUnitRow + (uint32_t)k * 16u + (uint32_t)(mn & 7) * 2u;
}
__device__ __forceinline__ uint64_t desc_ilv_mnmajor(uint32_t tile_saddr, int kk) {
  return ptx::smem_desc(tile_saddr + (uint32_t)kk * 256u, 128u, kIlvUnitRow, ptx::kSwizzleNone);
}

// Host: 2D bf16 tensor map [rows, cols] with a 64 x 128 box, 128B swizzle.
cudaError_t make_tmap_bf16(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows);
// Host: the same with a 64-column x box_rows box (box_rows <= 256).
cudaError_t make_tmap_bf16_box(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows, uint32_t box_rows);
// Host: 2D e4m3 tensor map with a 128-column (128-byte) x box_rows box, 128B swizzle.
cudaError_t make_tmap_e4m3_box(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows, uint32_t box_rows);
// Host: 2D bf16 tensor map with a 64-column x box_rows box, no swizzle.
cudaError_t make_tmap_bf16_plain(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows, uint32_t box_rows);
// 1-byte elements, box of 128 columns x box_rows, no swizzle
cudaError_t make_tmap_e4m3_plain(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows, uint32_t box_rows);
// Host: true on an sm_103 device with the tensor-map encoder available.
bool available();
// Host: forward with two query heads (sharing a KV head) per CTA.
cudaError_t launch_fwd_pair(const AttnArgs& a, const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                            cudaStream_t st);
// Host: single-token decode on the tensor cores (bf16 caches, head_dim 128,
// at most 16 query heads per KV head; a.chunk a multiple of 128, at most
// kDecTcMaxKeys): partials for decode_combine_kernel.
cudaError_t launch_decode_tc(const DecodeArgs& a, cudaStream_t st);
// Host: dQ as a GEMM over the dS^T tiles stored by the dK/dV kernel (a.ds).
cudaError_t launch_dq_gemm(const AttnArgs& a, const CUtensorMap& tk, cudaStream_t st);

}  // namespace tc
}  // namespace ism
