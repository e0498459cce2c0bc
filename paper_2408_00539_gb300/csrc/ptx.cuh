// Inline-PTX building blocks for sm_103a (Blackwell): mbarriers with bounded
// waits, TMA tiled loads, tcgen05 tensor-memory allocation / MMA / loads,
// and the descriptors they take.  Written from the public PTX ISA.
#pragma once

#include <cuda.h>
#include <stdint.h>

namespace ism {
namespace ptx {

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ bool elect_lane0() { return (threadIdx.x & 31) == 0; }

// ---------------------------------------------------------------- mbarrier

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("{\n .reg .b64 st;\n mbarrier.arrive.shared::cta.b64 st, [%0];\n}" ::"r"(smem_u32(bar))
               : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("{\n .reg .b64 st;\n mbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n}" ::"r"(
                   smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Non-blocking test of phase completion.
__device__ __forceinline__ bool mbar_test(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait: polls at most `limit` times (each poll may suspend the thread
// for a hardware-chosen interval).  Returns false on giving up.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, uint32_t limit) {
  for (uint32_t i = 0; i < limit; ++i)
    if (mbar_try_wait(bar, parity)) return true;
  return false;
}

// ---------------------------------------------------------------- fences

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// ---------------------------------------------------------------- TMA

__device__ __forceinline__ void tma_prefetch_desc(const void* tmap) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(tmap)) : "memory");
}

// 2D tiled load global -> shared, completion counted on `bar` in bytes.
// x is the innermost (contiguous) coordinate in elements, y the row.
__device__ __forceinline__ void tma_load_2d(void* smem_dst, const void* tmap, uint64_t* bar, int32_t x,
                                            int32_t y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], "
      "[%2];" ::"r"(smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(smem_u32(bar)), "r"(x), "r"(y)
      : "memory");
}

// Contiguous (non-tensor) bulk copy global -> shared of `bytes` (a multiple
// of 16; both addresses 16-byte aligned), completion counted on `bar`.
__device__ __forceinline__ void bulk_load(void* smem_dst, const void* gsrc, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(gsrc)), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// L2 eviction priorities for copies: a policy word from createpolicy, passed
// to the .L2::cache_hint forms below.  evict_first suits data read once
// (streamed), evict_last data that other CTAs read again soon.
__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t l2_policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ void st_global_v4_hint(void* gdst, const uint4& v, uint64_t policy) {
  asm volatile("st.global.L2::cache_hint.v4.b32 [%0], {%1, %2, %3, %4}, %5;" ::"l"(gdst), "r"(v.x), "r"(v.y),
               "r"(v.z), "r"(v.w), "l"(policy)
               : "memory");
}
__device__ __forceinline__ void tma_load_2d_hint(void* smem_dst, const void* tmap, uint64_t* bar, int32_t x,
                                                 int32_t y, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint [%0], "
      "[%1, {%3, %4}], [%2], %5;" ::"r"(smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(smem_u32(bar)), "r"(x), "r"(y), "l"(policy)
      : "memory");
}
__device__ __forceinline__ void bulk_load_hint(void* smem_dst, const void* gsrc, uint32_t bytes, uint64_t* bar,
                                               uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
          smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(gsrc)), "r"(bytes), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}

// ---------------------------------------------------------------- tcgen05

// Allocate `ncols` (power of two >= 32) TMEM columns; the base address is
// written to shared memory at `dst`.  Whole warp.
__device__ __forceinline__ void tmem_alloc(uint32_t* dst, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(dst)),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, kind::f16 (bf16/f16 inputs, fp32 accumulate).
__device__ __forceinline__ void mma_bf16_ss(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// D[tmem] (+)= A[tmem] * B[smem]^T: A read from tensor memory (row m in lane
// m, two bf16 of K per 32-bit column).
__device__ __forceinline__ void mma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Warp-converged forms: every lane of the warp executes the instruction and
// one lane chosen by elect.sync issues it.  The issuing warp stays converged,
// which keeps MMA issue at the tensor-pipe rate while other warps of the same
// scheduler are busy (a single-lane branch issuing MMAs loses about half of
// that rate there).  The whole warp must be converged at the call.
__device__ __forceinline__ void mma_bf16_ss_warp(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                                 uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred e, p;\n elect.sync _|e, 0xffffffff;\n setp.ne.b32 p, %4, 0;\n"
      " @e tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void mma_bf16_ts_warp(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                                 uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred e, p;\n elect.sync _|e, 0xffffffff;\n setp.ne.b32 p, %4, 0;\n"
      " @e tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// The eight k-steps (K = 128 in steps of 16) of one 128 x N contraction,
// issued by one elected lane of a converged warp: the other lanes branch past
// the block, so the whole sequence costs one election, and the operands of
// k-step kk are formed inside the block as the first ones plus a fixed offset
//   offset(kk) = (kk % 4) * kStep + (kk / 4) * kHalf
// (descriptors in units of 16 bytes: the address field is the low 14 bits and
// every tile lies inside the 256 KB it spans, so the sum never carries out;
// tensor-memory A operands in columns).  Layouts used:
//   KMajorSw128    K-major, 128-byte swizzled, two 64-column halves 16 KB apart
//   MnMajorSw128   MN-major, 128-byte swizzled, 2 KB a k-step
//   MnMajorIlv8    8-interleaved MN-major, 256 bytes a k-step
//   TmemPairs      bf16 pairs in tensor memory, 8 columns a k-step
//   TmemPairsGap32 the same with a 32-column gap after k-step 3
//   KMajorSw128Rows16  K-major, 128-byte swizzled, 16-row operand (halves 2 KB apart)
// k-step 0 accumulates when acc != 0, the others always.
struct KMajorSw128 { static constexpr uint32_t step = 2, half = 1024; };
struct MnMajorSw128 { static constexpr uint32_t step = 128, half = 512; };
struct MnMajorIlv8 { static constexpr uint32_t step = 16, half = 64; };
struct TmemPairs { static constexpr uint32_t step = 8, half = 32; };
struct TmemPairsGap32 { static constexpr uint32_t step = 8, half = 64; };
// K-major, 128-byte swizzled, 16 rows: two 64-column halves 2 KB apart
struct KMajorSw128Rows16 { static constexpr uint32_t step = 2, half = 128; };
template <class LA, class LB, uint32_t kAStep = LA::step, uint32_t kAHalf = LA::half, uint32_t kBStep = LB::step,
          uint32_t kBHalf = LB::half>
__device__ __forceinline__ void mma8_bf16_ss_warp(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                                  uint32_t acc) {
  asm volatile(
      "{\n .reg .pred e, p, t;\n .reg .b64 a1, a2, a3, a4, a5, a6, a7, b1, b2, b3, b4, b5, b6, b7;\n"
      " elect.sync _|e, 0xffffffff;\n @!e bra MMA8_SS_DONE;\n"
      " setp.ne.b32 p, %4, 0;\n setp.eq.u32 t, 0, 0;\n"
      " add.s64 a1, %1, %5; add.s64 a2, %1, %6; add.s64 a3, %1, %7; add.s64 a4, %1, %8;\n"
      " add.s64 a5, %1, %9; add.s64 a6, %1, %10; add.s64 a7, %1, %11;\n"
      " add.s64 b1, %2, %12; add.s64 b2, %2, %13; add.s64 b3, %2, %14; add.s64 b4, %2, %15;\n"
      " add.s64 b5, %2, %16; add.s64 b6, %2, %17; add.s64 b7, %2, %18;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], a1, b1, %3, t;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], a2, b2, %3, t;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], a3, b3, %3, t;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], a4, b4, %3, t;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], a5, b5, %3, t;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], a6, b6, %3, t;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], a7, b7, %3, t;\n"
      " MMA8_SS_DONE:\n}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(acc), "n"(kAStep), "n"(2 * kAStep), "n"(3 * kAStep), "n"(kAHalf),
      "n"(kAHalf + kAStep), "n"(kAHalf + 2 * kAStep), "n"(kAHalf + 3 * kAStep), "n"(kBStep), "n"(2 * kBStep),
      "n"(3 * kBStep), "n"(kBHalf), "n"(kBHalf + kBStep), "n"(kBHalf + 2 * kBStep), "n"(kBHalf + 3 * kBStep)
      : "memory");
}
template <class LA, class LB, uint32_t kAStep = LA::step, uint32_t kAHalf = LA::half, uint32_t kBStep = LB::step,
          uint32_t kBHalf = LB::half>
__device__ __forceinline__ void mma8_bf16_ts_warp(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                                  uint32_t acc) {
  asm volatile(
      "{\n .reg .pred e, p, t;\n .reg .b32 a1, a2, a3, a4, a5, a6, a7;\n"
      " .reg .b64 b1, b2, b3, b4, b5, b6, b7;\n"
      " elect.sync _|e, 0xffffffff;\n @!e bra MMA8_TS_DONE;\n"
      " setp.ne.b32 p, %4, 0;\n setp.eq.u32 t, 0, 0;\n"
      " add.u32 a1, %1, %5; add.u32 a2, %1, %6; add.u32 a3, %1, %7; add.u32 a4, %1, %8;\n"
      " add.u32 a5, %1, %9; add.u32 a6, %1, %10; add.u32 a7, %1, %11;\n"
      " add.s64 b1, %2, %12; add.s64 b2, %2, %13; add.s64 b3, %2, %14; add.s64 b4, %2, %15;\n"
      " add.s64 b5, %2, %16; add.s64 b6, %2, %17; add.s64 b7, %2, %18;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [a1], b1, %3, t;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [a2], b2, %3, t;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [a3], b3, %3, t;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [a4], b4, %3, t;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [a5], b5, %3, t;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [a6], b6, %3, t;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [a7], b7, %3, t;\n"
      " MMA8_TS_DONE:\n}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(acc), "n"(kAStep), "n"(2 * kAStep), "n"(3 * kAStep), "n"(kAHalf),
      "n"(kAHalf + kAStep), "n"(kAHalf + 2 * kAStep), "n"(kAHalf + 3 * kAStep), "n"(kBStep), "n"(2 * kBStep),
      "n"(3 * kBStep), "n"(kBHalf), "n"(kBHalf + kBStep), "n"(kBHalf + 2 * kBStep), "n"(kBHalf + 3 * kBStep)
      : "memory");
}
__device__ __forceinline__ void mma_commit_warp(uint64_t* bar) {
  asm volatile(
      "{\n .reg .pred e;\n elect.sync _|e, 0xffffffff;\n"
      " @e tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n}" ::"r"(smem_u32(bar))
      : "memory");
}
// mbarrier phase test by every lane of a converged warp, combined by a vote
// (warp-uniform result).
__device__ __forceinline__ bool mbar_test_warp(uint64_t* bar, uint32_t parity) {
  return __all_sync(0xffffffffu, mbar_test(bar, parity));
}

// Make `bar` track completion of all prior tcgen05.mma of this thread.
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   smem_u32(bar))
               : "memory");
}

// Each thread of the warp reads 32 consecutive 32-bit columns of its lane
// (lane = warp_in_quadrant*32 + laneid).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}

__device__ __forceinline__ void tmem_ld8(uint32_t taddr, uint32_t (&r)[8]) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
               : "r"(taddr));
}

__device__ __forceinline__ void tmem_ld4(uint32_t taddr, uint32_t (&r)[4]) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x4.b32 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(taddr));
}

__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
      "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]),
      "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]),
      "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}

__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// Ties registers written by an asynchronous tcgen05.ld to a point after
// tcgen05.wait::ld, so the compiler cannot move their uses above the wait.
template <int N>
__device__ __forceinline__ void reg_fence(uint32_t (&r)[N]) {
#pragma unroll
  for (int i = 0; i < N; ++i) asm volatile("" : "+r"(r[i]));
}
__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// Shared-memory matrix descriptor (tcgen05 format): start address, leading
// and stride byte offsets (all >> 4), version 1, swizzle mode.
enum : uint32_t { kSwizzleNone = 0, kSwizzle128B = 2, kSwizzle64B = 4, kSwizzle32B = 6 };
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr, uint32_t lbo_bytes, uint32_t sbo_bytes,
                                              uint32_t swizzle) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr >> 4) & 0x3FFFu);
  d |= (uint64_t)((lbo_bytes >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo_bytes >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1 << 46;  // descriptor version for tcgen05
  d |= (uint64_t)(swizzle & 0x7u) << 61;
  return d;
}

// Instruction descriptor for kind::f16 with bf16 A/B and fp32 D.
// a_mn / b_mn: operand is MN-major (transposed) instead of K-major.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(uint32_t m, uint32_t n, uint32_t a_mn, uint32_t b_mn) {
  return (1u << 4)            // D format: f32
         | (1u << 7)          // A format: bf16
         | (1u << 10)         // B format: bf16
         | (a_mn << 15)       // A major
         | (b_mn << 16)       // B major
         | ((n >> 3) << 17)   // N / 8
         | ((m >> 4) << 24);  // M / 16
}

// Four k-steps (K = 64) of a bf16 TS contraction, issued like mma8_bf16_ts_warp.
template <uint32_t kAStep, uint32_t kBStep>
__device__ __forceinline__ void mma4_bf16_ts_warp(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                                  uint32_t acc) {
  asm volatile(
      "{\n .reg .pred e, p, t;\n .reg .b32 a1, a2, a3;\n .reg .b64 b1, b2, b3;\n"
      " elect.sync _|e, 0xffffffff;\n @!e bra MMA4_BF_DONE;\n"
      " setp.ne.b32 p, %4, 0;\n setp.eq.u32 t, 0, 0;\n"
      " add.u32 a1, %1, %5; add.u32 a2, %1, %6; add.u32 a3, %1, %7;\n"
      " add.s64 b1, %2, %8; add.s64 b2, %2, %9; add.s64 b3, %2, %10;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [a1], b1, %3, t;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [a2], b2, %3, t;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [a3], b3, %3, t;\n"
      " MMA4_BF_DONE:\n}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(acc), "n"(kAStep), "n"(2 * kAStep), "n"(3 * kAStep), "n"(kBStep),
      "n"(2 * kBStep), "n"(3 * kBStep)
      : "memory");
}

// Instruction descriptor for kind::f8f6f4 with e4m3 A/B and fp32 D (K = 32 a step).
__host__ __device__ constexpr uint32_t idesc_e4m3_f32(uint32_t m, uint32_t n, uint32_t a_mn, uint32_t b_mn) {
  return (1u << 4)            // D format: f32
         | (0u << 7)          // A format: e4m3
         | (0u << 10)         // B format: e4m3
         | (a_mn << 15)       // A major
         | (b_mn << 16)       // B major
         | ((n >> 3) << 17)   // N / 8
         | ((m >> 4) << 24);  // M / 16
}

// The four k-steps (K = 128 in steps of 32) of one 128 x N e4m3 contraction
// (kind::f8f6f4), issued like mma8_bf16_*_warp: one elected lane, k-step kk
// at the first operands plus kk * kStep.  Layouts (kStep):
//   K-major, 128-byte swizzled, 128-byte rows:  2 (32 bytes)
//   MN-major, 128-byte swizzled, 128-byte rows: 256 (32 rows of 128 bytes)
//   e4m3 quads in tensor memory:                8 columns
template <uint32_t kAStep, uint32_t kBStep>
__device__ __forceinline__ void mma4_e4m3_ss_warp(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                                  uint32_t acc) {
  asm volatile(
      "{\n .reg .pred e, p, t;\n .reg .b64 a1, a2, a3, b1, b2, b3;\n"
      " elect.sync _|e, 0xffffffff;\n @!e bra MMA4_SS_DONE;\n"
      " setp.ne.b32 p, %4, 0;\n setp.eq.u32 t, 0, 0;\n"
      " add.s64 a1, %1, %5; add.s64 a2, %1, %6; add.s64 a3, %1, %7;\n"
      " add.s64 b1, %2, %8; add.s64 b2, %2, %9; add.s64 b3, %2, %10;\n"
      " tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n"
      " tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], a1, b1, %3, t;\n"
      " tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], a2, b2, %3, t;\n"
      " tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], a3, b3, %3, t;\n"
      " MMA4_SS_DONE:\n}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(acc), "n"(kAStep), "n"(2 * kAStep), "n"(3 * kAStep), "n"(kBStep),
      "n"(2 * kBStep), "n"(3 * kBStep)
      : "memory");
}
template <uint32_t kAStep, uint32_t kBStep>
__device__ __forceinline__ void mma4_e4m3_ts_warp(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                                  uint32_t acc) {
  asm volatile(
      "{\n .reg .pred e, p, t;\n .reg .b32 a1, a2, a3;\n .reg .b64 b1, b2, b3;\n"
      " elect.sync _|e, 0xffffffff;\n @!e bra MMA4_TS_DONE;\n"
      " setp.ne.b32 p, %4, 0;\n setp.eq.u32 t, 0, 0;\n"
      " add.u32 a1, %1, %5; add.u32 a2, %1, %6; add.u32 a3, %1, %7;\n"
      " add.s64 b1, %2, %8; add.s64 b2, %2, %9; add.s64 b3, %2, %10;\n"
      " tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], [%1], %2, %3, p;\n"
      " tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], [a1], b1, %3, t;\n"
      " tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], [a2], b2, %3, t;\n"
      " tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], [a3], b3, %3, t;\n"
      " MMA4_TS_DONE:\n}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(acc), "n"(kAStep), "n"(2 * kAStep), "n"(3 * kAStep), "n"(kBStep),
      "n"(2 * kBStep), "n"(3 * kBStep)
      : "memory");
}

// ---------------------------------------------------------------- CTA pairs (cluster of two)
// The pair's MMAs (cta_group::2) are issued by the even CTA; each CTA holds
// its half of A (rows) and of B (columns of N) at the same shared-memory
// offsets, and its own rows of D in its own tensor memory.

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// Every thread of both CTAs: arrive (release) and wait (acquire) at the cluster barrier.
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Shared-memory address of `p` (a shared::cta object) in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t cluster_addr(const void* p, uint32_t rank) {
  uint32_t a;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(a) : "r"(smem_u32(p)), "r"(rank));
  return a;
}
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_bar) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_bar) : "memory");
}
// Arrival without release semantics: for hand-offs whose data the sender has
// already completed by other means (tensor-memory stores waited for with
// tcgen05.wait::st), so that the arrival does not wait for the sender's
// unrelated global stores to become visible across the cluster.
__device__ __forceinline__ void mbar_arrive_cluster_relaxed(uint32_t cluster_bar) {
  asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_bar) : "memory");
}
__device__ __forceinline__ void st_cluster_u32(uint32_t cluster_addr_, uint32_t v) {
  asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(cluster_addr_), "r"(v) : "memory");
}
// Phase test with cluster-scope acquire (for barriers that CTAs of the pair arrive on).
__device__ __forceinline__ bool mbar_test_cluster(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.test_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool mbar_test_cluster_warp(uint64_t* bar, uint32_t parity) {
  return __all_sync(0xffffffffu, mbar_test_cluster(bar, parity));
}
// Tensor memory for the pair: one warp of each CTA, the same column count.
__device__ __forceinline__ void tmem_alloc_pair(uint32_t* dst, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(dst)), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish_pair() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
// Completion of the pair's MMAs issued so far, signalled on the barrier at
// the same offset in both CTAs.
__device__ __forceinline__ void mma_commit_pair_warp(uint64_t* bar) {
  asm volatile(
      "{\n .reg .pred e;\n elect.sync _|e, 0xffffffff;\n"
      " @e tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;\n}" ::"r"(
          smem_u32(bar)),
      "h"((uint16_t)3)
      : "memory");
}
// Eight k-steps of a pair MMA (M = 256), issued like mma8_bf16_ss_warp / _ts_warp.
template <class LA, class LB, uint32_t kAStep = LA::step, uint32_t kAHalf = LA::half, uint32_t kBStep = LB::step,
          uint32_t kBHalf = LB::half>
__device__ __forceinline__ void mma8_bf16_ss_pair_warp(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                                       uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n .reg .pred e, p, t;\n .reg .b64 a1, a2, a3, a4, a5, a6, a7, b1, b2, b3, b4, b5, b6, b7;\n"
      " elect.sync _|e, 0xffffffff;\n @!e bra MMA8_SSP_DONE;\n"
      " setp.ne.b32 p, %4, 0;\n setp.eq.u32 t, 0, 0;\n"
      " add.s64 a1, %1, %5; add.s64 a2, %1, %6; add.s64 a3, %1, %7; add.s64 a4, %1, %8;\n"
      " add.s64 a5, %1, %9; add.s64 a6, %1, %10; add.s64 a7, %1, %11;\n"
      " add.s64 b1, %2, %12; add.s64 b2, %2, %13; add.s64 b3, %2, %14; add.s64 b4, %2, %15;\n"
      " add.s64 b5, %2, %16; add.s64 b6, %2, %17; add.s64 b7, %2, %18;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], a1, b1, %3, t;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], a2, b2, %3, t;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], a3, b3, %3, t;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], a4, b4, %3, t;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], a5, b5, %3, t;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], a6, b6, %3, t;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], a7, b7, %3, t;\n"
      " MMA8_SSP_DONE:\n}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(acc), "n"(kAStep), "n"(2 * kAStep), "n"(3 * kAStep), "n"(kAHalf),
      "n"(kAHalf + kAStep), "n"(kAHalf + 2 * kAStep), "n"(kAHalf + 3 * kAStep), "n"(kBStep), "n"(2 * kBStep),
      "n"(3 * kBStep), "n"(kBHalf), "n"(kBHalf + kBStep), "n"(kBHalf + 2 * kBStep), "n"(kBHalf + 3 * kBStep)
      : "memory");
}
template <class LA, class LB, uint32_t kAStep = LA::step, uint32_t kAHalf = LA::half, uint32_t kBStep = LB::step,
          uint32_t kBHalf = LB::half>
__device__ __forceinline__ void mma8_bf16_ts_pair_warp(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc,
                                                       uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n .reg .pred e, p, t;\n .reg .b32 a1, a2, a3, a4, a5, a6, a7;\n"
      " .reg .b64 b1, b2, b3, b4, b5, b6, b7;\n"
      " elect.sync _|e, 0xffffffff;\n @!e bra MMA8_TSP_DONE;\n"
      " setp.ne.b32 p, %4, 0;\n setp.eq.u32 t, 0, 0;\n"
      " add.u32 a1, %1, %5; add.u32 a2, %1, %6; add.u32 a3, %1, %7; add.u32 a4, %1, %8;\n"
      " add.u32 a5, %1, %9; add.u32 a6, %1, %10; add.u32 a7, %1, %11;\n"
      " add.s64 b1, %2, %12; add.s64 b2, %2, %13; add.s64 b3, %2, %14; add.s64 b4, %2, %15;\n"
      " add.s64 b5, %2, %16; add.s64 b6, %2, %17; add.s64 b7, %2, %18;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], [%1], %2, %3, p;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], [a1], b1, %3, t;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], [a2], b2, %3, t;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], [a3], b3, %3, t;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], [a4], b4, %3, t;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], [a5], b5, %3, t;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], [a6], b6, %3, t;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], [a7], b7, %3, t;\n"
      " MMA8_TSP_DONE:\n}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(acc), "n"(kAStep), "n"(2 * kAStep), "n"(3 * kAStep), "n"(kAHalf),
      "n"(kAHalf + kAStep), "n"(kAHalf + 2 * kAStep), "n"(kAHalf + 3 * kAStep), "n"(kBStep), "n"(2 * kBStep),
      "n"(3 * kBStep), "n"(kBHalf), "n"(kBHalf + kBStep), "n"(kBHalf + 2 * kBStep), "n"(kBHalf + 3 * kBStep)
      : "memory");
}
// K-major, 128-byte swizzled, 64-row operand whose two 64-column halves are 8 KB apart
struct KMajorSw128Half8K { static constexpr uint32_t step = 2, half = 512; };

}  // namespace ptx
}  // namespace ism
