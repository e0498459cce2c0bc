// dQ of ISM attention as a GEMM over stored dS tiles (sm_103a).
//
// When the dK/dV kernel has kept every visible tile pair's dS (bf16, 128
// queries x 128 keys, 32 KiB a tile) in the workspace, dQ_t = scale *
// sum_c dS_tc K_c needs no recomputation of S, P or dP.  A persistent CTA per
// SM walks the (query tile, query head) items in cost order; for each it
// streams the (dS, K) tile pairs of the tile's non-empty key blocks through a
// 3-stage ring that runs on across items, and accumulates dQ in one of two
// tensor-memory accumulators, so the epilogue of one item overlaps the MMAs
// of the next.
// A dS tile is stored 8-interleaved (16-byte units of 8 consecutive queries
// of one key, the 128 keys of a query group adjacent), which is the no-swizzle
// MN-major operand layout: one contiguous bulk copy moves it into shared
// memory as the A operand (M = queries).  K arrives by TMA in the 128-byte
// swizzled layout as the MN-major B operand.
// Warps 0-3 epilogue (thread = query row), warp 4 copy producer, warp 5 MMA.
#include "ism_tc_common.cuh"

namespace ism {
namespace tc {
namespace {

constexpr int kThreads = 192;
constexpr int kStages = 3;
constexpr uint32_t kStageBytes = 2 * kTileBytes;  // dS tile + K tile
constexpr uint32_t OFF_BAR = kStages * kStageBytes;
constexpr uint32_t kSmemBytes = OFF_BAR + 128 + 1024;
constexpr uint32_t kTmemCols = 256;  // two 128-column dQ accumulators

struct Bars {
  uint64_t full[kStages], empty[kStages], acc_full[2], acc_empty[2], final_mma;
  uint32_t tmem_base;
  int32_t abort;
};
static_assert(sizeof(Bars) <= 128, "barrier block");

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}
__device__ __forceinline__ bool aborted(const int32_t* f) { return *reinterpret_cast<const volatile int32_t*>(f) != 0; }
__device__ __forceinline__ void set_abort(int32_t* f) { *reinterpret_cast<volatile int32_t*>(f) = 1; }

// Work item `item` = (query tile q_order[item / hq], query head item % hq).
struct Item {
  int h, g, t, nkb, gfirst;
  Tile w;
};
__device__ __forceinline__ Item decode(const AttnArgs& a, int64_t item) {
  Item it;
  int64_t tpos;
  bucket_item(item, a.nq, a.hq, tpos, it.h, a.hq == a.hkv);  // bucketed only when no two heads share K
  const int gq = a.q_order[tpos];
  it.w = a.qtiles[gq];
  it.g = it.h / (a.hq / a.hkv);
  it.nkb = it.w.a1;
  it.t = it.w.tile;
  it.gfirst = gq - it.t;  // q-tiles and k-tiles of a sequence are numbered alike
  return it;
}

__global__ void __launch_bounds__(kThreads, 1)
    dq_gemm_kernel(const __grid_constant__ CUtensorMap tmK, const AttnArgs a, int64_t n_items) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  Bars* bar = reinterpret_cast<Bars*>(smem + OFF_BAR);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      ptx::mbar_init(&bar->full[s], 1);
      ptx::mbar_init(&bar->empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      ptx::mbar_init(&bar->acc_full[b], 1);
      ptx::mbar_init(&bar->acc_empty[b], 128);
    }
    ptx::mbar_init(&bar->final_mma, 1);
    bar->abort = 0;
    ptx::fence_mbar_init();
  }
  if (warp == 5) {
    ptx::tmem_alloc(&bar->tmem_base, kTmemCols);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = bar->tmem_base;

  if (warp == 4) {
    // ------------------------------------------------ copies (the warp waits converged, lane 0 issues)
    uint32_t it = 0;  // stage uses so far, across items
    uint32_t nf[kStages] = {0, 0, 0};
    bool ok = true;
    // each dS tile is read once; K tiles are read by every query tile and head
    // of their sequence, so keep them in L2 ahead of the dS stream
    const uint64_t pol_ds = ptx::l2_policy_evict_first(), pol_k = ptx::l2_policy_evict_last();
    for (int64_t item = blockIdx.x; ok && item < n_items; item += gridDim.x) {
      const Item x = decode(a, item);
      for (int c = 0; c < x.nkb; ++c, ++it) {
        const int s = (int)(it % kStages);
        if (__any_sync(0xffffffffu, aborted(&bar->abort))) { ok = false; break; }
        if (it >= kStages && !wait_warp(&bar->empty[s], (it / kStages - 1) & 1, a.status)) {
          if (lane == 0) set_abort(&bar->abort);
          ok = false;
          break;
        }
        if (lane == 0) {
          const int gk = x.gfirst + c;
          const int64_t slot = ((int64_t)a.kpair_off[gk] + (x.t - a.ktiles[gk].a0)) * a.hq + x.h;
          const int32_t yk = x.w.k_base + c * kRows;
          uint8_t* st = smem + s * kStageBytes;
          ptx::mbar_expect_tx(&bar->full[s], kStageBytes);
          ptx::bulk_load_hint(st, static_cast<const uint8_t*>(a.ds) + slot * kTileBytes, kTileBytes, &bar->full[s],
                              pol_ds);
          ptx::tma_load_2d_hint(st + kTileBytes, &tmK, &bar->full[s], x.g * kD, yk, pol_k);
          ptx::tma_load_2d_hint(st + kTileBytes + kHalfBytes, &tmK, &bar->full[s], x.g * kD + 64, yk, pol_k);
        }
        __syncwarp();
        ++nf[s];
      }
    }
    if (!ok)
      for (int s = 0; s < kStages; ++s)
        if (nf[s]) wait_warp(&bar->full[s], (nf[s] - 1) & 1, a.status);
  } else if (warp == 5) {
    // ------------------------------------------------ MMA (the whole warp runs the loop,
    // one elected lane issues each instruction)
    constexpr uint32_t idesc = ptx::idesc_bf16_f32(128, 128, 1, 1);  // A and B MN-major
    uint32_t it = 0, local = 0;
    bool ok = true;
    for (int64_t item = blockIdx.x; ok && item < n_items; item += gridDim.x, ++local) {
      const Item x = decode(a, item);
      const uint32_t b = local & 1, acc = tmem + 128u * b;
      // the epilogue has read this accumulator's previous item
      if (local >= 2 && !wait_warp(&bar->acc_empty[b], ((local >> 1) - 1) & 1, a.status)) { ok = false; break; }
      ptx::tc_fence_after();
      for (int c = 0; c < x.nkb; ++c, ++it) {
        const int s = (int)(it % kStages);
        if (__shfl_sync(0xffffffffu, aborted(&bar->abort) ? 1 : 0, 0) ||
            !wait_warp(&bar->full[s], (it / kStages) & 1, a.status)) {
          ok = false;
          break;
        }
        ptx::tc_fence_after();
        const uint32_t sDS = ptx::smem_u32(smem + s * kStageBytes), sK = sDS + kTileBytes;
        ptx::mma8_bf16_ss_warp<ptx::MnMajorIlv8, ptx::MnMajorSw128>(acc, desc_ilv_mnmajor(sDS, 0), desc_mnmajor(sK, 0),
                                                                   idesc, c > 0 ? 1u : 0u);
        ptx::mma_commit_warp(&bar->empty[s]);
      }
      if (!ok) break;
      ptx::mma_commit_warp(&bar->acc_full[b]);
    }
    if (!ok && lane == 0) set_abort(&bar->abort);
    __syncwarp();
    ptx::mma_commit_warp(&bar->final_mma);
    wait_warp(&bar->final_mma, 0, a.status);
  } else {
    // ------------------------------------------------ epilogue: thread = query row
    const int r = threadIdx.x;
    const uint32_t lane_addr = (uint32_t)(warp * 32) << 16;
    uint32_t local = 0;
    // rotary encoding: the cosines and sines of the row's 64 pairs are loaded
    // one item ahead (at the end of the previous epilogue).  A table load
    // waited for inside the epilogue costs microseconds while the dS stream
    // keeps the memory system saturated, and the epilogues of the short
    // items at the end of the walk set the pace.
    float nc[64], ns[64];
    auto first_tables = [&](int64_t item) {
      if (item >= n_items) return;
      const Item y = decode(a, item);
      const int row = y.t * kRows + r;
      if (row < y.w.q_len) rope_row<64>(a.rope_cos + (int64_t)row * 64, a.rope_sin + (int64_t)row * 64, nc, ns);
    };
    if (a.rope_cos) first_tables(blockIdx.x);
    for (int64_t item = blockIdx.x; item < n_items; item += gridDim.x, ++local) {
      const Item x = decode(a, item);
      const uint32_t b = local & 1, acc = tmem + lane_addr + 128u * b;
      const int row = x.t * kRows + r;
      // one decision for the whole warp: the epilogue's loads and shuffles are warp-wide
      if (__any_sync(0xffffffffu, !wait(&bar->acc_full[b], (local >> 1) & 1, a.status) || aborted(&bar->abort))) {
        set_abort(&bar->abort);
        break;
      }
      ptx::tc_fence_after();
      // rows are stored by groups of four lanes (store_slice32)
      const int64_t rstride = (int64_t)a.hq * kD;
      __nv_bfloat16* const g0 =
          reinterpret_cast<__nv_bfloat16*>(a.dq) + ((int64_t)x.w.q_base + row - (lane & 3)) * rstride + x.h * kD;
      const int g_rows = x.w.q_len - (row - (lane & 3));
      if (a.rope_cos) {
        // rotary encoding: columns k and k + 64 of the row pair up
#pragma unroll
        for (int q2 = 0; q2 < 2; ++q2) {
          uint32_t lo[32], hi[32];
          if (x.nkb > 0) {
            ptx::tmem_ld32(acc + 32 * q2, lo);
            ptx::tmem_ld32(acc + 64 + 32 * q2, hi);
            ptx::tmem_ld_wait();
            ptx::reg_fence(lo);
            ptx::reg_fence(hi);
          } else {
#pragma unroll
            for (int k = 0; k < 32; ++k) lo[k] = hi[k] = 0u;
          }
          // (rows past the tile's end compute on stale tables and are not stored)
          uint32_t wl[16], wh[16];
          rope_back_pack(lo, hi, a.scale, nc + 32 * q2, ns + 32 * q2, wl, wh);
          store_slice32(wl, g0 + 32 * q2, rstride, g_rows);
          store_slice32(wh, g0 + 64 + 32 * q2, rstride, g_rows);
        }
        ptx::tc_fence_before();
        ptx::mbar_arrive(&bar->acc_empty[b]);
        first_tables(item + gridDim.x);
        continue;
      }
#pragma unroll 1
      for (int q4 = 0; q4 < 4; ++q4) {
        uint32_t v[32], w[16];
        if (x.nkb > 0) {
          ptx::tmem_ld32(acc + 32 * q4, v);
          ptx::tmem_ld_wait();
          ptx::reg_fence(v);
        } else {
#pragma unroll
          for (int k = 0; k < 32; ++k) v[k] = 0u;
        }
        pack_scaled32(v, a.scale, w);
        store_slice32(w, g0 + 32 * q4, rstride, g_rows);
      }
      ptx::tc_fence_before();
      ptx::mbar_arrive(&bar->acc_empty[b]);
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 5) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, kTmemCols);
  }
}

}  // namespace

cudaError_t launch_dq_gemm(const AttnArgs& a, const CUtensorMap& tk, cudaStream_t st) {
  cudaError_t e;
  if ((reinterpret_cast<uintptr_t>(a.ds) & 15u) != 0) return cudaErrorMisalignedAddress;
  if ((e = cudaFuncSetAttribute(dq_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes)) !=
      cudaSuccess)
    return e;
  const int64_t n_items = a.nq * a.hq;
  int grid = knobs().dq_grid > 0 ? knobs().dq_grid : sm_count();
  if (grid > n_items) grid = (int)n_items;
  if (grid <= 0) return cudaSuccess;
  dq_gemm_kernel<<<(unsigned)grid, kThreads, kSmemBytes, st>>>(tk, a, n_items);
  return cudaGetLastError();
}

}  // namespace tc
}  // namespace ism
