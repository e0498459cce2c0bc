// dK / dV of the ISM backward on a CTA pair (cta_group::2, cluster of two).
//
// The gradients are those of dkdv_kernel (ism_bwd_tc.cu): per key tile and KV
// head, over the query tiles that see the key tile and the query heads of the
// group, S^T = K Q^T, dP^T = V dO^T, P^T and dS^T back into tensor memory,
// dV += P^T dO and dK += dS^T Q.  Here the two CTAs of a cluster take two
// neighbouring key tiles of one sequence and KV head, and every contraction
// is one M = 256 MMA over both tiles, issued by the even CTA: the B operand
// (Q / dO) is split across the pair, so each CTA's tensor core reads half of
// it from its own shared memory.  What a CTA holds of a Q (dO) tile, in four
// 8 KB boxes of 64 rows x 64 columns (128-byte swizzle):
//   slot 0, 1: its half of the queries, dimensions 0-63 and 64-127 (the B of
//              S^T / dP^T, N split by queries);
//   slot 2, 3: all queries (0-63, 64-127) of its half of the dimensions (the
//              B of dV / dK, N split by dimensions).
// Both CTAs order the contraction dimension alike, as the pair MMA multiplies
// every A row of either CTA with every B row of either.
//
// Hand-offs across the pair: each CTA's TMA loads complete on its own
// barriers; the odd CTA's warp 9 forwards each completion to the even CTA
// (one remote arrival), whose MMA warp waits for both.  The compute warps of
// both CTAs hand P^T / dS^T to the even CTA's MMA warp with one remote
// arrival per warp.  The even CTA's MMA completions are multicast to the
// barriers of both CTAs.  The even CTA's load warp takes the work items and
// publishes each in the item rings of both CTAs.  Every wait is bounded.
#include "ism_tc_common.cuh"

namespace ism {
namespace tc {
namespace {

constexpr int kComputeThreads = 256;
constexpr uint32_t kTmemCols = 512;

__device__ __forceinline__ bool aborted(const int32_t* f) { return *reinterpret_cast<const volatile int32_t*>(f) != 0; }

// Bounded waits with cluster-scope acquire: the item ring (the even CTA writes
// the entries into this CTA's shared memory before arriving) and the final
// completion.  The hand-off barriers carry no data the waiter reads itself
// (the MMAs read tensor and shared memory through the async proxy), and use
// the CTA-scope waits of the single-CTA kernel.
__device__ __forceinline__ bool wait_c(uint64_t* bar, uint32_t parity, uint32_t* status) {
  if (ptx::mbar_test_cluster(bar, parity)) return true;
  const uint64_t t0 = globaltimer();
  while (true) {
#pragma unroll 1
    for (int i = 0; i < 64; ++i)
      if (ptx::mbar_test_cluster(bar, parity)) return true;
    if (globaltimer() - t0 > kWaitLimitNs) {
      atomicOr(status, kStatusTimeout);
      return false;
    }
  }
}
__device__ __forceinline__ bool wait_warp_c(uint64_t* bar, uint32_t parity, uint32_t* status) {
  if (ptx::mbar_test_cluster_warp(bar, parity)) return true;
  const uint64_t t0 = globaltimer();
  while (true) {
#pragma unroll 1
    for (int i = 0; i < 64; ++i)
      if (ptx::mbar_test_cluster_warp(bar, parity)) return true;
    if (__shfl_sync(0xffffffffu, (globaltimer() - t0 > kWaitLimitNs) ? 1 : 0, 0)) {
      if ((threadIdx.x & 31) == 0) atomicOr(status, kStatusTimeout);
      return false;
    }
  }
}

__device__ __forceinline__ void ld64(uint32_t taddr, uint32_t (&a)[32], uint32_t (&b)[32]) {
  ptx::tmem_ld32(taddr, a);
  ptx::tmem_ld32(taddr + 32, b);
}

namespace dkp {
constexpr int kQStages = 3;
constexpr uint32_t kSlot = 8192;  // one 64 x 64 box
constexpr uint32_t OFF_K = 0, OFF_V = kTileBytes, OFF_Q = 2 * kTileBytes, OFF_DO = 5 * kTileBytes,
                   OFF_META = 7 * kTileBytes;
constexpr uint32_t kMetaStage = 128 * 4 + 128 * 4 + 128;
constexpr uint32_t OFF_BAR = OFF_META + 2 * kMetaStage;
constexpr uint32_t kSmemBytes = OFF_BAR + 512;
constexpr uint32_t TM_S = 0, TM_DP = 128, TM_DV = 256, TM_DK = 384;
constexpr int kLoadWarp = 8, kMmaWarp = 9, kMetaWarp = 10;
constexpr int kThreads = 352;
constexpr int kItemSlots = 4;

struct Bars {
  uint64_t kv_full, kv_empty;
  uint64_t q_full[kQStages], q_empty[kQStages], do_full[2], do_empty[2], meta_full[2], meta_empty[2];
  uint64_t item_full[kItemSlots];
  uint64_t s_full, dp_full, pt_full, p_full, dv_done, dk_done, acc_full, final_mma;
  // the odd CTA's load completions, forwarded to the even CTA
  uint64_t peer_kv_full, peer_q_full[kQStages], peer_do_full[2];
  uint32_t tmem_base;
  int32_t abort;
  uint32_t full[2][2];
  int32_t items[kItemSlots];
};
static_assert(sizeof(Bars) <= 512, "barrier block");
static_assert(kSmemBytes <= 232448, "shared memory per CTA");
}  // namespace dkp

// Abort flag of both CTAs of the pair.
__device__ __forceinline__ void set_abort_pair(int32_t* f) {
  *reinterpret_cast<volatile int32_t*>(f) = 1;
  ptx::st_cluster_u32(ptx::cluster_addr(f, ptx::cluster_ctarank() ^ 1u), 1u);
}

__global__ void __launch_bounds__(dkp::kThreads, 1)
    dkdv_pair_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmdO,
                     const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                     const AttnArgs a) {
  using namespace dkp;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw;
  Bars* bar = reinterpret_cast<Bars*>(smem + OFF_BAR);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = ptx::cluster_ctarank();
  const bool lead = rank == 0;
  // alignment is a property of the launch, so both CTAs of the pair take the same branch
  if (ptx::smem_u32(smem) & 1023u) {
    if (threadIdx.x == 0) atomicOr(a.status, kStatusSmemAlign);
    return;
  }
  const int group = a.hq / a.hkv;
  const int64_t n_items = a.nkp * a.hkv;

  if (threadIdx.x == 0) {
    ptx::mbar_init(&bar->kv_full, 1);
    ptx::mbar_init(&bar->kv_empty, 1);
    for (int s = 0; s < kQStages; ++s) {
      ptx::mbar_init(&bar->q_full[s], 1);
      ptx::mbar_init(&bar->q_empty[s], 1);
      ptx::mbar_init(&bar->peer_q_full[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      ptx::mbar_init(&bar->do_full[s], 1);
      ptx::mbar_init(&bar->do_empty[s], 1);
      ptx::mbar_init(&bar->peer_do_full[s], 1);
      ptx::mbar_init(&bar->meta_full[s], 32);
      ptx::mbar_init(&bar->meta_empty[s], kComputeThreads);
    }
    for (int s = 0; s < kItemSlots; ++s) ptx::mbar_init(&bar->item_full[s], 1);
    ptx::mbar_init(&bar->peer_kv_full, 1);
    ptx::mbar_init(&bar->s_full, 1);
    ptx::mbar_init(&bar->dp_full, 1);
    ptx::mbar_init(&bar->pt_full, 16);  // one arrival per compute warp of either CTA
    ptx::mbar_init(&bar->p_full, 16);
    ptx::mbar_init(&bar->dv_done, 1);
    ptx::mbar_init(&bar->dk_done, 1);
    ptx::mbar_init(&bar->acc_full, 1);
    ptx::mbar_init(&bar->final_mma, 1);
    bar->abort = 0;
    ptx::fence_mbar_init();
  }
  if (warp == kMmaWarp) {
    ptx::tmem_alloc_pair(&bar->tmem_base, kTmemCols);
    ptx::tmem_relinquish_pair();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::cluster_sync();  // both CTAs: barriers initialised, tensor memory allocated
  ptx::tc_fence_after();
  const uint32_t tmem = bar->tmem_base;

  // Work items (key-tile pair kp_order[item / hkv], KV head item % hkv, in
  // cost order with bucket_item) come from a global counter that the even
  // CTA's load warp reads; it publishes each item in a small shared ring of
  // both CTAs, which every role follows.  A negative entry ends the walk.
  // CTA `rank` takes key tile c = (first tile of the pair) + rank; a pair
  // whose second tile lies past its sequence leaves the odd CTA with keys
  // that no query sees (masked, nothing stored).
  struct Item {
    int g, gk, c, qt0, qt_own, nqt, n_it;
    bool own;  // this CTA's key tile exists
    Tile w;
  };
  auto decode = [&](int item, Item& x) {
    int64_t kpos;
    bucket_item(item, a.nkp, a.hkv, kpos, x.g);
    const int gk0 = a.kp_order[kpos];
    x.w = a.ktiles[gk0];
    x.c = x.w.tile + (int)rank;
    x.own = x.c * kRows < x.w.k_len;
    x.gk = gk0 + (int)rank;
    x.qt0 = x.w.a0;
    x.nqt = x.w.a1;
    x.qt_own = x.own ? a.ktiles[x.gk].a0 : x.nqt;
    x.n_it = x.nqt > x.qt0 ? (x.nqt - x.qt0) * group : 0;
  };
  auto next_item = [&](uint32_t u, Item& x) -> bool {
    const int slot = (int)(u % kItemSlots);
    if (!wait_c(&bar->item_full[slot], (u / kItemSlots) & 1, a.status)) return false;
    const int item = *reinterpret_cast<volatile int32_t*>(&bar->items[slot]);
    if (item < 0) return false;
    decode(item, x);
    return true;
  };
  // Iteration i of an item visits query tile nqt - 1 - i / group of query
  // head g * group + i % group (last to first, as dkdv_kernel).  Barrier
  // phases count iterations (I) and items (u) across the whole walk.

  if (warp == kLoadWarp) {
    // ------------------------------------------------ work items (even CTA) and TMA loads (both)
    uint32_t I = 0, nq[kQStages] = {0, 0, 0}, ndo[2] = {0, 0}, nkv = 0;
    bool ok = true;
    for (uint32_t u = 0;;) {
      Item x;
      bool have;
      if (lead) {
        int item = -1;
        if (lane == 0) {
          item = ok && !aborted(&bar->abort) ? atomicAdd(a.work_counter, 1) : -1;
          if (item >= n_items) item = -1;
        }
        item = __shfl_sync(0xffffffffu, item, 0);
        if (item >= 0) {
          decode(item, x);
          if (x.n_it == 0) {
            // no query sees these keys (with ISM segments every key sees at least
            // itself, so this is only a guard): dK = dV = 0 for both tiles, not published
            for (int rr = lane; rr < 2 * kRows; rr += 32) {
              const int key = x.w.tile * kRows + rr;
              if (key >= x.w.k_len) break;
              const int64_t off = ((int64_t)x.w.k_base + key) * a.hkv * kD + x.g * kD;
              uint4* dk = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(a.dk) + off);
              uint4* dv = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(a.dv) + off);
              for (int k = 0; k < kD / 8; ++k) dk[k] = dv[k] = make_uint4(0u, 0u, 0u, 0u);
            }
            continue;
          }
        }
        // Published items all have iterations, so the load warp cannot run more
        // than one item ahead of the MMA warp (kv_empty) and a ring slot is never
        // rewritten before every role of either CTA has read it.
        if (lane == 0) {
          const int slot = (int)(u % kItemSlots);
          bar->items[slot] = item;
          ptx::st_cluster_u32(ptx::cluster_addr(&bar->items[slot], 1u), (uint32_t)item);
          ptx::mbar_arrive(&bar->item_full[slot]);
          ptx::mbar_arrive_cluster(ptx::cluster_addr(&bar->item_full[slot], 1u));
        }
        __syncwarp();
        ++u;
        have = item >= 0;
      } else {
        have = __all_sync(0xffffffffu, next_item(u, x));
        ++u;
      }
      if (!have) break;
      // this CTA's K and V once the previous item's S and dP MMAs are done with them
      if (nkv > 0 && !wait_warp(&bar->kv_empty, (nkv - 1) & 1, a.status)) {
        if (lane == 0) set_abort_pair(&bar->abort);
        ok = false;
        break;
      }
      const int32_t ky = x.w.k_base + x.c * kRows;  // past the tensor: zero fill; past the sequence: masked
      if (lane == 0) {
        ptx::mbar_expect_tx(&bar->kv_full, 2 * kTileBytes);
        ptx::tma_load_2d(smem + OFF_K, &tmK, &bar->kv_full, x.g * kD, ky);
        ptx::tma_load_2d(smem + OFF_K + kHalfBytes, &tmK, &bar->kv_full, x.g * kD + 64, ky);
        ptx::tma_load_2d(smem + OFF_V, &tmV, &bar->kv_full, x.g * kD, ky);
        ptx::tma_load_2d(smem + OFF_V + kHalfBytes, &tmV, &bar->kv_full, x.g * kD + 64, ky);
      }
      __syncwarp();
      ++nkv;
      for (int i = 0; i < x.n_it; ++i, ++I) {
        const int sq = (int)(I % kQStages), s = (int)(I & 1);
        const int h = x.g * group + i % group;
        const int32_t qy = x.w.q_base + (x.nqt - 1 - i / group) * kRows;
        if (__any_sync(0xffffffffu, aborted(&bar->abort))) { ok = false; break; }
        bool okq = I < kQStages || wait_warp(&bar->q_empty[sq], (I / kQStages - 1) & 1, a.status);
        if (okq) {
          if (lane == 0) {
            // slots 0, 1: this CTA's query half, both dimension halves; 2, 3: both query halves of its dimension half
            uint8_t* dst = smem + OFF_Q + sq * kTileBytes;
            ptx::mbar_expect_tx(&bar->q_full[sq], kTileBytes);
            ptx::tma_load_2d(dst, &tmQ, &bar->q_full[sq], h * kD, qy + 64 * (int)rank);
            ptx::tma_load_2d(dst + kSlot, &tmQ, &bar->q_full[sq], h * kD + 64, qy + 64 * (int)rank);
            ptx::tma_load_2d(dst + 2 * kSlot, &tmQ, &bar->q_full[sq], h * kD + 64 * (int)rank, qy);
            ptx::tma_load_2d(dst + 3 * kSlot, &tmQ, &bar->q_full[sq], h * kD + 64 * (int)rank, qy + 64);
          }
          __syncwarp();
          ++nq[sq];
          okq = I < 2 || wait_warp(&bar->do_empty[s], ((I >> 1) - 1) & 1, a.status);
        }
        if (okq) {
          if (lane == 0) {
            uint8_t* dst = smem + OFF_DO + s * kTileBytes;
            ptx::mbar_expect_tx(&bar->do_full[s], kTileBytes);
            ptx::tma_load_2d(dst, &tmdO, &bar->do_full[s], h * kD, qy + 64 * (int)rank);
            ptx::tma_load_2d(dst + kSlot, &tmdO, &bar->do_full[s], h * kD + 64, qy + 64 * (int)rank);
            ptx::tma_load_2d(dst + 2 * kSlot, &tmdO, &bar->do_full[s], h * kD + 64 * (int)rank, qy);
            ptx::tma_load_2d(dst + 3 * kSlot, &tmdO, &bar->do_full[s], h * kD + 64 * (int)rank, qy + 64);
          }
          __syncwarp();
          ++ndo[s];
        }
        if (!okq) {
          if (lane == 0) set_abort_pair(&bar->abort);
          ok = false;
          break;
        }
      }
      if (!ok) break;
    }
    if (!ok) {
      // every issued copy lands before the CTA exits
      if (nkv) wait_warp(&bar->kv_full, (nkv - 1) & 1, a.status);
      for (int s = 0; s < kQStages; ++s)
        if (nq[s]) wait_warp(&bar->q_full[s], (nq[s] - 1) & 1, a.status);
      for (int s = 0; s < 2; ++s)
        if (ndo[s]) wait_warp(&bar->do_full[s], (ndo[s] - 1) & 1, a.status);
    }
    __syncwarp();
  } else if (warp == kMmaWarp && !lead) {
    // ------------------------------------------------ odd CTA: forward each load completion to the even CTA
    const uint32_t r_kv = ptx::cluster_addr(&bar->peer_kv_full, 0u);
    uint32_t I = 0, nkv = 0;
    Item x;
    bool ok = true;
    for (uint32_t u = 0; ok && __all_sync(0xffffffffu, next_item(u, x)); ++u) {
      if (!wait_warp(&bar->kv_full, nkv & 1, a.status)) { ok = false; break; }
      ++nkv;
      if (lane == 0) ptx::mbar_arrive_cluster(r_kv);
      for (int i = 0; i < x.n_it; ++i, ++I) {
        const int sq = (int)(I % kQStages), s = (int)(I & 1);
        if (!wait_warp(&bar->q_full[sq], (I / kQStages) & 1, a.status)) { ok = false; break; }
        if (lane == 0) ptx::mbar_arrive_cluster(ptx::cluster_addr(&bar->peer_q_full[sq], 0u));
        if (!wait_warp(&bar->do_full[s], (I >> 1) & 1, a.status)) { ok = false; break; }
        if (lane == 0) ptx::mbar_arrive_cluster(ptx::cluster_addr(&bar->peer_do_full[s], 0u));
      }
    }
    if (!ok && lane == 0) set_abort_pair(&bar->abort);
    __syncwarp();
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------ even CTA: the pair's MMAs (the whole warp runs the
    // loop, one elected lane issues each instruction)
    constexpr uint32_t idesc_nt = ptx::idesc_bf16_f32(256, 128, 0, 0);
    constexpr uint32_t idesc_nn = ptx::idesc_bf16_f32(256, 128, 0, 1);
    const uint32_t sK = ptx::smem_u32(smem + OFF_K), sV = ptx::smem_u32(smem + OFF_V);
    uint32_t I0 = 0, nkv = 0;
    bool ok = true;
    // S^T = K Q^T: B = this CTA's query half (slots 0, 1: dimension halves 8 KB apart)
    auto issue_s = [&](uint32_t gi) {
      const uint32_t sQ = ptx::smem_u32(smem + OFF_Q + (gi % kQStages) * kTileBytes);
      ptx::mma8_bf16_ss_pair_warp<ptx::KMajorSw128, ptx::KMajorSw128Half8K>(
          tmem + TM_S, desc_kmajor(sK, 0), desc_kmajor(sQ, 0), idesc_nt, 0u);
      ptx::mma_commit_pair_warp(&bar->s_full);
    };
    auto issue_dp = [&](uint32_t gi) {
      const uint32_t sdO = ptx::smem_u32(smem + OFF_DO + (gi & 1) * kTileBytes);
      ptx::mma8_bf16_ss_pair_warp<ptx::KMajorSw128, ptx::KMajorSw128Half8K>(
          tmem + TM_DP, desc_kmajor(sV, 0), desc_kmajor(sdO, 0), idesc_nt, 0u);
      ptx::mma_commit_pair_warp(&bar->dp_full);
    };
    // dV += P^T dO: B = both query halves (slots 2, 3, 8 KB apart) of this CTA's dimension half
    auto issue_dv = [&](uint32_t gi, bool first) {
      const uint32_t s = gi & 1;
      const uint32_t sdO = ptx::smem_u32(smem + OFF_DO + s * kTileBytes + 2 * kSlot);
      ptx::mma8_bf16_ts_pair_warp<ptx::TmemPairsGap32, ptx::MnMajorSw128>(tmem + TM_DV, tmem + TM_S,
                                                                          desc_mnmajor(sdO, 0), idesc_nn,
                                                                          first ? 0u : 1u);
      ptx::mma_commit_pair_warp(&bar->do_empty[s]);
      ptx::mma_commit_pair_warp(&bar->dv_done);
    };
    auto issue_dk = [&](uint32_t gi, bool first) {
      const uint32_t sq = gi % kQStages;
      const uint32_t sQ = ptx::smem_u32(smem + OFF_Q + sq * kTileBytes + 2 * kSlot);
      ptx::mma8_bf16_ts_pair_warp<ptx::TmemPairsGap32, ptx::MnMajorSw128>(tmem + TM_DK, tmem + TM_DP,
                                                                          desc_mnmajor(sQ, 0), idesc_nn,
                                                                          first ? 0u : 1u);
      ptx::mma_commit_pair_warp(&bar->q_empty[sq]);
      ptx::mma_commit_pair_warp(&bar->dk_done);
    };
    Item x;
    for (uint32_t u = 0; ok; ++u) {
      if (!__all_sync(0xffffffffu, next_item(u, x))) break;
      const int n_it = x.n_it;
      if (!wait_warp(&bar->kv_full, nkv & 1, a.status) || !wait_warp(&bar->peer_kv_full, nkv & 1, a.status)) {
        ok = false;
        break;
      }
      ++nkv;
      // Event-driven issue in order of urgency, as dkdv_kernel: dK_i after dS^T_i
      // (p_full), dP_i after dK_{i-1} and both CTAs' dO_i, dV_i after P^T_i
      // (pt_full) and dP_i, S_i after dV_{i-1} and both CTAs' Q_i.  p_full and
      // pt_full count one arrival per compute warp of either CTA.
      const uint32_t end = I0 + (uint32_t)n_it;
      uint32_t ns = I0, np = I0, nv = I0, nk = I0;
      uint32_t qs = I0 % kQStages, qph = (I0 / kQStages) & 1;
      uint64_t t_idle = 0;
      while (ok && nk < end) {
        bool progressed = false;
        if (nk < nv && ptx::mbar_test_warp(&bar->p_full, nk & 1)) {
          ptx::tc_fence_after();
          issue_dk(nk, nk == I0);
          ++nk;
          progressed = true;
        }
        if (np < end && np <= nk && ptx::mbar_test_warp(&bar->do_full[np & 1], (np >> 1) & 1) &&
            ptx::mbar_test_warp(&bar->peer_do_full[np & 1], (np >> 1) & 1) &&
            (np == 0 || !(a.flags & kFlagDrainTmemReuse) || ptx::mbar_test_warp(&bar->dk_done, (np - 1) & 1))) {
          ptx::tc_fence_after();
          issue_dp(np);
          ++np;
          progressed = true;
          if (np == end && ns == end) ptx::mma_commit_pair_warp(&bar->kv_empty);
        }
        if (nv < np && ptx::mbar_test_warp(&bar->pt_full, nv & 1)) {
          ptx::tc_fence_after();
          issue_dv(nv, nv == I0);
          ++nv;
          progressed = true;
        }
        if (ns < end && ns <= nv && ptx::mbar_test_warp(&bar->q_full[qs], qph) &&
            ptx::mbar_test_warp(&bar->peer_q_full[qs], qph) &&
            (ns == 0 || !(a.flags & kFlagDrainTmemReuse) || ptx::mbar_test_warp(&bar->dv_done, (ns - 1) & 1))) {
          ptx::tc_fence_after();
          issue_s(ns);
          ++ns;
          if (++qs == kQStages) { qs = 0; qph ^= 1; }
          progressed = true;
          if (np == end && ns == end) ptx::mma_commit_pair_warp(&bar->kv_empty);
        }
        if (progressed) {
          t_idle = 0;
        } else {
          __nanosleep(16);
          const uint64_t now = globaltimer();
          if (t_idle == 0) t_idle = now;
          const bool expired = __shfl_sync(0xffffffffu, (now - t_idle > kWaitLimitNs || aborted(&bar->abort)) ? 1 : 0, 0);
          if (expired) {
            if (lane == 0) atomicOr(a.status, kStatusTimeout);
            ok = false;
          }
        }
      }
      if (!ok) break;
      ptx::mma_commit_pair_warp(&bar->acc_full);  // dV, dK of this item complete
      I0 = end;
    }
    if (!ok && lane == 0) set_abort_pair(&bar->abort);
    __syncwarp();
    ptx::mma_commit_pair_warp(&bar->final_mma);
    wait_warp_c(&bar->final_mma, 0, a.status);
    __syncwarp();
  } else if (warp == kMetaWarp) {
    // ------------------------------------------------ per-query metadata (all 32 lanes)
    uint32_t I = 0;
    Item x;
    for (uint32_t u = 0; next_item(u, x); ++u) {
      for (int i = 0; i < x.n_it; ++i, ++I) {
        const int s = (int)(I & 1);
        const int hh = i % group, t = x.nqt - 1 - i / group;
        const int h = x.g * group + hh;
        if (aborted(&bar->abort)) break;
        if (I >= 2 && !wait(&bar->meta_empty[s], ((I >> 1) - 1) & 1, a.status)) { set_abort_pair(&bar->abort); break; }
        uint8_t* meta = smem + OFF_META + s * kMetaStage;
        float* mlse = reinterpret_cast<float*>(meta);
        float* mdel = mlse + 128;
        uint8_t* mlim = reinterpret_cast<uint8_t*>(mdel + 128);
        bool all_full = true;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int j = lane * 4 + e;
          const int row = t * kRows + j;
          const bool valid = row < x.w.q_len;
          const int64_t grow = (int64_t)x.w.q_base + row;
          mlse[j] = valid ? a.lse_in[(int64_t)h * a.q_rows + grow] * kLog2e : 0.f;
          mdel[j] = valid ? a.delta[(int64_t)h * a.q_rows + grow] : 0.f;
          const int vis = valid ? a.kv_end[x.w.kv_base + row] - x.c * kRows : 0;
          mlim[j] = (uint8_t)(vis < 0 ? 0 : vis > 128 ? 128 : vis);
          all_full = all_full && vis >= 128;
        }
        // lanes 0-15 hold the queries of warpgroup 0, lanes 16-31 those of warpgroup 1
        const uint32_t fb = __ballot_sync(0xffffffffu, all_full);
        if (lane == 0) {
          bar->full[s][0] = (fb & 0xFFFFu) == 0xFFFFu;
          bar->full[s][1] = (fb >> 16) == 0xFFFFu;
        }
        ptx::mbar_arrive(&bar->meta_full[s]);
      }
      if (aborted(&bar->abort)) break;
    }
  } else {
    // ------------------------------------------------ compute: thread = key row r, warpgroup wg owns queries [64 wg, 64 wg + 64)
    const int wg = threadIdx.x >> 7, r = threadIdx.x & 127;
    const uint32_t lane_addr = (uint32_t)((warp & 3) * 32) << 16;
    const uint32_t tS = tmem + lane_addr + TM_S + 64u * wg, tP = tmem + lane_addr + TM_DP + 64u * wg;
    const float sl2 = a.scale * kLog2e;
    // the stored dS is read back only by the dQ GEMM, after this kernel: its
    // lines go first when L2 needs room, ahead of the Q / dO tiles other CTAs reuse
    const uint64_t pol_ds = ptx::l2_policy_evict_first();
    // hand-offs to the even CTA's MMA warp: one arrival per warp, relaxed: the
    // P^T / dS^T stores are complete (tcgen05.wait::st) and the MMA reads nothing
    // else these threads wrote; a release would wait for their dS stores to reach L2
    const uint32_t r_pt_full = ptx::cluster_addr(&bar->pt_full, 0u), r_p_full = ptx::cluster_addr(&bar->p_full, 0u);
    bool ok = true;
    uint32_t I = 0, nacc = 0;
    Item x;
    for (uint32_t u = 0; ok && next_item(u, x); ++u) {
      const int n_it = x.n_it;
      // dS^T stores of the previous iteration left for after this iteration's P
      // phase (half of them), where the compute warps wait for dP^T anyway
      uint4* ds_dst = nullptr;
      uint32_t ds_rest[16];
      for (int i = 0; ok && i < n_it; ++i, ++I) {
        const int s = (int)(I & 1);
        if (!wait(&bar->meta_full[s], (I >> 1) & 1, a.status) || !wait(&bar->s_full, I & 1, a.status)) {
          ok = false;
          break;
        }
        ptx::tc_fence_after();
        const uint8_t* meta = smem + OFF_META + s * kMetaStage;
        const float4* mlse4 = reinterpret_cast<const float4*>(meta) + wg * 16;
        const float4* mdel4 = reinterpret_cast<const float4*>(meta + 512) + wg * 16;
        const uint32_t* mlim4 = reinterpret_cast<const uint32_t*>(meta + 1024) + wg * 16;
        // phase 1: P from S^T (dP^T may still be in flight)
        uint32_t pp[32];  // pp[k]: queries 64 wg + 2k, 64 wg + 2k + 1 (bf16)
        {
          uint32_t sv[2][32];
          ld64(tS, sv[0], sv[1]);
          ptx::tmem_ld_wait();
          ptx::reg_fence(sv[0]);
          ptx::reg_fence(sv[1]);
          if (bar->full[s][wg]) {
            // every key of the tile is visible to every query of this warpgroup
            const float2 sl2x2 = make_float2(sl2, sl2);
#pragma unroll
            for (int q4 = 0; q4 < 16; ++q4) {
              const float4 l4 = mlse4[q4];
              const uint32_t* sq = &sv[q4 >> 3][(q4 & 7) * 4];
              const float2 a01 = fma2(make_float2(__uint_as_float(sq[0]), __uint_as_float(sq[1])), sl2x2,
                                      make_float2(-l4.x, -l4.y));
              const float2 a23 = fma2(make_float2(__uint_as_float(sq[2]), __uint_as_float(sq[3])), sl2x2,
                                      make_float2(-l4.z, -l4.w));
              pp[q4 * 2] = pack_bf16(ex2(a01.x), ex2(a01.y));
              pp[q4 * 2 + 1] = pack_bf16(ex2(a23.x), ex2(a23.y));
            }
          } else {
#pragma unroll
            for (int q4 = 0; q4 < 16; ++q4) {
              const float4 l4 = mlse4[q4];
              const uint32_t lim = mlim4[q4];
              const float lv[4] = {l4.x, l4.y, l4.z, l4.w};
              float p[4];
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const int vis = (int)((lim >> (8 * e)) & 0xFFu);
                p[e] = r < vis ? ex2(__uint_as_float(sv[q4 >> 3][(q4 & 7) * 4 + e]) * sl2 - lv[e]) : 0.f;
              }
              pp[q4 * 2] = pack_bf16(p[0], p[1]);
              pp[q4 * 2 + 1] = pack_bf16(p[2], p[3]);
            }
          }
        }
        // P^T over this warpgroup's (already read) S^T columns; dV may start
        ptx::tmem_st32(tS, pp);
        ptx::tmem_st_wait();
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive_cluster_relaxed(r_pt_full);
        if (ds_dst) {
#pragma unroll
          for (int k = 0; k < 4; ++k)
            ptx::st_global_v4_hint(ds_dst + (k + 4) * kRows,
                                   make_uint4(ds_rest[4 * k], ds_rest[4 * k + 1], ds_rest[4 * k + 2], ds_rest[4 * k + 3]),
                                   pol_ds);
          ds_dst = nullptr;
        }
        // phase 2: dS from dP^T
        if (!wait(&bar->dp_full, I & 1, a.status)) { ok = false; break; }
        ptx::tc_fence_after();
        uint32_t pd[32];
        {
          uint32_t dv[2][32];
          ld64(tP, dv[0], dv[1]);
          ptx::tmem_ld_wait();
          ptx::reg_fence(dv[0]);
          ptx::reg_fence(dv[1]);
#pragma unroll
          for (int q4 = 0; q4 < 16; ++q4) {
            const float4 d4 = mdel4[q4];
            const uint32_t w0 = pp[q4 * 2], w1 = pp[q4 * 2 + 1];
            const int b = (q4 & 7) * 4, hv = q4 >> 3;
            const float2 v01 = mul2(make_float2(__uint_as_float(w0 << 16), __uint_as_float(w0 & 0xFFFF0000u)),
                                    add2(make_float2(__uint_as_float(dv[hv][b + 0]), __uint_as_float(dv[hv][b + 1])),
                                         make_float2(-d4.x, -d4.y)));
            const float2 v23 = mul2(make_float2(__uint_as_float(w1 << 16), __uint_as_float(w1 & 0xFFFF0000u)),
                                    add2(make_float2(__uint_as_float(dv[hv][b + 2]), __uint_as_float(dv[hv][b + 3])),
                                         make_float2(-d4.z, -d4.w)));
            pd[q4 * 2] = pack_bf16(v01.x, v01.y);
            pd[q4 * 2 + 1] = pack_bf16(v23.x, v23.y);
          }
        }
        ptx::mbar_arrive(&bar->meta_empty[s]);
        // dS^T over this warpgroup's (already read) dP^T columns
        ptx::tmem_st32(tP, pd);
        ptx::tmem_st_wait();
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive_cluster_relaxed(r_p_full);
        if (a.ds && x.own && x.nqt - 1 - i / group >= x.qt_own) {
          // keep dS^T row r, queries [64 wg, 64 wg + 64), for the dQ GEMM, in
          // the 8-interleaved layout (16-byte unit (query group, key)): the 32
          // lanes of a warp store 512 contiguous bytes per instruction.  Issued
          // after the hand-off so that the dV/dK MMAs do not wait for it.
          const int hh = i % group, t = x.nqt - 1 - i / group;
          const int64_t slot = ((int64_t)a.kpair_off[x.gk] + (t - x.qt_own)) * a.hq + (x.g * group + hh);
          uint4* dst = reinterpret_cast<uint4*>(static_cast<uint8_t*>(a.ds) + slot * kTileBytes) + wg * 8 * kRows + r;
#pragma unroll
          for (int k = 0; k < 4; ++k)
            ptx::st_global_v4_hint(dst + k * kRows, make_uint4(pd[4 * k], pd[4 * k + 1], pd[4 * k + 2], pd[4 * k + 3]),
                                   pol_ds);
#pragma unroll
          for (int k = 0; k < 16; ++k) ds_rest[k] = pd[16 + k];
          ds_dst = dst;
        }
      }
      if (ds_dst) {
#pragma unroll
        for (int k = 0; k < 4; ++k)
          ptx::st_global_v4_hint(ds_dst + (k + 4) * kRows,
                                 make_uint4(ds_rest[4 * k], ds_rest[4 * k + 1], ds_rest[4 * k + 2], ds_rest[4 * k + 3]),
                                 pol_ds);
      }
      if (!ok) break;
      // epilogue of the item: dV, dK from tensor memory
      const int key = x.c * kRows + r;
      const bool kvalid = key < x.w.k_len;
      // one decision for the whole warp: the epilogue's loads and shuffles are warp-wide
      if (!__all_sync(0xffffffffu, wait(&bar->acc_full, nacc & 1, a.status))) { ok = false; break; }
      ++nacc;
      ptx::tc_fence_after();
      // rows are stored by groups of four lanes (store_slice32): the group of
      // this lane starts at key - (lane & 3)
      const int64_t rstride = (int64_t)a.hkv * kD;
      const int64_t grow = (int64_t)x.w.k_base + key - (lane & 3);
      const int g_rows = x.w.k_len - (key - (lane & 3));
      __nv_bfloat16* const dvg = reinterpret_cast<__nv_bfloat16*>(a.dv) + grow * rstride + x.g * kD;
      __nv_bfloat16* const dkg = reinterpret_cast<__nv_bfloat16*>(a.dk) + grow * rstride + x.g * kD;
      if (wg == 1 && a.rope_cos) {
#pragma unroll 1
        for (int q2 = 0; q2 < 2; ++q2) {
          uint32_t lo[32], hi[32];
          ptx::tmem_ld32(tmem + lane_addr + TM_DK + q2 * 32, lo);
          ptx::tmem_ld32(tmem + lane_addr + TM_DK + 64 + q2 * 32, hi);
          ptx::tmem_ld_wait();
          ptx::reg_fence(lo);
          ptx::reg_fence(hi);
          float rc[32], rs[32];
          if (kvalid) {
            rope_row<32>(a.rope_cos + (int64_t)key * 64 + 32 * q2, a.rope_sin + (int64_t)key * 64 + 32 * q2, rc, rs);
          } else {
#pragma unroll
            for (int k = 0; k < 32; ++k) rc[k] = rs[k] = 0.f;
          }
          uint32_t wl[16], wh[16];
          rope_back_pack(lo, hi, a.scale, rc, rs, wl, wh);
          store_slice32(wl, dkg + q2 * 32, rstride, g_rows);
          store_slice32(wh, dkg + 64 + q2 * 32, rstride, g_rows);
        }
        ptx::tc_fence_before();
        continue;
      }
      // warpgroup 0 writes dV, warpgroup 1 writes dK (scaled)
#pragma unroll 1
      for (int q4 = 0; q4 < 4; ++q4) {
        uint32_t v[32], w[16];
        ptx::tmem_ld32(tmem + lane_addr + (wg == 0 ? TM_DV : TM_DK) + 32 * q4, v);
        ptx::tmem_ld_wait();
        ptx::reg_fence(v);
        pack_scaled32(v, wg == 0 ? 1.f : a.scale, w);
        store_slice32(w, (wg == 0 ? dvg : dkg) + 32 * q4, rstride, g_rows);
      }
      ptx::tc_fence_before();
    }
    if (!ok) set_abort_pair(&bar->abort);
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::cluster_sync();  // neither CTA frees its tensor memory or exits while the pair's MMAs could use it
  if (warp == kMmaWarp) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc_pair(tmem, kTmemCols);
  }
}

}  // namespace
}  // namespace tc
}  // namespace ism

namespace ism {
namespace tc {

// dK / dV on CTA pairs over the key-tile pairs of a.kp_order (a.nkp of them);
// tk / tv are the K / V tensor maps of dkdv_kernel (64-column x 128-row boxes).
cudaError_t launch_dkdv_pair(const AttnArgs& a, const CUtensorMap& tk, const CUtensorMap& tv, cudaStream_t st) {
  using namespace dkp;
  CUtensorMap tq, tdo;  // 64-column x 64-row boxes: the quarters of a Q / dO tile
  cudaError_t e;
  if ((e = make_tmap_bf16_box(&tq, a.q, (uint64_t)a.hq * kD, (uint64_t)a.q_rows, 64)) != cudaSuccess) return e;
  if ((e = make_tmap_bf16_box(&tdo, a.dout, (uint64_t)a.hq * kD, (uint64_t)a.q_rows, 64)) != cudaSuccess) return e;
  if ((e = cudaFuncSetAttribute(dkdv_pair_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes)) !=
      cudaSuccess)
    return e;
  int64_t grid = knobs().dkdv_grid > 0 ? knobs().dkdv_grid : sm_count();
  if (grid > 2 * a.nkp * a.hkv) grid = 2 * a.nkp * a.hkv;
  grid &= ~int64_t(1);
  if (grid < 2) grid = 2;
  if (!a.work_counter || !a.kp_order) return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kSmemBytes;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, dkdv_pair_kernel, tq, tdo, tk, tv, a);
}

}  // namespace tc
}  // namespace ism
