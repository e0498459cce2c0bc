// ISM attention backward on sm_103a tensor cores: the standard softmax
// attention gradients over the Eq. (e_ISM) mask, with P recomputed from the
// forward's log-sum-exp.
//
//   delta_kernel   Delta_j = sum_d dO_jd O_jd                      (HBM-bound)
//   dq_kernel      per (query tile, query head), over the tile's non-empty
//                  key blocks: S = Q K^T, dP = dO V^T (TMEM), dS = P (dP - Delta)
//                  back into TMEM, dQ += dS K (TMEM); dQ = scale * dQ.
//   dkdv_kernel    per (key tile, KV head), over the query heads of the group
//                  and the query tiles that see the key tile: S^T = K Q^T and
//                  dP^T = V dO^T (TMEM), P^T and dS^T back into TMEM (A operands
//                  of the next MMAs), dV += P^T dO, dK += dS^T Q (TMEM
//                  accumulators); dK = scale * dK.
// Warp roles in both MMA kernels: warps 0..7 compute (two warpgroups, each
// owning 64 of the 128 columns of a tile; thread = TMEM lane = tile row),
// warp 8 loads (TMA), warp 9 owns TMEM and issues the MMAs.
#include "ism_tc_common.cuh"

namespace ism {
namespace tc {
namespace {

constexpr int kThreads = 320;
constexpr int kComputeThreads = 256;
constexpr uint32_t kTmemCols = 512;

__device__ __forceinline__ bool aborted(const int32_t* f) { return *reinterpret_cast<const volatile int32_t*>(f) != 0; }
__device__ __forceinline__ void set_abort(int32_t* f) { *reinterpret_cast<volatile int32_t*>(f) = 1; }

__device__ __forceinline__ void ld64(uint32_t taddr, uint32_t (&a)[32], uint32_t (&b)[32]) {
  ptx::tmem_ld32(taddr, a);
  ptx::tmem_ld32(taddr + 32, b);
}

// ------------------------------------------------------------------ delta
// One 16-lane group per (row, head): 8 bf16 per lane, D = 128.  A group takes
// four (row, head) pairs per round with all eight loads issued before any
// use (more bytes in flight per thread: the kernel only streams O and dO).
// The reductions shuffle within the group's own 16 lanes, so the two groups
// of a warp may run different numbers of rounds.
__global__ void delta_kernel(const __nv_bfloat16* __restrict__ O, const __nv_bfloat16* __restrict__ dO,
                             float* __restrict__ delta, int64_t rows, int hq) {
  constexpr int kUnroll = 4;
  const int64_t n = rows * hq;
  const int sub = threadIdx.x & 15;
  const uint32_t group_mask = 0xFFFFu << (threadIdx.x & 16);
  const int64_t groups = ((int64_t)gridDim.x * blockDim.x) >> 4;
  for (int64_t i0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 4; i0 < n; i0 += groups * kUnroll) {
    uint4 a[kUnroll], b[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int64_t i = i0 + u * groups;
      if (i < n) {
        a[u] = reinterpret_cast<const uint4*>(O + i * kD)[sub];
        b[u] = reinterpret_cast<const uint4*>(dO + i * kD)[sub];
      }
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int64_t i = i0 + u * groups;
      if (i >= n) break;
      const __nv_bfloat162* pa = reinterpret_cast<const __nv_bfloat162*>(&a[u]);
      const __nv_bfloat162* pb = reinterpret_cast<const __nv_bfloat162*>(&b[u]);
      float acc = 0.f;
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const float2 x = __bfloat1622float2(pa[k]), y = __bfloat1622float2(pb[k]);
        acc = fmaf(x.x, y.x, fmaf(x.y, y.y, acc));
      }
#pragma unroll
      for (int o = 8; o > 0; o >>= 1) acc += __shfl_xor_sync(group_mask, acc, o);
      if (sub == 0) {
        const int64_t row = i / hq;
        const int h = (int)(i % hq);
        delta[(int64_t)h * rows + row] = acc;
      }
    }
  }
}

// ------------------------------------------------------------------ dQ
// dS goes back into tensor memory over the S it came from and is the A
// operand of dQ += dS K, so shared memory holds Q, dO, a 3-stage K ring (K is
// read by the first and the last MMA of a block) and a 2-stage V ring.  S is
// double-buffered in tensor memory: S_{c+1} is computed while block c's
// scores are turned into dS.
namespace dq {
constexpr int kKStages = 3;
constexpr uint32_t OFF_Q = 0, OFF_DO = kTileBytes, OFF_K = 2 * kTileBytes, OFF_V = 5 * kTileBytes,
                   OFF_BAR = 7 * kTileBytes;
constexpr uint32_t kSmemBytes = OFF_BAR + 256 + 1024;
constexpr uint32_t TM_S = 0, TM_DP = 256, TM_DQ = 384;  // S regions at 0 and 128

struct Bars {
  uint64_t qdo_full;
  uint64_t k_full[kKStages], k_empty[kKStages], v_full[2], v_empty[2];
  uint64_t s_full[2], p_full[2], dq_done[2];  // per S region
  uint64_t dp_full, dp_read, final_mma;
  uint32_t tmem_base;
  int32_t abort;
};
static_assert(sizeof(Bars) <= 256, "barrier block");
}  // namespace dq

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

__global__ void __launch_bounds__(kThreads, 1)
    dq_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmdO,
              const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV, const AttnArgs a) {
  using namespace dq;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  Bars* bar = reinterpret_cast<Bars*>(smem + OFF_BAR);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int64_t tpos;
  int h;
  bucket_item(blockIdx.x, a.nq, a.hq, tpos, h, a.hq == a.hkv);  // blocks start roughly in index order
  const Tile w = a.qtiles[a.q_order[tpos]];
  const int g = h / (a.hq / a.hkv);
  const int nkb = w.a1, kfull = w.a0;

  if (threadIdx.x == 0) {
    ptx::mbar_init(&bar->qdo_full, 1);
    for (int s = 0; s < kKStages; ++s) {
      ptx::mbar_init(&bar->k_full[s], 1);
      ptx::mbar_init(&bar->k_empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      ptx::mbar_init(&bar->v_full[s], 1);
      ptx::mbar_init(&bar->v_empty[s], 1);
      ptx::mbar_init(&bar->s_full[s], 1);
      ptx::mbar_init(&bar->p_full[s], kComputeThreads);
      ptx::mbar_init(&bar->dq_done[s], 1);
    }
    ptx::mbar_init(&bar->dp_full, 1);
    ptx::mbar_init(&bar->dp_read, kComputeThreads);
    ptx::mbar_init(&bar->final_mma, 1);
    bar->abort = 0;
    ptx::fence_mbar_init();
  }
  if (warp == 9) {
    ptx::tmem_alloc(&bar->tmem_base, kTmemCols);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = bar->tmem_base;

  if (warp == 8) {
    // the warp waits converged, lane 0 issues the copies
    if (nkb > 0) {
      if (lane == 0) {
        ptx::tma_prefetch_desc(&tmK);
        ptx::tma_prefetch_desc(&tmV);
        const int32_t qy = w.q_base + w.tile * kRows;
        ptx::mbar_expect_tx(&bar->qdo_full, 2 * kTileBytes);
        ptx::tma_load_2d(smem + OFF_Q, &tmQ, &bar->qdo_full, h * kD, qy);
        ptx::tma_load_2d(smem + OFF_Q + kHalfBytes, &tmQ, &bar->qdo_full, h * kD + 64, qy);
        ptx::tma_load_2d(smem + OFF_DO, &tmdO, &bar->qdo_full, h * kD, qy);
        ptx::tma_load_2d(smem + OFF_DO + kHalfBytes, &tmdO, &bar->qdo_full, h * kD + 64, qy);
      }
      __syncwarp();
      uint32_t nk[kKStages] = {0, 0, 0}, nv[2] = {0, 0};
      for (int c = 0; c < nkb; ++c) {
        const int sk = c % kKStages, sv = c & 1;
        if (__any_sync(0xffffffffu, aborted(&bar->abort))) break;
        const int32_t ky = w.k_base + c * kRows;
        if (c >= kKStages && !wait_warp(&bar->k_empty[sk], (uint32_t)(c / kKStages - 1) & 1, a.status)) {
          if (lane == 0) set_abort(&bar->abort);
          break;
        }
        if (lane == 0) {
          ptx::mbar_expect_tx(&bar->k_full[sk], kTileBytes);
          ptx::tma_load_2d(smem + OFF_K + sk * kTileBytes, &tmK, &bar->k_full[sk], g * kD, ky);
          ptx::tma_load_2d(smem + OFF_K + sk * kTileBytes + kHalfBytes, &tmK, &bar->k_full[sk], g * kD + 64, ky);
        }
        __syncwarp();
        ++nk[sk];
        if (c >= 2 && !wait_warp(&bar->v_empty[sv], (uint32_t)((c >> 1) - 1) & 1, a.status)) {
          if (lane == 0) set_abort(&bar->abort);
          break;
        }
        if (lane == 0) {
          ptx::mbar_expect_tx(&bar->v_full[sv], kTileBytes);
          ptx::tma_load_2d(smem + OFF_V + sv * kTileBytes, &tmV, &bar->v_full[sv], g * kD, ky);
          ptx::tma_load_2d(smem + OFF_V + sv * kTileBytes + kHalfBytes, &tmV, &bar->v_full[sv], g * kD + 64, ky);
        }
        __syncwarp();
        ++nv[sv];
      }
      if (__any_sync(0xffffffffu, aborted(&bar->abort))) {
        wait_warp(&bar->qdo_full, 0, a.status);
        for (int s = 0; s < kKStages; ++s)
          if (nk[s]) wait_warp(&bar->k_full[s], (nk[s] - 1) & 1, a.status);
        for (int s = 0; s < 2; ++s)
          if (nv[s]) wait_warp(&bar->v_full[s], (nv[s] - 1) & 1, a.status);
      }
    }
  } else if (warp == 9) {
    // the whole warp runs the loop, one elected lane issues each instruction
    if (nkb > 0) {
      constexpr uint32_t idesc_nt = ptx::idesc_bf16_f32(128, 128, 0, 0);  // A K-major, B K-major
      constexpr uint32_t idesc_nn = ptx::idesc_bf16_f32(128, 128, 0, 1);  // A K-major, B MN-major
      const uint32_t sQ = ptx::smem_u32(smem + OFF_Q), sdO = ptx::smem_u32(smem + OFF_DO);
      auto issue_s = [&](int c) {
        const uint32_t sK = ptx::smem_u32(smem + OFF_K + (c % kKStages) * kTileBytes);
        ptx::mma8_bf16_ss_warp<ptx::KMajorSw128, ptx::KMajorSw128>(tmem + TM_S + 128u * (c & 1), desc_kmajor(sQ, 0),
                                                                  desc_kmajor(sK, 0), idesc_nt, 0u);
        ptx::mma_commit_warp(&bar->s_full[c & 1]);
      };
      auto issue_dp = [&](int c) {
        const int sv = c & 1;
        const uint32_t sV = ptx::smem_u32(smem + OFF_V + sv * kTileBytes);
        ptx::mma8_bf16_ss_warp<ptx::KMajorSw128, ptx::KMajorSw128>(tmem + TM_DP, desc_kmajor(sdO, 0), desc_kmajor(sV, 0),
                                                                  idesc_nt, 0u);
        ptx::mma_commit_warp(&bar->dp_full);
        ptx::mma_commit_warp(&bar->v_empty[sv]);
      };
      auto issue_dq = [&](int c) {
        const int R = c & 1;
        const uint32_t sK = ptx::smem_u32(smem + OFF_K + (c % kKStages) * kTileBytes);
        // dQ += dS K_c: dS (bf16, keys packed two per column) in S region R, keys [0,64) at
        // columns [0,32) and [64,128) at columns [64,96)
        ptx::mma8_bf16_ts_warp<ptx::TmemPairsGap32, ptx::MnMajorSw128>(tmem + TM_DQ, tmem + TM_S + 128u * R,
                                                                      desc_mnmajor(sK, 0), idesc_nn, c > 0 ? 1u : 0u);
        ptx::mma_commit_warp(&bar->dq_done[R]);
        ptx::mma_commit_warp(&bar->k_empty[c % kKStages]);
      };
      // Event-driven issue: S_c, dP_c, dQ_c go out as soon as their inputs are
      // ready, so no wait blocks an unrelated MMA.
      //   S_c  needs K_c and dQ_{c-2} issued (it overwrites the dS that dQ_{c-2}
      //        reads; MMAs of this thread execute in order, or, with
      //        kFlagDrainTmemReuse, dQ_{c-2} completed)
      //   dP_c needs V_c and dP_{c-1} read by the compute warps
      //   dQ_c needs dS_c written
      bool ok = wait_warp(&bar->qdo_full, 0, a.status) && wait_warp(&bar->k_full[0], 0, a.status) &&
                wait_warp(&bar->v_full[0], 0, a.status);
      if (ok) {
        ptx::tc_fence_after();
        issue_s(0);
        issue_dp(0);
      }
      int ns = 1, nd = 1, nq = 0;
      uint64_t t_idle = 0;
      while (ok && nq < nkb) {
        bool progressed = false;
        if (ns < nkb && (ns < 2 || nq > ns - 2) &&
            (ns < 2 || !(a.flags & kFlagDrainTmemReuse) ||
             ptx::mbar_test_warp(&bar->dq_done[ns & 1], (uint32_t)((ns - 2) >> 1) & 1)) &&
            ptx::mbar_test_warp(&bar->k_full[ns % kKStages], (uint32_t)(ns / kKStages) & 1)) {
          ptx::tc_fence_after();
          issue_s(ns++);
          progressed = true;
        }
        if (nd < nkb && ptx::mbar_test_warp(&bar->dp_read, (uint32_t)(nd - 1) & 1) &&
            ptx::mbar_test_warp(&bar->v_full[nd & 1], (uint32_t)(nd >> 1) & 1)) {
          ptx::tc_fence_after();
          issue_dp(nd++);
          progressed = true;
        }
        if (nq < ns && nq < nd && ptx::mbar_test_warp(&bar->p_full[nq & 1], (uint32_t)(nq >> 1) & 1)) {
          ptx::tc_fence_after();
          issue_dq(nq++);
          progressed = true;
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
      if (!ok && lane == 0) set_abort(&bar->abort);
      __syncwarp();
      ptx::mma_commit_warp(&bar->final_mma);
      wait_warp(&bar->final_mma, 0, a.status);
    }
    __syncwarp();
  } else {
    // compute: thread = query row r of the tile; warpgroup wg owns key columns [64 wg, 64 wg + 64)
    const int wg = threadIdx.x >> 7, r = threadIdx.x & 127;
    const uint32_t lane_addr = (uint32_t)((warp & 3) * 32) << 16;
    const int row = w.tile * kRows + r;
    const bool valid = row < w.q_len;
    const int64_t grow = (int64_t)w.q_base + row;
    const int ke = valid ? a.kv_end[w.kv_base + row] : 0;
    const float lse2 = valid ? a.lse_in[(int64_t)h * a.q_rows + grow] * kLog2e : 0.f;
    const float dl = valid ? a.delta[(int64_t)h * a.q_rows + grow] : 0.f;
    const float sl2 = a.scale * kLog2e;
    bool ok = nkb > 0;
    for (int c = 0; ok && c < nkb; ++c) {
      const int R = c & 1;
      const uint32_t tS = tmem + lane_addr + TM_S + 128u * R + 64u * wg;
      if (!wait(&bar->s_full[R], (uint32_t)(c >> 1) & 1, a.status) || !wait(&bar->dp_full, (uint32_t)c & 1, a.status)) {
        ok = false;
        break;
      }
      ptx::tc_fence_after();
      uint32_t s0[32], s1[32], d0[32], d1[32];
      ld64(tS, s0, s1);
      ld64(tmem + lane_addr + TM_DP + 64u * wg, d0, d1);
      ptx::tmem_ld_wait();
      ptx::reg_fence(s0);
      ptx::reg_fence(s1);
      ptx::reg_fence(d0);
      ptx::reg_fence(d1);
      ptx::tc_fence_before();
      ptx::mbar_arrive(&bar->dp_read);
      const int lim = (c < kfull) ? 128 : ke - c * kRows - wg * 64;  // visible columns of this half
      uint32_t pk[32];  // pk[k] holds columns 2k and 2k+1 of this half
#pragma unroll
      for (int k = 0; k < 32; ++k) {
        float v[2];
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int jj = 2 * k + e;
          const float sv = __uint_as_float(jj < 32 ? s0[jj] : s1[jj - 32]);
          const float dv = __uint_as_float(jj < 32 ? d0[jj] : d1[jj - 32]);
          const float p = jj < lim ? ex2(sv * sl2 - lse2) : 0.f;
          v[e] = p * (dv - dl);
        }
        pk[k] = pack_bf16(v[0], v[1]);
      }
      // dS over the first 32 columns of this half of S (already read)
      ptx::tmem_st32(tS, pk);
      ptx::tmem_st_wait();
      ptx::tc_fence_before();
      ptx::mbar_arrive(&bar->p_full[R]);
    }
    // rotary encoding: this warpgroup's 32 pairs of the row's tables, loaded
    // while the last dQ MMAs run
    float rc[32], rs[32];
    if (valid && a.rope_cos) {
      const int64_t pos = (int64_t)w.tile * kRows + r;
      rope_row<32>(a.rope_cos + pos * 64 + wg * 32, a.rope_sin + pos * 64 + wg * 32, rc, rs);
    }
    if (ok) ok = wait(&bar->final_mma, 0, a.status);
    if (!ok) {
      set_abort(&bar->abort);
    } else {
      ptx::tc_fence_after();
      uint32_t q0[32], q1[32];
      if (a.rope_cos) {
        // rotary encoding: warpgroup wg takes columns wg*32.. and 64 + wg*32.., which pair up
        ptx::tmem_ld32(tmem + lane_addr + TM_DQ + wg * 32, q0);
        ptx::tmem_ld32(tmem + lane_addr + TM_DQ + 64 + wg * 32, q1);
      } else {
        ld64(tmem + lane_addr + TM_DQ + wg * 64, q0, q1);
      }
      ptx::tmem_ld_wait();
      ptx::reg_fence(q0);
      ptx::reg_fence(q1);
      // rows are stored by groups of four lanes (store_slice32)
      const int64_t rstride = (int64_t)a.hq * kD;
      __nv_bfloat16* const g0 = reinterpret_cast<__nv_bfloat16*>(a.dq) + (grow - (lane & 3)) * rstride + h * kD;
      const int g_rows = w.q_len - (row - (lane & 3));
      uint32_t w0[16], w1[16];
      if (a.rope_cos) {
        if (!valid) {
#pragma unroll
          for (int k = 0; k < 32; ++k) rc[k] = rs[k] = 0.f;
        }
        rope_back_pack(q0, q1, a.scale, rc, rs, w0, w1);
        store_slice32(w0, g0 + 32 * wg, rstride, g_rows);
        store_slice32(w1, g0 + 64 + 32 * wg, rstride, g_rows);
      } else {
        pack_scaled32(q0, a.scale, w0);
        pack_scaled32(q1, a.scale, w1);
        store_slice32(w0, g0 + 64 * wg, rstride, g_rows);
        store_slice32(w1, g0 + 64 * wg + 32, rstride, g_rows);
      }
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 9) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, kTmemCols);
  }
}

// ------------------------------------------------------------------ dK / dV
namespace dkv {
// Q is read by the first (S^T) and the last (dK) MMA of an iteration, so it
// gets a 3-stage ring; dO (dP^T early, dV late) 2 stages.  P^T lives in tensor
// memory over the S^T it came from and dS^T over the dP^T it came from, so dV
// can start as soon as P is written and dP^T of the next tile only waits for dK.
constexpr int kQStages = 3;
constexpr uint32_t OFF_K = 0, OFF_V = kTileBytes, OFF_Q = 2 * kTileBytes, OFF_DO = 5 * kTileBytes,
                   OFF_META = 7 * kTileBytes;
// per stage: lse2[128] f32, delta[128] f32, visible-key count[128] u8
constexpr uint32_t kMetaStage = 128 * 4 + 128 * 4 + 128;
constexpr uint32_t OFF_BAR = OFF_META + 2 * kMetaStage;
constexpr uint32_t kSmemBytes = OFF_BAR + 512;  // needs a 1024-aligned dynamic shared base
constexpr uint32_t TM_S = 0, TM_DP = 128, TM_DV = 256, TM_DK = 384;
// warps 0-7 compute, 8 work items + TMA loads, 9 TMEM + MMA issue, 10 per-query metadata
constexpr int kLoadWarp = 8, kMmaWarp = 9, kMetaWarp = 10;
constexpr int kThreads = 352;
constexpr int kItemSlots = 4;  // work items published ahead of the roles that follow them

struct Bars {
  uint64_t kv_full, kv_empty;
  uint64_t q_full[kQStages], q_empty[kQStages], do_full[2], do_empty[2], meta_full[2], meta_empty[2];
  uint64_t item_full[kItemSlots];
  uint64_t s_full, dp_full, pt_full, p_full, dv_done, dk_done, acc_full, final_mma;
  uint32_t tmem_base;
  int32_t abort;
  uint32_t full[2][2];  // per meta stage and warpgroup: all 64 queries see all 128 keys
  int32_t items[kItemSlots];
};
static_assert(sizeof(Bars) <= 512, "barrier block");
static_assert(kSmemBytes <= 232448, "shared memory per CTA");
}  // namespace dkv

__global__ void __launch_bounds__(dkv::kThreads, 1)
    dkdv_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmdO,
                const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV, const AttnArgs a) {
  using namespace dkv;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw;
  Bars* bar = reinterpret_cast<Bars*>(smem + OFF_BAR);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (ptx::smem_u32(smem) & 1023u) {  // the swizzled tiles need 1024-byte alignment
    if (threadIdx.x == 0) atomicOr(a.status, kStatusSmemAlign);
    return;
  }
  const int group = a.hq / a.hkv;
  const int64_t n_items = a.nk * a.hkv;

  if (threadIdx.x == 0) {
    ptx::mbar_init(&bar->kv_full, 1);
    ptx::mbar_init(&bar->kv_empty, 1);
    for (int s = 0; s < kQStages; ++s) {
      ptx::mbar_init(&bar->q_full[s], 1);
      ptx::mbar_init(&bar->q_empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      ptx::mbar_init(&bar->do_full[s], 1);
      ptx::mbar_init(&bar->do_empty[s], 1);
      ptx::mbar_init(&bar->meta_full[s], 32);
      ptx::mbar_init(&bar->meta_empty[s], kComputeThreads);
    }
    for (int s = 0; s < kItemSlots; ++s) ptx::mbar_init(&bar->item_full[s], 1);
    ptx::mbar_init(&bar->s_full, 1);
    ptx::mbar_init(&bar->dp_full, 1);
    ptx::mbar_init(&bar->pt_full, kComputeThreads);
    ptx::mbar_init(&bar->p_full, kComputeThreads);
    ptx::mbar_init(&bar->dv_done, 1);
    ptx::mbar_init(&bar->dk_done, 1);
    ptx::mbar_init(&bar->acc_full, 1);
    ptx::mbar_init(&bar->final_mma, 1);
    bar->abort = 0;
    ptx::fence_mbar_init();
  }
  if (warp == kMmaWarp) {
    ptx::tmem_alloc(&bar->tmem_base, kTmemCols);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = bar->tmem_base;

  // Work items (k-tile k_order[item / hkv], KV head item % hkv) come from a
  // global counter, most expensive first; the load warp takes them and
  // publishes each in a small shared ring that the other roles follow, so
  // every role of the CTA walks the same items.  A negative entry ends the walk.
  struct Item {
    int g, gk, c, qt0, nqt, n_it;
    Tile w;
  };
  auto decode = [&](int item, Item& x) {
    int64_t kpos;
    bucket_item(item, a.nk, a.hkv, kpos, x.g);
    x.gk = a.k_order[kpos];
    x.w = a.ktiles[x.gk];
    x.c = x.w.tile;
    x.qt0 = x.w.a0;
    x.nqt = x.w.a1;
    x.n_it = x.nqt > x.qt0 ? (x.nqt - x.qt0) * group : 0;
  };
  // the item of slot u, waited for by every role but the load warp (false: stop)
  auto next_item = [&](uint32_t u, Item& x) -> bool {
    const int slot = (int)(u % kItemSlots);
    if (!wait(&bar->item_full[slot], (u / kItemSlots) & 1, a.status)) return false;
    const int item = *reinterpret_cast<volatile int32_t*>(&bar->items[slot]);
    if (item < 0) return false;
    decode(item, x);
    return true;
  };
  // Iteration i of an item visits query tile nqt - 1 - i / group of query head
  // g * group + i % group: the key tiles of a sequence all start at its last
  // query tile and move down together, so the CTAs running at the same time
  // read the same Q / dO tiles and mostly hit L2.  Barrier phases count
  // iterations (I) and items (u) across the whole walk.

  if (warp == kLoadWarp) {
    // ------------------------------------------------ work items and TMA loads (the warp waits
    // converged, lane 0 issues)
    uint32_t I = 0, nq[kQStages] = {0, 0, 0}, ndo[2] = {0, 0}, nkv = 0;
    bool ok = true;
    for (uint32_t u = 0;;) {
      int item = -1;
      if (lane == 0) {
        item = ok && !aborted(&bar->abort) ? atomicAdd(a.work_counter, 1) : -1;
        if (item >= n_items) item = -1;
      }
      item = __shfl_sync(0xffffffffu, item, 0);
      Item x;
      if (item >= 0) {
        decode(item, x);
        if (x.n_it == 0) {
          // no query sees these keys (with ISM segments every key sees at least
          // itself, so this is only a guard): dK = dV = 0, and the item is not published
          for (int rr = lane; rr < kRows; rr += 32) {
            const int key = x.c * kRows + rr;
            if (key >= x.w.k_len) break;
            const int64_t off = ((int64_t)x.w.k_base + key) * a.hkv * kD + x.g * kD;
            uint4* dk = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(a.dk) + off);
            uint4* dv = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(a.dv) + off);
            for (int k = 0; k < kD / 8; ++k) dk[k] = dv[k] = make_uint4(0u, 0u, 0u, 0u);
          }
          continue;
        }
      }
      // Every published item has iterations, so the load warp cannot run more
      // than one item ahead of the MMA warp (kv_empty) and a ring slot is never
      // rewritten before every role has read it.
      if (lane == 0) {
        const int slot = (int)(u % kItemSlots);
        bar->items[slot] = item;
        ptx::mbar_arrive(&bar->item_full[slot]);  // release: the entry is visible to the waiters
      }
      __syncwarp();
      ++u;
      if (item < 0) break;
      // K and V of this item once the previous item's S and dP MMAs are done with them
      if (nkv > 0 && !wait_warp(&bar->kv_empty, (nkv - 1) & 1, a.status)) {
        if (lane == 0) set_abort(&bar->abort);
        ok = false;
        continue;
      }
      const int32_t ky = x.w.k_base + x.c * kRows;
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
            ptx::mbar_expect_tx(&bar->q_full[sq], kTileBytes);
            ptx::tma_load_2d(smem + OFF_Q + sq * kTileBytes, &tmQ, &bar->q_full[sq], h * kD, qy);
            ptx::tma_load_2d(smem + OFF_Q + sq * kTileBytes + kHalfBytes, &tmQ, &bar->q_full[sq], h * kD + 64, qy);
          }
          __syncwarp();
          ++nq[sq];
          okq = I < 2 || wait_warp(&bar->do_empty[s], ((I >> 1) - 1) & 1, a.status);
        }
        if (okq) {
          if (lane == 0) {
            ptx::mbar_expect_tx(&bar->do_full[s], kTileBytes);
            ptx::tma_load_2d(smem + OFF_DO + s * kTileBytes, &tmdO, &bar->do_full[s], h * kD, qy);
            ptx::tma_load_2d(smem + OFF_DO + s * kTileBytes + kHalfBytes, &tmdO, &bar->do_full[s], h * kD + 64, qy);
          }
          __syncwarp();
          ++ndo[s];
        }
        if (!okq) {
          if (lane == 0) set_abort(&bar->abort);
          ok = false;
          break;
        }
      }
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
        if (I >= 2 && !wait(&bar->meta_empty[s], ((I >> 1) - 1) & 1, a.status)) { set_abort(&bar->abort); break; }
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
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------ MMA issue (the whole warp runs the
    // loop, one elected lane issues each instruction)
    constexpr uint32_t idesc_nt = ptx::idesc_bf16_f32(128, 128, 0, 0);
    constexpr uint32_t idesc_nn = ptx::idesc_bf16_f32(128, 128, 0, 1);
    const uint32_t sK = ptx::smem_u32(smem + OFF_K), sV = ptx::smem_u32(smem + OFF_V);
    uint32_t I0 = 0, nkv = 0;  // iterations of earlier items; items with K / V loaded
    bool ok = true;
    auto issue_s = [&](uint32_t gi) {
      const uint32_t sQ = ptx::smem_u32(smem + OFF_Q + (gi % kQStages) * kTileBytes);
      ptx::mma8_bf16_ss_warp<ptx::KMajorSw128, ptx::KMajorSw128>(tmem + TM_S, desc_kmajor(sK, 0), desc_kmajor(sQ, 0), idesc_nt, 0u);
      ptx::mma_commit_warp(&bar->s_full);
    };
    auto issue_dp = [&](uint32_t gi) {
      const uint32_t sdO = ptx::smem_u32(smem + OFF_DO + (gi & 1) * kTileBytes);
      ptx::mma8_bf16_ss_warp<ptx::KMajorSw128, ptx::KMajorSw128>(tmem + TM_DP, desc_kmajor(sV, 0), desc_kmajor(sdO, 0), idesc_nt, 0u);
      ptx::mma_commit_warp(&bar->dp_full);
    };
    // P^T (bf16, two queries per column) sits in the S^T columns and dS^T in the dP^T
    // columns: warpgroup wg's queries [64 wg, 64 wg + 64) at column 64 wg + [0, 32)
    auto issue_dv = [&](uint32_t gi, bool first) {
      const uint32_t s = gi & 1;
      const uint32_t sdO = ptx::smem_u32(smem + OFF_DO + s * kTileBytes);
      ptx::mma8_bf16_ts_warp<ptx::TmemPairsGap32, ptx::MnMajorSw128>(tmem + TM_DV, tmem + TM_S, desc_mnmajor(sdO, 0), idesc_nn, first ? 0u : 1u);
      ptx::mma_commit_warp(&bar->do_empty[s]);
      ptx::mma_commit_warp(&bar->dv_done);
    };
    auto issue_dk = [&](uint32_t gi, bool first) {
      const uint32_t sq = gi % kQStages;
      const uint32_t sQ = ptx::smem_u32(smem + OFF_Q + sq * kTileBytes);
      ptx::mma8_bf16_ts_warp<ptx::TmemPairsGap32, ptx::MnMajorSw128>(tmem + TM_DK, tmem + TM_DP, desc_mnmajor(sQ, 0), idesc_nn, first ? 0u : 1u);
      ptx::mma_commit_warp(&bar->q_empty[sq]);
      ptx::mma_commit_warp(&bar->dk_done);
    };
    Item x;
    for (uint32_t u = 0; ok; ++u) {
      if (!__all_sync(0xffffffffu, next_item(u, x))) break;
      const int n_it = x.n_it;
      if (!wait_warp(&bar->kv_full, nkv & 1, a.status)) { ok = false; break; }
      ++nkv;
      // Event-driven issue, in order of urgency (the tensor pipe runs MMAs in
      // issue order, so whatever is issued first runs first):
      //   dK_i  needs dS^T_i written (p_full)
      //   dP_i  needs dO_i and dK_{i-1} issued (it overwrites the dS^T dK_{i-1}
      //         reads; MMAs of this thread execute in order, or, with
      //         kFlagDrainTmemReuse, dK_{i-1} completed)
      //   dV_i  needs P^T_i written (pt_full) and dP_i issued (both read dO_i)
      //   S_i   needs Q_i and dV_{i-1} issued (it overwrites the P^T dV_{i-1}
      //         reads; in order, or with the flag, dV_{i-1} completed)
      // The first dV / dK of an item restart the accumulators, which the
      // compute warps have read out (their epilogue of the previous item comes
      // before the P^T / dS^T writes these MMAs wait for).
      // counters of issued S, dP, dV, dK over the whole walk; this item ends at `end`
      const uint32_t end = I0 + (uint32_t)n_it;
      uint32_t ns = I0, np = I0, nv = I0, nk = I0;
      uint32_t qs = I0 % kQStages, qph = (I0 / kQStages) & 1;  // Q stage and phase of S_ns
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
            (np == 0 || !(a.flags & kFlagDrainTmemReuse) || ptx::mbar_test_warp(&bar->dk_done, (np - 1) & 1))) {
          ptx::tc_fence_after();
          issue_dp(np);
          ++np;
          progressed = true;
          // the last MMAs reading this item's K and V are issued: the next K / V may load
          if (np == end && ns == end) ptx::mma_commit_warp(&bar->kv_empty);
        }
        if (nv < np && ptx::mbar_test_warp(&bar->pt_full, nv & 1)) {
          ptx::tc_fence_after();
          issue_dv(nv, nv == I0);
          ++nv;
          progressed = true;
        }
        if (ns < end && ns <= nv && ptx::mbar_test_warp(&bar->q_full[qs], qph) &&
            (ns == 0 || !(a.flags & kFlagDrainTmemReuse) || ptx::mbar_test_warp(&bar->dv_done, (ns - 1) & 1))) {
          ptx::tc_fence_after();
          issue_s(ns);
          ++ns;
          if (++qs == kQStages) { qs = 0; qph ^= 1; }
          progressed = true;
          if (np == end && ns == end) ptx::mma_commit_warp(&bar->kv_empty);
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
      ptx::mma_commit_warp(&bar->acc_full);  // dV, dK of this item complete
      I0 = end;
    }
    if (!ok && lane == 0) set_abort(&bar->abort);
    __syncwarp();
    ptx::mma_commit_warp(&bar->final_mma);
    wait_warp(&bar->final_mma, 0, a.status);
    __syncwarp();
  } else {
    // ------------------------------------------------ compute: thread = key row r, warpgroup wg owns queries [64 wg, 64 wg + 64)
    const int wg = threadIdx.x >> 7, r = threadIdx.x & 127;
    const uint32_t lane_addr = (uint32_t)((warp & 3) * 32) << 16;
    const uint32_t tS = tmem + lane_addr + TM_S + 64u * wg, tP = tmem + lane_addr + TM_DP + 64u * wg;
    const float sl2 = a.scale * kLog2e;
    // the stored dS is read back only by the dQ GEMM, after this kernel: its
    // lines go first when L2 needs room, ahead of the Q / dO tiles other CTAs reuse
    const uint64_t pol_ds = ptx::l2_policy_evict_first();
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
        ptx::mbar_arrive(&bar->pt_full);
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
        ptx::mbar_arrive(&bar->p_full);
        if (a.ds) {
          // keep dS^T row r, queries [64 wg, 64 wg + 64), for the dQ GEMM, in
          // the 8-interleaved layout (16-byte unit (query group, key)): the 32
          // lanes of a warp store 512 contiguous bytes per instruction.  Issued
          // after the hand-off so that the dV/dK MMAs do not wait for it.
          const int hh = i % group, t = x.nqt - 1 - i / group;
          const int64_t slot = ((int64_t)a.kpair_off[x.gk] + (t - x.qt0)) * a.hq + (x.g * group + hh);
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
    if (!ok) set_abort(&bar->abort);
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, kTmemCols);
  }
}

}  // namespace

cudaError_t launch_dkdv_pair(const AttnArgs& a, const CUtensorMap& tk, const CUtensorMap& tv, cudaStream_t st);

cudaError_t launch_bwd(const AttnArgs& a, int64_t k_rows, cudaStream_t st) {
  cudaError_t e;
  if (a.q_rows > 0) {
    int64_t groups = a.q_rows * a.hq;
    int grid = (int)((groups * 16 + 255) / 256);
    if (grid > 152 * 16) grid = 152 * 16;
    timer_begin(ISM_KERNEL_BWD_PRE, st);
    delta_kernel<<<grid, 256, 0, st>>>((const __nv_bfloat16*)a.o, (const __nv_bfloat16*)a.dout, a.delta, a.q_rows,
                                       a.hq);
    timer_end(ISM_KERNEL_BWD_PRE, st);
    count_launch();
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  CUtensorMap tq, tdo, tk, tv;
  if ((e = make_tmap_bf16(&tq, a.q, (uint64_t)a.hq * kD, (uint64_t)a.q_rows)) != cudaSuccess) return e;
  if ((e = make_tmap_bf16(&tdo, a.dout, (uint64_t)a.hq * kD, (uint64_t)a.q_rows)) != cudaSuccess) return e;
  if ((e = make_tmap_bf16(&tk, a.k, (uint64_t)a.hkv * kD, (uint64_t)k_rows)) != cudaSuccess) return e;
  if ((e = make_tmap_bf16(&tv, a.v, (uint64_t)a.hkv * kD, (uint64_t)k_rows)) != cudaSuccess) return e;
  // Recompute path: dQ recomputes S, P and dP itself and runs before dK/dV.
  // Stored-dS path: dK/dV writes the dS^T tiles, then dQ is a GEMM over them.
  if (a.nq && !a.ds) {
    if ((e = cudaFuncSetAttribute(dq_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dq::kSmemBytes)) !=
        cudaSuccess)
      return e;
    timer_begin(ISM_KERNEL_BWD_DQ, st);
    dq_kernel<<<(unsigned)(a.nq * a.hq), kThreads, dq::kSmemBytes, st>>>(tq, tdo, tk, tv, a);
    timer_end(ISM_KERNEL_BWD_DQ, st);
    count_launch();
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  if (a.nk && knobs().dkdv_pair && a.kp_order) {
    // the CTA-pair kernel (ism_dkdv2_tc.cu)
    timer_begin(ISM_KERNEL_BWD_DKDV, st);
    if ((e = launch_dkdv_pair(a, tk, tv, st)) != cudaSuccess) return e;
    timer_end(ISM_KERNEL_BWD_DKDV, st);
    count_launch();
  } else if (a.nk) {
    if ((e = cudaFuncSetAttribute(dkdv_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)dkv::kSmemBytes)) != cudaSuccess)
      return e;
    // persistent: one CTA per SM takes (k-tile, KV head) items from the work counter
    int64_t grid = knobs().dkdv_grid > 0 ? knobs().dkdv_grid : sm_count();
    if (grid > a.nk * a.hkv) grid = a.nk * a.hkv;
    if (!a.work_counter) return cudaErrorInvalidValue;
    timer_begin(ISM_KERNEL_BWD_DKDV, st);
    dkdv_kernel<<<(unsigned)grid, dkv::kThreads, dkv::kSmemBytes, st>>>(tq, tdo, tk, tv, a);
    timer_end(ISM_KERNEL_BWD_DKDV, st);
    count_launch();
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  if (a.nq && a.ds) {
    timer_begin(ISM_KERNEL_BWD_DQ, st);
    if ((e = launch_dq_gemm(a, tk, st)) != cudaSuccess) return e;
    timer_end(ISM_KERNEL_BWD_DQ, st);
    count_launch();
  }
  return cudaSuccess;
}

}  // namespace tc

bool tc_bwd_available() { return tc::available(); }
cudaError_t launch_tc_bwd(const AttnArgs& a, int64_t k_rows, cudaStream_t st) { return tc::launch_bwd(a, k_rows, st); }

}  // namespace ism
