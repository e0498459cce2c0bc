// Single-token decode on the tensor cores (sm_103a), bf16 caches, head_dim 128.
//
// A decode step (Section 2.3: the new answer token attends to the whole reused
// cache plus itself) reads every cached key and value of a (sequence, KV head)
// once, so it is bound by HBM.  The CUDA-core decode spends most of its issue
// slots on dot products and the reductions that assemble them; here both
// contractions run on the tensor cores and the threads only do the softmax.
//
// Work item: (sequence b, KV head g, split) = keys [k0, k1) of the cache, in
// tiles of 128 keys.  A persistent CTA per SM walks the items; per item
//   pass 1: S^T_t = K_t Q^T for every tile t (M = 128 keys, N = 16 query
//           heads of the group, zero or foreign rows past the group), all
//           tiles kept in tensor memory (16 columns each); the softmax
//           warps fold each ring tile's scores into a running maximum as
//           soon as its MMAs complete, while the next K tiles stream in;
//   the exact maximum per head over the item's keys;
//   pass 2: P_t = exp2(S_t * scale * log2 e - m) as bf16 into a 128-byte
//           swizzled MN-major operand in shared memory (rows = keys, the
//           heads contiguous: a thread stores its key's 16 heads as whole
//           16-byte chunks), then O += P_t V_t (M = 128 with the group in
//           rows 0-15, N = 128 dimensions, K = 128 keys; V MN-major as it
//           arrives).
// With the exact maximum known before any P, no rescaling of O is needed.
// The item's (max, sum, unnormalised O) per head go to the split partials,
// which decode_combine_kernel merges as for the CUDA-core kernels.
// Warps 0-3: softmax and epilogue (thread = key of a tile, TMEM lane);
// warp 4: TMA loads (Q of the item, then its K tiles, then its V tiles,
// through one ring); warp 5: MMA issue.
// e4m3 caches (kE4M3): Q, K, V, P in e4m3 (kind::f8f6f4 MMAs, K = 32 a step,
// 128-byte rows: one swizzled box per 128 keys), scores scaled by qk_descale,
// O by v_descale.  A ring tile holds 256 keys (two 128-key boxes, 32 KB, the
// size of a bf16 tile): each hand-off between the loads, the MMAs and the
// softmax warps then covers as many bytes as in bf16.  With 128-key e4m3
// tiles the per-tile chain, not DRAM, set the pace (0.77 of the copy
// bandwidth, the same with a deeper ring).  The last tile of an item may hold
// one 128-key half only; the other half is neither loaded nor multiplied.
#include "ism_tc_common.cuh"

namespace ism {
namespace tc {
namespace {

constexpr int kMaxStages = 8;
constexpr int kHeadsPad = 16;  // N of S^T = K Q^T
constexpr int kMaxTiles = kDecTcMaxKeys / 128;
constexpr int kThreads = 192;
constexpr int kLoadWarp = 4, kMmaWarp = 5;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t TM_O = 0, TM_S = 128;
static_assert(TM_S + kHeadsPad * kMaxTiles <= kTmemCols, "S tiles fit in tensor memory");

// Shared-memory plan: ring of K / V tiles, two P operands, two Q tiles, barriers.
template <bool kE4M3>
struct DecCfg {
  static constexpr int kStages = 4;
  static constexpr int kSub = kE4M3 ? 2 : 1;          // 128-key sub-tiles of a ring tile
  static constexpr uint32_t kTile = kTileBytes;       // bf16: 128 keys x 128 dims; e4m3: 256 keys x 128 dims
  static constexpr uint32_t kSubBytes = kTile / kSub;  // one 128-key sub-tile
  static constexpr uint32_t kQHalf = kHeadsPad * 128;                  // 16 rows x 128 bytes
  static constexpr uint32_t kQBytes = kE4M3 ? kQHalf : 2 * kQHalf;
  static constexpr uint32_t OFF_RING = 0, OFF_P = kStages * kTile, OFF_Q = OFF_P + 2 * kTile,
                            OFF_BAR = OFF_Q + 2 * kQBytes;
  static constexpr uint32_t kSmemBytes = OFF_BAR + 2048 + 1024;  // barrier block + 1024-byte alignment slack
  static_assert(kStages <= kMaxStages, "ring");
  static_assert(kSmemBytes <= 232448, "shared memory per CTA");
};

struct Bars {
  uint64_t full[kMaxStages], empty[kMaxStages];
  uint64_t q_full[2], q_empty[2];
  // S of ring tile n complete (s_tile[n % 4]) / read by the softmax warps (s_seen[n % 4]); the
  // MMA warp runs at most four ring tiles ahead, so a phase parity is never ambiguous
  uint64_t s_tile[4], s_seen[4];
  uint64_t s_free, p_ready[2], p_free[2], o_full, o_free, final_mma;
  uint64_t red_m_full, red_l_full;  // the four softmax warps' partial maxima / sums are written
  uint32_t tmem_base;
  int32_t abort;
  // per item parity: warp 0's epilogue of item u reads them while the other
  // warps may already fold the scores of item u + 1
  float red_m[2][4][kHeadsPad], red_l[2][4][kHeadsPad];
};
static_assert(sizeof(Bars) <= 2048, "barrier block");

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}
__device__ __forceinline__ bool aborted(const int32_t* f) { return *reinterpret_cast<const volatile int32_t*>(f) != 0; }
__device__ __forceinline__ void set_abort(int32_t* f) { *reinterpret_cast<volatile int32_t*>(f) = 1; }

struct DecItem {
  int b, g, split, k0, k1;
  int nt;    // ring tiles (kSub sub-tiles of 128 keys each, the last possibly short)
  int nsub;  // 128-key sub-tiles
};
// item = (split * batch + b) * hkv + g: consecutive CTAs take the KV heads of
// one (sequence, split), whose rows lie side by side in the cache
// ([B, cap, Hkv, D]): CTAs that start together read neighbouring pieces of
// the same cache rows, which keeps DRAM pages open across their requests
// (an e4m3 head row is only 128 bytes of a 1 KB cache row)
template <int kSub>
__device__ __forceinline__ DecItem dec_item(const DecodeArgs& a, int64_t item) {
  DecItem x;
  x.g = (int)(item % a.hkv);
  const int64_t rest = item / a.hkv;
  x.b = (int)(rest % a.batch);
  x.split = (int)(rest / a.batch);
  const int kv_len = a.c_snap[x.b] + 1;
  x.k0 = x.split * a.chunk;
  x.k1 = min(kv_len, x.k0 + a.chunk);
  x.nsub = x.k1 > x.k0 ? (x.k1 - x.k0 + 127) / 128 : 0;
  x.nt = (x.nsub + kSub - 1) / kSub;
  return x;
}

// The P operand is stored MN-major (128-byte swizzled rows = keys, the heads
// contiguous along a row, as the V tile stores dimensions): the thread of key
// k writes its 16 heads as whole 16-byte chunks (bf16: chunks 0 and 1 of the
// row, e4m3: chunk 0), swizzled by k & 7.  Heads past 16 (M up to 128) are
// never written; they only feed output rows that are not read.
__device__ __forceinline__ uint32_t p_chunk(uint32_t k, uint32_t c) { return k * 128u + ((c ^ (k & 7u)) << 4); }

// The scores of the first G heads of a 128-key sub-tile (thread = key).
template <int G>
__device__ __forceinline__ void ld_scores(uint32_t taddr, uint32_t (&v)[G]) {
  if constexpr (G == 4)
    ptx::tmem_ld4(taddr, v);
  else if constexpr (G == 8)
    ptx::tmem_ld8(taddr, v);
  else
    ptx::tmem_ld16(taddr, v);
}

// kG: the heads the softmax warps process (4, 8 or 16, at least the group);
// the score MMAs always compute 16 (N = 16), the columns past kG are not read.
template <bool kE4M3, int kG>
__global__ void __launch_bounds__(kThreads, 1)
    decode_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                     const __grid_constant__ CUtensorMap tmV, const DecodeArgs a, int64_t n_items) {
  using Cfg = DecCfg<kE4M3>;
  constexpr int kStages = Cfg::kStages, kSub = Cfg::kSub;
  constexpr uint32_t kTile = Cfg::kTile, kSubBytes = Cfg::kSubBytes, kQHalf = Cfg::kQHalf, kQBytes = Cfg::kQBytes;
  constexpr uint32_t OFF_RING = Cfg::OFF_RING, OFF_P = Cfg::OFF_P, OFF_Q = Cfg::OFF_Q, OFF_BAR = Cfg::OFF_BAR;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  Bars* bar = reinterpret_cast<Bars*>(smem + OFF_BAR);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      ptx::mbar_init(&bar->full[s], 1);
      ptx::mbar_init(&bar->empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      ptx::mbar_init(&bar->q_full[i], 1);
      ptx::mbar_init(&bar->q_empty[i], 1);
      ptx::mbar_init(&bar->p_ready[i], 128);
      ptx::mbar_init(&bar->p_free[i], 1);
    }
    for (int i = 0; i < 4; ++i) {
      ptx::mbar_init(&bar->s_tile[i], 1);
      ptx::mbar_init(&bar->s_seen[i], 128);
    }
    ptx::mbar_init(&bar->s_free, 128);
    ptx::mbar_init(&bar->o_full, 1);
    ptx::mbar_init(&bar->o_free, 32);
    ptx::mbar_init(&bar->final_mma, 1);
    ptx::mbar_init(&bar->red_m_full, 128);
    ptx::mbar_init(&bar->red_l_full, 128);
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
  // launched as a programmatic dependent of the cache write: the set-up above
  // overlaps it; the cache lengths and the new rows are read only after it
  // has completed.  The combine kernel after this one may start early and
  // waits for this grid in turn.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (warp == kLoadWarp) {
    // ------------------------------------------------ TMA loads (the warp waits converged, lane 0 issues)
    uint32_t nl = 0, nu = 0;  // ring tiles issued; non-empty items
    uint32_t nf[kStages] = {}, nq[2] = {0, 0};
    bool ok = true;
    const uint64_t pol = ptx::l2_policy_evict_first();  // the cache is streamed once per step
    if (lane == 0) {
      ptx::tma_prefetch_desc(&tmK);
      ptx::tma_prefetch_desc(&tmV);
    }
    for (int64_t item = blockIdx.x; ok && item < n_items; item += gridDim.x) {
      const DecItem x = dec_item<Cfg::kSub>(a, item);
      if (x.nt == 0) continue;
      const uint32_t qb = nu & 1;
      if (__any_sync(0xffffffffu, aborted(&bar->abort)) ||
          (nu >= 2 && !wait_warp(&bar->q_empty[qb], ((nu >> 1) - 1) & 1, a.status))) {
        ok = false;
        break;
      }
      if (lane == 0) {
        // the 16 query rows from the group's first head (rows past the group
        // are other heads' queries or zero fill; their outputs are not used)
        const int32_t qy = x.b * a.hq + x.g * a.group;
        uint8_t* dq = smem + OFF_Q + qb * kQBytes;
        ptx::mbar_expect_tx(&bar->q_full[qb], kQBytes);
        ptx::tma_load_2d(dq, &tmQ, &bar->q_full[qb], 0, qy);
        if (!kE4M3) ptx::tma_load_2d(dq + kQHalf, &tmQ, &bar->q_full[qb], 64, qy);
      }
      __syncwarp();
      ++nq[qb];
      ++nu;
      for (int pass = 0; ok && pass < 2; ++pass) {
        const CUtensorMap* map = pass ? &tmV : &tmK;
        for (int t = 0; t < x.nt; ++t, ++nl) {
          const uint32_t s = nl % kStages;
          if (__any_sync(0xffffffffu, aborted(&bar->abort)) ||
              (nl >= kStages && !wait_warp(&bar->empty[s], ((nl / kStages) - 1) & 1, a.status))) {
            ok = false;
            break;
          }
          if (lane == 0) {
            // a 128-key sub-tile starts at a multiple of 128 keys and lies in one page
            const int nh = min(kSub, x.nsub - t * kSub);
            uint8_t* dst = smem + OFF_RING + s * kTile;
            ptx::mbar_expect_tx(&bar->full[s], (uint32_t)nh * kSubBytes);
            for (int hh = 0; hh < nh; ++hh) {
              const int64_t p = (int64_t)x.k0 + (int64_t)(t * kSub + hh) * 128;
              const int32_t y =
                  a.pages.table ? (int32_t)paged_row(a.pages, x.b, p) : (int32_t)((int64_t)x.b * a.cap + p);
              ptx::tma_load_2d_hint(dst + hh * kSubBytes, map, &bar->full[s], x.g * kD, y, pol);
              if (!kE4M3) ptx::tma_load_2d_hint(dst + kHalfBytes, map, &bar->full[s], x.g * kD + 64, y, pol);
            }
          }
          __syncwarp();
          ++nf[s];
        }
      }
    }
    if (!ok) {
      if (lane == 0) set_abort(&bar->abort);
      // every issued copy lands before the CTA exits
      for (int s = 0; s < kStages; ++s)
        if (nf[s]) wait_warp(&bar->full[s], (nf[s] - 1) & 1, a.status);
      for (int i = 0; i < 2; ++i)
        if (nq[i]) wait_warp(&bar->q_full[i], (nq[i] - 1) & 1, a.status);
    }
    __syncwarp();
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------ MMA issue (the whole warp runs the loop,
    // one elected lane issues each instruction)
    constexpr uint32_t idesc_s =
        kE4M3 ? ptx::idesc_e4m3_f32(128, kHeadsPad, 0, 0) : ptx::idesc_bf16_f32(128, kHeadsPad, 0, 0);
    constexpr uint32_t idesc_pv = kE4M3 ? ptx::idesc_e4m3_f32(128, 128, 1, 1) : ptx::idesc_bf16_f32(128, 128, 1, 1);
    uint32_t nl = 0, nu = 0, T = 0, TS = 0;  // ring tiles consumed; non-empty items; P tiles; S tiles
    bool ok = true;
    for (int64_t item = blockIdx.x; ok && item < n_items; item += gridDim.x) {
      const DecItem x = dec_item<Cfg::kSub>(a, item);
      if (x.nt == 0) continue;
      const uint32_t qb = nu & 1;
      // Q landed; the softmax warps have read the previous item's S
      if (!wait_warp(&bar->q_full[qb], (nu >> 1) & 1, a.status) ||
          (nu >= 1 && !wait_warp(&bar->s_free, (nu - 1) & 1, a.status))) {
        ok = false;
        break;
      }
      ptx::tc_fence_after();
      const uint32_t sQ = ptx::smem_u32(smem + OFF_Q + qb * kQBytes);
      for (int t = 0; t < x.nt; ++t, ++nl) {
        const uint32_t s = nl % kStages;
        if (__shfl_sync(0xffffffffu, aborted(&bar->abort) ? 1 : 0, 0) ||
            !wait_warp(&bar->full[s], (nl / kStages) & 1, a.status)) {
          ok = false;
          break;
        }
        // the softmax warps have read S of the ring tile four back (its barrier is reused)
        if (TS >= 4 && !wait_warp(&bar->s_seen[TS & 3], ((TS >> 2) - 1) & 1, a.status)) {
          ok = false;
          break;
        }
        ptx::tc_fence_after();
        const uint32_t sK = ptx::smem_u32(smem + OFF_RING + s * kTile);
        if constexpr (kE4M3) {  // 128-byte rows: four k-steps of 32 bytes in one box, per 128-key sub-tile
          const int nh = min(kSub, x.nsub - t * kSub);
          for (int hh = 0; hh < nh; ++hh)
            ptx::mma4_e4m3_ss_warp<2, 2>(tmem + TM_S + kHeadsPad * (uint32_t)(t * kSub + hh),
                                         desc_kmajor(sK + hh * kSubBytes, 0), desc_kmajor(sQ, 0), idesc_s, 0u);
        } else {
          ptx::mma8_bf16_ss_warp<ptx::KMajorSw128, ptx::KMajorSw128Rows16>(
              tmem + TM_S + kHeadsPad * (uint32_t)t, desc_kmajor(sK, 0), desc_kmajor(sQ, 0), idesc_s, 0u);
        }
        ptx::mma_commit_warp(&bar->empty[s]);
        ptx::mma_commit_warp(&bar->s_tile[TS & 3]);
        ++TS;
      }
      if (!ok) break;
      ptx::mma_commit_warp(&bar->q_empty[qb]);
      // the epilogue has read the previous item's O
      if (nu >= 1 && !wait_warp(&bar->o_free, (nu - 1) & 1, a.status)) {
        ok = false;
        break;
      }
      ptx::tc_fence_after();
      for (int t = 0; t < x.nt; ++t, ++nl, ++T) {
        const uint32_t s = nl % kStages, pb = T & 1;
        if (__shfl_sync(0xffffffffu, aborted(&bar->abort) ? 1 : 0, 0) ||
            !wait_warp(&bar->p_ready[pb], (T >> 1) & 1, a.status) ||
            !wait_warp(&bar->full[s], (nl / kStages) & 1, a.status)) {
          ok = false;
          break;
        }
        ptx::tc_fence_after();
        const uint32_t sP = ptx::smem_u32(smem + OFF_P + pb * kTile);
        const uint32_t sV = ptx::smem_u32(smem + OFF_RING + s * kTile);
        if constexpr (kE4M3) {  // V MN-major: 32 keys of 128 bytes a k-step, per 128-key sub-tile
          const int nh = min(kSub, x.nsub - t * kSub);
          for (int hh = 0; hh < nh; ++hh)
            ptx::mma4_e4m3_ss_warp<256, 256>(tmem + TM_O, desc_kmajor(sP + hh * kSubBytes, 0),
                                           desc_kmajor(sV + hh * kSubBytes, 0), idesc_pv,
                                           (t > 0 || hh > 0) ? 1u : 0u);
        } else
          ptx::mma8_bf16_ss_warp<ptx::MnMajorSw128, ptx::MnMajorSw128>(tmem + TM_O, desc_mnmajor(sP, 0),
                                                                      desc_mnmajor(sV, 0), idesc_pv, t > 0 ? 1u : 0u);
        ptx::mma_commit_warp(&bar->empty[s]);
        ptx::mma_commit_warp(&bar->p_free[pb]);
      }
      if (!ok) break;
      ptx::mma_commit_warp(&bar->o_full);
      ++nu;
    }
    if (!ok && lane == 0) set_abort(&bar->abort);
    __syncwarp();
    ptx::mma_commit_warp(&bar->final_mma);
    wait_warp(&bar->final_mma, 0, a.status);
    __syncwarp();
  } else {
    // ------------------------------------------------ softmax and epilogue: thread r = key r of a tile
    const int r = threadIdx.x;
    const uint32_t lane_addr = (uint32_t)(warp * 32) << 16;
    const float c2 = a.scale * kLog2e * (kE4M3 ? a.qk_descale : 1.f);
    const float o_scale = kE4M3 ? a.v_descale : 1.f;
    const int group = a.group;
    uint32_t nu = 0, T = 0, TS = 0;
    bool ok = true;
    for (int64_t item = blockIdx.x; ok && item < n_items; item += gridDim.x) {
      const DecItem x = dec_item<Cfg::kSub>(a, item);
      const int64_t pbase = ((int64_t)x.b * a.hq + (int64_t)x.g * group) * a.splits + x.split;
      if (x.nt == 0) {
        // a split past the sequence's keys: a partial the combine skips
        if (warp == 0 && lane < group) {
          a.part_ml[(pbase + (int64_t)lane * a.splits) * 2] = -INFINITY;
          a.part_ml[(pbase + (int64_t)lane * a.splits) * 2 + 1] = 0.f;
        }
        continue;
      }
      // pass 1: maximum of the scaled scores per head over the item's keys,
      // ring tile by ring tile as the score MMAs complete
      static_assert(kG == 4 || kG == 8 || kG == kHeadsPad, "heads per softmax pass");
      float mx[kG];
#pragma unroll
      for (int h = 0; h < kG; ++h) mx[h] = -INFINITY;
      for (int t = 0; t < x.nt; ++t, ++TS) {
        if (!wait(&bar->s_tile[TS & 3], (TS >> 2) & 1, a.status)) {
          ok = false;
          break;
        }
        ptx::tc_fence_after();
        const int nh = min(kSub, x.nsub - t * kSub);
        for (int hh = 0; hh < nh; ++hh) {
          const int j = t * kSub + hh;
          uint32_t v[kG];
          ld_scores<kG>(tmem + lane_addr + TM_S + kHeadsPad * (uint32_t)j, v);
          ptx::tmem_ld_wait();
          ptx::reg_fence(v);
          if (x.k0 + j * 128 + r < x.k1) {
#pragma unroll
            for (int h = 0; h < kG; ++h) mx[h] = fmaxf(mx[h], __uint_as_float(v[h]));
          }
        }
        ptx::tc_fence_before();
        ptx::mbar_arrive(&bar->s_seen[TS & 3]);
      }
      if (!ok) break;
#pragma unroll
      for (int h = 0; h < kG; ++h) {
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) mx[h] = fmaxf(mx[h], __shfl_xor_sync(0xffffffffu, mx[h], o));
      }
      if (lane == 0) {
#pragma unroll
        for (int h = 0; h < kG; ++h) bar->red_m[nu & 1][warp][h] = mx[h];
      }
      ptx::mbar_arrive(&bar->red_m_full);
      if (!wait(&bar->red_m_full, nu & 1, a.status)) {
        ok = false;
        break;
      }
      float m2[kG];  // max of scale * log2(e) * S per head (finite: every item has a key)
#pragma unroll
      for (int h = 0; h < kG; ++h)
        m2[h] = fmaxf(fmaxf(bar->red_m[nu & 1][0][h], bar->red_m[nu & 1][1][h]),
                      fmaxf(bar->red_m[nu & 1][2][h], bar->red_m[nu & 1][3][h])) *
                c2;
      // pass 2: P as bf16 into the A operand of O += P V (rows = heads, columns = keys)
      float l[kG];
#pragma unroll
      for (int h = 0; h < kG; ++h) l[h] = 0.f;
      for (int t = 0; t < x.nt; ++t, ++T) {
        const uint32_t pb = T & 1;
        if (T >= 2 && !wait(&bar->p_free[pb], ((T >> 1) - 1) & 1, a.status)) {
          ok = false;
          break;
        }
        uint8_t* P = smem + OFF_P + pb * kTile;
        if constexpr (kE4M3) {
          const int nh = min(kSub, x.nsub - t * kSub);
          for (int hh = 0; hh < nh; ++hh) {
            const int j = t * kSub + hh;
            uint32_t v[kG];
            ld_scores<kG>(tmem + lane_addr + TM_S + kHeadsPad * (uint32_t)j, v);
            ptx::tmem_ld_wait();
            ptx::reg_fence(v);
            const bool valid = x.k0 + j * 128 + r < x.k1;
            uint32_t b4[4] = {0u, 0u, 0u, 0u};  // heads past kG: zero
#pragma unroll
            for (int h = 0; h < kG; h += 4) {
              float p4[4];
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                p4[e] = (valid && h + e < group) ? ex2(__uint_as_float(v[h + e]) * c2 - m2[h + e]) : 0.f;
                l[h + e] += p4[e];
              }
              b4[h >> 2] = pack_e4m3x4(p4[0], p4[1], p4[2], p4[3]);
            }
            *reinterpret_cast<uint4*>(P + hh * kSubBytes + p_chunk((uint32_t)r, 0u)) =
                make_uint4(b4[0], b4[1], b4[2], b4[3]);
          }
        } else {
          uint32_t v[kG];
          ld_scores<kG>(tmem + lane_addr + TM_S + kHeadsPad * (uint32_t)t, v);
          ptx::tmem_ld_wait();
          ptx::reg_fence(v);
          const bool valid = x.k0 + t * 128 + r < x.k1;
          uint32_t pk[kHeadsPad / 2] = {};  // heads past kG: zero
#pragma unroll
          for (int h = 0; h < kG; h += 2) {
            const float p0 = (valid && h < group) ? ex2(__uint_as_float(v[h]) * c2 - m2[h]) : 0.f;
            const float p1 = (valid && h + 1 < group) ? ex2(__uint_as_float(v[h + 1]) * c2 - m2[h + 1]) : 0.f;
            pk[h >> 1] = pack_bf16(p0, p1);
            l[h] += __uint_as_float(pk[h >> 1] << 16);  // the sum of the P that enters P V
            l[h + 1] += __uint_as_float(pk[h >> 1] & 0xFFFF0000u);
          }
          *reinterpret_cast<uint4*>(P + p_chunk((uint32_t)r, 0u)) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
          // heads 8-15 feed only output rows that are not read when kG is 8 or less
          if constexpr (kG > 8)
            *reinterpret_cast<uint4*>(P + p_chunk((uint32_t)r, 1u)) = make_uint4(pk[4], pk[5], pk[6], pk[7]);
        }
        ptx::fence_proxy_async_smem();
        ptx::mbar_arrive(&bar->p_ready[pb]);
      }
      if (!ok) break;
      ptx::tc_fence_before();
      ptx::mbar_arrive(&bar->s_free);
#pragma unroll
      for (int h = 0; h < kG; ++h) {
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) l[h] += __shfl_xor_sync(0xffffffffu, l[h], o);
      }
      if (lane == 0) {
#pragma unroll
        for (int h = 0; h < kG; ++h) bar->red_l[nu & 1][warp][h] = l[h];
      }
      ptx::mbar_arrive(&bar->red_l_full);
      if (!wait(&bar->red_l_full, nu & 1, a.status)) {
        ok = false;
        break;
      }
      if (warp == 0) {
        // epilogue: lane h holds row h of O = the unnormalised output of head h
        if (!wait(&bar->o_full, nu & 1, a.status)) {
          ok = false;
          break;
        }
        ptx::tc_fence_after();
        const bool mine = lane < group;
        float* dst = a.part_o + (pbase + (int64_t)(mine ? lane : 0) * a.splits) * kD;
#pragma unroll 1
        for (int q4 = 0; q4 < 4; ++q4) {
          uint32_t o[32];
          ptx::tmem_ld32(tmem + TM_O + 32u * q4, o);
          ptx::tmem_ld_wait();
          ptx::reg_fence(o);
          if (mine) {
#pragma unroll
            for (int i = 0; i < 8; ++i)
              reinterpret_cast<float4*>(dst + 32 * q4)[i] =
                  make_float4(__uint_as_float(o[4 * i]) * o_scale, __uint_as_float(o[4 * i + 1]) * o_scale,
                              __uint_as_float(o[4 * i + 2]) * o_scale, __uint_as_float(o[4 * i + 3]) * o_scale);
          }
        }
        if (mine) {
          float mh = -INFINITY, lh = 0.f;
#pragma unroll
          for (int w = 0; w < 4; ++w) {
            mh = fmaxf(mh, bar->red_m[nu & 1][w][lane]);
            lh += bar->red_l[nu & 1][w][lane];
          }
          a.part_ml[(pbase + (int64_t)lane * a.splits) * 2] = mh * c2;
          a.part_ml[(pbase + (int64_t)lane * a.splits) * 2 + 1] = lh;
        }
        ptx::tc_fence_before();
        ptx::mbar_arrive(&bar->o_free);
      }
      ++nu;
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

template <bool kE4M3, int kG>
cudaError_t launch_decode_tc_t(const DecodeArgs& a, cudaStream_t st) {
  using Cfg = DecCfg<kE4M3>;
  CUtensorMap tq, tk, tv;
  cudaError_t e;
  if constexpr (kE4M3) {
    if ((e = make_tmap_e4m3_box(&tq, a.q, (uint64_t)kD, (uint64_t)a.batch * a.hq, kHeadsPad)) != cudaSuccess) return e;
    if ((e = make_tmap_e4m3_box(&tk, a.k_cache, (uint64_t)a.hkv * kD, (uint64_t)a.kv_rows, 128)) != cudaSuccess) return e;
    if ((e = make_tmap_e4m3_box(&tv, a.v_cache, (uint64_t)a.hkv * kD, (uint64_t)a.kv_rows, 128)) != cudaSuccess) return e;
  } else {
    if ((e = make_tmap_bf16_box(&tq, a.q, (uint64_t)kD, (uint64_t)a.batch * a.hq, kHeadsPad)) != cudaSuccess) return e;
    if ((e = make_tmap_bf16(&tk, a.k_cache, (uint64_t)a.hkv * kD, (uint64_t)a.kv_rows)) != cudaSuccess) return e;
    if ((e = make_tmap_bf16(&tv, a.v_cache, (uint64_t)a.hkv * kD, (uint64_t)a.kv_rows)) != cudaSuccess) return e;
  }
  if ((e = cudaFuncSetAttribute(decode_tc_kernel<kE4M3, kG>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)Cfg::kSmemBytes)) != cudaSuccess)
    return e;
  const int64_t sms = sm_count();
  const int64_t n_items = (int64_t)a.batch * a.hkv * a.splits;
  int64_t grid = sms < n_items ? sms : n_items;
  if (grid <= 0) return cudaSuccess;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = Cfg::kSmemBytes;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, decode_tc_kernel<kE4M3, kG>, tq, tk, tv, a, n_items);
}

}  // namespace

cudaError_t launch_decode_tc(const DecodeArgs& a, cudaStream_t st) {
  if (a.d != kD || (a.dtype != ISM_BF16 && a.dtype != ISM_E4M3) || a.group > kHeadsPad || a.chunk % 128 != 0 ||
      a.chunk > kDecTcMaxKeys)
    return cudaErrorInvalidValue;
  // the softmax warps process the group's heads rounded up to 4, 8 or 16
  if (a.dtype == ISM_E4M3)
    return a.group <= 4 ? launch_decode_tc_t<true, 4>(a, st)
           : a.group <= 8 ? launch_decode_tc_t<true, 8>(a, st)
                          : launch_decode_tc_t<true, kHeadsPad>(a, st);
  return a.group <= 4 ? launch_decode_tc_t<false, 4>(a, st)
         : a.group <= 8 ? launch_decode_tc_t<false, 8>(a, st)
                        : launch_decode_tc_t<false, kHeadsPad>(a, st);
}

}  // namespace tc
}  // namespace ism
