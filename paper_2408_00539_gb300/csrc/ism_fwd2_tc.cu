// ISM attention forward, two (query head, query tile) units per CTA that
// read the same K/V (sm_103a tensor cores).
//
// When the query heads come in pairs that share a KV head (grouped-query
// attention with an even group size), one CTA computes the same 128-row
// query tile for both heads of a pair.  Otherwise (a.pair_order set) it
// computes two neighbouring query tiles of one head; the second tile sees at
// least the keys of the first, so it runs the same key blocks and possibly
// more.  Either way every K/V block is loaded once and used by both units.  The two heads' softmax warpgroups alternate with the tensor
// core (while one warpgroup turns S_A into P_A, the tensor core computes
// S_B, and so on).  P is written back into tensor memory over the S it came
// from and read there as the A operand of O += P V.
//
// Tensor memory (512 columns): S_A [0,128) O_A [128,256) S_B [256,384)
// O_B [384,512).  Shared memory: Q_A, Q_B, and a 2-stage K / V ring.
// Warps 0-3 softmax of head A, 4-7 of head B, 8 TMA producer, 9 MMA issuer.
// The mask and the lazy-rescale online softmax are those of the one-head
// kernel (Eq. e_ISM with the bound of Eq. fj; full tiles unmasked).
#include "ism_tc_common.cuh"

namespace ism {
namespace tc {
namespace {

constexpr int kThreads = 320;
constexpr uint32_t kTmemCols = 512;
// Shared memory: Q_A, Q_B, K ring (2), V ring (2), barriers.  A 128 x 128 tile
// is 32 KB in bf16 (two 64-column swizzled halves) and 16 KB in e4m3 (one).
template <bool kE4M3>
struct PairLayout {
  static constexpr uint32_t TB = kE4M3 ? 16384u : kTileBytes;
  static constexpr uint32_t QA = 0, QB = TB, K = 2 * TB, V = 4 * TB, BAR = 6 * TB;
  static constexpr uint32_t SMEM = BAR + 256 + 1024;
};

struct Bars {
  uint64_t q_full, q_empty;
  uint64_t k_full[2], k_empty[2], v_full[2], v_empty[2];
  uint64_t s_full[2], p_half[2], p_full[2], pv_done[2];  // per head of the pair
  uint64_t final_mma;
  uint32_t tmem_base;
  int32_t abort;
};

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}
__device__ __forceinline__ bool aborted(const int32_t* f) { return *reinterpret_cast<const volatile int32_t*>(f) != 0; }
__device__ __forceinline__ void set_abort(int32_t* f) { *reinterpret_cast<volatile int32_t*>(f) = 1; }

// One unit of work: two (query head, query tile) pairs that read the same
// K / V blocks, over key tiles [jb, jb + max(nkb0, nkb1)).
struct Unit {
  Tile w0, w1;
  int h0, h1, nkb0, nkb1;
  int jb, half;     // first key tile; half of a split item (-1: the whole item)
  int64_t split_k;  // index of a split item among the split ones
  __device__ int nkb() const { return nkb0 > nkb1 ? nkb0 : nkb1; }
};

template <bool kTilePairs, bool kSplit>
__device__ __forceinline__ Unit decode_unit(const AttnArgs& a, int64_t u) {
  Unit x;
  x.jb = 0;
  x.half = -1;
  x.split_k = 0;
  if constexpr (!kTilePairs) {
    const int npairs = a.hq >> 1;
    int64_t item = u;
    if (kSplit && item >= a.split_whole) {
      x.split_k = (item - a.split_whole) >> 1;
      x.half = (int)((item - a.split_whole) & 1);
      item = a.split_whole + x.split_k;
    }
    int64_t tpos;
    int hp;
    bucket_item(item, a.nq, npairs, tpos, hp, false);  // head pairs of a tile share K / V
    x.w0 = x.w1 = a.qtiles[a.q_order[tpos]];
    x.h0 = 2 * hp;
    x.h1 = x.h0 + 1;
    x.nkb0 = x.nkb1 = x.w0.a1;
    if (x.half >= 0) {  // key tiles [0, mid) or [mid, a1)
      const int mid = x.w0.a1 / 2;
      x.jb = x.half ? mid : 0;
      x.nkb0 = x.nkb1 = x.half ? x.w0.a1 - mid : mid;
    }
  } else {
    int64_t ppos;
    bucket_item(u, a.npairs, a.hq, ppos, x.h0, a.hq == a.hkv);  // one query head per KV head: bucketed
    x.h1 = x.h0;
    const int gq = a.pair_order[ppos];
    x.w0 = a.qtiles[gq];
    bool second = false;
    if (gq + 1 < a.nq) {
      x.w1 = a.qtiles[gq + 1];
      second = x.w1.q_base == x.w0.q_base && x.w1.tile == x.w0.tile + 1;
    }
    if (!second) x.w1 = x.w0;
    x.nkb0 = x.w0.a1;
    x.nkb1 = second ? x.w1.a1 : 0;
  }
  return x;
}

// The k-th unit of this CTA in a snake walk over the cost-ordered units
// (round r takes position b in even rounds, G - 1 - b in odd ones), so the
// CTAs' totals stay close; -1 past the end.
__device__ __forceinline__ int64_t unit_of(int64_t k, int64_t n_units) {
  const int64_t G = gridDim.x, b = blockIdx.x;
  const int64_t u = k * G + ((k & 1) ? G - 1 - b : b);
  return u < n_units ? u : -1;
}

// kE4M3: Q, K, V in e4m3 (kind::f8f6f4 MMAs, K = 32 a step); the scores are
// scaled by qk_descale, P is rounded to e4m3 for O += P V and O is scaled by
// v_descale (per-tensor dequantisation factors of the inputs).
// kSplit: the launch runs items past a.split_whole as two key-range halves
// (head pairs only); the instantiation without it is the plain kernel.
// Persistent: each CTA walks its units (unit_of) with one set of barriers
// whose phases run on across units.  The next unit's Q is loaded as soon as
// the last score MMA of the current unit has read Q, and its first score MMAs
// are issued right behind the current unit's last P V, so they overlap the
// output epilogue; the first P V of the next unit (which overwrites O) waits
// for the softmax warps' first P of that unit, which they write only after
// reading the previous O.
template <bool kTilePairs, bool kE4M3, bool kSplit = false>
__global__ void __launch_bounds__(kThreads, 1)
    fwd_pair_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                    const __grid_constant__ CUtensorMap tmV, const AttnArgs a, int64_t n_units) {
  using L = PairLayout<kE4M3>;
  constexpr uint32_t kTB = L::TB;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  Bars* bar = reinterpret_cast<Bars*>(smem + L::BAR);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    ptx::mbar_init(&bar->q_full, 1);
    ptx::mbar_init(&bar->q_empty, 1);
    for (int s = 0; s < 2; ++s) {
      ptx::mbar_init(&bar->k_full[s], 1);
      ptx::mbar_init(&bar->k_empty[s], 1);
      ptx::mbar_init(&bar->v_full[s], 1);
      ptx::mbar_init(&bar->v_empty[s], 1);
      ptx::mbar_init(&bar->s_full[s], 1);
      ptx::mbar_init(&bar->p_half[s], 128);
      ptx::mbar_init(&bar->p_full[s], 128);
      ptx::mbar_init(&bar->pv_done[s], 1);
    }
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
    // ------------------------------------------------------------ producer (the warp waits
    // converged, lane 0 issues the copies)
    // one 128 x 128 tile: two 64-column boxes in bf16, one 128-column box in e4m3
    auto load_tile = [&](uint8_t* dst, const CUtensorMap* map, uint64_t* b, int32_t x, int32_t y) {
      ptx::tma_load_2d(dst, map, b, x, y);
      if (!kE4M3) ptx::tma_load_2d(dst + kHalfBytes, map, b, x + 64, y);
    };
    if (lane == 0) {
      ptx::tma_prefetch_desc(&tmQ);
      ptx::tma_prefetch_desc(&tmK);
      ptx::tma_prefetch_desc(&tmV);
    }
    uint32_t nq = 0, it = 0;           // Q loads and K / V blocks so far (all units)
    uint32_t nk[2] = {0, 0}, nv[2] = {0, 0};
    bool ok = true;
    for (int64_t k = 0; ok; ++k) {
      const int64_t u = unit_of(k, n_units);
      if (u < 0) break;
      const Unit x = decode_unit<kTilePairs, kSplit>(a, u);
      const int nkb = x.nkb();
      if (nkb == 0) continue;
      const int g = x.h0 / (a.hq / a.hkv);
      const int k_first = x.jb * kRows;
      // the previous unit's score MMAs have read its Q
      if (nq > 0 && !wait_warp(&bar->q_empty, (nq - 1) & 1, a.status)) {
        if (lane == 0) set_abort(&bar->abort);
        ok = false;
        break;
      }
      if (lane == 0) {
        const int32_t qy0 = x.w0.q_base + x.w0.tile * kRows, qy1 = x.w1.q_base + x.w1.tile * kRows;
        ptx::mbar_expect_tx(&bar->q_full, (x.nkb1 > 0 ? 2 : 1) * kTB);
        load_tile(smem + L::QA, &tmQ, &bar->q_full, x.h0 * kD, qy0);
        if (x.nkb1 > 0) load_tile(smem + L::QB, &tmQ, &bar->q_full, x.h1 * kD, qy1);
      }
      __syncwarp();
      ++nq;
      for (int j = 0; j < nkb; ++j, ++it) {
        const int s = it & 1;
        const uint32_t n = it >> 1;
        if (__any_sync(0xffffffffu, aborted(&bar->abort))) { ok = false; break; }
        const int32_t ky = a.pages.table
                               ? (int32_t)paged_row(a.pages, x.w0.k_base, (int64_t)k_first + j * kRows)
                               : x.w0.k_base + k_first + j * kRows;
        if (it >= 2 && !wait_warp(&bar->k_empty[s], (n - 1) & 1, a.status)) {
          if (lane == 0) set_abort(&bar->abort);
          ok = false;
          break;
        }
        if (lane == 0) {
          ptx::mbar_expect_tx(&bar->k_full[s], kTB);
          load_tile(smem + L::K + s * kTB, &tmK, &bar->k_full[s], g * kD, ky);
        }
        __syncwarp();
        ++nk[s];
        if (it >= 2 && !wait_warp(&bar->v_empty[s], (n - 1) & 1, a.status)) {
          if (lane == 0) set_abort(&bar->abort);
          ok = false;
          break;
        }
        if (lane == 0) {
          ptx::mbar_expect_tx(&bar->v_full[s], kTB);
          load_tile(smem + L::V + s * kTB, &tmV, &bar->v_full[s], g * kD, ky);
        }
        __syncwarp();
        ++nv[s];
      }
    }
    if (!ok || __any_sync(0xffffffffu, aborted(&bar->abort))) {
      // let the copies in flight land before the CTA exits
      if (nq) wait_warp(&bar->q_full, (nq - 1) & 1, a.status);
      for (int s = 0; s < 2; ++s) {
        if (nk[s]) wait_warp(&bar->k_full[s], (nk[s] - 1) & 1, a.status);
        if (nv[s]) wait_warp(&bar->v_full[s], (nv[s] - 1) & 1, a.status);
      }
    }
  } else if (warp == 9) {
    // ------------------------------------------------------------ MMA issuer (the whole
    // warp runs the loop, one elected lane issues each instruction)
    constexpr uint32_t idesc_qk = kE4M3 ? ptx::idesc_e4m3_f32(128, 128, 0, 0) : ptx::idesc_bf16_f32(128, 128, 0, 0);
    constexpr uint32_t idesc_pv = kE4M3 ? ptx::idesc_e4m3_f32(128, 128, 0, 1) : ptx::idesc_bf16_f32(128, 128, 0, 1);
    const uint32_t sQ0 = ptx::smem_u32(smem + L::QA);
    uint32_t nq = 0, it = 0;       // units with key blocks, K / V blocks (all units)
    uint32_t nb[2] = {0, 0};       // blocks of unit x so far (P hand-offs)
    // head x: Q at sQ0 + x * kTB, S at tmem + 256 x, O at tmem + 128 + 256 x
    auto issue_s = [&](int x, uint32_t blk) {
      const uint32_t sK = ptx::smem_u32(smem + L::K + (blk & 1) * kTB);
      const uint32_t sQ = sQ0 + (uint32_t)x * kTB, tS = tmem + 256u * (uint32_t)x;
      if constexpr (kE4M3)  // 128-byte rows: k-steps of 32 bytes
        ptx::mma4_e4m3_ss_warp<2, 2>(tS, desc_kmajor(sQ, 0), desc_kmajor(sK, 0), idesc_qk, 0u);
      else
        ptx::mma8_bf16_ss_warp<ptx::KMajorSw128, ptx::KMajorSw128>(tS, desc_kmajor(sQ, 0), desc_kmajor(sK, 0),
                                                                  idesc_qk, 0u);
      ptx::mma_commit_warp(&bar->s_full[x]);
    };
    // P V in two halves of 64 keys for bf16: the first as soon as the softmax
    // warps have written P of keys [0, 64) (p_half), the second after p_full
    auto issue_pv = [&](int x, uint32_t blk, bool first) -> bool {
      const uint32_t sV = ptx::smem_u32(smem + L::V + (blk & 1) * kTB);
      const uint32_t tS = tmem + 256u * (uint32_t)x, tO = tS + 128u;
      if (!wait_warp(&bar->p_half[x], nb[x] & 1, a.status)) return false;
      ptx::tc_fence_after();
      if constexpr (!kE4M3) ptx::mma4_bf16_ts_warp<8, 128>(tO, tS, desc_mnmajor(sV, 0), idesc_pv, first ? 0u : 1u);
      if (!wait_warp(&bar->p_full[x], nb[x] & 1, a.status)) return false;
      ptx::tc_fence_after();
      if constexpr (kE4M3)  // P: four e4m3 a column; V MN-major, 32 rows of 128 bytes a k-step
        ptx::mma4_e4m3_ts_warp<8, 256>(tO, tS, desc_kmajor(sV, 0), idesc_pv, first ? 0u : 1u);
      else  // keys [64, 128): P columns 32 + 8 kk, V rows 64 + 16 kk
        ptx::mma4_bf16_ts_warp<8, 128>(tO, tS + 32, desc_mnmajor(sV, 4), idesc_pv, 1u);
      ptx::mma_commit_warp(&bar->pv_done[x]);
      ++nb[x];
      return true;
    };
    bool ok = true;
    for (int64_t k = 0; ok; ++k) {
      const int64_t u = unit_of(k, n_units);
      if (u < 0) break;
      const Unit x = decode_unit<kTilePairs, kSplit>(a, u);
      const int nkb = x.nkb();
      if (nkb == 0) continue;
      // unit y runs key blocks [0, nkb_y); the last unit reading block j
      // releases its K / V stages (unit 1 whenever it has the block: nkb1 is
      // either equal to nkb0, at least nkb0, or 0)
      auto last_user = [&](int j) { return j < x.nkb1 ? 1 : 0; };
      if (__shfl_sync(0xffffffffu, aborted(&bar->abort) ? 1 : 0, 0) ||
          !wait_warp(&bar->q_full, nq & 1, a.status) || !wait_warp(&bar->k_full[it & 1], (it >> 1) & 1, a.status)) {
        ok = false;
        break;
      }
      ++nq;
      // S of block 0 overwrites the previous unit's last P: issued after that
      // unit's last P V (in issue order; the drained variant waits for it)
      if (a.flags & kFlagDrainTmemReuse)
        for (int y = 0; ok && y < 2; ++y)
          if (nb[y] > 0 && !wait_warp(&bar->pv_done[y], (nb[y] - 1) & 1, a.status)) ok = false;
      if (!ok) break;
      ptx::tc_fence_after();
      if (x.nkb0 > 0) issue_s(0, it);
      if (x.nkb1 > 0) issue_s(1, it);
      ptx::mma_commit_warp(&bar->k_empty[it & 1]);
      if (nkb == 1) ptx::mma_commit_warp(&bar->q_empty);  // every score MMA of the unit is issued
      // Per block: PV_A(j), S_A(j+1), PV_B(j), S_B(j+1).  S_x(j+1) overwrites
      // the P_x(j) that PV_x(j) reads; MMAs issued by this thread execute in
      // order, so S_x(j+1) follows PV_x(j) without a wait (kFlagDrainTmemReuse
      // makes it wait for PV_x(j) to complete instead).
      for (int j = 0; ok && j < nkb; ++j) {
        const uint32_t blk = it + (uint32_t)j;
        const int s = blk & 1, s1 = (blk + 1) & 1;
        const bool more = j + 1 < nkb;
        if (__shfl_sync(0xffffffffu, aborted(&bar->abort) ? 1 : 0, 0)) { ok = false; break; }
        if (!wait_warp(&bar->v_full[s], (blk >> 1) & 1, a.status)) { ok = false; break; }
        if (more && !wait_warp(&bar->k_full[s1], ((blk + 1) >> 1) & 1, a.status)) { ok = false; break; }
        for (int y = 0; y < 2; ++y) {
          const int nkby = y ? x.nkb1 : x.nkb0;
          if (j >= nkby) continue;
          if (!issue_pv(y, blk, j == 0)) { ok = false; break; }
          if (y == last_user(j)) ptx::mma_commit_warp(&bar->v_empty[s]);
          if (j + 1 < nkby) {
            if ((a.flags & kFlagDrainTmemReuse) && !wait_warp(&bar->pv_done[y], (nb[y] - 1) & 1, a.status)) {
              ok = false;
              break;
            }
            ptx::tc_fence_after();
            issue_s(y, blk + 1);
            if (y == last_user(j + 1)) {
              ptx::mma_commit_warp(&bar->k_empty[s1]);
              if (j + 2 == nkb) ptx::mma_commit_warp(&bar->q_empty);  // the unit's last score MMA
            }
          }
        }
      }
      it += (uint32_t)nkb;
    }
    if (!ok && lane == 0) set_abort(&bar->abort);
    __syncwarp();
    ptx::mma_commit_warp(&bar->final_mma);
    wait_warp(&bar->final_mma, 0, a.status);
    __syncwarp();
  } else {
    // ------------------------------------------------------------ softmax of head x
    const int xh = warp >> 2;
    const int r = threadIdx.x & 127;
    const uint32_t lane_addr = (uint32_t)((warp & 3) * 32) << 16;
    const uint32_t tS = tmem + lane_addr + (xh ? 256u : 0u), tO = tmem + lane_addr + (xh ? 384u : 128u);
    const float sl2 = a.scale * kLog2e * (kE4M3 ? a.qk_descale : 1.f);
    uint32_t nb = 0;  // blocks of this head so far (all units)
    bool ok = true;
    for (int64_t k = 0; ok; ++k) {
      const int64_t u = unit_of(k, n_units);
      if (u < 0) break;
      const Unit x = decode_unit<kTilePairs, kSplit>(a, u);
      const int h = xh ? x.h1 : x.h0;
      const Tile wm = xh ? x.w1 : x.w0;
      const int nkbm = xh ? x.nkb1 : x.nkb0, kfull = wm.a0 - x.jb;  // key tiles counted from the unit's first
      const int k_first = x.jb * kRows;
      const int row = wm.tile * kRows + r;
      const bool valid = row < wm.q_len;
      const int ke = a.kv_end[wm.kv_base + (valid ? row : wm.q_len - 1)] - k_first;
      float m_use = -INFINITY, l = 0.f;
      for (int j = 0; ok && j < nkbm; ++j) {
        const uint32_t blk = nb + (uint32_t)j;
        if (!wait(&bar->s_full[xh], blk & 1, a.status)) { ok = false; break; }
        ptx::tc_fence_after();
        float xs[128];
        {
          uint32_t t[4][32];
#pragma unroll
          for (int c = 0; c < 4; ++c) ptx::tmem_ld32(tS + c * 32, t[c]);
          ptx::tmem_ld_wait();
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            ptx::reg_fence(t[c]);
#pragma unroll
            for (int i = 0; i < 32; ++i) xs[c * 32 + i] = __uint_as_float(t[c][i]);
          }
        }
        // row max on the raw scores (the scale is positive), masked keys at -inf;
        // eight independent partial maxima keep the dependency chain short
        float mr[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) mr[q] = -INFINITY;
        if (j >= kfull) {
          const int lim = ke - j * kRows;
#pragma unroll
          for (int c = 0; c < 128; ++c) {
            xs[c] = c < lim ? xs[c] : -INFINITY;
            mr[c & 7] = fmaxf(mr[c & 7], xs[c]);
          }
        } else {
#pragma unroll
          for (int c = 0; c < 128; ++c) mr[c & 7] = fmaxf(mr[c & 7], xs[c]);
        }
        const float mraw = fmaxf(fmaxf(fmaxf(mr[0], mr[1]), fmaxf(mr[2], mr[3])),
                                 fmaxf(fmaxf(mr[4], mr[5]), fmaxf(mr[6], mr[7])));
        const float m_new = fmaxf(m_use, mraw * sl2);
        if (j == 0) {
          m_use = m_new;
        } else if (m_new > m_use + 8.f) {
          // bring O (complete through PV(j-1)) and l to the new max
          if (!wait(&bar->pv_done[xh], (blk - 1) & 1, a.status)) { ok = false; break; }
          ptx::tc_fence_after();
          const float f = ex2(m_use - m_new);
          l *= f;
#pragma unroll 1
          for (int c = 0; c < 4; ++c) {
            uint32_t o[32];
            ptx::tmem_ld32(tO + c * 32, o);
            ptx::tmem_ld_wait();
            ptx::reg_fence(o);
#pragma unroll
            for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * f);
            ptx::tmem_st32(tO + c * 32, o);
          }
          m_use = m_new;
        }
        // P over the first 64 columns of S (already read), 32 columns at a time
        float2 rsv[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
        const float2 sl2x2 = make_float2(sl2, sl2), negm = make_float2(-m_use, -m_use);
        if constexpr (kE4M3) {
          // P as e4m3 over the first 32 columns of S: column c holds keys 4c .. 4c + 3
          uint32_t pk[32];
#pragma unroll
          for (int c = 0; c < 32; ++c) {
            const float2 a01 = fma2(make_float2(xs[4 * c], xs[4 * c + 1]), sl2x2, negm);
            const float2 a23 = fma2(make_float2(xs[4 * c + 2], xs[4 * c + 3]), sl2x2, negm);
            const float2 p01 = make_float2(ex2(a01.x), ex2(a01.y)), p23 = make_float2(ex2(a23.x), ex2(a23.y));
            rsv[0] = add2(rsv[0], p01);
            rsv[1] = add2(rsv[1], p23);
            pk[c] = pack_e4m3x4(p01.x, p01.y, p23.x, p23.y);
          }
          ptx::tmem_st32(tS, pk);
          ptx::tmem_st_wait();
          ptx::tc_fence_before();
          ptx::mbar_arrive(&bar->p_half[xh]);
        } else {
#pragma unroll
          for (int hf = 0; hf < 2; ++hf) {
            uint32_t pk[32];
#pragma unroll
            for (int c = 0; c < 32; ++c) {
              const float2 arg = fma2(make_float2(xs[64 * hf + 2 * c], xs[64 * hf + 2 * c + 1]), sl2x2, negm);
              const float2 pr = make_float2(ex2(arg.x), ex2(arg.y));
              rsv[c & 1] = add2(rsv[c & 1], pr);
              pk[c] = pack_bf16(pr.x, pr.y);
            }
            ptx::tmem_st32(tS + 32 * hf, pk);
            if (hf == 0) {  // keys [0, 64): the first half of P V may start
              ptx::tmem_st_wait();
              ptx::tc_fence_before();
              ptx::mbar_arrive(&bar->p_half[xh]);
            }
          }
        }
        l += (rsv[0].x + rsv[0].y) + (rsv[1].x + rsv[1].y);
        ptx::tmem_st_wait();
        ptx::tc_fence_before();
        ptx::mbar_arrive(&bar->p_full[xh]);
      }
      if (!ok) break;
      if (nkbm > 0) {
        nb += (uint32_t)nkbm;
        // one decision for the whole warp: the epilogue's loads and shuffles are warp-wide
        if (!__all_sync(0xffffffffu, wait(&bar->pv_done[xh], (nb - 1) & 1, a.status))) { ok = false; break; }
        ptx::tc_fence_after();
      }
      if (kSplit && x.half >= 0) {
        // half of a split item: unnormalised O and (max, sum) for the merge; a
        // half without key tiles leaves max -inf (weight 0, its O is not read)
        const int64_t pu = ((x.split_k * 2 + x.half) * 2 + xh) * kRows + r;
        a.part_ml[pu * 2] = nkbm > 0 ? m_use : -INFINITY;
        a.part_ml[pu * 2 + 1] = nkbm > 0 ? l : 0.f;
        if (nkbm > 0) {
          const float f = kE4M3 ? a.v_descale : 1.f;
          float4* dst = reinterpret_cast<float4*>(a.part_o + pu * kD);
#pragma unroll 1
          for (int c = 0; c < 4; ++c) {
            uint32_t o[32];
            ptx::tmem_ld32(tO + c * 32, o);
            ptx::tmem_ld_wait();
            ptx::reg_fence(o);
#pragma unroll
            for (int i = 0; i < 8; ++i)
              dst[c * 8 + i] = make_float4(__uint_as_float(o[4 * i]) * f, __uint_as_float(o[4 * i + 1]) * f,
                                           __uint_as_float(o[4 * i + 2]) * f, __uint_as_float(o[4 * i + 3]) * f);
          }
        }
      } else if (nkbm > 0) {
        const float inv = (kE4M3 ? a.v_descale : 1.f) / l;
        const int64_t orow = (int64_t)wm.q_base + row;
        // rows are stored by groups of four lanes (store_slice32)
        const int li = r & 3;
        const int64_t rstride = (int64_t)a.hq * kD;
        __nv_bfloat16* const g0 = reinterpret_cast<__nv_bfloat16*>(a.out) + (orow - li) * rstride + h * kD;
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          uint32_t o[32], w[16];
          ptx::tmem_ld32(tO + c * 32, o);
          ptx::tmem_ld_wait();
          ptx::reg_fence(o);
          pack_scaled32(o, inv, w);
          store_slice32(w, g0 + 32 * c, rstride, wm.q_len - (row - li));
        }
        if (valid && a.lse) a.lse[(int64_t)h * a.q_rows + orow] = (m_use + log2f(l)) * kLn2;
      }
    }
    if (!ok) set_abort(&bar->abort);
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 9) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, kTmemCols);
  }
}

// Merge of the two halves of each split item: block (split item k, head x,
// row r) of 128 threads (dimensions).  m in the base-2 scaled units of the
// forward, so O = (w0 O0 + w1 O1) / (w0 l0 + w1 l1) with w = 2^(m - M), and
// LSE = (M + log2 L) ln 2, as the whole-item epilogue writes them.
__global__ void __launch_bounds__(128) fwd_split_merge_kernel(const AttnArgs a) {
  const int64_t b = blockIdx.x;
  const int r = (int)(b % kRows), x = (int)((b / kRows) & 1);
  const int64_t k = b / (2 * kRows);
  const int npairs = a.hq >> 1;
  const int64_t item = a.split_whole + k;
  int64_t tpos;
  int hp;
  bucket_item(item, a.nq, npairs, tpos, hp, false);  // as fwd_pair_kernel decodes its items
  const Tile w = a.qtiles[a.q_order[tpos]];
  const int h = 2 * hp + x;
  const int row = w.tile * kRows + r;
  if (row >= w.q_len) return;
  const int d = threadIdx.x;
  const int64_t p0 = ((k * 2 + 0) * 2 + x) * kRows + r, p1 = ((k * 2 + 1) * 2 + x) * kRows + r;
  const float m0 = a.part_ml[p0 * 2], l0 = a.part_ml[p0 * 2 + 1];
  const float m1 = a.part_ml[p1 * 2], l1 = a.part_ml[p1 * 2 + 1];
  const float M = fmaxf(m0, m1);
  const float f0 = m0 == -INFINITY ? 0.f : exp2f(m0 - M), f1 = m1 == -INFINITY ? 0.f : exp2f(m1 - M);
  const float o0 = f0 != 0.f ? a.part_o[p0 * kD + d] : 0.f, o1 = f1 != 0.f ? a.part_o[p1 * kD + d] : 0.f;
  const float L = (f0 != 0.f ? f0 * l0 : 0.f) + (f1 != 0.f ? f1 * l1 : 0.f);
  const int64_t orow = (int64_t)w.q_base + row;
  reinterpret_cast<__nv_bfloat16*>(a.out)[(orow * a.hq + h) * kD + d] = __float2bfloat16_rn((f0 * o0 + f1 * o1) / L);
  if (d == 0 && a.lse) a.lse[(int64_t)h * a.q_rows + orow] = (M + log2f(L)) * kLn2;
}

template <bool kE4M3>
cudaError_t launch_fwd_pair_t(const AttnArgs& a, const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                              cudaStream_t st) {
  cudaError_t e;
  const bool tile_pairs = a.pair_order != nullptr;
  const bool split_launch = !tile_pairs && a.split_items > 0;
  auto kern = tile_pairs ? fwd_pair_kernel<true, kE4M3>
                         : (split_launch ? fwd_pair_kernel<false, kE4M3, true> : fwd_pair_kernel<false, kE4M3>);
  constexpr uint32_t smem = PairLayout<kE4M3>::SMEM;
  if ((e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) != cudaSuccess)
    return e;
  const int64_t items = tile_pairs ? a.npairs * a.hq : a.nq * (a.hq / 2);
  if (items == 0) return cudaSuccess;
  const bool split = !tile_pairs && a.split_items > 0;
  if (split && (a.split_whole + a.split_items != items || !a.part_o || !a.part_ml)) return cudaErrorInvalidValue;
  const int64_t n_units = split ? a.split_whole + 2 * a.split_items : items;
  // persistent: one CTA per SM walks its share of the units
  const int64_t grid = n_units < sm_count() ? n_units : sm_count();
  kern<<<(unsigned)grid, kThreads, smem, st>>>(tq, tk, tv, a, n_units);
  if ((e = cudaGetLastError()) != cudaSuccess || !split) return e;
  fwd_split_merge_kernel<<<(unsigned)(a.split_items * 2 * kRows), 128, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_fwd_pair(const AttnArgs& a, const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                            cudaStream_t st) {
  return a.dtype == ISM_E4M3 ? launch_fwd_pair_t<true>(a, tq, tk, tv, st) : launch_fwd_pair_t<false>(a, tq, tk, tv, st);
}

}  // namespace tc
}  // namespace ism
