// Fused ISM attention forward on sm_103a tensor cores (Eq. e_ISM with the
// bound f(j) of Eq. fj, softmax form of Section 2.3).
//
// One CTA computes a 128-row query tile of one head over the tile's
// non-empty key blocks [0, kt_end): the leading kt_full_end blocks run
// without a mask, the rest apply key < kv_end[row].  Warp roles:
//   warp 4      TMA producer: Q once, then K/V blocks into a 2-stage ring
//   warp 5      TMEM owner and MMA issuer: S = Q K^T into one of two TMEM
//               S buffers, O += P V into the TMEM O accumulator
//   warps 0..3  softmax: thread r owns query row r (TMEM lane r); online
//               softmax in base 2 with a lazily updated running max (the
//               accumulator is rescaled only when the max grows by more
//               than 2^8), P written to shared memory in the MMA's
//               swizzled K-major layout; epilogue O / l and LSE.
// The MMA warp issues S_{j+1} before PV_j so the tensor core works on the
// next block while the softmax warps process the current one.
#include <cstdlib>
#include <mutex>

#include "ism_tc_common.cuh"

namespace ism {
namespace tc {

namespace {

constexpr int kStages = 2;
constexpr uint32_t OFF_Q = 0;
constexpr uint32_t OFF_K = kTileBytes;
constexpr uint32_t OFF_V = OFF_K + kStages * kTileBytes;
constexpr uint32_t OFF_P = OFF_V + kStages * kTileBytes;
constexpr uint32_t OFF_BAR = OFF_P + 2 * kTileBytes;
constexpr uint32_t kSmemBytes = OFF_BAR + 256 + 1024;  // barriers + alignment slack
constexpr int kThreads = 192;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t TM_S = 0, TM_O = 256;  // S buffers at columns 0 and 128, O at 256

struct Bars {
  uint64_t q_full;
  uint64_t k_full[kStages], k_empty[kStages];
  uint64_t v_full[kStages], v_empty[kStages];
  uint64_t s_full[2], s_free[2];
  uint64_t p_full[2], p_free[2];
  uint64_t final_mma;
  uint32_t tmem_base;
  int32_t abort;
};
static_assert(sizeof(Bars) <= 256, "barrier block");

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

__device__ __forceinline__ bool aborted(Bars* b) { return *reinterpret_cast<volatile int32_t*>(&b->abort) != 0; }
__device__ __forceinline__ void set_abort(Bars* b) { *reinterpret_cast<volatile int32_t*>(&b->abort) = 1; }

__global__ void __launch_bounds__(kThreads, 1)
    fwd_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
               const __grid_constant__ CUtensorMap tmV, const AttnArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  Bars* bar = reinterpret_cast<Bars*>(smem + OFF_BAR);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.x % a.hq;
  const Tile w = a.qtiles[a.q_order[blockIdx.x / a.hq]];
  const int g = h / (a.hq / a.hkv);
  const int nkb = w.a1, kfull = w.a0;
  const uint32_t sQ = ptx::smem_u32(smem + OFF_Q);

  if (threadIdx.x == 0) {
    ptx::mbar_init(&bar->q_full, 1);
    for (int s = 0; s < kStages; ++s) {
      ptx::mbar_init(&bar->k_full[s], 1);
      ptx::mbar_init(&bar->k_empty[s], 1);
      ptx::mbar_init(&bar->v_full[s], 1);
      ptx::mbar_init(&bar->v_empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      ptx::mbar_init(&bar->s_full[s], 1);
      ptx::mbar_init(&bar->s_free[s], 128);
      ptx::mbar_init(&bar->p_full[s], 128);
      ptx::mbar_init(&bar->p_free[s], 1);
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
    // ------------------------------------------------------------ producer (the warp waits
    // converged, lane 0 issues the copies)
    if (nkb > 0) {
      if (lane == 0) {
        ptx::tma_prefetch_desc(&tmQ);
        ptx::tma_prefetch_desc(&tmK);
        ptx::tma_prefetch_desc(&tmV);
        const int32_t qy = w.q_base + w.tile * kRows;
        ptx::mbar_expect_tx(&bar->q_full, kTileBytes);
        ptx::tma_load_2d(smem + OFF_Q, &tmQ, &bar->q_full, h * kD, qy);
        ptx::tma_load_2d(smem + OFF_Q + kHalfBytes, &tmQ, &bar->q_full, h * kD + 64, qy);
      }
      __syncwarp();
      uint32_t nk[kStages] = {0, 0}, nv[kStages] = {0, 0};  // loads issued per stage barrier
      for (int j = 0; j < nkb; ++j) {
        const int s = j & 1;
        const uint32_t n = (uint32_t)(j >> 1);
        if (__any_sync(0xffffffffu, aborted(bar))) break;
        const int32_t ky = a.pages.table ? (int32_t)paged_row(a.pages, w.k_base, (int64_t)j * kRows)
                                         : w.k_base + j * kRows;
        if (j >= kStages && !wait_warp(&bar->k_empty[s], (n - 1) & 1, a.status)) {
          if (lane == 0) set_abort(bar);
          break;
        }
        if (lane == 0) {
          ptx::mbar_expect_tx(&bar->k_full[s], kTileBytes);
          ptx::tma_load_2d(smem + OFF_K + s * kTileBytes, &tmK, &bar->k_full[s], g * kD, ky);
          ptx::tma_load_2d(smem + OFF_K + s * kTileBytes + kHalfBytes, &tmK, &bar->k_full[s], g * kD + 64, ky);
        }
        __syncwarp();
        ++nk[s];
        if (j >= kStages && !wait_warp(&bar->v_empty[s], (n - 1) & 1, a.status)) {
          if (lane == 0) set_abort(bar);
          break;
        }
        if (lane == 0) {
          ptx::mbar_expect_tx(&bar->v_full[s], kTileBytes);
          ptx::tma_load_2d(smem + OFF_V + s * kTileBytes, &tmV, &bar->v_full[s], g * kD, ky);
          ptx::tma_load_2d(smem + OFF_V + s * kTileBytes + kHalfBytes, &tmV, &bar->v_full[s], g * kD + 64, ky);
        }
        __syncwarp();
        ++nv[s];
      }
      if (__any_sync(0xffffffffu, aborted(bar))) {
        // wait (bounded) for this warp's own copies still in flight
        wait_warp(&bar->q_full, 0, a.status);
        for (int s = 0; s < kStages; ++s) {
          if (nk[s]) wait_warp(&bar->k_full[s], (nk[s] - 1) & 1, a.status);
          if (nv[s]) wait_warp(&bar->v_full[s], (nv[s] - 1) & 1, a.status);
        }
      }
    }
  } else if (warp == 5) {
    // ------------------------------------------------------------ MMA issuer (the whole
    // warp runs the loop, one elected lane issues each instruction)
    if (nkb > 0) {
      constexpr uint32_t idesc_qk = ptx::idesc_bf16_f32(128, 128, 0, 0);
      constexpr uint32_t idesc_pv = ptx::idesc_bf16_f32(128, 128, 0, 1);
      bool ok = wait_warp(&bar->q_full, 0, a.status);
      auto issue_pv = [&](int i) -> bool {
        const int s = i & 1;
        const uint32_t n = (uint32_t)(i >> 1);
        if (!wait_warp(&bar->p_full[s], n & 1, a.status)) return false;
        if (!wait_warp(&bar->v_full[s], n & 1, a.status)) return false;
        ptx::tc_fence_after();
        const uint32_t sP = ptx::smem_u32(smem + OFF_P + s * kTileBytes);
        const uint32_t sV = ptx::smem_u32(smem + OFF_V + s * kTileBytes);
        ptx::mma8_bf16_ss_warp<ptx::KMajorSw128, ptx::MnMajorSw128>(tmem + TM_O, desc_kmajor(sP, 0), desc_mnmajor(sV, 0),
                                                                   idesc_pv, i > 0 ? 1u : 0u);
        ptx::mma_commit_warp(&bar->p_free[s]);
        ptx::mma_commit_warp(&bar->v_empty[s]);
        return true;
      };
      for (int j = 0; ok && j < nkb; ++j) {
        const int s = j & 1;
        const uint32_t n = (uint32_t)(j >> 1);
        if (__shfl_sync(0xffffffffu, aborted(bar) ? 1 : 0, 0)) { ok = false; break; }
        if (!wait_warp(&bar->k_full[s], n & 1, a.status)) { ok = false; break; }
        if (j >= 2 && !wait_warp(&bar->s_free[s], (n - 1) & 1, a.status)) { ok = false; break; }
        ptx::tc_fence_after();
        const uint32_t sK = ptx::smem_u32(smem + OFF_K + s * kTileBytes);
        ptx::mma8_bf16_ss_warp<ptx::KMajorSw128, ptx::KMajorSw128>(tmem + TM_S + s * 128, desc_kmajor(sQ, 0),
                                                                  desc_kmajor(sK, 0), idesc_qk, 0u);
        ptx::mma_commit_warp(&bar->s_full[s]);
        ptx::mma_commit_warp(&bar->k_empty[s]);
        if (j >= 1 && !issue_pv(j - 1)) { ok = false; break; }
      }
      if (ok && !__shfl_sync(0xffffffffu, aborted(bar) ? 1 : 0, 0)) ok = issue_pv(nkb - 1);
      if (!ok && lane == 0) set_abort(bar);
      __syncwarp();
      // all MMAs of this thread complete before TMEM is released
      ptx::mma_commit_warp(&bar->final_mma);
      wait_warp(&bar->final_mma, 0, a.status);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ softmax
    const int r = threadIdx.x;  // row of the tile == TMEM lane
    const int row = w.tile * kRows + r;
    const bool valid = row < w.q_len;
    const int ke = a.kv_end[w.kv_base + (valid ? row : w.q_len - 1)];
    const float sl2 = a.scale * kLog2e;
    const uint32_t lane_addr = (uint32_t)(warp * 32) << 16;
    float m_use = -INFINITY, l = 0.f;
    bool ok = nkb > 0;
    for (int j = 0; ok && j < nkb; ++j) {
      const int s = j & 1;
      const uint32_t n = (uint32_t)(j >> 1);
      if (!wait(&bar->s_full[s], n & 1, a.status)) { ok = false; break; }
      ptx::tc_fence_after();
      float x[128];
      {
        uint32_t t[4][32];
#pragma unroll
        for (int c = 0; c < 4; ++c) ptx::tmem_ld32(tmem + lane_addr + TM_S + s * 128 + c * 32, t[c]);
        ptx::tmem_ld_wait();
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          ptx::reg_fence(t[c]);
#pragma unroll
          for (int i = 0; i < 32; ++i) x[c * 32 + i] = __uint_as_float(t[c][i]);
        }
      }
      ptx::tc_fence_before();
      ptx::mbar_arrive(&bar->s_free[s]);
      // row max on the raw scores (the scale is positive), masked keys at -inf;
      // eight independent partial maxima keep the dependency chain short
      float mr[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) mr[k] = -INFINITY;
      if (j >= kfull) {
        const int lim = ke - j * kRows;
#pragma unroll
        for (int c = 0; c < 128; ++c) {
          x[c] = c < lim ? x[c] : -INFINITY;
          mr[c & 7] = fmaxf(mr[c & 7], x[c]);
        }
      } else {
#pragma unroll
        for (int c = 0; c < 128; ++c) mr[c & 7] = fmaxf(mr[c & 7], x[c]);
      }
      const float mraw = fmaxf(fmaxf(fmaxf(mr[0], mr[1]), fmaxf(mr[2], mr[3])),
                               fmaxf(fmaxf(mr[4], mr[5]), fmaxf(mr[6], mr[7])));
      const float m_new = fmaxf(m_use, mraw * sl2);
      if (j == 0) {
        m_use = m_new;
      } else if (m_new > m_use + 8.f) {
        // the max grew a lot: bring O (complete through PV_{j-1}) and l to the new max
        const int sp = (j - 1) & 1;
        if (!wait(&bar->p_free[sp], (uint32_t)((j - 1) >> 1) & 1, a.status)) { ok = false; break; }
        ptx::tc_fence_after();
        const float f = ex2(m_use - m_new);
        l *= f;
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          uint32_t o[32];
          ptx::tmem_ld32(tmem + lane_addr + TM_O + c * 32, o);
          ptx::tmem_ld_wait();
          ptx::reg_fence(o);
#pragma unroll
          for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * f);
          ptx::tmem_st32(tmem + lane_addr + TM_O + c * 32, o);
        }
        ptx::tmem_st_wait();
        m_use = m_new;
      }
      float rsv[4] = {0.f, 0.f, 0.f, 0.f};
      uint32_t pk[64];
#pragma unroll
      for (int c = 0; c < 64; ++c) {
        const float p0 = ex2(fmaf(x[2 * c], sl2, -m_use));
        const float p1 = ex2(fmaf(x[2 * c + 1], sl2, -m_use));
        rsv[c & 3] += p0 + p1;
        pk[c] = pack_bf16(p0, p1);
      }
      l += (rsv[0] + rsv[1]) + (rsv[2] + rsv[3]);
      if (j >= 2 && !wait(&bar->p_free[s], (n - 1) & 1, a.status)) { ok = false; break; }
      uint8_t* prow = smem + OFF_P + s * kTileBytes + r * 128;
#pragma unroll
      for (int hh = 0; hh < 2; ++hh)
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          uint4 v4 = make_uint4(pk[hh * 32 + c * 4], pk[hh * 32 + c * 4 + 1], pk[hh * 32 + c * 4 + 2],
                                pk[hh * 32 + c * 4 + 3]);
          *reinterpret_cast<uint4*>(prow + hh * kHalfBytes + ((c ^ (r & 7)) << 4)) = v4;
        }
      ptx::fence_proxy_async_smem();
      ptx::tc_fence_before();
      ptx::mbar_arrive(&bar->p_full[s]);
    }
    if (ok) {
      const int jl = nkb - 1;
      ok = wait(&bar->p_free[jl & 1], (uint32_t)(jl >> 1) & 1, a.status);
    }
    // one decision for the whole warp: the epilogue's loads and shuffles are warp-wide
    ok = __all_sync(0xffffffffu, ok);
    if (!ok) {
      set_abort(bar);
    } else {
      ptx::tc_fence_after();
      const float inv = 1.f / l;
      const int64_t orow = (int64_t)w.q_base + row;
      // rows are stored by groups of four lanes (store_slice32)
      const int li = r & 3;
      const int64_t rstride = (int64_t)a.hq * kD;
      __nv_bfloat16* const g0 = reinterpret_cast<__nv_bfloat16*>(a.out) + (orow - li) * rstride + h * kD;
#pragma unroll 1
      for (int c = 0; c < 4; ++c) {
        uint32_t o[32], wo[16];
        ptx::tmem_ld32(tmem + lane_addr + TM_O + c * 32, o);
        ptx::tmem_ld_wait();
        ptx::reg_fence(o);
        pack_scaled32(o, inv, wo);
        store_slice32(wo, g0 + 32 * c, rstride, w.q_len - (row - li));
      }
      if (valid && a.lse) a.lse[(int64_t)h * a.q_rows + orow] = (m_use + log2f(l)) * kLn2;
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 5) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, kTmemCols);
  }
}

// ---------------------------------------------------------------- diagnostic
// One 128x128x128 tile: C = A * B^T (B given as [N, K], K-major) or C = A * B
// (B given as [K, N], MN-major).  Operands staged by plain stores in the
// swizzled layout (modes 0/1), by TMA (modes 2/3), or A in tensor memory and
// B by plain stores (modes 4/5); mode 6: A given as [K, M] (MN-major) and B
// as [K, N], C = A^T B; mode 7: as mode 6 with A in the 8-interleaved
// MN-major layout without swizzle.  Bit 3 of the mode: the same with the eight
// k-steps issued by warp 0 through the batched (one election) form.
__global__ void __launch_bounds__(128, 1)
    mma_tile_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    const __nv_bfloat16* A, const __nv_bfloat16* B, float* C, int mode, uint32_t* status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sa = smem;
  uint8_t* sb = smem + kTileBytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + 2 * kTileBytes);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 2);
  const int warp = threadIdx.x >> 5;
  const bool batched = (mode & 8) != 0;
  mode &= 7;
  const bool a_mn = mode == 6 || mode == 7;
  const bool a_ilv = mode == 7;
  const bool b_mn = (mode & 1) != 0 || mode == 6;
  const bool a_tmem = mode == 4 || mode == 5;
  if (threadIdx.x == 0) {
    ptx::mbar_init(&bars[0], 1);
    ptx::mbar_init(&bars[1], 1);
    ptx::fence_mbar_init();
  }
  if (warp == 0) {
    ptx::tmem_alloc(tslot, 256);
    ptx::tmem_relinquish();
  }
  if (mode < 2 || a_tmem || a_mn) {
    for (int i = threadIdx.x; i < 128 * 128; i += blockDim.x) {
      const int r = i >> 7, c = i & 127;
      *reinterpret_cast<__nv_bfloat16*>(sa + (a_ilv ? ilv_offset(c, r) : swz_offset(r, c))) = A[i];
      *reinterpret_cast<__nv_bfloat16*>(sb + swz_offset(r, c)) = B[i];
    }
    ptx::fence_proxy_async_smem();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tslot;
  const uint32_t lane_addr = (uint32_t)(warp * 32) << 16;
  if (a_tmem) {
    // row r of A into lane r, columns [128, 192): two bf16 of K per column
    const int r = threadIdx.x;
    for (int half = 0; half < 2; ++half) {
      uint32_t v[32];
      for (int i = 0; i < 32; ++i) {
        const __nv_bfloat16 lo = A[r * 128 + half * 64 + 2 * i], hi = A[r * 128 + half * 64 + 2 * i + 1];
        v[i] = (uint32_t)__bfloat16_as_ushort(lo) | ((uint32_t)__bfloat16_as_ushort(hi) << 16);
      }
      ptx::tmem_st32(tmem + lane_addr + 128 + half * 32, v);
    }
    ptx::tmem_st_wait();
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
  }
  bool ok = true;
  if (batched ? warp == 0 : threadIdx.x == 0) {
    if (mode == 2 || mode == 3) {
      if (threadIdx.x == 0) {
        ptx::mbar_expect_tx(&bars[0], 2 * kTileBytes);
        ptx::tma_load_2d(sa, &tmA, &bars[0], 0, 0);
        ptx::tma_load_2d(sa + kHalfBytes, &tmA, &bars[0], 64, 0);
        ptx::tma_load_2d(sb, &tmB, &bars[0], 0, 0);
        ptx::tma_load_2d(sb + kHalfBytes, &tmB, &bars[0], 64, 0);
      }
      ok = wait(&bars[0], 0, status);
    }
    const uint32_t idesc = ptx::idesc_bf16_f32(128, 128, a_mn ? 1u : 0u, b_mn ? 1u : 0u);
    const uint32_t saa = ptx::smem_u32(sa), sbb = ptx::smem_u32(sb);
    if (batched) {
      // the whole warp, converged; one elected lane issues and commits
      ok = __all_sync(0xffffffffu, ok);
      if (ok) {
        using namespace ptx;
        const uint64_t bd = b_mn ? desc_mnmajor(sbb, 0) : desc_kmajor(sbb, 0);
        if (a_tmem && b_mn)
          mma8_bf16_ts_warp<TmemPairs, MnMajorSw128>(tmem, tmem + 128, bd, idesc, 0u);
        else if (a_tmem)
          mma8_bf16_ts_warp<TmemPairs, KMajorSw128>(tmem, tmem + 128, bd, idesc, 0u);
        else if (a_ilv)
          mma8_bf16_ss_warp<MnMajorIlv8, MnMajorSw128>(tmem, desc_ilv_mnmajor(saa, 0), bd, idesc, 0u);
        else if (a_mn)
          mma8_bf16_ss_warp<MnMajorSw128, MnMajorSw128>(tmem, desc_mnmajor(saa, 0), bd, idesc, 0u);
        else if (b_mn)
          mma8_bf16_ss_warp<KMajorSw128, MnMajorSw128>(tmem, desc_kmajor(saa, 0), bd, idesc, 0u);
        else
          mma8_bf16_ss_warp<KMajorSw128, KMajorSw128>(tmem, desc_kmajor(saa, 0), bd, idesc, 0u);
      }
      ptx::mma_commit_warp(&bars[1]);
    } else if (ok) {
      for (int kk = 0; kk < 8; ++kk) {
        const uint64_t bd = b_mn ? desc_mnmajor(sbb, kk) : desc_kmajor(sbb, kk);
        if (a_tmem)
          ptx::mma_bf16_ts(tmem, tmem + 128 + 8 * kk, bd, idesc, kk > 0 ? 1u : 0u);
        else
          ptx::mma_bf16_ss(tmem,
                           a_ilv ? desc_ilv_mnmajor(saa, kk) : a_mn ? desc_mnmajor(saa, kk) : desc_kmajor(saa, kk),
                           bd, idesc, kk > 0 ? 1u : 0u);
      }
    }
    if (!batched) ptx::mma_commit(&bars[1]);
    ok = wait(&bars[1], 0, status) && ok;
  }
  __syncthreads();
  ptx::tc_fence_after();
  for (int c = 0; c < 4; ++c) {
    uint32_t v[32];
    ptx::tmem_ld32(tmem + lane_addr + c * 32, v);
    ptx::tmem_ld_wait();
    ptx::reg_fence(v);
    for (int i = 0; i < 32; ++i) C[threadIdx.x * 128 + c * 32 + i] = __uint_as_float(v[i]);
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, 256);
  }
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

}  // namespace

cudaError_t make_tmap_bf16_plain(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows, uint32_t box_rows) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return cudaErrorNotSupported;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t es[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

cudaError_t make_tmap_e4m3_plain(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows, uint32_t box_rows) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return cudaErrorNotSupported;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols};
  cuuint32_t box[2] = {128, box_rows};
  cuuint32_t es[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(base), dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

cudaError_t make_tmap_bf16(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return cudaErrorNotSupported;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {64, 128};
  cuuint32_t es[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

cudaError_t make_tmap_bf16_box(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows, uint32_t box_rows) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return cudaErrorNotSupported;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t es[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

cudaError_t make_tmap_e4m3_box(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows, uint32_t box_rows) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return cudaErrorNotSupported;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols};
  cuuint32_t box[2] = {128, box_rows};
  cuuint32_t es[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(base), dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// 2D e4m3 tensor map [rows, cols] with a 128 x 128 box (128-byte rows), 128B swizzle.
cudaError_t make_tmap_e4m3(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return cudaErrorNotSupported;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols};
  cuuint32_t box[2] = {128, 128};
  cuuint32_t es[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(base), dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

cudaError_t launch_fwd(const AttnArgs& a, int64_t k_rows, cudaStream_t st) {
  if (a.nq == 0) return cudaSuccess;
  CUtensorMap tq, tk, tv;
  cudaError_t e;
  if (a.dtype == ISM_E4M3) {  // only the paired kernel has the e4m3 form
    if ((e = make_tmap_e4m3(&tq, a.q, (uint64_t)a.hq * kD, (uint64_t)a.q_rows)) != cudaSuccess) return e;
    if ((e = make_tmap_e4m3(&tk, a.k, (uint64_t)a.hkv * kD, (uint64_t)k_rows)) != cudaSuccess) return e;
    if ((e = make_tmap_e4m3(&tv, a.v, (uint64_t)a.hkv * kD, (uint64_t)k_rows)) != cudaSuccess) return e;
    return launch_fwd_pair(a, tq, tk, tv, st);
  }
  if ((e = make_tmap_bf16(&tq, a.q, (uint64_t)a.hq * kD, (uint64_t)a.q_rows)) != cudaSuccess) return e;
  if ((e = make_tmap_bf16(&tk, a.k, (uint64_t)a.hkv * kD, (uint64_t)k_rows)) != cudaSuccess) return e;
  if ((e = make_tmap_bf16(&tv, a.v, (uint64_t)a.hkv * kD, (uint64_t)k_rows)) != cudaSuccess) return e;
  if (((a.hq / a.hkv) % 2 == 0 || a.pair_order) && !knobs().fwd_one_head)
    return launch_fwd_pair(a, tq, tk, tv, st);
  if ((e = cudaFuncSetAttribute(fwd_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes)) !=
      cudaSuccess)
    return e;
  fwd_kernel<<<(unsigned)(a.nq * a.hq), kThreads, kSmemBytes, st>>>(tq, tk, tv, a);
  return cudaGetLastError();
}

cudaError_t launch_mma_tile(const void* A, const void* B, float* C, int mode, uint32_t* status, cudaStream_t st) {
  CUtensorMap ta, tb;
  memset(&ta, 0, sizeof(ta));
  memset(&tb, 0, sizeof(tb));
  cudaError_t e;
  if ((mode & 7) == 2 || (mode & 7) == 3) {
    if ((e = make_tmap_bf16(&ta, A, 128, 128)) != cudaSuccess) return e;
    if ((e = make_tmap_bf16(&tb, B, 128, 128)) != cudaSuccess) return e;
  }
  const uint32_t smem = 2 * kTileBytes + 64 + 1024;
  if ((e = cudaFuncSetAttribute(mma_tile_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) !=
      cudaSuccess)
    return e;
  mma_tile_kernel<<<1, 128, smem, st>>>(ta, tb, (const __nv_bfloat16*)A, (const __nv_bfloat16*)B, C, mode, status);
  return cudaGetLastError();
}

bool available() {
  static int cached = -1;
  static std::mutex mu;
  std::lock_guard<std::mutex> lk(mu);
  if (cached < 0) {
    int dev = 0, major = 0, minor = 0;
    cached = 0;
    if (cudaGetDevice(&dev) == cudaSuccess &&
        cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) == cudaSuccess &&
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) == cudaSuccess)
      cached = (major == 10 && minor == 3 && encode_fn() != nullptr) ? 1 : 0;
  }
  return cached == 1;
}

}  // namespace tc

bool tc_available() { return tc::available(); }
cudaError_t launch_tc_fwd(const AttnArgs& a, int64_t k_rows, cudaStream_t st) { return tc::launch_fwd(a, k_rows, st); }
cudaError_t launch_tc_mma_tile(const void* a, const void* b, float* c, int mode, uint32_t* status, cudaStream_t st) {
  return tc::launch_mma_tile(a, b, c, mode, status, st);
}

}  // namespace ism
