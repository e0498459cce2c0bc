// Segment metadata kernels: per-token key bound kv_end (Eq. fj, Section 2.1),
// the (q-tile, k-tile) classification, work lists for the attention kernels
// ordered most expensive first, and the append-prefill plan (Section 2.3).
#include "ism_internal.cuh"

namespace ism {
namespace {

__device__ __forceinline__ int upper_bound_i32(const int32_t* a, int n, int32_t x) {
  // first index i in [0, n) with a[i] > x (n if none); a non-decreasing
  int lo = 0, hi = n;
  while (lo < hi) {
    int mid = (lo + hi) >> 1;
    if (a[mid] > x) hi = mid; else lo = mid + 1;
  }
  return lo;
}

// Inclusive prefix sum of one value per thread over the block (blockDim.x a
// multiple of 32, at most 1024): shuffle scans within each warp, then warp 0
// scans the warp totals.  *total receives the block's sum.  Every thread of
// the block calls it (it holds __syncthreads).
template <typename T>
__device__ T block_inclusive_scan(T v, T* total) {
  __shared__ T wsum[32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const T t = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += t;
  }
  if (lane == 31) wsum[warp] = v;
  __syncthreads();
  if (warp == 0) {
    T w = lane < nw ? wsum[lane] : T(0);
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const T t = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += t;
    }
    wsum[lane] = w;  // inclusive over the warps
  }
  __syncthreads();
  const T add = warp > 0 ? wsum[warp - 1] : T(0);
  *total = wsum[nw - 1];
  __syncthreads();  // wsum is free for the next call
  return v + add;
}

// Per-sequence tile offsets computed by every block into shared memory:
// qoff/koff [B+1] (q-tiles / k-tiles before sequence b) and toff [B+1]
// (tile_class bytes before sequence b).  Block-wide scans over chunks of
// blockDim.x sequences with a running carry.
__device__ void seq_offsets_smem(const SegsDev& s, int bm, int bn, int32_t* qoff, int32_t* koff, int64_t* toff) {
  if (threadIdx.x == 0) { qoff[0] = 0; koff[0] = 0; toff[0] = 0; }
  int32_t cq = 0, ck = 0;  // carries, the same in every thread
  int64_t ct = 0;
  for (int base = 0; base < s.num_seqs; base += blockDim.x) {
    const int b = base + threadIdx.x;
    int32_t nq = 0, nk = 0;
    if (b < s.num_seqs) {
      const int32_t L = s.cu_seqlens[b + 1] - s.cu_seqlens[b];
      nq = (L + bm - 1) / bm;
      nk = (L + bn - 1) / bn;
    }
    int32_t tq, tk;
    int64_t tt;
    const int32_t iq = block_inclusive_scan<int32_t>(nq, &tq), ik = block_inclusive_scan<int32_t>(nk, &tk);
    const int64_t it = block_inclusive_scan<int64_t>((int64_t)nq * nk, &tt);
    if (b < s.num_seqs) {
      qoff[b + 1] = cq + iq;
      koff[b + 1] = ck + ik;
      toff[b + 1] = ct + it;
    }
    cq += tq;
    ck += tk;
    ct += tt;
  }
  __syncthreads();
}

// kv_end of every token (Eq. fj): a token of a query segment is bounded by
// the end of its segment, a token of an answer segment by itself.  One block
// per segment (grid-stride); threads over the segment's tokens.
__global__ void kv_end_kernel(SegsDev s, int32_t* kv_end) {
  for (int seg = blockIdx.x; seg < s.num_segs; seg += gridDim.x) {
    int b = upper_bound_i32(s.cu_segs, s.num_seqs + 1, seg) - 1;
    int32_t start = seg > s.cu_segs[b] ? s.seg_end[seg - 1] : 0;
    int32_t end = s.seg_end[seg];
    int32_t base = s.cu_seqlens[b];
    bool query = s.seg_type[seg] == ISM_SEG_QUERY;
    for (int32_t j = start + threadIdx.x; j < end; j += blockDim.x)
      kv_end[base + j] = query ? end : j + 1;
  }
}

// q-tile and k-tile descriptors plus the optional public tile-map arrays.
// Since kv_end is non-decreasing within a sequence, q-tile t has
// floor(kv_end[first row] / bn) leading FULL tiles when all of its rows lie
// inside the sequence (0 otherwise), and ceil(kv_end[last row] / bn)
// non-empty tiles; k-tile c is first reached by the q-tile holding the first
// row whose kv_end exceeds c*bn.
// `dyn` holds the per-sequence offsets ((num_seqs + 1) * 16 bytes).
__device__ void tiles_body(const SegsDev& s, int bm, int bn, const int32_t* __restrict__ kv_end, int64_t nq,
                           int64_t nk, Tile* qtiles, Tile* ktiles, uint8_t* tile_class, int32_t* kt_full_end,
                           int32_t* kt_end, int32_t* qt_begin, unsigned char* dyn) {
  int64_t* toff = reinterpret_cast<int64_t*>(dyn);
  int32_t* qoff = reinterpret_cast<int32_t*>(toff + s.num_seqs + 1);
  int32_t* koff = qoff + s.num_seqs + 1;
  seq_offsets_smem(s, bm, bn, qoff, koff, toff);
  int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; g < nq; g += stride) {
    int b = upper_bound_i32(qoff, s.num_seqs + 1, (int32_t)g) - 1;
    int32_t t = (int32_t)g - qoff[b];
    int32_t base = s.cu_seqlens[b];
    int32_t L = s.cu_seqlens[b + 1] - base;
    int32_t r0 = t * bm;
    int32_t rl = min(L, r0 + bm) - 1;
    int32_t full = (r0 + bm <= L) ? kv_end[base + r0] / bn : 0;
    int32_t ne = (kv_end[base + rl] + bn - 1) / bn;
    if (qtiles) {
      Tile w;
      w.q_base = base; w.k_base = base; w.q_len = L; w.k_len = L; w.tile = t;
      w.a0 = full; w.a1 = ne; w.kv_base = base;
      qtiles[g] = w;
    }
    if (kt_full_end) kt_full_end[g] = full;
    if (kt_end) kt_end[g] = ne;
    if (tile_class) {
      int32_t nkt = (L + bn - 1) / bn;
      uint8_t* row = tile_class + toff[b] + (int64_t)t * nkt;
      for (int32_t c = 0; c < nkt; ++c)
        row[c] = c < full ? (uint8_t)ISM_TILE_FULL : c < ne ? (uint8_t)ISM_TILE_PARTIAL : (uint8_t)ISM_TILE_EMPTY;
    }
  }
  for (int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; g < nk; g += stride) {
    int b = upper_bound_i32(koff, s.num_seqs + 1, (int32_t)g) - 1;
    int32_t c = (int32_t)g - koff[b];
    int32_t base = s.cu_seqlens[b];
    int32_t L = s.cu_seqlens[b + 1] - base;
    // first row that sees key x = c*bn: kv_end is non-decreasing, and under
    // Eq. fj the first segment ending after x starts that row when it is a
    // query segment, else the row is max(segment start, x)
    const int32_t x = c * bn;
    const int s0 = s.cu_segs[b], s1 = s.cu_segs[b + 1];
    const int seg = s0 + upper_bound_i32(s.seg_end + s0, s1 - s0, x);
    const int32_t start = seg > s0 ? s.seg_end[seg - 1] : 0;
    int32_t j = s.seg_type[seg] == ISM_SEG_QUERY ? start : (x > start ? x : start);
    int32_t qb = j / bm;
    if (qt_begin) qt_begin[g] = qb;
    if (ktiles) {
      Tile w;
      w.q_base = base; w.k_base = base; w.q_len = L; w.k_len = L; w.tile = c;
      w.a0 = qb; w.a1 = (L + bm - 1) / bm; w.kv_base = base;
      ktiles[g] = w;
    }
  }
}

__global__ void __launch_bounds__(256) tiles_kernel(SegsDev s, int bm, int bn, const int32_t* __restrict__ kv_end,
                             int64_t nq, int64_t nk, Tile* qtiles, Tile* ktiles, uint8_t* tile_class,
                             int32_t* kt_full_end, int32_t* kt_end, int32_t* qt_begin) {
  extern __shared__ __align__(16) unsigned char dyn[];
  tiles_body(s, bm, bn, kv_end, nq, nk, qtiles, ktiles, tile_class, kt_full_end, kt_end, qt_begin, dyn);
}

// Work lists ordered by decreasing cost (counting sort, one block).  Cost of
// a q-tile = its non-empty k-tiles; of a k-tile = its non-empty q-tiles.  The
// optional third list holds the q-tiles with an even index in their sequence
// (the first of each pair of neighbouring q-tiles), costed by the pair's
// larger count (the second tile's, kv_end being non-decreasing); the optional
// fourth the k-tiles with an even index (pairs of neighbouring k-tiles),
// costed by the first tile's count, which covers the second's (its first
// non-empty q-tile comes no earlier).
// Items of equal cost come in arbitrary order; results do not depend on it.
__device__ __forceinline__ bool pair_head(const Tile* qtiles, int64_t nq, int64_t i, int* cost) {
  const Tile w = qtiles[i];
  if (w.tile & 1) return false;
  int c = w.a1;
  if (i + 1 < nq) {
    const Tile n = qtiles[i + 1];
    if (n.q_base == w.q_base && n.tile == w.tile + 1) c = max(c, n.a1);
  }
  *cost = c;
  return true;
}

__device__ void order_body(const Tile* __restrict__ qtiles, int64_t nq, const Tile* __restrict__ ktiles, int64_t nk,
                           int max_cost, int32_t* q_order, int32_t* k_order, int32_t* pair_order, int32_t* hist,
                           int32_t* kp_order = nullptr) {
  for (int pass = 0; pass < 4; ++pass) {
    const Tile* items = pass == 1 || pass == 3 ? ktiles : qtiles;
    int64_t n = pass == 1 || pass == 3 ? nk : nq;
    int32_t* order = pass == 0 ? q_order : pass == 1 ? k_order : pass == 2 ? pair_order : kp_order;
    if (items == nullptr || order == nullptr || n == 0) continue;
    for (int i = threadIdx.x; i <= max_cost; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    for (int64_t i = threadIdx.x; i < n; i += blockDim.x) {
      int cost;
      if (pass == 2) {
        if (!pair_head(items, n, i, &cost)) continue;
      } else {
        const Tile w = items[i];
        if (pass == 3 && (w.tile & 1)) continue;  // k-tile pairs: the even tile, costed by its query tiles
        cost = pass == 0 ? w.a1 : w.a1 - w.a0;
      }
      cost = min(max(cost, 0), max_cost);
      atomicAdd(&hist[cost], 1);
    }
    __syncthreads();
    // exclusive scan from the highest cost down (each thread rewrites the
    // entries it read, so no barrier is needed between the read and the write)
    int32_t run = 0;
    for (int base = 0; base <= max_cost; base += blockDim.x) {
      const int c = max_cost - (base + (int)threadIdx.x);
      const int32_t h = c >= 0 ? hist[c] : 0;
      int32_t tot;
      const int32_t incl = block_inclusive_scan<int32_t>(h, &tot);
      if (c >= 0) hist[c] = run + incl - h;
      run += tot;
    }
    __syncthreads();
    for (int64_t i = threadIdx.x; i < n; i += blockDim.x) {
      int cost;
      if (pass == 2) {
        if (!pair_head(items, n, i, &cost)) continue;
      } else {
        const Tile w = items[i];
        if (pass == 3 && (w.tile & 1)) continue;  // k-tile pairs: the even tile, costed by its query tiles
        cost = pass == 0 ? w.a1 : w.a1 - w.a0;
      }
      cost = min(max(cost, 0), max_cost);
      order[atomicAdd(&hist[cost], 1)] = (int32_t)i;
    }
    __syncthreads();
  }
}

__global__ void order_kernel(const Tile* __restrict__ qtiles, int64_t nq, const Tile* __restrict__ ktiles,
                             int64_t nk, int max_cost, int32_t* q_order, int32_t* k_order, int32_t* pair_order) {
  extern __shared__ int32_t hist[];  // [max_cost + 1]
  order_body(qtiles, nq, ktiles, nk, max_cost, q_order, k_order, pair_order, hist);
}

// Exclusive prefix over k-tiles of their non-empty q-tile counts (a1 - a0):
// the first (k-tile, q-tile) pair slot of each k-tile.  One block, chunks of
// blockDim.x with a running carry.
__device__ void pair_offsets_body(const Tile* __restrict__ ktiles, int64_t nk, int32_t* kpair_off) {
  int32_t carry = 0;  // the same in every thread
  for (int64_t base = 0; base < nk; base += blockDim.x) {
    const int64_t i = base + threadIdx.x;
    int32_t v = 0;
    if (i < nk) {
      const Tile w = ktiles[i];
      v = w.a1 - w.a0 > 0 ? w.a1 - w.a0 : 0;
    }
    int32_t tot;
    const int32_t incl = block_inclusive_scan<int32_t>(v, &tot);
    if (i < nk) kpair_off[i] = carry + incl - v;
    carry += tot;
  }
}

__global__ void pair_offsets_kernel(const Tile* __restrict__ ktiles, int64_t nk, int32_t* kpair_off) {
  pair_offsets_body(ktiles, nk, kpair_off);
}

// All metadata of one attention pass in a single block: kv_end per token
// (Eq. fj, a warp per segment), the q-/k-tile descriptors, the cost-ordered work lists and, for
// the stored-dS backward, the pair offsets.  Global writes of one phase are
// visible to the block's threads after __syncthreads.
__global__ void __launch_bounds__(1024)
    pass_meta_kernel(SegsDev s, int32_t* kv_end, int bm, int bn, int64_t nq, int64_t nk, Tile* qtiles,
                     Tile* ktiles, int max_cost, int32_t* q_order, int32_t* k_order, int32_t* pair_order,
                     int32_t* kpair_off, int32_t* counters, int n_counters, int32_t* kp_order) {
  extern __shared__ __align__(16) unsigned char dyn[];
  if ((int)threadIdx.x < n_counters) counters[threadIdx.x] = 0;  // work counters of the kernels that follow
  // kv_end: one warp per segment, lanes over its tokens
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nwarps = blockDim.x >> 5;
  for (int seg = warp; seg < s.num_segs; seg += nwarps) {
    const int b = upper_bound_i32(s.cu_segs, s.num_seqs + 1, seg) - 1;
    const int32_t start = seg > s.cu_segs[b] ? s.seg_end[seg - 1] : 0;
    const int32_t end = s.seg_end[seg];
    const int32_t base = s.cu_seqlens[b];
    const bool query = s.seg_type[seg] == ISM_SEG_QUERY;
    for (int32_t j = start + lane; j < end; j += 32) kv_end[base + j] = query ? end : j + 1;
  }
  __syncthreads();
  tiles_body(s, bm, bn, kv_end, nq, nk, qtiles, ktiles, nullptr, nullptr, nullptr, nullptr, dyn);
  __syncthreads();
  order_body(qtiles, nq, ktiles, nk, max_cost, q_order, k_order, pair_order, reinterpret_cast<int32_t*>(dyn),
             kp_order);
  if (kpair_off) pair_offsets_body(ktiles, nk, kpair_off);
}

__device__ __forceinline__ int32_t chunk_kv_end(const AppendSegs& sg, int32_t j) {
  int32_t start = 0;
  for (int i = 0; i < sg.n; ++i) {
    int32_t e = sg.end[i];
    if (j < e && j >= start) return sg.type[i] == ISM_SEG_QUERY ? e : j + 1;
    start = e;
  }
  return j + 1;
}

// Append plan (one block): snapshot cache_len, advance it by l_new, write the
// absolute key bound of every new row (all cached keys plus Eq. fj within
// the chunk) and one q-tile descriptor per (sequence, chunk tile).
__global__ void append_plan_kernel(AppendSegs sg, int batch, int64_t kbase_stride, int bm, int bn,
                                   int32_t* cache_len, int32_t* c_snap, int32_t* kv_end,
                                   Tile* qtiles, int32_t* q_order, int32_t* pair_order) {
  __shared__ int32_t cs[1024];
  const int32_t Ln = sg.l_new;
  for (int base = 0; base < batch; base += 1024) {
    // (batch > 1024 is handled in chunks; every thread sees its own chunk)
    int b = base + threadIdx.x;
    if (threadIdx.x < 1024 && b < batch) cs[threadIdx.x] = cache_len[b];
    __syncthreads();
    int nb = min(1024, batch - base);
    for (int i = threadIdx.x; i < nb * Ln; i += blockDim.x) {
      int bl = i / Ln, j = i % Ln;
      kv_end[(int64_t)(base + bl) * Ln + j] = cs[bl] + chunk_kv_end(sg, j);
    }
    int nqt = (Ln + bm - 1) / bm;
    for (int i = threadIdx.x; i < nb * nqt; i += blockDim.x) {
      int bl = i / nqt, t = i % nqt;
      int32_t c = cs[bl];
      int32_t r0 = t * bm, rl = min(Ln, r0 + bm) - 1;
      Tile w;
      w.q_base = (base + bl) * Ln; w.k_base = (int32_t)((base + bl) * kbase_stride);
      w.q_len = Ln; w.k_len = c + Ln; w.tile = t;
      w.a0 = (r0 + bm <= Ln) ? (c + chunk_kv_end(sg, r0)) / bn : 0;
      w.a1 = (c + chunk_kv_end(sg, rl) + bn - 1) / bn;
      w.kv_base = (base + bl) * Ln;
      int64_t g = (int64_t)(base + bl) * nqt + t;
      qtiles[g] = w;
      q_order[g] = (int32_t)g;
    }
    // q-tile pairs (2i, 2i + 1) of each sequence's chunk for the paired forward
    const int npt = (nqt + 1) / 2;
    if (pair_order)
      for (int i = threadIdx.x; i < nb * npt; i += blockDim.x) {
        const int bl = i / npt, p = i % npt;
        pair_order[(int64_t)(base + bl) * npt + p] = (int32_t)((int64_t)(base + bl) * nqt + 2 * p);
      }
    __syncthreads();
    if (threadIdx.x < nb) {
      c_snap[base + threadIdx.x] = cs[threadIdx.x];
      cache_len[base + threadIdx.x] = cs[threadIdx.x] + Ln;
    }
    __syncthreads();
  }
}

// K_new/V_new rows into the caches at [c_snap[b], c_snap[b] + l_new) (rows of
// sequence b from b * cap, or through the page table).
// The attention kernels read keys in tiles of 128 from key 0, so the last
// tile of a sequence runs past its last key.  Masked keys get P = 0, but the
// P V contraction still multiplies those rows of V, and unwritten cache
// memory may hold NaN or Inf bit patterns (0 * NaN = NaN).  Value rows
// [c + l_new, round_up(c + l_new, 128)) are therefore set to zero by every
// cache write (clipped to the capacity of a contiguous cache; a paged tile
// lies within one page).  Keys need no such care: masked scores are replaced,
// not multiplied.
// Single-token steps run without the plan kernel: the cache write reads the
// cache lengths itself (c_snap = cache_len, unchanged until the decode's
// combine kernel advances it) and records them in snap_out for the decode.
__device__ __forceinline__ void copy_snapshot(int batch, const int32_t* __restrict__ c_snap, int32_t* snap_out) {
  if (!snap_out) return;
  for (int64_t b = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; b < batch; b += (int64_t)gridDim.x * blockDim.x)
    snap_out[b] = c_snap[b];
}

__device__ __forceinline__ void zero_value_tail(int batch, int l_new, int vec_per_row, int64_t cap,
                                                const KvPages& pages, const int32_t* __restrict__ c_snap,
                                                uint4* v_cache) {
  const int64_t total = (int64_t)batch * 128 * vec_per_row;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t row = i / vec_per_row;
    const int col = (int)(i % vec_per_row);
    const int b = (int)(row / 128);
    const int64_t end = (int64_t)c_snap[b] + l_new;
    const int64_t p = end + row % 128;
    int64_t stop = (end + 127) / 128 * 128;
    if (!pages.table && stop > cap) stop = cap;
    if (p >= stop) continue;
    const int64_t dst = (pages.table ? paged_row(pages, b, p) : (int64_t)b * cap + p) * vec_per_row + col;
    v_cache[dst] = make_uint4(0u, 0u, 0u, 0u);
  }
}

__global__ void cache_write_kernel(int batch, int l_new, int row_bytes, int64_t cap, KvPages pages,
                                   const int32_t* __restrict__ c_snap, const uint4* __restrict__ k_new,
                                   const uint4* __restrict__ v_new, uint4* k_cache, uint4* v_cache,
                                   int32_t* snap_out) {
  // a decode kernel launched as a programmatic dependent may start its set-up now
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int vec_per_row = row_bytes / 16;
  copy_snapshot(batch, c_snap, snap_out);
  const int64_t total = (int64_t)batch * l_new * vec_per_row;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (int64_t)gridDim.x * blockDim.x) {
    int64_t row = i / vec_per_row;
    int col = (int)(i % vec_per_row);
    int b = (int)(row / l_new);
    int j = (int)(row % l_new);
    const int64_t p = (int64_t)c_snap[b] + j;
    int64_t dst = (pages.table ? paged_row(pages, b, p) : (int64_t)b * cap + p) * vec_per_row + col;
    k_cache[dst] = k_new[i];
    v_cache[dst] = v_new[i];
  }
  zero_value_tail(batch, l_new, vec_per_row, cap, pages, c_snap, v_cache);
}

// Rotary encoding fused with the cache write.  One thread takes eight
// consecutive coordinates k0..k0+7 of the first half of one head row and
// their partners k0+D/2.. (a query head, a key head, or a value head, which
// is copied as is).  Position of new token j of sequence b: c_snap[b] + j.
// The rotation is in fp32; the results are rounded once to the cache's type:
// bf16, or e4m3 after division by the tensor's dequantisation factor
// (q_descale for the rotated queries, k_descale / v_descale for the cache).
__device__ __forceinline__ void load8(const __nv_bfloat16* p, float (&x)[8]) {
  const uint4 u = *reinterpret_cast<const uint4*>(p);
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float2 f = __bfloat1622float2(h[e]);
    x[2 * e] = f.x;
    x[2 * e + 1] = f.y;
  }
}
__device__ __forceinline__ uint32_t e4m3x2(float lo, float hi) {
  uint16_t r;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(r) : "f"(hi), "f"(lo));
  return r;
}
// Eight values stored in the element type of the output: bf16 (descale
// ignored) or e4m3 (x / descale, round to nearest, saturating).
template <bool kE4M3>
__device__ __forceinline__ void store8(void* base, int64_t elem, const float (&x)[8], float descale) {
  if constexpr (kE4M3) {
    uint2 u;
    u.x = e4m3x2(x[0] / descale, x[1] / descale) | (e4m3x2(x[2] / descale, x[3] / descale) << 16);
    u.y = e4m3x2(x[4] / descale, x[5] / descale) | (e4m3x2(x[6] / descale, x[7] / descale) << 16);
    *reinterpret_cast<uint2*>(static_cast<uint8_t*>(base) + elem) = u;
  } else {
    uint4 u;
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&u);
#pragma unroll
    for (int e = 0; e < 4; ++e) h[e] = __floats2bfloat162_rn(x[2 * e], x[2 * e + 1]);
    *reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(base) + elem) = u;
  }
}

template <bool kE4M3>
__global__ void rope_cache_write_kernel(int batch, int l_new, int hq, int hkv, int d, int64_t cap, KvPages pages,
                                        const int32_t* __restrict__ c_snap, const __nv_bfloat16* __restrict__ q_new,
                                        const __nv_bfloat16* __restrict__ k_new,
                                        const __nv_bfloat16* __restrict__ v_new, const float* __restrict__ cos_t,
                                        const float* __restrict__ sin_t, float q_descale, float k_descale,
                                        float v_descale, void* q_rot, void* k_cache, void* v_cache,
                                        int32_t* snap_out) {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  copy_snapshot(batch, c_snap, snap_out);
  const int half = d / 2;
  const int units = half / 8;  // 8-coordinate units in one half of a head row
  const int per_row = (hq + 2 * hkv) * units;
  const int64_t total = (int64_t)batch * l_new * per_row;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t row = i / per_row;  // b * l_new + j
    const int r = (int)(i % per_row);
    const int head = r / units;
    const int k0 = (r % units) * 8;
    const int b = (int)(row / l_new);
    const int64_t p = (int64_t)c_snap[b] + row % l_new;
    const int64_t dst_row = pages.table ? paged_row(pages, b, p) : (int64_t)b * cap + p;
    const __nv_bfloat16* src;
    void* dst;
    int64_t off;  // element offset of the head row in dst
    float descale;
    if (head < hq) {
      src = q_new + (row * hq + head) * d;
      dst = q_rot;
      off = (row * hq + head) * d;
      descale = q_descale;
    } else if (head < hq + hkv) {
      src = k_new + (row * hkv + (head - hq)) * d;
      dst = k_cache;
      off = (dst_row * hkv + (head - hq)) * d;
      descale = k_descale;
    } else {
      src = v_new + (row * hkv + (head - hq - hkv)) * d;
      off = (dst_row * hkv + (head - hq - hkv)) * d;
      float lo[8], hi[8];
      load8(src + k0, lo);
      load8(src + half + k0, hi);
      store8<kE4M3>(v_cache, off + k0, lo, v_descale);
      store8<kE4M3>(v_cache, off + half + k0, hi, v_descale);
      continue;
    }
    float lo[8], hi[8], c[8], s[8];
    load8(src + k0, lo);
    load8(src + half + k0, hi);
    const float4* cp = reinterpret_cast<const float4*>(cos_t + p * half + k0);
    const float4* sp = reinterpret_cast<const float4*>(sin_t + p * half + k0);
    const float4 c0 = __ldg(cp), c1 = __ldg(cp + 1), s0 = __ldg(sp), s1 = __ldg(sp + 1);
    c[0] = c0.x; c[1] = c0.y; c[2] = c0.z; c[3] = c0.w; c[4] = c1.x; c[5] = c1.y; c[6] = c1.z; c[7] = c1.w;
    s[0] = s0.x; s[1] = s0.y; s[2] = s0.z; s[3] = s0.w; s[4] = s1.x; s[5] = s1.y; s[6] = s1.z; s[7] = s1.w;
    float ol[8], oh[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      ol[e] = lo[e] * c[e] - hi[e] * s[e];
      oh[e] = hi[e] * c[e] + lo[e] * s[e];
    }
    store8<kE4M3>(dst, off + k0, ol, descale);
    store8<kE4M3>(dst, off + half + k0, oh, descale);
  }
  zero_value_tail(batch, l_new, hkv * d * (kE4M3 ? 1 : 2) / 16, cap, pages, c_snap, reinterpret_cast<uint4*>(v_cache));
}

}  // namespace

cudaError_t launch_kv_end(const SegsDev& s, int32_t* kv_end, cudaStream_t st) {
  if (s.num_segs == 0) return cudaSuccess;
  int grid = s.num_segs < 4096 ? s.num_segs : 4096;
  kv_end_kernel<<<grid, 256, 0, st>>>(s, kv_end);
  return cudaGetLastError();
}

cudaError_t launch_tiles(const SegsDev& s, int bm, int bn, const int32_t* kv_end, int64_t nq, int64_t nk,
                         Tile* qtiles, Tile* ktiles, uint8_t* tile_class, int32_t* kt_full_end,
                         int32_t* kt_end, int32_t* qt_begin, cudaStream_t st) {
  int64_t n = nq > nk ? nq : nk;
  if (n == 0) return cudaSuccess;
  int grid = (int)((n + 255) / 256);
  if (grid > 608) grid = 608;
  size_t smem = (size_t)(s.num_seqs + 1) * (sizeof(int64_t) + 2 * sizeof(int32_t));
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(tiles_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  tiles_kernel<<<grid, 256, smem, st>>>(s, bm, bn, kv_end, nq, nk, qtiles, ktiles, tile_class, kt_full_end,
                                        kt_end, qt_begin);
  return cudaGetLastError();
}

cudaError_t launch_order(const Tile* qtiles, int64_t nq, const Tile* ktiles, int64_t nk, int max_cost,
                         int32_t* q_order, int32_t* k_order, cudaStream_t st, int32_t* pair_order) {
  size_t smem = sizeof(int32_t) * (size_t)(max_cost + 1);
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(order_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  order_kernel<<<1, 1024, smem, st>>>(qtiles, nq, ktiles, nk, max_cost, q_order, k_order, pair_order);
  return cudaGetLastError();
}

cudaError_t launch_pass_meta(const SegsDev& s, int32_t* kv_end, int bm, int bn, int64_t nq, int64_t nk,
                             Tile* qtiles, Tile* ktiles, int max_cost, int32_t* q_order, int32_t* k_order,
                             int32_t* pair_order, int32_t* kpair_off, int32_t* counters, int n_counters,
                             cudaStream_t st, int32_t* kp_order) {
  size_t a = (size_t)(s.num_seqs + 1) * (sizeof(int64_t) + 2 * sizeof(int32_t));
  size_t b = sizeof(int32_t) * (size_t)(max_cost + 1);
  size_t smem = a > b ? a : b;
  // opted in well below 48 KB: the kernel's static shared memory (the block
  // scans' warp totals) and the dynamic part together must fit what a launch
  // gets without opting in
  if (smem > 16 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(pass_meta_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  pass_meta_kernel<<<1, 1024, smem, st>>>(s, kv_end, bm, bn, nq, nk, qtiles, ktiles, max_cost, q_order, k_order,
                                          pair_order, kpair_off, counters, n_counters, kp_order);
  return cudaGetLastError();
}

cudaError_t launch_pair_offsets(const Tile* ktiles, int64_t nk, int32_t* kpair_off, cudaStream_t st) {
  if (nk == 0) return cudaSuccess;
  pair_offsets_kernel<<<1, 1024, 0, st>>>(ktiles, nk, kpair_off);
  return cudaGetLastError();
}

cudaError_t launch_append_plan(const AppendSegs& segs, int batch, int64_t kbase_stride, int bm, int bn,
                               int32_t* cache_len, int32_t* c_snap, int32_t* kv_end, Tile* qtiles,
                               int32_t* q_order, int32_t* pair_order, cudaStream_t st) {
  append_plan_kernel<<<1, 1024, 0, st>>>(segs, batch, kbase_stride, bm, bn, cache_len, c_snap, kv_end, qtiles,
                                         q_order, pair_order);
  return cudaGetLastError();
}

cudaError_t launch_cache_write(int dtype, int batch, int l_new, int hkv, int d, int64_t cap, const KvPages& pages,
                               const int32_t* c_snap, const void* k_new, const void* v_new,
                               void* k_cache, void* v_cache, cudaStream_t st, int32_t* snap_out) {
  int elem = dtype == ISM_BF16 ? 2 : dtype == ISM_E4M3 ? 1 : 4;
  int row_bytes = hkv * d * elem;
  int64_t total = (int64_t)batch * l_new * (row_bytes / 16);
  if (total == 0) return cudaSuccess;
  const int64_t tail = (int64_t)batch * 128 * (row_bytes / 16);  // value rows zeroed past the new end
  if (tail > total) total = tail;
  int grid = (int)((total + 255) / 256);
  if (grid > 152 * 16) grid = 152 * 16;
  cache_write_kernel<<<grid, 256, 0, st>>>(batch, l_new, row_bytes, cap, pages, c_snap, (const uint4*)k_new,
                                           (const uint4*)v_new, (uint4*)k_cache, (uint4*)v_cache, snap_out);
  return cudaGetLastError();
}

cudaError_t launch_rope_cache_write(int dtype, int batch, int l_new, int hq, int hkv, int d, int64_t cap,
                                   const KvPages& pages, const int32_t* c_snap, const void* q_new,
                                   const void* k_new, const void* v_new, const float* cos_t, const float* sin_t,
                                   float q_descale, float k_descale, float v_descale, void* q_rot, void* k_cache,
                                   void* v_cache, cudaStream_t st, int32_t* snap_out) {
  int64_t total = (int64_t)batch * l_new * (hq + 2 * hkv) * (d / 16);
  if (total == 0) return cudaSuccess;
  const bool e4m3 = dtype == ISM_E4M3;
  const int64_t tail = (int64_t)batch * 128 * (hkv * d * (e4m3 ? 1 : 2) / 16);  // value rows zeroed past the new end
  if (tail > total) total = tail;
  int grid = (int)((total + 255) / 256);
  if (grid > 152 * 16) grid = 152 * 16;
  auto kern = e4m3 ? rope_cache_write_kernel<true> : rope_cache_write_kernel<false>;
  kern<<<grid, 256, 0, st>>>(batch, l_new, hq, hkv, d, cap, pages, c_snap, (const __nv_bfloat16*)q_new,
                             (const __nv_bfloat16*)k_new, (const __nv_bfloat16*)v_new, cos_t, sin_t, q_descale,
                             k_descale, v_descale, q_rot, k_cache, v_cache, snap_out);
  return cudaGetLastError();
}

}  // namespace ism
