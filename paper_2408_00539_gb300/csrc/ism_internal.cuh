// Internal declarations shared by the libism translation units.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "../../include/ism.h"

namespace ism {

// One tile of work for the attention kernels.  A "sequence" here is one
// query stream attending to one key stream: a packed dialogue for the
// one-pass forward/backward, or (new chunk of sequence b, its KV cache) for
// append-prefill.  Key positions (and kv_end values) are relative to k_base.
struct Tile {
  int32_t q_base;   // global Q/O/dO row of query row 0 of the sequence
  int32_t k_base;   // global K/V row of key 0 of the sequence
  int32_t q_len;    // query rows of the sequence
  int32_t k_len;    // keys of the sequence
  int32_t tile;     // q-tile index t (or k-tile index c) within the sequence
  int32_t a0;       // q-tile: number of leading FULL k-tiles; k-tile: first non-empty q-tile
  int32_t a1;       // q-tile: one past the last non-empty k-tile; k-tile: number of q-tiles
  int32_t kv_base;  // index of the sequence's query row 0 in the kv_end array
};
static_assert(sizeof(Tile) == 32, "Tile layout");

// Paged K/V cache (append-prefill and decode): key p of sequence b sits in
// row table[b * max_pages + p / page_size] * page_size + p % page_size of the
// pools.  With table == nullptr the cache is contiguous: the rows of sequence
// b start at b * cap (append kernels) or at Tile::k_base (attention kernels).
struct KvPages {
  const int32_t* table;
  int32_t page_size, max_pages;
};
__device__ __forceinline__ int64_t paged_row(const KvPages& pg, int b, int64_t p) {
  return (int64_t)__ldg(pg.table + (int64_t)b * pg.max_pages + p / pg.page_size) * pg.page_size + p % pg.page_size;
}

// Device view of the segment arrays (device pointers only).
struct SegsDev {
  int32_t num_seqs;
  int32_t num_segs;
  const int32_t* cu_seqlens;
  const int32_t* cu_segs;
  const int32_t* seg_end;
  const uint8_t* seg_type;
};

// Chunk segments of an append, passed to kernels by value.
constexpr int kMaxAppendSegs = 256;
struct AppendSegs {
  int32_t n;
  int32_t l_new;
  int32_t end[kMaxAppendSegs];
  uint8_t type[kMaxAppendSegs];
};

// Meta arrays carved out of a workspace.
struct Meta {
  int32_t* kv_end;      // [kv rows]
  Tile* qtiles;         // [nq]
  Tile* ktiles;         // [nk] (may be null)
  int32_t* q_order;     // [nq] q-tile indices, most expensive first
  int32_t* k_order;     // [nk]
  int64_t nq, nk;
};

// Status word bits recorded by device code.
enum : uint32_t { kStatusTimeout = 1u, kStatusSmemAlign = 2u };

// ---------------------------------------------------------------- launches
// Each returns cudaSuccess or the launch error.

// Tile-map kernels (ism_meta.cu).
cudaError_t launch_kv_end(const SegsDev& s, int32_t* kv_end, cudaStream_t st);
// At most kMaxSeqs sequences (per-sequence offsets are kept in shared memory).
constexpr int kMaxSeqs = 8192;
cudaError_t launch_tiles(const SegsDev& s, int bm, int bn, const int32_t* kv_end, int64_t nq, int64_t nk,
                         Tile* qtiles, Tile* ktiles, uint8_t* tile_class, int32_t* kt_full_end,
                         int32_t* kt_end, int32_t* qt_begin, cudaStream_t st);
cudaError_t launch_order(const Tile* qtiles, int64_t nq, const Tile* ktiles, int64_t nk, int max_cost,
                         int32_t* q_order, int32_t* k_order, cudaStream_t st, int32_t* pair_order = nullptr);
cudaError_t launch_pair_offsets(const Tile* ktiles, int64_t nk, int32_t* kpair_off, cudaStream_t st);
// kv_end, tiles, work lists (and pair offsets when kpair_off is set, the
// k-tile pair list when kp_order is set) in one launch.
cudaError_t launch_pass_meta(const SegsDev& s, int32_t* kv_end, int bm, int bn, int64_t nq, int64_t nk,
                             Tile* qtiles, Tile* ktiles, int max_cost, int32_t* q_order, int32_t* k_order,
                             int32_t* pair_order, int32_t* kpair_off, int32_t* counters, int n_counters,
                             cudaStream_t st, int32_t* kp_order = nullptr);
// k_base of sequence b's tiles = b * kbase_stride (the cache capacity, or 1 for a paged cache)
cudaError_t launch_append_plan(const AppendSegs& segs, int batch, int64_t kbase_stride, int bm, int bn,
                               int32_t* cache_len, int32_t* c_snap, int32_t* kv_end, Tile* qtiles,
                               int32_t* q_order, int32_t* pair_order, cudaStream_t st);
// c_snap: cache lengths before the append.  snap_out (nullable): receives a
// copy of them (single-token steps pass cache_len itself as c_snap).
cudaError_t launch_cache_write(int dtype, int batch, int l_new, int hkv, int d, int64_t cap, const KvPages& pages,
                               const int32_t* c_snap, const void* k_new, const void* v_new,
                               void* k_cache, void* v_cache, cudaStream_t st, int32_t* snap_out = nullptr);
// Cache write with the rotary encoding of the new queries and keys (bf16
// inputs, head_dim a multiple of 16): rotated keys and plain values into the
// cache, rotated queries into q_rot [batch * l_new, hq, d], all in the cache's
// type: bf16, or e4m3 (dtype ISM_E4M3) after division by the descales.
cudaError_t launch_rope_cache_write(int dtype, int batch, int l_new, int hq, int hkv, int d, int64_t cap,
                                   const KvPages& pages, const int32_t* c_snap, const void* q_new,
                                   const void* k_new, const void* v_new, const float* cos_t, const float* sin_t,
                                   float q_descale, float k_descale, float v_descale, void* q_rot, void* k_cache,
                                   void* v_cache, cudaStream_t st, int32_t* snap_out = nullptr);

// Rotary encoding of the one-pass path (ism_rope.cu): rotates every query and
// key head row of a packed batch by its position inside its sequence (pairs
// k, k + d/2; tables [rows, d/2] fp32), from q_src / k_src into q_dst / k_dst
// (in place allowed).  sin_sign = -1 applies the transposed rotation.  bf16
// or fp32 rows, d a multiple of 16.
cudaError_t launch_rope_rows(const int32_t* cu_seqlens, int num_seqs, int64_t T, int hq, int hkv, int d, int dtype,
                             const void* q_src, const void* k_src, void* q_dst, void* k_dst, const float* cos_t,
                             const float* sin_t, float sin_sign, cudaStream_t st);

// CUDA-core attention (ism_simt.cu), fp32 or bf16 storage, fp32 math.
struct AttnArgs {
  const void* q; const void* k; const void* v; const void* o; const void* dout;
  void* out; float* lse; const float* lse_in;
  void* dq; void* dk; void* dv;
  float* delta;
  int32_t hq, hkv, d, dtype;
  int64_t q_rows;      // rows of Q (LSE row stride)
  float scale;
  const int32_t* kv_end;
  const Tile* qtiles; const int32_t* q_order; int64_t nq;
  const Tile* ktiles; const int32_t* k_order; int64_t nk;
  uint32_t* status;
  // Stored-dS backward: when ds is set, dK/dV also writes each bf16 dS tile
  // (128 queries x 128 keys, 8-query-interleaved, 32 KiB) of (k-tile gk,
  // q-tile t, head h) to slot (kpair_off[gk] + t - qt_begin(gk)) * hq + h,
  // and dQ is a GEMM over them.
  void* ds;
  const int32_t* kpair_off;
  int64_t ds_slots;
  // Query-tile pairs for the paired forward when the query heads of a KV head
  // are odd in number: pair_order lists the even-indexed q-tiles (each with
  // the next q-tile of its sequence, when there is one) in cost order.
  const int32_t* pair_order;
  int64_t npairs;
  // Work counter of the persistent dK/dV kernel (zeroed by the metadata pass).
  int32_t* work_counter;
  // dK/dV on CTA pairs: kp_order lists the even-indexed k-tiles (each with the
  // next k-tile of its sequence, when there is one) in cost order; nkp of them.
  const int32_t* kp_order;
  int64_t nkp;
  // Paged K/V (forward over an appended chunk only): Tile::k_base holds the
  // sequence index and key p's row is paged_row(pages, k_base, p).
  KvPages pages;
  // e4m3 forward: per-tensor dequantisation factors (scores scaled by
  // q_descale * k_descale, the output by v_descale).
  float qk_descale, v_descale;
  // Key-range split of the paired forward (head pairs only): launch items
  // [0, split_whole) run whole; each later item runs as two CTAs over the
  // first and the second half of its key tiles, writing unnormalised O and
  // (max, sum) to part_o / part_ml, merged by a second kernel.  Off when
  // split_items == 0.
  int64_t split_whole, split_items;
  float* part_o;    // [split_items][2 halves][2 heads][128 rows][128] fp32
  float* part_ml;   // [split_items][2 halves][2 heads][128 rows][2] fp32
  // Rotary encoding (tensor-core backward only): when rope_cos is set, the dQ
  // and dK epilogues store the gradients of the unrotated queries and keys,
  // applying the transposed rotation of the row's position in its sequence
  // (tables [rows, 64] fp32, the angle of pair k of position p at p * 64 + k).
  const float* rope_cos;
  const float* rope_sin;
  // Bit 0: before an MMA that overwrites tensor memory an earlier MMA reads
  // as its A operand, wait for that earlier MMA to complete.  Clear: rely on
  // MMAs issued by one thread executing in issue order.
  uint32_t flags;
};
enum : uint32_t { kFlagDrainTmemReuse = 1u };
cudaError_t launch_simt_fwd(const AttnArgs& a, cudaStream_t st);
cudaError_t launch_simt_bwd(const AttnArgs& a, cudaStream_t st);

// Split-KV decode for single-token appends (ism_decode.cu).
struct DecodeArgs {
  const void* q;         // [B, Hq, D]
  const void* k_cache;   // [B, cap, Hkv, D], or the page pools [pages * page_size, Hkv, D]
  const void* v_cache;
  KvPages pages;         // table == nullptr: contiguous caches
  void* out;             // [B, Hq, D]
  float* lse;            // [Hq, B] or null
  const int32_t* c_snap; // cache length before the append, per sequence
  int32_t batch, hq, hkv, d, dtype;
  int32_t group;         // query heads per KV head (the kernels pad it to a power of two)
  float qk_descale, v_descale;  // e4m3: dequantisation of the scores and of the output
  int64_t cap;
  int64_t kv_rows;       // rows of the K / V tensors: batch * cap, or pages * page_size
  float scale;
  int32_t splits, chunk;
  float* part_o;         // [B, Hq, splits, D]
  float* part_ml;        // [B, Hq, splits, 2]
  int32_t tma;           // stream the cache with TMA (head_dim 128, sm_103)
  int32_t tc;            // tensor-core kernel (bf16 or e4m3, head_dim 128, group <= 16; chunk a multiple of 128)
  uint32_t* status;      // device status word (bounded waits)
  int32_t* cache_len;    // nullable: the combine kernel advances it by one (single-token steps)
};
// Keys one work item of the tensor-core decode covers at most (its scores of
// 24 tiles of 128 keys stay in tensor memory).
constexpr int kDecTcMaxKeys = 24 * 128;
cudaError_t launch_decode(const DecodeArgs& a, cudaStream_t st);

// Tensor-core kernels (ism_fwd_tc.cu / ism_bwd_tc.cu), bf16 only.
bool tc_available();
bool tc_bwd_available();
cudaError_t launch_tc_mma_tile(const void* a, const void* b, float* c, int mode, uint32_t* status, cudaStream_t st);
namespace tc {
cudaError_t launch_mma_tile_e4m3(const void* a, const void* b, float* c, int mode, uint32_t* status, cudaStream_t st);
}
cudaError_t launch_tc_fwd(const AttnArgs& a, int64_t k_rows, cudaStream_t st);
cudaError_t launch_tc_bwd(const AttnArgs& a, int64_t k_rows, cudaStream_t st);

cudaError_t launch_timeout_probe(uint32_t spin_limit, uint32_t* status, cudaStream_t st);

// Debug and tuning switches from the environment (ISM_*), read once when the
// library is loaded and again by ism_debug_reload_env(), so that no call reads
// the environment.
struct Knobs {
  bool force_cuda_cores;   // ISM_FORCE_CUDA_CORES=1: CUDA-core kernels for bf16 too
  bool drain_tmem_reuse;   // ISM_DRAIN_TMEM_REUSE=1: wait for A-operand readers before overwriting TMEM
  bool fwd_one_head;       // ISM_FWD_ONE_HEAD=1: one-head forward kernel
  bool bwd_recompute_dq;   // ISM_BWD_RECOMPUTE_DQ=1: recompute backward even with a stored-dS workspace
  bool decode_no_tma;      // ISM_DECODE_NO_TMA=1: register-load CUDA-core decode
  bool decode_no_tc;       // ISM_DECODE_NO_TC=1: CUDA-core decode kernels
  int64_t prefill_split;   // ISM_PREFILL_SPLIT=n: n key-range split items in a prefill (-1: chosen by the library)
  int32_t dkdv_grid;       // ISM_DKDV_GRID=n: CTAs of the persistent dK/dV kernel (0: one per SM)
  int32_t dq_grid;         // ISM_DQ_GRID=n: CTAs of the persistent dQ kernel (0: one per SM)
  bool dkdv_pair;          // ISM_DKDV_PAIR=1: dK/dV on CTA pairs (cta_group::2)
};
const Knobs& knobs();
void reload_knobs();
// Multiprocessor count of the current device (looked up once per device).
int sm_count();

// Measurement hooks (ism_api.cu): events recorded around launches of one
// kernel kind on the calling host thread, and a count of every launch.
void timer_begin(int kernel_id, cudaStream_t st);
void timer_end(int kernel_id, cudaStream_t st);
void count_launch(int n = 1);
// Sets the message returned by ism_last_error() on this host thread.
void set_error(const char* msg);

}  // namespace ism
