/*
 * ism.h -- C ABI of libism: softmax attention under the Intermittent
 * Semi-working Mask (ISM, arXiv 2408.00539) on NVIDIA GB300 (sm_103a).
 *
 * The mask (Section 2.1, Eq. e_ISM with the bound f(j) of Eq. fj): a
 * dialogue [P, Q1, A1, ..., Q_{n-1}, A_{n-1}, Q_n] is cut into segments.
 * A token of a query segment (the prompt P belongs to the first one) sees
 * every key up to the end of its own query segment; a token of an answer
 * segment sees keys up to and including itself; no token sees past the end
 * of its own segment.  In 0-based indices row j of a sequence sees keys
 * [0, kv_end[j]) with kv_end[j] = f(j+1).
 *
 * Conventions shared by every entry point
 *  - Pointers without a `_host` suffix are DEVICE pointers; `_host` ones are
 *    host mirrors of the same data, used for validation and sizing without a
 *    device synchronisation.  Both must hold identical values.
 *  - Tensors are dense, row-major and 16-byte aligned.  Q and O are
 *    [tokens, Hq, D]; K and V are [tokens, Hkv, D]; LSE is [Hq, tokens] fp32
 *    (natural log of the sum of exp(scale * q.k) over visible keys).
 *  - Grouped-query attention: query head h uses KV head h / (Hq / Hkv).
 *  - The caller owns and allocates every buffer, workspaces included.  The
 *    library allocates no device memory and keeps no state between calls
 *    except one device status word per device (see ism_check_status).
 *  - Every call is asynchronous on `stream` (a cudaStream_t; NULL is the
 *    legacy default stream).  Only ism_check_status synchronises.
 *  - Arguments are validated on the host before anything is launched; on an
 *    error nothing is launched, outputs are untouched, and ism_last_error()
 *    describes the problem.
 */
#ifndef ISM_H_
#define ISM_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* ism_stream_t; /* identical to cudaStream_t */

typedef enum {
  ISM_OK = 0,
  ISM_ERR_INVALID_ARG = 1,  /* null/misaligned pointer, malformed segments, size overflow */
  ISM_ERR_UNSUPPORTED = 2,  /* valid but not implemented (head_dim, dtype, tile size) */
  ISM_ERR_CUDA = 3,         /* a CUDA runtime call or kernel launch failed */
  ISM_ERR_TIMEOUT = 4,      /* a bounded device-side wait gave up (reported by ism_check_status) */
  ISM_ERR_WORKSPACE = 5     /* workspace pointer null/misaligned or smaller than required */
} ism_status_t;

typedef enum { ISM_BF16 = 0, ISM_FP32 = 1, ISM_E4M3 = 2 } ism_dtype_t;

enum { ISM_SEG_QUERY = 0, ISM_SEG_ANSWER = 1 };
enum { ISM_TILE_EMPTY = 0, ISM_TILE_FULL = 1, ISM_TILE_PARTIAL = 2 };

/* Turn boundaries of a varlen batch (Section 2.1: the cumulative ends
 * m_p, m_{q_k}, m_{a_k} of the dialogue's prompt, queries and answers).
 *   cu_seqlens [num_seqs+1]  token offset of each packed sequence; cu_seqlens[0] = 0,
 *                            non-decreasing.  Sequences never attend to each other.
 *   cu_segs    [num_seqs+1]  segment offset of each sequence; cu_segs[0] = 0,
 *                            cu_segs[num_seqs] = num_segs.
 *   seg_end    [num_segs]    exclusive end of each segment relative to its
 *                            sequence, non-decreasing within the sequence; the
 *                            last one equals the sequence length.  Zero-length
 *                            segments are allowed.
 *   seg_type   [num_segs]    ISM_SEG_QUERY or ISM_SEG_ANSWER.  Consecutive query
 *                            segments are separate bidirectional blocks.
 * A sequence of length 0 has no segments or only zero-length ones. */
typedef struct {
  int32_t num_seqs;
  int32_t num_segs;
  const int32_t* cu_seqlens;
  const int32_t* cu_seqlens_host;
  const int32_t* cu_segs;
  const int32_t* cu_segs_host;
  const int32_t* seg_end;
  const int32_t* seg_end_host;
  const uint8_t* seg_type;
  const uint8_t* seg_type_host;
} ism_segments_t;

/* Heads and element type.  Supported: head_dim 64 or 128; Hq % Hkv == 0;
 * ISM_BF16 (fp32 accumulation) or ISM_FP32 (fp32 CUDA-core path); ISM_E4M3
 * (fp8 inputs, head_dim 128) only for the e4m3 entry points and their
 * workspace queries.  The tensor-core kernels serve bf16 and e4m3 at
 * head_dim 128; bf16 at head_dim 64 runs the CUDA-core kernels (correct, but
 * far from the tensor-core rate), as does fp32.  softmax_scale multiplies q.k before the softmax (the paper omits
 * the factor, Section 2.1; 1/sqrt(head_dim) is the usual choice). */
typedef struct {
  int32_t num_heads_q;
  int32_t num_heads_kv;
  int32_t head_dim;
  int32_t dtype; /* ism_dtype_t */
  float softmax_scale;
} ism_attn_shape_t;

/* Rotary position encoding tables (positional encoding is outside the
 * operation of Section 2.1, which leaves it out; models that take up ISM,
 * Section 2.3, rotate queries and keys by their positions before attention).
 * For a head row x at position p and k < D/2, the pair (x_k, x_{k+D/2}) is
 * turned by the angle whose cosine and sine are cos[p * D/2 + k] and
 * sin[p * D/2 + k]:
 *     y_k = x_k cos - x_{k+D/2} sin,     y_{k+D/2} = x_{k+D/2} cos + x_k sin
 * (the rotary encoding of RoFormer in its rotate-half form), in fp32 with one
 * rounding to the element type.  cos / sin: fp32 device tables [rows, D/2],
 * 16-byte aligned, read only.  Any angles are accepted. */
typedef struct {
  const float* cos;
  const float* sin;
  int32_t rows;
} ism_rope_t;

/* ---------------------------------------------------------------------------
 * Tile map.  Classifies each (q-tile, k-tile) rectangle of each sequence:
 * rows [t*bm, t*bm+bm) and keys [c*bn, c*bn+bn) relative to the sequence.
 * FULL: inside the sequence and every pair visible (run without a mask);
 * EMPTY: no in-bounds pair visible (skipped); PARTIAL otherwise.  Because
 * kv_end is non-decreasing (Eq. fj), each q-tile row of the map reads
 * FULL* PARTIAL* EMPTY*.  No counterpart in the paper: it is a classification
 * of the Eq. (fj) mask.
 * ------------------------------------------------------------------------- */

/* Sizes of the tile-map arrays: n_tiles = sum_b nqt_b*nkt_b, n_qtiles =
 * sum_b ceil(L_b/bm), n_ktiles = sum_b ceil(L_b/bn).  bm, bn in {16,...,256}
 * multiples of 16.  Host-only; reads the _host mirrors. */
ism_status_t ism_tile_map_size(const ism_segments_t* segs, int32_t bm, int32_t bn,
                               int64_t* n_tiles, int64_t* n_qtiles, int64_t* n_ktiles);

/* Builds the tile map on the device (kernels on `stream`).  Outputs (device,
 * any may be NULL to skip):
 *   tile_class  [n_tiles]  uint8, per sequence a row-major [nqt_b, nkt_b] block
 *   kt_full_end [n_qtiles] number of leading FULL k-tiles of each q-tile
 *   kt_end      [n_qtiles] one past the last non-EMPTY k-tile
 *   qt_begin    [n_ktiles] first non-EMPTY q-tile of each k-tile column
 *   kv_end      [total_tokens] per-token exclusive key bound, sequence-relative
 * Cited: Eq. (fj), Section 2.1. */
ism_status_t ism_build_tile_map(const ism_segments_t* segs, int32_t bm, int32_t bn,
                                uint8_t* tile_class, int32_t* kt_full_end, int32_t* kt_end,
                                int32_t* qt_begin, int32_t* kv_end, ism_stream_t stream);

/* ---------------------------------------------------------------------------
 * Forward over whole packed dialogues in one pass (Eq. e_ISM with softmax;
 * Section 2.3 applies ISM by replacing the causal mask of a softmax LLM).
 *   q [T, Hq, D], k/v [T, Hkv, D] (dtype), o [T, Hq, D] (dtype, written),
 *   lse [Hq, T] fp32 (written; may be NULL only if no backward follows).
 *   workspace: device scratch of at least ism_attn_fwd_workspace_size bytes,
 *   256-byte aligned; its contents on entry do not matter.
 * ------------------------------------------------------------------------- */
ism_status_t ism_attn_fwd_workspace_size(const ism_segments_t* segs, const ism_attn_shape_t* shape,
                                         size_t* bytes);
ism_status_t ism_attn_fwd(const ism_segments_t* segs, const ism_attn_shape_t* shape,
                          const void* q, const void* k, const void* v, void* o, float* lse,
                          void* workspace, size_t workspace_bytes, ism_stream_t stream);

/* ---------------------------------------------------------------------------
 * Forward with e4m3 (fp8) Q, K, V: the operation of ism_attn_fwd (Eq. e_ISM,
 * the bound of Eq. fj) on the dequantised inputs q * q_descale, k * k_descale,
 * v * v_descale (one factor per tensor).  shape->dtype must be ISM_E4M3 and
 * head_dim 128; q [T, Hq, 128], k/v [T, Hkv, 128] e4m3 (OCP fp8 E4M3FN);
 * o [T, Hq, 128] bf16 (written); lse [Hq, T] fp32 or NULL.  The score
 * contraction and O += P V run on the fp8 tensor cores (kind::f8f6f4) with
 * fp32 accumulation; P is rounded to e4m3 (round to nearest) for P V, the
 * softmax statistics stay fp32.  Workspace: ism_attn_fwd_workspace_size with
 * the same shape.  Errors as ism_attn_fwd, plus ISM_ERR_UNSUPPORTED without
 * the sm_103 tensor cores and ISM_ERR_INVALID_ARG for a descale that is not
 * a positive finite number.
 * ------------------------------------------------------------------------- */
ism_status_t ism_attn_fwd_e4m3(const ism_segments_t* segs, const ism_attn_shape_t* shape,
                               const void* q, const void* k, const void* v,
                               float q_descale, float k_descale, float v_descale,
                               void* o, float* lse, void* workspace, size_t workspace_bytes,
                               ism_stream_t stream);

/* Forward without a caller-provided workspace (the paper has no counterpart;
 * this is a deployment convenience).  Some callers cannot allocate device
 * memory at the point where they run attention: inference servers that carve
 * all device memory into their own pools once at start-up and may not grow
 * them afterwards (a late cudaMalloc can fail there, and it synchronises the
 * device), and hosts that drive the GPU only through this C interface, with
 * no device allocator of their own.  This variant takes the forward's scratch
 * from a fixed array of ism_attn_fwd_noalloc_max_workspace() bytes (4 MiB)
 * that the library keeps in device memory on every GPU that loads it, until
 * the process exits.  It calls no allocator.
 *  - Same arguments and results as ism_attn_fwd, minus the workspace.
 *  - Batches whose forward workspace (ism_attn_fwd_workspace_size) exceeds
 *    the array return ISM_ERR_WORKSPACE before anything is launched.
 *  - The first call on a device looks the array's device address up
 *    (cudaGetSymbolAddress, a host-side query) with that device current.
 *  - All calls share the one array: calls whose kernels may overlap on the
 *    GPU (different streams without ordering) race on it. */
size_t ism_attn_fwd_noalloc_max_workspace(void);
ism_status_t ism_attn_fwd_noalloc(const ism_segments_t* segs, const ism_attn_shape_t* shape,
                                  const void* q, const void* k, const void* v, void* o, float* lse,
                                  ism_stream_t stream);

/* ---------------------------------------------------------------------------
 * Backward: gradients of sum(O * dO) with respect to Q, K, V, given the
 * forward's O and LSE.  dq [T, Hq, D], dk/dv [T, Hkv, D] (dtype, written;
 * dk/dv summed over the query heads that share a KV head).  Standard
 * softmax-attention calculus over the Eq. (e_ISM) mask.
 *
 * Two schedules, chosen by the workspace the caller passes:
 *  - stored-dS (bf16, head_dim 128, tensor cores): the dK/dV kernel also
 *    keeps every visible 128x128 tile of dS^T (bf16) in the workspace and dQ
 *    is a GEMM over those tiles; 32 KiB per visible (query tile, key tile,
 *    query head) on top of the minimum.  Taken when workspace_bytes is at
 *    least ism_attn_bwd_workspace_size; ISM_BWD_RECOMPUTE_DQ=1 in the
 *    environment disables it.
 *  - recompute: the dQ kernel recomputes S, P and dP; needs only
 *    ism_attn_bwd_workspace_size_min bytes.
 * ism_attn_bwd_workspace_size reports the stored-dS size where that schedule
 * applies and the minimum otherwise.  Both schedules give dQ from the same
 * bf16-rounded dS, so they differ only in fp32 summation order.
 * ------------------------------------------------------------------------- */
ism_status_t ism_attn_bwd_workspace_size(const ism_segments_t* segs, const ism_attn_shape_t* shape,
                                         size_t* bytes);
ism_status_t ism_attn_bwd_workspace_size_min(const ism_segments_t* segs, const ism_attn_shape_t* shape,
                                             size_t* bytes);
ism_status_t ism_attn_bwd(const ism_segments_t* segs, const ism_attn_shape_t* shape,
                          const void* q, const void* k, const void* v, const void* o,
                          const float* lse, const void* dout,
                          void* dq, void* dk, void* dv,
                          void* workspace, size_t workspace_bytes, ism_stream_t stream);

/* ---------------------------------------------------------------------------
 * One-pass forward and backward with rotary encoding (see ism_rope_t).  The
 * positions of a packed batch restart at every sequence: token t of sequence
 * b sits at position t - cu_seqlens[b]; rope->rows must be at least the
 * longest sequence.  bf16 or fp32 inputs, head_dim 64 or 128.
 *
 * ism_attn_fwd_rope rotates q [T, Hq, D] and k [T, Hkv, D] (unrotated) into
 * q_rot / k_rot (same shapes and dtype, written; they may be q / k themselves
 * for a rotation in place) in one pass over both, then runs ism_attn_fwd on
 * q_rot, k_rot and v.  A training step keeps q_rot and k_rot for the
 * backward, which takes them instead of q and k.
 *
 * ism_attn_bwd_rope is ism_attn_bwd on q_rot, k_rot (as written by the
 * forward), v, o, lse, dout, except that dq and dk are the gradients with
 * respect to the UNROTATED q and k: the gradients of the rotated rows go back
 * through the transposed rotation (the rotation by the opposite angle).  On
 * the tensor cores (bf16, head_dim 128) that happens in the dQ and dK
 * epilogues; otherwise one more pass rotates dq and dk in place.
 * Workspaces: ism_attn_fwd_workspace_size / ism_attn_bwd_workspace_size (or
 * _min) of the same segments and shape.  Errors as ism_attn_fwd /
 * ism_attn_bwd, plus ISM_ERR_INVALID_ARG for a missing or misaligned table,
 * tables too short for the longest sequence, or e4m3 inputs.
 * ------------------------------------------------------------------------- */
ism_status_t ism_attn_fwd_rope(const ism_segments_t* segs, const ism_attn_shape_t* shape,
                               const void* q, const void* k, const void* v, const ism_rope_t* rope,
                               void* q_rot, void* k_rot, void* o, float* lse,
                               void* workspace, size_t workspace_bytes, ism_stream_t stream);
ism_status_t ism_attn_bwd_rope(const ism_segments_t* segs, const ism_attn_shape_t* shape,
                               const void* q_rot, const void* k_rot, const void* v, const void* o,
                               const float* lse, const void* dout, const ism_rope_t* rope,
                               void* dq, void* dk, void* dv,
                               void* workspace, size_t workspace_bytes, ism_stream_t stream);

/* ---------------------------------------------------------------------------
 * Plans: the metadata of one batch of segments, built once and shared by the
 * forward and the backward of every attention layer over those segments
 * with the same head counts.  The metadata is what ism_attn_fwd and
 * ism_attn_bwd otherwise rebuild at the start of every call: the per-token
 * key bounds (Eq. fj), the (query tile, key tile) descriptors and the work
 * lists in cost order.  A training step then runs one metadata pass for all
 * of its layers instead of two per layer.
 *
 * ism_attn_plan_size: device bytes of the plan for these segments and shape
 *   (head counts; dtype ISM_BF16 or ISM_FP32; head_dim as for ism_attn_fwd).
 * ism_attn_plan_build: runs the metadata pass into `plan` (device memory of
 *   at least that size, 256-byte aligned, owned by the caller) on `stream`
 *   and fills *plan_info on the host: a fingerprint of the segments' host
 *   arrays and the head counts, and the plan's size.
 * ism_attn_fwd_planned / ism_attn_bwd_planned: ism_attn_fwd / ism_attn_bwd
 *   on the plan's metadata, with identical results.  The segments and shape
 *   must be those of the build (same host arrays and head counts; the
 *   softmax scale may differ): a mismatch of the fingerprint returns
 *   ISM_ERR_INVALID_ARG before any launch.  The forward needs no workspace;
 *   the backward takes a workspace as ism_attn_bwd does
 *   (ism_attn_bwd_workspace_size for the stored-dS schedule, _min for the
 *   recompute schedule: both cover what the planned call uses).
 * ism_attn_fwd_rope_planned / ism_attn_bwd_rope_planned: the same for
 *   ism_attn_fwd_rope / ism_attn_bwd_rope (arguments as there).
 * The plan must stay unchanged while a call that uses it may run, and calls
 * that share a plan run in stream order (the backward resets a work counter
 * held in the plan).  No counterpart in the paper.
 * ------------------------------------------------------------------------- */
typedef struct {
  uint64_t fingerprint;
  size_t bytes;
} ism_attn_plan_info_t;

ism_status_t ism_attn_plan_size(const ism_segments_t* segs, const ism_attn_shape_t* shape, size_t* bytes);
ism_status_t ism_attn_plan_build(const ism_segments_t* segs, const ism_attn_shape_t* shape, void* plan,
                                 size_t plan_bytes, ism_attn_plan_info_t* plan_info, ism_stream_t stream);
ism_status_t ism_attn_fwd_planned(const ism_segments_t* segs, const ism_attn_shape_t* shape, const void* plan,
                                  const ism_attn_plan_info_t* plan_info, const void* q, const void* k,
                                  const void* v, void* o, float* lse, ism_stream_t stream);
ism_status_t ism_attn_bwd_planned(const ism_segments_t* segs, const ism_attn_shape_t* shape, void* plan,
                                  const ism_attn_plan_info_t* plan_info, const void* q, const void* k,
                                  const void* v, const void* o, const float* lse, const void* dout, void* dq,
                                  void* dk, void* dv, void* workspace, size_t workspace_bytes,
                                  ism_stream_t stream);
ism_status_t ism_attn_fwd_rope_planned(const ism_segments_t* segs, const ism_attn_shape_t* shape, const void* plan,
                                       const ism_attn_plan_info_t* plan_info, const void* q, const void* k,
                                       const void* v, const ism_rope_t* rope, void* q_rot, void* k_rot, void* o,
                                       float* lse, ism_stream_t stream);
ism_status_t ism_attn_bwd_rope_planned(const ism_segments_t* segs, const ism_attn_shape_t* shape, void* plan,
                                       const ism_attn_plan_info_t* plan_info, const void* q_rot, const void* k_rot,
                                       const void* v, const void* o, const float* lse, const void* dout,
                                       const ism_rope_t* rope, void* dq, void* dk, void* dv, void* workspace,
                                       size_t workspace_bytes, ism_stream_t stream);

/* ---------------------------------------------------------------------------
 * Append-prefill of a new turn against a reused KV cache (Section 2.3: the
 * history's keys/values C_h are reused, the new chunk's C_q are computed and
 * [C_h; C_q] concatenated).  Valid because no token sees past the end of its
 * own segment (prose after Eq. fj).  One call:
 *   1. writes k_new/v_new into k_cache/v_cache at rows [cache_len[b], cache_len[b]+l_new);
 *   2. computes, for every new token j of sequence b, attention over cache
 *      keys [0, cache_len[b] + kv_end_new[j]) where kv_end_new is Eq. (fj)
 *      applied to the chunk's own segments (all cached keys are visible);
 *   3. advances the device cache_len[b] by l_new (the caller advances its
 *      host mirror).
 * A decode step is l_new = 1 with one ANSWER segment.
 *   q_new [B, l_new, Hq, D], k_new/v_new [B, l_new, Hkv, D] (dtype)
 *   new_seg_end_host/new_seg_type_host [n_new_segs]: chunk-relative segments,
 *     the same for every sequence, last end == l_new, n_new_segs <= 256
 *   k_cache/v_cache [B, cache_capacity, Hkv, D] (dtype, in/out)
 *   cache_len [B] int32 device (in/out), cache_len_host [B] its host mirror;
 *     cache_len_host[b] + l_new <= cache_capacity is required.
 *   o_new [B, l_new, Hq, D] (dtype, written); lse_new [Hq, B, l_new] fp32 or NULL.
 * If a cache ends inside a query segment its old rows would differ from a
 * full pass once the segment grows; the new rows are still exact.
 * The attention reads the cache in tiles of 128 keys from key 0; so that rows
 * past the new end never reach the P V contraction with NaN or Inf bit
 * patterns, the call also sets v_cache rows [cache_len[b] + l_new,
 * round_up(cache_len[b] + l_new, 128)) to zero (within the capacity; the same
 * holds for the paged, e4m3 and RoPE appends).  Nothing else past the new end
 * is read or written.
 * ------------------------------------------------------------------------- */
ism_status_t ism_attn_prefill_append_workspace_size(const ism_attn_shape_t* shape, int32_t batch,
                                                    int32_t l_new, size_t* bytes);
ism_status_t ism_attn_prefill_append(const ism_attn_shape_t* shape, int32_t batch,
                                     const void* q_new, const void* k_new, const void* v_new,
                                     int32_t l_new, const int32_t* new_seg_end_host,
                                     const uint8_t* new_seg_type_host, int32_t n_new_segs,
                                     void* k_cache, void* v_cache, int64_t cache_capacity,
                                     int32_t* cache_len, const int32_t* cache_len_host,
                                     void* o_new, float* lse_new,
                                     void* workspace, size_t workspace_bytes, ism_stream_t stream);

/* ---------------------------------------------------------------------------
 * Append-prefill and decode with e4m3 (fp8) queries and KV caches: the
 * operation of ism_attn_prefill_append on q * q_descale, k * k_descale,
 * v * v_descale, where k_descale / v_descale are the factors of the whole
 * cache (the caller quantises k_new / v_new with them).  shape->dtype must be
 * ISM_E4M3, head_dim 128.  q_new, k_new, v_new and the caches are e4m3;
 * o_new is bf16 [B, l_new, Hq, 128]; lse_new [Hq, B, l_new] fp32 or NULL.
 * The attention runs on the fp8 tensor cores (the kernel of
 * ism_attn_fwd_e4m3; P rounded to e4m3), including single-token steps.
 * Workspace: ism_attn_prefill_append_workspace_size with the same shape.
 * ------------------------------------------------------------------------- */
ism_status_t ism_attn_prefill_append_e4m3(const ism_attn_shape_t* shape, int32_t batch,
                                          const void* q_new, const void* k_new, const void* v_new,
                                          int32_t l_new, const int32_t* new_seg_end_host,
                                          const uint8_t* new_seg_type_host, int32_t n_new_segs,
                                          void* k_cache, void* v_cache, int64_t cache_capacity,
                                          int32_t* cache_len, const int32_t* cache_len_host,
                                          float q_descale, float k_descale, float v_descale,
                                          void* o_new, float* lse_new,
                                          void* workspace, size_t workspace_bytes, ism_stream_t stream);

/* ---------------------------------------------------------------------------
 * Append-prefill and decode against a paged KV cache: the same operation as
 * ism_attn_prefill_append (Section 2.3, Eq. fj on the new chunk, every cached
 * key visible), with the keys and values of sequence b kept in fixed-size
 * pages of a shared pool instead of one contiguous row range.  Key position p
 * of sequence b lives in row  block_table[b * max_pages + p / page_size] *
 * page_size + p % page_size  of the pools.
 *   k_pool/v_pool [num_pages * page_size, Hkv, D] (dtype, in/out)
 *   page_size: a multiple of 128 (a 128-key tile never spans two pages)
 *   block_table [B, max_pages] int32 device, block_table_host its host mirror:
 *     the pages of sequence b, in key order; entries that cover keys
 *     [0, cache_len[b] + l_new) must lie in [0, num_pages), the rest are not read.
 *     Two sequences may share a page only where both only read it.
 *   cache_len / cache_len_host as for ism_attn_prefill_append;
 *     cache_len_host[b] + l_new <= max_pages * page_size is required.
 * The other arguments, the outputs and the workspace
 * (ism_attn_prefill_append_workspace_size) are those of ism_attn_prefill_append.
 * Results equal those of ism_attn_prefill_append on the gathered cache.
 * Errors: ISM_ERR_INVALID_ARG for a page_size that is not a positive multiple
 * of 128, a block-table entry outside the pool, or too few pages.
 * ------------------------------------------------------------------------- */
ism_status_t ism_attn_prefill_append_paged(const ism_attn_shape_t* shape, int32_t batch,
                                           const void* q_new, const void* k_new, const void* v_new,
                                           int32_t l_new, const int32_t* new_seg_end_host,
                                           const uint8_t* new_seg_type_host, int32_t n_new_segs,
                                           void* k_pool, void* v_pool, int32_t num_pages, int32_t page_size,
                                           const int32_t* block_table, const int32_t* block_table_host,
                                           int32_t max_pages, int32_t* cache_len, const int32_t* cache_len_host,
                                           void* o_new, float* lse_new,
                                           void* workspace, size_t workspace_bytes, ism_stream_t stream);

/* ---------------------------------------------------------------------------
 * Append-prefill and decode with rotary position encoding applied on the way
 * into the cache (see ism_rope_t).  Token j of sequence b sits at position
 * p = cache_len[b] + j; its query and its key are rotated there, in fp32, and
 * rounded once to bf16.  The rotated keys are what the cache stores, values
 * are stored unchanged, and the new rows attend exactly as in
 * ism_attn_prefill_append, with the rotated queries.  The rotation runs inside
 * the pass that writes the cache (no extra launch); the rotated queries go to
 * the workspace.
 *   rope->cos / rope->sin: fp32 device tables [rope->rows, D/2], 16-byte
 *     aligned, read only; cache_len_host[b] + l_new <= rope->rows is required.
 *   shape->dtype must be ISM_BF16; head_dim 64 or 128.
 *   q_new / k_new are the unrotated values; every other argument is that of
 *   ism_attn_prefill_append (contiguous caches).
 * Workspace: ism_attn_prefill_append_rope_workspace_size (the append's
 * workspace plus B * l_new * Hq * D bf16 for the rotated queries).
 * Errors: ISM_ERR_INVALID_ARG for a missing or misaligned table, rows too few
 * for the positions written, or a dtype other than ISM_BF16.
 * ------------------------------------------------------------------------- */
ism_status_t ism_attn_prefill_append_rope_workspace_size(const ism_attn_shape_t* shape, int32_t batch,
                                                         int32_t l_new, size_t* bytes);
ism_status_t ism_attn_prefill_append_rope(const ism_attn_shape_t* shape, int32_t batch,
                                          const void* q_new, const void* k_new, const void* v_new,
                                          int32_t l_new, const int32_t* new_seg_end_host,
                                          const uint8_t* new_seg_type_host, int32_t n_new_segs,
                                          void* k_cache, void* v_cache, int64_t cache_capacity,
                                          int32_t* cache_len, const int32_t* cache_len_host,
                                          const ism_rope_t* rope, void* o_new, float* lse_new,
                                          void* workspace, size_t workspace_bytes, ism_stream_t stream);

/* ---------------------------------------------------------------------------
 * The rotary append on the other cache layouts: the operation of
 * ism_attn_prefill_append_rope (Section 2.3 with rotary encoding, see
 * ism_rope_t; token j of sequence b at position cache_len[b] + j) against a
 * paged bf16 cache (the layout and arguments of ism_attn_prefill_append_paged)
 * or an e4m3 cache (those of ism_attn_prefill_append_e4m3).
 *
 * ism_attn_prefill_append_paged_rope: shape->dtype ISM_BF16; results equal
 * those of ism_attn_prefill_append_rope on the gathered cache.
 *
 * ism_attn_prefill_append_e4m3_rope: shape->dtype ISM_E4M3 (the caches and the
 * attention), head_dim 128, but q_new, k_new and v_new are bf16 and
 * UNROTATED: the pass that writes the cache rotates queries and keys in fp32
 * and then quantises, so that the stored keys are rounded once.  Rotated keys
 * are stored as round(k_rot / k_descale), values as round(v / v_descale)
 * (e4m3, round to nearest, saturating at +-448), and the rotated queries
 * round(q_rot / q_descale) go to the workspace; the attention is that of
 * ism_attn_prefill_append_e4m3 with these factors.  A rotation can raise a
 * coordinate up to sqrt(2) times the largest input coordinate; choose the
 * factors with that headroom.
 *
 * Workspace (both): ism_attn_prefill_append_rope_workspace_size with the same
 * shape.  Errors as the append they extend, plus ISM_ERR_INVALID_ARG for a
 * NULL rope, a missing or misaligned table, or tables shorter than the
 * positions written.
 * ------------------------------------------------------------------------- */
ism_status_t ism_attn_prefill_append_paged_rope(const ism_attn_shape_t* shape, int32_t batch,
                                                const void* q_new, const void* k_new, const void* v_new,
                                                int32_t l_new, const int32_t* new_seg_end_host,
                                                const uint8_t* new_seg_type_host, int32_t n_new_segs,
                                                void* k_pool, void* v_pool, int32_t num_pages, int32_t page_size,
                                                const int32_t* block_table, const int32_t* block_table_host,
                                                int32_t max_pages, int32_t* cache_len, const int32_t* cache_len_host,
                                                const ism_rope_t* rope, void* o_new, float* lse_new,
                                                void* workspace, size_t workspace_bytes, ism_stream_t stream);
ism_status_t ism_attn_prefill_append_e4m3_rope(const ism_attn_shape_t* shape, int32_t batch,
                                               const void* q_new, const void* k_new, const void* v_new,
                                               int32_t l_new, const int32_t* new_seg_end_host,
                                               const uint8_t* new_seg_type_host, int32_t n_new_segs,
                                               void* k_cache, void* v_cache, int64_t cache_capacity,
                                               int32_t* cache_len, const int32_t* cache_len_host,
                                               float q_descale, float k_descale, float v_descale,
                                               const ism_rope_t* rope, void* o_new, float* lse_new,
                                               void* workspace, size_t workspace_bytes, ism_stream_t stream);

/* ---------------------------------------------------------------------------
 * Status and diagnostics.
 * ------------------------------------------------------------------------- */

/* Synchronises `stream`, then reads and clears the current device's status
 * word.  Returns ISM_ERR_TIMEOUT if any kernel gave up a bounded wait since
 * the last check (the kernel exits early and its outputs are undefined),
 * ISM_ERR_CUDA on a CUDA error, ISM_OK otherwise. */
ism_status_t ism_check_status(ism_stream_t stream);

/* Test hook for the bounded-wait machinery: launches one kernel that waits on
 * a barrier nothing ever signals, with a spin limit of `spin_limit` polls,
 * gives up, records ISM_ERR_TIMEOUT in the status word and returns.  Lets a
 * test observe the timeout path without hanging a GPU. */
ism_status_t ism_debug_timeout_probe(uint32_t spin_limit, ism_stream_t stream);

/* Measurement hooks (no counterpart in the paper).
 * ism_set_kernel_timer: while set, every launch of kernel kind `kernel_id`
 * issued by this host thread is bracketed by cudaEventRecord(start_event)
 * and cudaEventRecord(stop_event) on the launch's stream (the events are
 * cudaEvent_t handles owned by the caller; NULL clears the timer).
 * ism_kernel_launches: number of kernels this library has launched in the
 * process so far (all threads). */
enum {
  ISM_KERNEL_FWD = 1,        /* one-pass forward (and append-prefill over a chunk) */
  ISM_KERNEL_BWD_DKDV = 2,   /* backward dK/dV */
  ISM_KERNEL_BWD_DQ = 3,     /* backward dQ */
  ISM_KERNEL_BWD_PRE = 4,    /* backward preprocessing (Delta) */
  ISM_KERNEL_DECODE = 5,     /* single-token append (split-KV + merge) */
  ISM_KERNEL_META = 6,       /* tile map / work lists */
  ISM_KERNEL_ROPE = 7        /* rotary encoding pass of the one-pass forward (and CUDA-core backward) */
};
ism_status_t ism_set_kernel_timer(int32_t kernel_id, void* start_event, void* stop_event);
uint64_t ism_kernel_launches(void);

/* Debug and tuning switches (no counterpart in the paper).  The library reads
 * its ISM_* environment variables once, when it is loaded, so that no call
 * spends host time on them.  ism_debug_reload_env reads them again (for tests
 * that change a switch in a running process); it must not run concurrently
 * with other calls of the library. */
void ism_debug_reload_env(void);

/* Diagnostic of the tensor-core building blocks (no counterpart in the
 * paper): one 128x128x128 bf16 tile product on tcgen05 with fp32 result.
 *   a [128,128] bf16 row-major (M x K); c [128,128] fp32 row-major (written)
 *   mode 0/2/4: b [128,128] is N x K and c = a * b^T
 *   mode 1/3/5: b [128,128] is K x N and c = a * b
 *   modes 0/1 stage the operands with plain stores, 2/3 with TMA, 4/5 put
 *   a in tensor memory (the A-from-TMEM form of the MMA)
 *   mode 6: a [128,128] is K x M and b is K x N (both MN-major), c = a^T * b
 *   mode 7: as mode 6, a staged in the 8-interleaved layout without swizzle.
 *   mode 8 + m: as mode m with the eight k-steps issued by one warp through
 *   the batched form the attention kernels use (one election, descriptors
 *   advanced by fixed offsets). */
ism_status_t ism_debug_mma_tile(const void* a, const void* b, float* c, int32_t mode, ism_stream_t stream);
/* The same for e4m3 operands (kind::f8f6f4, K = 32 a step), the layouts of
 * the e4m3 forward: a [128,128] e4m3 row-major (M x K), c fp32 [128,128].
 *   mode 0: b [128,128] is N x K, c = a * b^T (both K-major in shared memory)
 *   mode 1: b is K x N (MN-major), c = a * b
 *   mode 2: as mode 1 with a in tensor memory (four e4m3 a column). */
ism_status_t ism_debug_mma_tile_e4m3(const void* a, const void* b, float* c, int32_t mode, ism_stream_t stream);

const char* ism_status_string(ism_status_t status);
/* Human-readable detail of the last failing call on this host thread. */
const char* ism_last_error(void);
/* 1 if the library was built with the sm_103a tensor-core kernels. */
int32_t ism_has_tensor_cores(void);

#ifdef __cplusplus
}
#endif
#endif /* ISM_H_ */
