// Host side of the C ABI: argument validation on the host mirrors, workspace
// layout, kernel dispatch and the device status word.
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <atomic>
#include <mutex>
#include <string>
#include <vector>

#include "ism_internal.cuh"

namespace ism {
namespace {

thread_local std::string g_last_error;

ism_status_t fail(ism_status_t st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return st;
}

ism_status_t cuda_fail(cudaError_t e, const char* where) {
  return fail(ISM_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
}

#define ISM_TRY_CUDA(expr, where)                 \
  do {                                            \
    cudaError_t e_ = (expr);                      \
    if (e_ != cudaSuccess) return cuda_fail(e_, where); \
  } while (0)

// One status word per device; the library's only persistent device state.
__device__ uint32_t g_status_word;

std::mutex g_status_mu;
std::vector<uint32_t*> g_status_ptr;

ism_status_t status_ptr(uint32_t** out) {
  int dev = 0;
  ISM_TRY_CUDA(cudaGetDevice(&dev), "cudaGetDevice");
  std::lock_guard<std::mutex> lk(g_status_mu);
  if ((int)g_status_ptr.size() <= dev) g_status_ptr.resize(dev + 1, nullptr);
  if (!g_status_ptr[dev]) {
    void* p = nullptr;
    ISM_TRY_CUDA(cudaGetSymbolAddress(&p, g_status_word), "cudaGetSymbolAddress(status)");
    g_status_ptr[dev] = static_cast<uint32_t*>(p);
  }
  *out = g_status_ptr[dev];
  return ISM_OK;
}

// ---------------------------------------------------------------- measurement

constexpr int kTimerSlots = 8;
thread_local cudaEvent_t g_timer_start[kTimerSlots];
thread_local cudaEvent_t g_timer_stop[kTimerSlots];
std::atomic<uint64_t> g_launches{0};

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

constexpr int kTile = 128;       // q/k tile rows of the attention kernels and their work lists
constexpr int kMaxSplits = 64;   // split-KV chunks per (sequence, KV head) for decode

struct SegInfo {
  int64_t total_tokens = 0;
  int64_t max_len = 0;
};

ism_status_t check_segments(const ism_segments_t* s, SegInfo* info) {
  if (!s) return fail(ISM_ERR_INVALID_ARG, "segments is NULL");
  if (s->num_seqs < 0 || s->num_segs < 0) return fail(ISM_ERR_INVALID_ARG, "negative counts");
  if (s->num_seqs > kMaxSeqs) return fail(ISM_ERR_UNSUPPORTED, "num_seqs %d > %d", s->num_seqs, kMaxSeqs);
  if (!s->cu_seqlens_host || !s->cu_segs_host || !s->cu_seqlens || !s->cu_segs)
    return fail(ISM_ERR_INVALID_ARG, "cu_seqlens / cu_segs (device and host) must be non-NULL");
  if (s->num_segs > 0 && (!s->seg_end || !s->seg_end_host || !s->seg_type || !s->seg_type_host))
    return fail(ISM_ERR_INVALID_ARG, "seg_end / seg_type (device and host) must be non-NULL");
  const int32_t* cs = s->cu_seqlens_host;
  const int32_t* cg = s->cu_segs_host;
  if (cs[0] != 0 || cg[0] != 0) return fail(ISM_ERR_INVALID_ARG, "cu_seqlens[0] and cu_segs[0] must be 0");
  if (cg[s->num_seqs] != s->num_segs)
    return fail(ISM_ERR_INVALID_ARG, "cu_segs[num_seqs]=%d != num_segs=%d", cg[s->num_seqs], s->num_segs);
  int64_t max_len = 0;
  for (int b = 0; b < s->num_seqs; ++b) {
    int64_t L = (int64_t)cs[b + 1] - cs[b];
    if (L < 0) return fail(ISM_ERR_INVALID_ARG, "cu_seqlens decreases at sequence %d", b);
    if (cg[b + 1] < cg[b]) return fail(ISM_ERR_INVALID_ARG, "cu_segs decreases at sequence %d", b);
    int32_t prev = 0;
    for (int i = cg[b]; i < cg[b + 1]; ++i) {
      int32_t e = s->seg_end_host[i];
      if (e < prev) return fail(ISM_ERR_INVALID_ARG, "seq %d: seg_end not non-decreasing at segment %d", b, i);
      if (s->seg_type_host[i] > 1) return fail(ISM_ERR_INVALID_ARG, "segment %d: type %d is not QUERY/ANSWER", i,
                                               (int)s->seg_type_host[i]);
      prev = e;
    }
    if (prev != L)
      return fail(ISM_ERR_INVALID_ARG, "seq %d: segments end at %d but the sequence has %lld tokens", b, prev,
                  (long long)L);
    if (L > max_len) max_len = L;
  }
  info->total_tokens = cs[s->num_seqs];
  info->max_len = max_len;
  return ISM_OK;
}

ism_status_t check_shape(const ism_attn_shape_t* sh, bool allow_e4m3 = false) {
  if (!sh) return fail(ISM_ERR_INVALID_ARG, "shape is NULL");
  if (sh->num_heads_q <= 0 || sh->num_heads_kv <= 0) return fail(ISM_ERR_INVALID_ARG, "head counts must be > 0");
  if (sh->num_heads_q % sh->num_heads_kv)
    return fail(ISM_ERR_INVALID_ARG, "num_heads_q (%d) is not a multiple of num_heads_kv (%d)", sh->num_heads_q,
                sh->num_heads_kv);
  if (sh->head_dim != 64 && sh->head_dim != 128)
    return fail(ISM_ERR_UNSUPPORTED, "head_dim %d (supported: 64, 128)", sh->head_dim);
  if (sh->dtype == ISM_E4M3) {
    if (!allow_e4m3) return fail(ISM_ERR_UNSUPPORTED, "e4m3 inputs only in ism_attn_fwd_e4m3");
    if (sh->head_dim != 128) return fail(ISM_ERR_UNSUPPORTED, "e4m3 needs head_dim 128");
  } else if (sh->dtype != ISM_BF16 && sh->dtype != ISM_FP32) {
    return fail(ISM_ERR_UNSUPPORTED, "dtype %d", sh->dtype);
  }
  if (!(sh->softmax_scale > 0.f) || sh->softmax_scale != sh->softmax_scale)
    return fail(ISM_ERR_INVALID_ARG, "softmax_scale must be a positive number");
  return ISM_OK;
}

SegsDev dev_view(const ism_segments_t* s) {
  SegsDev d;
  d.num_seqs = s->num_seqs;
  d.num_segs = s->num_segs;
  d.cu_seqlens = s->cu_seqlens;
  d.cu_segs = s->cu_segs;
  d.seg_end = s->seg_end;
  d.seg_type = s->seg_type;
  return d;
}

// Bump allocator over a caller-provided workspace (256-byte aligned pieces).
struct Carve {
  uintptr_t base;
  size_t off = 0;
  explicit Carve(void* p) : base(reinterpret_cast<uintptr_t>(p)) {}
  template <typename T>
  T* take(int64_t n) {
    off = (off + 255) & ~size_t(255);
    T* p = reinterpret_cast<T*>(base + off);
    off += sizeof(T) * (size_t)(n > 0 ? n : 0);
    return p;
  }
};

struct Counts {
  int64_t nq = 0, nk = 0, ntiles = 0;
  int64_t npairs = 0;  // q-tile pairs (neighbouring q-tiles of a sequence, the last one may be alone)
  int max_cost = 0;
};

Counts count_tiles(const ism_segments_t* s, int bm, int bn) {
  Counts c;
  for (int b = 0; b < s->num_seqs; ++b) {
    int64_t L = (int64_t)s->cu_seqlens_host[b + 1] - s->cu_seqlens_host[b];
    int64_t nq = (L + bm - 1) / bm, nk = (L + bn - 1) / bn;
    c.nq += nq;
    c.nk += nk;
    c.npairs += (nq + 1) / 2;
    c.ntiles += nq * nk;
    int mc = (int)(nq > nk ? nq : nk);
    if (mc > c.max_cost) c.max_cost = mc;
  }
  return c;
}

// Visible (k-tile, q-tile) pairs over all sequences at kTile x kTile tiles:
// k-tile c pairs with every q-tile from the one holding the first row whose
// kv_end exceeds c*kTile to the last.  Under Eq. fj that row is the start of
// the first segment ending after c*kTile when it is a query segment, else
// max(segment start, c*kTile).  Host walk over segments and k-tiles.
int64_t count_pairs(const ism_segments_t* s) {
  int64_t pairs = 0;
  for (int b = 0; b < s->num_seqs; ++b) {
    const int32_t L = s->cu_seqlens_host[b + 1] - s->cu_seqlens_host[b];
    const int32_t nt = (L + kTile - 1) / kTile;
    int32_t seg = s->cu_segs_host[b], start = 0;
    const int32_t seg1 = s->cu_segs_host[b + 1];
    for (int32_t c = 0; c < nt; ++c) {
      const int32_t x = c * kTile;
      while (seg < seg1 && s->seg_end_host[seg] <= x) start = s->seg_end_host[seg++];
      if (seg == seg1) break;
      const int32_t j = s->seg_type_host[seg] == ISM_SEG_QUERY ? start : (x > start ? x : start);
      pairs += nt - j / kTile;
    }
  }
  return pairs;
}

// Workspace of the one-pass forward/backward.  ds_slots > 0 adds the
// stored-dS backward's pair offsets and bf16 dS^T tiles (32 KiB a slot).
struct PassLayout {
  int32_t* kv_end;
  Tile *qtiles, *ktiles;
  int32_t *q_order, *k_order;
  float* delta;
  int32_t* kpair_off;
  void* ds;
  int32_t* pair_order;
  int32_t* kp_order;  // k-tile pairs in cost order (backward only)
  int32_t* counters;  // work counters of the persistent backward kernels (backward only)
  size_t bytes;
};
constexpr int kPassCounters = 2;

PassLayout pass_layout(void* ws, const ism_segments_t* s, const Counts& c, int64_t T, int hq, bool bwd,
                       int64_t ds_slots = 0, bool tile_pairs = false) {
  Carve cv(ws);
  PassLayout L;
  L.kv_end = cv.take<int32_t>(T);
  L.qtiles = cv.take<Tile>(c.nq);
  L.q_order = cv.take<int32_t>(c.nq);
  L.ktiles = bwd ? cv.take<Tile>(c.nk) : nullptr;
  L.k_order = bwd ? cv.take<int32_t>(c.nk) : nullptr;
  L.delta = bwd ? cv.take<float>((int64_t)hq * T) : nullptr;
  L.kpair_off = ds_slots > 0 ? cv.take<int32_t>(c.nk) : nullptr;
  L.ds = ds_slots > 0 ? static_cast<void*>(cv.take<uint16_t>(ds_slots * kTile * kTile)) : nullptr;
  L.pair_order = tile_pairs ? cv.take<int32_t>(c.npairs) : nullptr;
  L.kp_order = bwd ? cv.take<int32_t>(c.npairs) : nullptr;  // k-tile pairs number as q-tile pairs here
  L.counters = bwd ? cv.take<int32_t>(kPassCounters) : nullptr;
  L.bytes = ((cv.off + 255) & ~size_t(255)) + 256;
  return L;
}

// Device layout of a plan (ism_attn_plan_build): the metadata of both
// passes for one batch of segments and head counts, without the backward's
// Delta and dS tiles, which stay in the backward's workspace.
bool fwd_tile_pairs(const ism_attn_shape_t* sh);
PassLayout plan_layout(void* plan, const Counts& c, int64_t T, bool tile_pairs) {
  Carve cv(plan);
  PassLayout L{};
  L.kv_end = cv.take<int32_t>(T);
  L.qtiles = cv.take<Tile>(c.nq);
  L.q_order = cv.take<int32_t>(c.nq);
  L.ktiles = cv.take<Tile>(c.nk);
  L.k_order = cv.take<int32_t>(c.nk);
  L.kpair_off = cv.take<int32_t>(c.nk);
  L.pair_order = tile_pairs ? cv.take<int32_t>(c.npairs) : nullptr;
  L.counters = cv.take<int32_t>(kPassCounters);
  L.bytes = ((cv.off + 255) & ~size_t(255)) + 256;
  return L;
}

// What a plan was built for: FNV-1a over the segments' host arrays, the head
// counts and whether the forward pairs query tiles (the work lists differ).
uint64_t plan_fingerprint(const ism_segments_t* s, const ism_attn_shape_t* sh, bool tile_pairs) {
  uint64_t h = 1469598103934665603ull;
  auto mix = [&](const void* p, size_t n) {
    const unsigned char* b = static_cast<const unsigned char*>(p);
    for (size_t i = 0; i < n; ++i) h = (h ^ b[i]) * 1099511628211ull;
  };
  const int32_t head[4] = {s->num_seqs, s->num_segs, sh->num_heads_q, sh->num_heads_kv};
  mix(head, sizeof(head));
  const uint8_t tp = tile_pairs ? 1 : 0;
  mix(&tp, 1);
  mix(s->cu_seqlens_host, sizeof(int32_t) * (size_t)(s->num_seqs + 1));
  mix(s->cu_segs_host, sizeof(int32_t) * (size_t)(s->num_seqs + 1));
  if (s->num_segs > 0) {
    mix(s->seg_end_host, sizeof(int32_t) * (size_t)s->num_segs);
    mix(s->seg_type_host, (size_t)s->num_segs);
  }
  return h;
}

bool force_cuda_cores() { return knobs().force_cuda_cores; }

uint32_t tc_flags() { return knobs().drain_tmem_reuse ? kFlagDrainTmemReuse : 0u; }

bool use_tc(const ism_attn_shape_t* sh) {
  return sh->dtype == ISM_BF16 && sh->head_dim == 128 && tc_available() && !force_cuda_cores();
}
bool use_tc_bwd(const ism_attn_shape_t* sh) { return use_tc(sh) && tc_bwd_available(); }

// The tensor-core forward pairs two query heads of a KV head per CTA; with an
// odd number of query heads per KV head it pairs neighbouring query tiles of
// one head instead, from a work list the metadata pass builds.
bool fwd_tile_pairs(const ism_attn_shape_t* sh) {
  if ((sh->num_heads_q / sh->num_heads_kv) % 2 == 0) return false;
  if (sh->dtype == ISM_E4M3) return true;  // the e4m3 forward runs only the paired kernel
  if (!use_tc(sh)) return false;
  return !knobs().fwd_one_head;
}

// dS tile slots of the stored-dS backward (pairs x query heads), or 0 where
// that path does not apply: CUDA-core backward, ISM_BWD_RECOMPUTE_DQ=1, or
// more pairs than the 32-bit pair offsets hold.
int64_t stored_ds_slots(const ism_segments_t* s, const ism_attn_shape_t* sh) {
  if (!use_tc_bwd(sh)) return 0;
  if (knobs().bwd_recompute_dq) return 0;
  const int64_t pairs = count_pairs(s);
  if (pairs >= (int64_t(1) << 31)) return 0;
  return pairs * sh->num_heads_q;
}

ism_status_t check_ws(void* ws, size_t have, size_t need) {
  if (have < need) return fail(ISM_ERR_WORKSPACE, "workspace of %zu bytes, %zu required", have, need);
  if (need && !ws) return fail(ISM_ERR_WORKSPACE, "workspace is NULL");
  if (reinterpret_cast<uintptr_t>(ws) & 255u) return fail(ISM_ERR_WORKSPACE, "workspace must be 256-byte aligned");
  return ISM_OK;
}

ism_status_t build_pass_meta(const ism_segments_t* s, const Counts& c, const PassLayout& L, bool bwd,
                             cudaStream_t st) {
  SegsDev d = dev_view(s);
  timer_begin(ISM_KERNEL_META, st);
  ISM_TRY_CUDA(launch_pass_meta(d, L.kv_end, kTile, kTile, c.nq, bwd ? c.nk : 0, L.qtiles, bwd ? L.ktiles : nullptr,
                                c.max_cost, L.q_order, bwd ? L.k_order : nullptr, L.pair_order, L.kpair_off,
                                L.counters, L.counters ? kPassCounters : 0, st,
                                knobs().dkdv_pair ? L.kp_order : nullptr),
               "metadata launch");
  timer_end(ISM_KERNEL_META, st);
  count_launch(1);
  return ISM_OK;
}

}  // namespace

void timer_begin(int id, cudaStream_t st) {
  if (id > 0 && id < kTimerSlots && g_timer_start[id]) cudaEventRecord(g_timer_start[id], st);
}
void timer_end(int id, cudaStream_t st) {
  if (id > 0 && id < kTimerSlots && g_timer_stop[id]) cudaEventRecord(g_timer_stop[id], st);
}
void count_launch(int n) { g_launches.fetch_add((uint64_t)n, std::memory_order_relaxed); }
void set_error(const char* msg) { g_last_error = msg; }

namespace {
bool env_on(const char* name) {
  const char* e = getenv(name);
  return e && e[0] == '1';
}
int64_t env_int(const char* name, int64_t unset) {
  const char* e = getenv(name);
  return (e && e[0]) ? atoll(e) : unset;
}
Knobs read_knobs() {
  Knobs k;
  k.force_cuda_cores = env_on("ISM_FORCE_CUDA_CORES");
  k.drain_tmem_reuse = env_on("ISM_DRAIN_TMEM_REUSE");
  k.fwd_one_head = env_on("ISM_FWD_ONE_HEAD");
  k.bwd_recompute_dq = env_on("ISM_BWD_RECOMPUTE_DQ");
  k.decode_no_tma = env_on("ISM_DECODE_NO_TMA");
  k.decode_no_tc = env_on("ISM_DECODE_NO_TC");
  const int64_t split = env_int("ISM_PREFILL_SPLIT", -1);
  k.prefill_split = split < 0 ? -1 : split;
  const int64_t g1 = env_int("ISM_DKDV_GRID", 0), g2 = env_int("ISM_DQ_GRID", 0);
  k.dkdv_grid = g1 > 0 && g1 < (1 << 20) ? (int32_t)g1 : 0;
  k.dq_grid = g2 > 0 && g2 < (1 << 20) ? (int32_t)g2 : 0;
  k.dkdv_pair = env_on("ISM_DKDV_PAIR");
  return k;
}
Knobs g_knobs = read_knobs();  // read when the library is loaded

std::mutex g_sm_mu;
std::vector<int> g_sm_count;
}  // namespace

const Knobs& knobs() { return g_knobs; }
void reload_knobs() { g_knobs = read_knobs(); }

int sm_count() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 152;
  std::lock_guard<std::mutex> lk(g_sm_mu);
  if ((int)g_sm_count.size() <= dev) g_sm_count.resize(dev + 1, 0);
  if (!g_sm_count[dev]) {
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0) return 152;
    g_sm_count[dev] = sms;
  }
  return g_sm_count[dev];
}

}  // namespace ism

using namespace ism;

extern "C" {

const char* ism_status_string(ism_status_t s) {
  switch (s) {
    case ISM_OK: return "ISM_OK";
    case ISM_ERR_INVALID_ARG: return "ISM_ERR_INVALID_ARG";
    case ISM_ERR_UNSUPPORTED: return "ISM_ERR_UNSUPPORTED";
    case ISM_ERR_CUDA: return "ISM_ERR_CUDA";
    case ISM_ERR_TIMEOUT: return "ISM_ERR_TIMEOUT";
    case ISM_ERR_WORKSPACE: return "ISM_ERR_WORKSPACE";
  }
  return "ISM_ERR_UNKNOWN";
}

const char* ism_last_error(void) { return g_last_error.c_str(); }

int32_t ism_has_tensor_cores(void) { return tc_available() ? 1 : 0; }

ism_status_t ism_set_kernel_timer(int32_t kernel_id, void* start_event, void* stop_event) {
  if (kernel_id <= 0 || kernel_id >= kTimerSlots) return fail(ISM_ERR_INVALID_ARG, "kernel_id %d", kernel_id);
  if ((start_event == nullptr) != (stop_event == nullptr))
    return fail(ISM_ERR_INVALID_ARG, "give both events or neither");
  g_timer_start[kernel_id] = static_cast<cudaEvent_t>(start_event);
  g_timer_stop[kernel_id] = static_cast<cudaEvent_t>(stop_event);
  return ISM_OK;
}

uint64_t ism_kernel_launches(void) { return g_launches.load(); }

void ism_debug_reload_env(void) { reload_knobs(); }

ism_status_t ism_tile_map_size(const ism_segments_t* segs, int32_t bm, int32_t bn, int64_t* n_tiles,
                               int64_t* n_qtiles, int64_t* n_ktiles) {
  SegInfo info;
  ism_status_t r = check_segments(segs, &info);
  if (r != ISM_OK) return r;
  if (bm < 16 || bn < 16 || bm > 256 || bn > 256 || bm % 16 || bn % 16)
    return fail(ISM_ERR_UNSUPPORTED, "tile sizes must be multiples of 16 in [16, 256]");
  Counts c = count_tiles(segs, bm, bn);
  if (n_tiles) *n_tiles = c.ntiles;
  if (n_qtiles) *n_qtiles = c.nq;
  if (n_ktiles) *n_ktiles = c.nk;
  return ISM_OK;
}

ism_status_t ism_build_tile_map(const ism_segments_t* segs, int32_t bm, int32_t bn, uint8_t* tile_class,
                                int32_t* kt_full_end, int32_t* kt_end, int32_t* qt_begin, int32_t* kv_end,
                                ism_stream_t stream) {
  int64_t nt, nq, nk;
  ism_status_t r = ism_tile_map_size(segs, bm, bn, &nt, &nq, &nk);
  if (r != ISM_OK) return r;
  if (segs->cu_seqlens_host[segs->num_seqs] == 0) return ISM_OK;
  if (!kv_end) return fail(ISM_ERR_INVALID_ARG, "kv_end output is required (the tile classes are derived from it)");
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  SegsDev d = dev_view(segs);
  ISM_TRY_CUDA(launch_kv_end(d, kv_end, st), "kv_end launch");
  if (tile_class || kt_full_end || kt_end || qt_begin)
    ISM_TRY_CUDA(launch_tiles(d, bm, bn, kv_end, nq, qt_begin ? nk : 0, nullptr, nullptr, tile_class, kt_full_end,
                              kt_end, qt_begin, st),
                 "tiles launch");
  return ISM_OK;
}

ism_status_t ism_attn_fwd_workspace_size(const ism_segments_t* segs, const ism_attn_shape_t* shape,
                                         size_t* bytes) {
  SegInfo info;
  ism_status_t r = check_segments(segs, &info);
  if (r != ISM_OK) return r;
  if ((r = check_shape(shape, true)) != ISM_OK) return r;
  if (!bytes) return fail(ISM_ERR_INVALID_ARG, "bytes is NULL");
  Counts c = count_tiles(segs, kTile, kTile);
  *bytes = pass_layout(nullptr, segs, c, info.total_tokens, shape->num_heads_q, false, 0, fwd_tile_pairs(shape)).bytes;
  return ISM_OK;
}

ism_status_t ism_attn_bwd_workspace_size(const ism_segments_t* segs, const ism_attn_shape_t* shape,
                                         size_t* bytes) {
  SegInfo info;
  ism_status_t r = check_segments(segs, &info);
  if (r != ISM_OK) return r;
  if ((r = check_shape(shape)) != ISM_OK) return r;
  if (!bytes) return fail(ISM_ERR_INVALID_ARG, "bytes is NULL");
  Counts c = count_tiles(segs, kTile, kTile);
  *bytes = pass_layout(nullptr, segs, c, info.total_tokens, shape->num_heads_q, true, stored_ds_slots(segs, shape))
               .bytes;
  return ISM_OK;
}

ism_status_t ism_attn_bwd_workspace_size_min(const ism_segments_t* segs, const ism_attn_shape_t* shape,
                                             size_t* bytes) {
  SegInfo info;
  ism_status_t r = check_segments(segs, &info);
  if (r != ISM_OK) return r;
  if ((r = check_shape(shape)) != ISM_OK) return r;
  if (!bytes) return fail(ISM_ERR_INVALID_ARG, "bytes is NULL");
  Counts c = count_tiles(segs, kTile, kTile);
  *bytes = pass_layout(nullptr, segs, c, info.total_tokens, shape->num_heads_q, true).bytes;
  return ISM_OK;
}

}  // extern "C"

namespace {

// Checks the rotary tables of a one-pass call: present, aligned, covering
// every position of the batch (the longest sequence), for bf16 / fp32 inputs.
ism_status_t check_rope_pass(const ism_rope_t* rope, const ism_attn_shape_t* shape, const SegInfo& info) {
  if (!rope) return fail(ISM_ERR_INVALID_ARG, "rope is NULL");
  if (shape->dtype != ISM_BF16 && shape->dtype != ISM_FP32)
    return fail(ISM_ERR_INVALID_ARG, "rotary encoding on the one-pass path needs bf16 or fp32 inputs");
  if (!rope->cos || !rope->sin || !aligned16(rope->cos) || !aligned16(rope->sin))
    return fail(ISM_ERR_INVALID_ARG, "rope tables must be non-NULL and 16-byte aligned");
  if (info.max_len > rope->rows)
    return fail(ISM_ERR_INVALID_ARG, "rope tables cover %d positions, the longest sequence has %lld tokens", rope->rows,
                (long long)info.max_len);
  return ISM_OK;
}

// The one-pass forward for bf16 / fp32 (ism_attn_fwd) and e4m3 inputs
// (ism_attn_fwd_e4m3; qk_descale = q_descale * k_descale); with rope set,
// q and k are first rotated into q_rot / k_rot and the attention reads those.
ism_status_t fwd_impl(const ism_segments_t* segs, const ism_attn_shape_t* shape, const void* q, const void* k,
                      const void* v, void* o, float* lse, void* workspace, size_t workspace_bytes, ism_stream_t stream,
                      float qk_descale, float v_descale, const ism_rope_t* rope = nullptr, void* q_rot = nullptr,
                      void* k_rot = nullptr, const PassLayout* pre = nullptr) {
  SegInfo info;
  ism_status_t r = check_segments(segs, &info);
  if (r != ISM_OK) return r;
  const bool e4m3 = shape && shape->dtype == ISM_E4M3;
  if ((r = check_shape(shape, e4m3)) != ISM_OK) return r;
  if (e4m3 && !tc_available()) return fail(ISM_ERR_UNSUPPORTED, "e4m3 forward needs the sm_103 tensor cores");
  if (rope && (r = check_rope_pass(rope, shape, info)) != ISM_OK) return r;
  if (info.total_tokens == 0) return ISM_OK;
  if (!q || !k || !v || !o) return fail(ISM_ERR_INVALID_ARG, "q, k, v, o must be non-NULL");
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o) || (lse && !aligned16(lse)))
    return fail(ISM_ERR_INVALID_ARG, "tensors must be 16-byte aligned");
  if (rope && (!q_rot || !k_rot || !aligned16(q_rot) || !aligned16(k_rot)))
    return fail(ISM_ERR_INVALID_ARG, "q_rot and k_rot must be non-NULL and 16-byte aligned");
  Counts c = count_tiles(segs, kTile, kTile);
  // pre: the metadata of a plan (ism_attn_plan_build), already on the device
  PassLayout L = pre ? *pre
                     : pass_layout(workspace, segs, c, info.total_tokens, shape->num_heads_q, false, 0,
                                   fwd_tile_pairs(shape));
  if (!pre && (r = check_ws(workspace, workspace_bytes, L.bytes)) != ISM_OK) return r;
  uint32_t* status;
  if ((r = status_ptr(&status)) != ISM_OK) return r;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (rope) {
    timer_begin(ISM_KERNEL_ROPE, st);
    ISM_TRY_CUDA(launch_rope_rows(segs->cu_seqlens, segs->num_seqs, info.total_tokens, shape->num_heads_q,
                                  shape->num_heads_kv, shape->head_dim, shape->dtype, q, k, q_rot, k_rot, rope->cos,
                                  rope->sin, 1.f, st),
                 "rope launch");
    timer_end(ISM_KERNEL_ROPE, st);
    count_launch(1);
    q = q_rot;
    k = k_rot;
  }
  if (!pre && (r = build_pass_meta(segs, c, L, false, st)) != ISM_OK) return r;

  AttnArgs a{};
  a.q = q; a.k = k; a.v = v; a.out = o; a.lse = lse;
  a.hq = shape->num_heads_q; a.hkv = shape->num_heads_kv; a.d = shape->head_dim; a.dtype = shape->dtype;
  a.q_rows = info.total_tokens; a.scale = shape->softmax_scale;
  a.qk_descale = qk_descale; a.v_descale = v_descale;
  a.kv_end = L.kv_end; a.qtiles = L.qtiles; a.q_order = L.q_order; a.nq = c.nq;
  a.pair_order = L.pair_order; a.npairs = L.pair_order ? c.npairs : 0;
  a.status = status;
  a.flags = tc_flags();
  timer_begin(ISM_KERNEL_FWD, st);
  if (use_tc(shape) || e4m3) {
    ISM_TRY_CUDA(launch_tc_fwd(a, info.total_tokens, st), "tensor-core forward launch");
  } else {
    ISM_TRY_CUDA(launch_simt_fwd(a, st), "forward launch");
  }
  timer_end(ISM_KERNEL_FWD, st);
  count_launch(1);
  return ISM_OK;
}

bool valid_descales(float q_descale, float k_descale, float v_descale) {
  const float ds[3] = {q_descale, k_descale, v_descale};
  for (float x : ds)
    if (!(x > 0.f) || x > 3.0e38f) return false;
  return true;
}

}  // namespace

extern "C" {

ism_status_t ism_attn_fwd(const ism_segments_t* segs, const ism_attn_shape_t* shape, const void* q,
                          const void* k, const void* v, void* o, float* lse, void* workspace,
                          size_t workspace_bytes, ism_stream_t stream) {
  if (shape && shape->dtype == ISM_E4M3)
    return fail(ISM_ERR_UNSUPPORTED, "e4m3 inputs only in ism_attn_fwd_e4m3");
  return fwd_impl(segs, shape, q, k, v, o, lse, workspace, workspace_bytes, stream, 1.f, 1.f);
}

ism_status_t ism_attn_fwd_e4m3(const ism_segments_t* segs, const ism_attn_shape_t* shape, const void* q,
                               const void* k, const void* v, float q_descale, float k_descale, float v_descale,
                               void* o, float* lse, void* workspace, size_t workspace_bytes, ism_stream_t stream) {
  if (!shape || shape->dtype != ISM_E4M3)
    return fail(ISM_ERR_INVALID_ARG, "ism_attn_fwd_e4m3 needs shape->dtype ISM_E4M3");
  if (!valid_descales(q_descale, k_descale, v_descale))
    return fail(ISM_ERR_INVALID_ARG, "descales must be positive finite numbers");
  return fwd_impl(segs, shape, q, k, v, o, lse, workspace, workspace_bytes, stream, q_descale * k_descale, v_descale);
}

ism_status_t ism_attn_fwd_rope(const ism_segments_t* segs, const ism_attn_shape_t* shape, const void* q,
                               const void* k, const void* v, const ism_rope_t* rope, void* q_rot, void* k_rot,
                               void* o, float* lse, void* workspace, size_t workspace_bytes, ism_stream_t stream) {
  if (shape && shape->dtype == ISM_E4M3)
    return fail(ISM_ERR_INVALID_ARG, "rotary encoding on the one-pass path needs bf16 or fp32 inputs");
  if (!rope) return fail(ISM_ERR_INVALID_ARG, "rope is NULL");
  return fwd_impl(segs, shape, q, k, v, o, lse, workspace, workspace_bytes, stream, 1.f, 1.f, rope, q_rot, k_rot);
}

}  // extern "C"

namespace {

ism_status_t bwd_impl(const ism_segments_t* segs, const ism_attn_shape_t* shape, const void* q, const void* k,
                      const void* v, const void* o, const float* lse, const void* dout, void* dq, void* dk, void* dv,
                      void* workspace, size_t workspace_bytes, ism_stream_t stream, const ism_rope_t* rope,
                      const PassLayout* pre = nullptr) {
  SegInfo info;
  ism_status_t r = check_segments(segs, &info);
  if (r != ISM_OK) return r;
  if ((r = check_shape(shape)) != ISM_OK) return r;
  if (rope && (r = check_rope_pass(rope, shape, info)) != ISM_OK) return r;
  if (info.total_tokens == 0) return ISM_OK;
  if (!q || !k || !v || !o || !lse || !dout || !dq || !dk || !dv)
    return fail(ISM_ERR_INVALID_ARG, "q, k, v, o, lse, dout, dq, dk, dv must be non-NULL");
  const void* ptrs[] = {q, k, v, o, lse, dout, dq, dk, dv};
  for (const void* p : ptrs)
    if (!aligned16(p)) return fail(ISM_ERR_INVALID_ARG, "tensors must be 16-byte aligned");
  Counts c = count_tiles(segs, kTile, kTile);
  // the stored-dS path when the workspace holds its tiles, else recompute
  int64_t slots = stored_ds_slots(segs, shape);
  PassLayout L;
  if (pre) {
    // metadata from a plan; Delta and the dS tiles from the workspace
    L = *pre;
    Carve cv(workspace);
    L.delta = cv.take<float>((int64_t)shape->num_heads_q * info.total_tokens);
    const size_t need_min = ((cv.off + 255) & ~size_t(255)) + 256;
    void* ds = slots > 0 ? static_cast<void*>(cv.take<uint16_t>(slots * kTile * kTile)) : nullptr;
    const size_t need_full = ((cv.off + 255) & ~size_t(255)) + 256;
    L.ds = ds && workspace_bytes >= need_full ? ds : nullptr;
    if (!L.ds) slots = 0;
    L.bytes = L.ds ? need_full : need_min;
  } else {
    L = pass_layout(workspace, segs, c, info.total_tokens, shape->num_heads_q, true, slots);
    if (slots > 0 && workspace_bytes < L.bytes) {
      L = pass_layout(workspace, segs, c, info.total_tokens, shape->num_heads_q, true);
      slots = 0;
    }
  }
  if ((r = check_ws(workspace, workspace_bytes, L.bytes)) != ISM_OK) return r;
  uint32_t* status;
  if ((r = status_ptr(&status)) != ISM_OK) return r;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (pre) {
    // the plan's work counters start at zero for this call
    ISM_TRY_CUDA(cudaMemsetAsync(L.counters, 0, kPassCounters * sizeof(int32_t), st), "work counter reset");
  } else if ((r = build_pass_meta(segs, c, L, true, st)) != ISM_OK) {
    return r;
  }

  AttnArgs a{};
  a.q = q; a.k = k; a.v = v; a.o = o; a.dout = dout; a.lse_in = lse;
  a.dq = dq; a.dk = dk; a.dv = dv; a.delta = L.delta;
  a.hq = shape->num_heads_q; a.hkv = shape->num_heads_kv; a.d = shape->head_dim; a.dtype = shape->dtype;
  a.q_rows = info.total_tokens; a.scale = shape->softmax_scale;
  a.kv_end = L.kv_end; a.qtiles = L.qtiles; a.q_order = L.q_order; a.nq = c.nq;
  a.ktiles = L.ktiles; a.k_order = L.k_order; a.nk = c.nk;
  a.ds = L.ds; a.kpair_off = L.kpair_off; a.ds_slots = L.ds ? slots : 0;
  a.work_counter = L.counters;
  // the k-tile pair list exists only when the CTA-pair dK/dV kernel will run
  // (and a plan holds none)
  a.kp_order = knobs().dkdv_pair && !pre ? L.kp_order : nullptr;
  a.nkp = a.kp_order ? c.npairs : 0;
  a.status = status;
  a.flags = tc_flags();
  if (use_tc_bwd(shape)) {
    if (rope) {  // the dQ and dK epilogues rotate the gradients back
      a.rope_cos = rope->cos;
      a.rope_sin = rope->sin;
    }
    ISM_TRY_CUDA(launch_tc_bwd(a, info.total_tokens, st), "tensor-core backward launch");
  } else {
    ISM_TRY_CUDA(launch_simt_bwd(a, st), "backward launch");
    if (rope) {  // gradients of the rotated rows, rotated back in place
      timer_begin(ISM_KERNEL_ROPE, st);
      ISM_TRY_CUDA(launch_rope_rows(segs->cu_seqlens, segs->num_seqs, info.total_tokens, shape->num_heads_q,
                                    shape->num_heads_kv, shape->head_dim, shape->dtype, dq, dk, dq, dk, rope->cos,
                                    rope->sin, -1.f, st),
                   "rope launch");
      timer_end(ISM_KERNEL_ROPE, st);
      count_launch(1);
    }
  }
  return ISM_OK;
}

}  // namespace

extern "C" {

ism_status_t ism_attn_bwd(const ism_segments_t* segs, const ism_attn_shape_t* shape, const void* q,
                          const void* k, const void* v, const void* o, const float* lse, const void* dout,
                          void* dq, void* dk, void* dv, void* workspace, size_t workspace_bytes,
                          ism_stream_t stream) {
  return bwd_impl(segs, shape, q, k, v, o, lse, dout, dq, dk, dv, workspace, workspace_bytes, stream, nullptr);
}

ism_status_t ism_attn_bwd_rope(const ism_segments_t* segs, const ism_attn_shape_t* shape, const void* q_rot,
                               const void* k_rot, const void* v, const void* o, const float* lse, const void* dout,
                               const ism_rope_t* rope, void* dq, void* dk, void* dv, void* workspace,
                               size_t workspace_bytes, ism_stream_t stream) {
  if (!rope) return fail(ISM_ERR_INVALID_ARG, "rope is NULL");
  return bwd_impl(segs, shape, q_rot, k_rot, v, o, lse, dout, dq, dk, dv, workspace, workspace_bytes, stream, rope);
}

// ---------------------------------------------------------------- plans

ism_status_t ism_attn_plan_size(const ism_segments_t* segs, const ism_attn_shape_t* shape, size_t* bytes) {
  SegInfo info;
  ism_status_t r = check_segments(segs, &info);
  if (r != ISM_OK) return r;
  if ((r = check_shape(shape)) != ISM_OK) return r;
  if (!bytes) return fail(ISM_ERR_INVALID_ARG, "bytes is NULL");
  Counts c = count_tiles(segs, kTile, kTile);
  *bytes = plan_layout(nullptr, c, info.total_tokens, fwd_tile_pairs(shape)).bytes;
  return ISM_OK;
}

ism_status_t ism_attn_plan_build(const ism_segments_t* segs, const ism_attn_shape_t* shape, void* plan,
                                 size_t plan_bytes, ism_attn_plan_info_t* plan_info, ism_stream_t stream) {
  SegInfo info;
  ism_status_t r = check_segments(segs, &info);
  if (r != ISM_OK) return r;
  if ((r = check_shape(shape)) != ISM_OK) return r;
  if (!plan_info) return fail(ISM_ERR_INVALID_ARG, "plan_info is NULL");
  Counts c = count_tiles(segs, kTile, kTile);
  const bool tile_pairs = fwd_tile_pairs(shape);
  PassLayout L = plan_layout(plan, c, info.total_tokens, tile_pairs);
  if ((r = check_ws(plan, plan_bytes, L.bytes)) != ISM_OK) return r;
  if (info.total_tokens > 0) {
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if ((r = build_pass_meta(segs, c, L, true, st)) != ISM_OK) return r;
  }
  plan_info->fingerprint = plan_fingerprint(segs, shape, tile_pairs);
  plan_info->bytes = L.bytes;
  return ISM_OK;
}

}  // extern "C"

namespace {

// The layout of a plan for these segments and shape, after checking that the
// plan was built for them.
ism_status_t planned_layout(const ism_segments_t* segs, const ism_attn_shape_t* shape, const void* plan,
                            const ism_attn_plan_info_t* plan_info, PassLayout* L) {
  SegInfo info;
  ism_status_t r = check_segments(segs, &info);
  if (r != ISM_OK) return r;
  if ((r = check_shape(shape)) != ISM_OK) return r;
  if (!plan || !plan_info) return fail(ISM_ERR_INVALID_ARG, "plan and plan_info must be non-NULL");
  if (reinterpret_cast<uintptr_t>(plan) & 255u) return fail(ISM_ERR_INVALID_ARG, "plan must be 256-byte aligned");
  const bool tile_pairs = fwd_tile_pairs(shape);
  if (plan_fingerprint(segs, shape, tile_pairs) != plan_info->fingerprint)
    return fail(ISM_ERR_INVALID_ARG, "the plan was built for other segments or head counts");
  Counts c = count_tiles(segs, kTile, kTile);
  *L = plan_layout(const_cast<void*>(plan), c, info.total_tokens, tile_pairs);
  if (plan_info->bytes < L->bytes) return fail(ISM_ERR_INVALID_ARG, "plan_info does not describe this plan");
  return ISM_OK;
}

}  // namespace

extern "C" {

ism_status_t ism_attn_fwd_planned(const ism_segments_t* segs, const ism_attn_shape_t* shape, const void* plan,
                                  const ism_attn_plan_info_t* plan_info, const void* q, const void* k,
                                  const void* v, void* o, float* lse, ism_stream_t stream) {
  PassLayout L;
  ism_status_t r = planned_layout(segs, shape, plan, plan_info, &L);
  if (r != ISM_OK) return r;
  return fwd_impl(segs, shape, q, k, v, o, lse, nullptr, 0, stream, 1.f, 1.f, nullptr, nullptr, nullptr, &L);
}

ism_status_t ism_attn_bwd_planned(const ism_segments_t* segs, const ism_attn_shape_t* shape, void* plan,
                                  const ism_attn_plan_info_t* plan_info, const void* q, const void* k,
                                  const void* v, const void* o, const float* lse, const void* dout, void* dq,
                                  void* dk, void* dv, void* workspace, size_t workspace_bytes,
                                  ism_stream_t stream) {
  PassLayout L;
  ism_status_t r = planned_layout(segs, shape, plan, plan_info, &L);
  if (r != ISM_OK) return r;
  return bwd_impl(segs, shape, q, k, v, o, lse, dout, dq, dk, dv, workspace, workspace_bytes, stream, nullptr, &L);
}

ism_status_t ism_attn_fwd_rope_planned(const ism_segments_t* segs, const ism_attn_shape_t* shape, const void* plan,
                                       const ism_attn_plan_info_t* plan_info, const void* q, const void* k,
                                       const void* v, const ism_rope_t* rope, void* q_rot, void* k_rot, void* o,
                                       float* lse, ism_stream_t stream) {
  if (!rope) return fail(ISM_ERR_INVALID_ARG, "rope is NULL");
  PassLayout L;
  ism_status_t r = planned_layout(segs, shape, plan, plan_info, &L);
  if (r != ISM_OK) return r;
  return fwd_impl(segs, shape, q, k, v, o, lse, nullptr, 0, stream, 1.f, 1.f, rope, q_rot, k_rot, &L);
}

ism_status_t ism_attn_bwd_rope_planned(const ism_segments_t* segs, const ism_attn_shape_t* shape, void* plan,
                                       const ism_attn_plan_info_t* plan_info, const void* q_rot, const void* k_rot,
                                       const void* v, const void* o, const float* lse, const void* dout,
                                       const ism_rope_t* rope, void* dq, void* dk, void* dv, void* workspace,
                                       size_t workspace_bytes, ism_stream_t stream) {
  if (!rope) return fail(ISM_ERR_INVALID_ARG, "rope is NULL");
  PassLayout L;
  ism_status_t r = planned_layout(segs, shape, plan, plan_info, &L);
  if (r != ISM_OK) return r;
  return bwd_impl(segs, shape, q_rot, k_rot, v, o, lse, dout, dq, dk, dv, workspace, workspace_bytes, stream, rope,
                  &L);
}

// ---------------------------------------------------------------- append

namespace {

struct AppendLayout {
  int32_t* c_snap;
  int32_t* kv_end;
  Tile* qtiles;
  int32_t* q_order;
  int32_t* pair_order;  // neighbouring q-tiles of a chunk, for the paired forward
  int64_t npairs;
  float* part_o;
  float* part_ml;
  void* q_rot;  // rotated queries of a RoPE append (bf16 [batch * l_new, Hq, D]), else null
  // partials of the forward's key-range split (prefill): up to split_cap items
  float* part_fo;
  float* part_fml;
  int64_t split_cap;
  size_t bytes;
};

// Forward items (query tile, head pair) that may run as two key-range halves.
constexpr int64_t kMaxSplitItems = 256;

AppendLayout append_layout(void* ws, const ism_attn_shape_t* sh, int batch, int l_new, bool rope = false) {
  Carve cv(ws);
  AppendLayout L;
  const int64_t nqt_seq = (l_new + kTile - 1) / kTile;
  int64_t nqt = (int64_t)batch * nqt_seq;
  L.c_snap = cv.take<int32_t>(batch);
  L.kv_end = cv.take<int32_t>((int64_t)batch * l_new);
  L.qtiles = cv.take<Tile>(nqt);
  L.q_order = cv.take<int32_t>(nqt);
  L.npairs = (int64_t)batch * ((nqt_seq + 1) / 2);
  L.pair_order = cv.take<int32_t>(L.npairs);
  if (l_new == 1) {
    L.part_o = cv.take<float>((int64_t)batch * sh->num_heads_q * kMaxSplits * sh->head_dim);
    L.part_ml = cv.take<float>((int64_t)batch * sh->num_heads_q * kMaxSplits * 2);
  } else {
    L.part_o = L.part_ml = nullptr;
  }
  L.q_rot = rope ? (void*)cv.take<__nv_bfloat16>((int64_t)batch * l_new * sh->num_heads_q * sh->head_dim) : nullptr;
  if (l_new > 1 && sh->num_heads_q % 2 == 0) {
    const int64_t items = nqt * (sh->num_heads_q / 2);
    L.split_cap = items < kMaxSplitItems ? items : kMaxSplitItems;
    L.part_fo = cv.take<float>(L.split_cap * 2 * 2 * kTile * 128);
    L.part_fml = cv.take<float>(L.split_cap * 2 * 2 * kTile * 2);
  } else {
    L.split_cap = 0;
    L.part_fo = L.part_fml = nullptr;
  }
  L.bytes = ((cv.off + 255) & ~size_t(255)) + 256;
  return L;
}

}  // namespace

ism_status_t ism_attn_prefill_append_workspace_size(const ism_attn_shape_t* shape, int32_t batch, int32_t l_new,
                                                    size_t* bytes) {
  ism_status_t r = check_shape(shape, true);
  if (r != ISM_OK) return r;
  if (batch < 0 || l_new < 0) return fail(ISM_ERR_INVALID_ARG, "batch and l_new must be >= 0");
  if (!bytes) return fail(ISM_ERR_INVALID_ARG, "bytes is NULL");
  *bytes = append_layout(nullptr, shape, batch, l_new).bytes;  // (e4m3 shapes included)
  return ISM_OK;
}

ism_status_t ism_attn_prefill_append_rope_workspace_size(const ism_attn_shape_t* shape, int32_t batch,
                                                         int32_t l_new, size_t* bytes) {
  ism_status_t r = check_shape(shape, true);
  if (r != ISM_OK) return r;
  if (batch < 0 || l_new < 0) return fail(ISM_ERR_INVALID_ARG, "batch and l_new must be >= 0");
  if (!bytes) return fail(ISM_ERR_INVALID_ARG, "bytes is NULL");
  *bytes = append_layout(nullptr, shape, batch, l_new, true).bytes;
  return ISM_OK;
}

}  // extern "C"

namespace {

// Cache geometry of one append call: contiguous [B, cap] caches, or pages.
constexpr int kMaxDecodeGroup = 16;

struct CacheGeom {
  int64_t cap;       // contiguous: rows per sequence
  int64_t kv_rows;   // rows of the K / V tensors (tensor-map extent)
  int64_t max_keys;  // keys a sequence can hold
  KvPages pages;     // table == nullptr: contiguous
};

ism_status_t append_impl(const ism_attn_shape_t* shape, int32_t batch, const void* q_new, const void* k_new,
                         const void* v_new, int32_t l_new, const int32_t* new_seg_end_host,
                         const uint8_t* new_seg_type_host, int32_t n_new_segs, void* k_cache, void* v_cache,
                         const CacheGeom& cg, int32_t* cache_len, const int32_t* cache_len_host, void* o_new,
                         float* lse_new, void* workspace, size_t workspace_bytes, cudaStream_t st,
                         float q_descale = 1.f, float k_descale = 1.f, float v_descale = 1.f,
                         const ism_rope_t* rope = nullptr) {
  const float qk_descale = q_descale * k_descale;
  ism_status_t r;
  if (!q_new || !k_new || !v_new || !k_cache || !v_cache || !cache_len || !cache_len_host || !o_new)
    return fail(ISM_ERR_INVALID_ARG, "q_new, k_new, v_new, caches, cache_len (device+host), o_new must be non-NULL");
  const void* ptrs[] = {q_new, k_new, v_new, k_cache, v_cache, o_new};
  for (const void* p : ptrs)
    if (!aligned16(p)) return fail(ISM_ERR_INVALID_ARG, "tensors must be 16-byte aligned");
  if (lse_new && !aligned16(lse_new)) return fail(ISM_ERR_INVALID_ARG, "lse_new must be 16-byte aligned");
  if (!new_seg_end_host || !new_seg_type_host || n_new_segs <= 0 || n_new_segs > kMaxAppendSegs)
    return fail(ISM_ERR_INVALID_ARG, "chunk needs 1..%d segments", kMaxAppendSegs);
  AppendSegs sg;
  memset(&sg, 0, sizeof(sg));
  sg.n = n_new_segs;
  sg.l_new = l_new;
  int32_t prev = 0;
  for (int i = 0; i < n_new_segs; ++i) {
    if (new_seg_end_host[i] < prev) return fail(ISM_ERR_INVALID_ARG, "chunk seg_end not non-decreasing");
    if (new_seg_type_host[i] > 1) return fail(ISM_ERR_INVALID_ARG, "chunk segment type %d", (int)new_seg_type_host[i]);
    sg.end[i] = prev = new_seg_end_host[i];
    sg.type[i] = new_seg_type_host[i];
  }
  if (prev != l_new) return fail(ISM_ERR_INVALID_ARG, "chunk segments end at %d, l_new is %d", prev, l_new);
  if ((int64_t)batch * l_new >= (int64_t(1) << 31)) return fail(ISM_ERR_INVALID_ARG, "batch * l_new too large");
  int32_t max_c = 0;
  for (int b = 0; b < batch; ++b) {
    int32_t c = cache_len_host[b];
    if (c < 0 || (int64_t)c + l_new > cg.max_keys)
      return fail(ISM_ERR_INVALID_ARG, "sequence %d: cache_len %d + l_new %d exceeds capacity %lld", b, c, l_new,
                  (long long)cg.max_keys);
    if (c > max_c) max_c = c;
  }
  if (rope) {
    if (!rope->cos || !rope->sin || !aligned16(rope->cos) || !aligned16(rope->sin))
      return fail(ISM_ERR_INVALID_ARG, "rope tables must be non-NULL and 16-byte aligned");
    if ((int64_t)max_c + l_new > rope->rows)
      return fail(ISM_ERR_INVALID_ARG, "rope tables cover %d positions, the append writes up to %lld", rope->rows,
                  (long long)max_c + l_new);
  }
  AppendLayout L = append_layout(workspace, shape, batch, l_new, rope != nullptr);
  if ((r = check_ws(workspace, workspace_bytes, L.bytes)) != ISM_OK) return r;
  uint32_t* status;
  if ((r = status_ptr(&status)) != ISM_OK) return r;
  const int hq = shape->num_heads_q, hkv = shape->num_heads_kv, d = shape->head_dim;
  const bool paged = cg.pages.table != nullptr;

  // decode kernels serve up to kMaxDecodeGroup query heads per KV head; larger
  // groups take the forward kernels (one query row per tile)
  const bool decode = l_new == 1 && (shape->dtype == ISM_BF16 || shape->dtype == ISM_E4M3) && !force_cuda_cores() &&
                      hq / hkv <= kMaxDecodeGroup;
  // A single-token step needs no tile plan: the cache write reads the cache
  // lengths and snapshots them, and the decode's combine kernel advances them.
  timer_begin(ISM_KERNEL_META, st);
  if (!decode)
    ISM_TRY_CUDA(launch_append_plan(sg, batch, paged ? 1 : cg.cap, kTile, kTile, cache_len, L.c_snap, L.kv_end,
                                    L.qtiles, L.q_order, L.pair_order, st),
                 "append plan launch");
  const int32_t* c_src = decode ? cache_len : L.c_snap;
  int32_t* snap_out = decode ? L.c_snap : nullptr;
  if (rope) {
    ISM_TRY_CUDA(launch_rope_cache_write(shape->dtype, batch, l_new, hq, hkv, d, cg.cap, cg.pages, c_src, q_new,
                                         k_new, v_new, rope->cos, rope->sin, q_descale, k_descale, v_descale,
                                         L.q_rot, k_cache, v_cache, st, snap_out),
                 "rope cache write launch");
    q_new = L.q_rot;  // the attention below reads the rotated queries
  } else {
    ISM_TRY_CUDA(launch_cache_write(shape->dtype, batch, l_new, hkv, d, cg.cap, cg.pages, c_src, k_new, v_new,
                                    k_cache, v_cache, st, snap_out),
                 "cache write launch");
  }
  timer_end(ISM_KERNEL_META, st);
  count_launch(decode ? 1 : 2);
  if (decode) {
    DecodeArgs a{};
    a.cache_len = cache_len;
    a.q = q_new; a.k_cache = k_cache; a.v_cache = v_cache; a.pages = cg.pages; a.out = o_new; a.lse = lse_new;
    a.c_snap = L.c_snap;
    a.batch = batch; a.hq = hq; a.hkv = hkv; a.d = d; a.dtype = shape->dtype; a.cap = cg.cap;
    a.group = hq / hkv;
    a.qk_descale = qk_descale; a.v_descale = v_descale;
    a.kv_rows = cg.kv_rows;
    a.scale = shape->softmax_scale;
    // chunks of a multiple of 64 keys, as many as fill whole waves of resident
    // CTAs: 4 per SM for the register kernel (one wave), 2 per SM for the TMA
    // kernel (four waves, so each CTA's ring runs several tiles)
    int64_t kv_max = (int64_t)max_c + 1;
    int64_t pairs = (int64_t)batch * hkv;
    const int sms = sm_count();
    a.tma = (d == 128 && tc_available() && !knobs().decode_no_tma) ? 1 : 0;
    a.tc = (a.tma && !knobs().decode_no_tc &&
            kv_max <= (int64_t)kMaxSplits * kDecTcMaxKeys)
               ? 1
               : 0;
    int64_t splits, chunk;
    if (a.tc) {
      // persistent tensor-core kernel: the split count that minimises the
      // busiest CTA's work, (items per CTA) x (128-key tiles per item + 1 for
      // the item's hand-offs), over chunks of whole tiles up to kDecTcMaxKeys
      int64_t best = -1;
      splits = chunk = 0;
      for (int64_t sp = 1; sp <= kMaxSplits; ++sp) {
        const int64_t ch = ((kv_max + sp - 1) / sp + 127) / 128 * 128;
        if (ch > kDecTcMaxKeys) continue;
        const int64_t used = (kv_max + ch - 1) / ch;
        const int64_t per_cta = (pairs * used + sms - 1) / sms;
        const int64_t cost = per_cta * (ch / 128 + 1);
        if (best < 0 || cost < best) {
          best = cost;
          splits = used;
          chunk = ch;
        }
      }
    } else {
      int64_t want = (a.tma ? 8 * (int64_t)sms : 4 * (int64_t)sms) / pairs;
      splits = want < 1 ? 1 : want > kMaxSplits ? kMaxSplits : want;
      chunk = (kv_max + splits - 1) / splits;
      chunk = (chunk + 63) / 64 * 64;
      splits = (kv_max + chunk - 1) / chunk;
    }
    a.splits = (int32_t)splits;
    a.chunk = (int32_t)chunk;
    a.part_o = L.part_o; a.part_ml = L.part_ml;
    a.status = status;
    timer_begin(ISM_KERNEL_DECODE, st);
    ISM_TRY_CUDA(launch_decode(a, st), "decode launch");
    timer_end(ISM_KERNEL_DECODE, st);
    count_launch(2);
    return ISM_OK;
  }
  AttnArgs a{};
  a.q = q_new; a.k = k_cache; a.v = v_cache; a.out = o_new; a.lse = lse_new;
  a.hq = hq; a.hkv = hkv; a.d = d; a.dtype = shape->dtype;
  a.q_rows = (int64_t)batch * l_new; a.scale = shape->softmax_scale;
  a.kv_end = L.kv_end; a.qtiles = L.qtiles; a.q_order = L.q_order;
  a.nq = (int64_t)batch * ((l_new + kTile - 1) / kTile);
  a.pages = cg.pages;
  if (shape->dtype == ISM_E4M3) {
    // the e4m3 forward is the paired kernel: neighbouring q-tiles for an odd group
    a.qk_descale = qk_descale;
    a.v_descale = v_descale;
    if ((hq / hkv) % 2) {
      a.pair_order = L.pair_order;
      a.npairs = L.npairs;
    }
  }
  a.status = status;
  a.flags = tc_flags();
  // The items of the paired forward (query tile, head pair) all cost about the
  // same in a prefill; those that would leave a last round with idle SMs run
  // as two halves of their key range instead, when the items are long enough
  // (at least 64 key tiles) for the halves to outweigh the merge.  Measured
  // on the 8 x 16K prefill with the persistent forward: bf16 0.795 -> 0.719
  // ms, e4m3 0.668 -> 0.595 ms; 40-token chunks over 4000 keys stay whole.
  // ISM_PREFILL_SPLIT=n forces n split items.
  if ((use_tc(shape) || shape->dtype == ISM_E4M3) && d == 128 && (hq / hkv) % 2 == 0 && !a.pair_order &&
      L.split_cap > 0) {
    const int64_t items = a.nq * (hq / 2);
    int64_t n_split = 0;
    if (knobs().prefill_split >= 0) {
      n_split = knobs().prefill_split;
    } else {
      const int sms = sm_count();
      const int64_t key_tiles = ((int64_t)max_c + l_new + kTile - 1) / kTile;
      if (items > sms && key_tiles >= 64) n_split = items % sms;
    }
    if (n_split > L.split_cap) n_split = L.split_cap;
    if (n_split > 0) {
      a.split_items = n_split;
      a.split_whole = items - n_split;
      a.part_o = L.part_fo;
      a.part_ml = L.part_fml;
    }
  }
  timer_begin(ISM_KERNEL_FWD, st);
  if (use_tc(shape) || shape->dtype == ISM_E4M3) {
    ISM_TRY_CUDA(launch_tc_fwd(a, cg.kv_rows, st), "tensor-core prefill launch");
  } else {
    ISM_TRY_CUDA(launch_simt_fwd(a, st), "prefill launch");
  }
  timer_end(ISM_KERNEL_FWD, st);
  count_launch(a.split_items > 0 ? 2 : 1);  // the key-range halves are merged by a second kernel
  return ISM_OK;
}

}  // namespace

extern "C" {

ism_status_t ism_attn_prefill_append(const ism_attn_shape_t* shape, int32_t batch, const void* q_new,
                                     const void* k_new, const void* v_new, int32_t l_new,
                                     const int32_t* new_seg_end_host, const uint8_t* new_seg_type_host,
                                     int32_t n_new_segs, void* k_cache, void* v_cache, int64_t cache_capacity,
                                     int32_t* cache_len, const int32_t* cache_len_host, void* o_new,
                                     float* lse_new, void* workspace, size_t workspace_bytes,
                                     ism_stream_t stream) {
  ism_status_t r = check_shape(shape);
  if (r != ISM_OK) return r;
  if (batch < 0 || l_new < 0) return fail(ISM_ERR_INVALID_ARG, "batch and l_new must be >= 0");
  if (batch == 0 || l_new == 0) return ISM_OK;
  if (cache_capacity <= 0 || (int64_t)batch * cache_capacity >= (int64_t(1) << 31))
    return fail(ISM_ERR_INVALID_ARG, "batch * cache_capacity must be in (0, 2^31)");
  CacheGeom cg;
  cg.cap = cache_capacity;
  cg.kv_rows = (int64_t)batch * cache_capacity;
  cg.max_keys = cache_capacity;
  cg.pages = KvPages{nullptr, 0, 0};
  return append_impl(shape, batch, q_new, k_new, v_new, l_new, new_seg_end_host, new_seg_type_host, n_new_segs,
                     k_cache, v_cache, cg, cache_len, cache_len_host, o_new, lse_new, workspace, workspace_bytes,
                     reinterpret_cast<cudaStream_t>(stream));
}

ism_status_t ism_attn_prefill_append_e4m3(const ism_attn_shape_t* shape, int32_t batch, const void* q_new,
                                          const void* k_new, const void* v_new, int32_t l_new,
                                          const int32_t* new_seg_end_host, const uint8_t* new_seg_type_host,
                                          int32_t n_new_segs, void* k_cache, void* v_cache, int64_t cache_capacity,
                                          int32_t* cache_len, const int32_t* cache_len_host, float q_descale,
                                          float k_descale, float v_descale, void* o_new, float* lse_new,
                                          void* workspace, size_t workspace_bytes, ism_stream_t stream) {
  ism_status_t r = check_shape(shape, true);
  if (r != ISM_OK) return r;
  if (shape->dtype != ISM_E4M3) return fail(ISM_ERR_INVALID_ARG, "ism_attn_prefill_append_e4m3 needs ISM_E4M3");
  if (!valid_descales(q_descale, k_descale, v_descale))
    return fail(ISM_ERR_INVALID_ARG, "descales must be positive finite numbers");
  if (!tc_available()) return fail(ISM_ERR_UNSUPPORTED, "e4m3 attention needs the sm_103 tensor cores");
  if (batch < 0 || l_new < 0) return fail(ISM_ERR_INVALID_ARG, "batch and l_new must be >= 0");
  if (batch == 0 || l_new == 0) return ISM_OK;
  if (cache_capacity <= 0 || (int64_t)batch * cache_capacity >= (int64_t(1) << 31))
    return fail(ISM_ERR_INVALID_ARG, "batch * cache_capacity must be in (0, 2^31)");
  CacheGeom cg;
  cg.cap = cache_capacity;
  cg.kv_rows = (int64_t)batch * cache_capacity;
  cg.max_keys = cache_capacity;
  cg.pages = KvPages{nullptr, 0, 0};
  return append_impl(shape, batch, q_new, k_new, v_new, l_new, new_seg_end_host, new_seg_type_host, n_new_segs,
                     k_cache, v_cache, cg, cache_len, cache_len_host, o_new, lse_new, workspace, workspace_bytes,
                     reinterpret_cast<cudaStream_t>(stream), q_descale, k_descale, v_descale);
}

ism_status_t ism_attn_prefill_append_rope(const ism_attn_shape_t* shape, int32_t batch, const void* q_new,
                                          const void* k_new, const void* v_new, int32_t l_new,
                                          const int32_t* new_seg_end_host, const uint8_t* new_seg_type_host,
                                          int32_t n_new_segs, void* k_cache, void* v_cache, int64_t cache_capacity,
                                          int32_t* cache_len, const int32_t* cache_len_host, const ism_rope_t* rope,
                                          void* o_new, float* lse_new, void* workspace, size_t workspace_bytes,
                                          ism_stream_t stream) {
  ism_status_t r = check_shape(shape);
  if (r != ISM_OK) return r;
  if (shape->dtype != ISM_BF16) return fail(ISM_ERR_INVALID_ARG, "ism_attn_prefill_append_rope needs ISM_BF16");
  if (!rope) return fail(ISM_ERR_INVALID_ARG, "rope is NULL");
  if (batch < 0 || l_new < 0) return fail(ISM_ERR_INVALID_ARG, "batch and l_new must be >= 0");
  if (batch == 0 || l_new == 0) return ISM_OK;
  if (cache_capacity <= 0 || (int64_t)batch * cache_capacity >= (int64_t(1) << 31))
    return fail(ISM_ERR_INVALID_ARG, "batch * cache_capacity must be in (0, 2^31)");
  CacheGeom cg;
  cg.cap = cache_capacity;
  cg.kv_rows = (int64_t)batch * cache_capacity;
  cg.max_keys = cache_capacity;
  cg.pages = KvPages{nullptr, 0, 0};
  return append_impl(shape, batch, q_new, k_new, v_new, l_new, new_seg_end_host, new_seg_type_host, n_new_segs,
                     k_cache, v_cache, cg, cache_len, cache_len_host, o_new, lse_new, workspace, workspace_bytes,
                     reinterpret_cast<cudaStream_t>(stream), 1.f, 1.f, 1.f, rope);
}

ism_status_t ism_attn_prefill_append_e4m3_rope(const ism_attn_shape_t* shape, int32_t batch, const void* q_new,
                                               const void* k_new, const void* v_new, int32_t l_new,
                                               const int32_t* new_seg_end_host, const uint8_t* new_seg_type_host,
                                               int32_t n_new_segs, void* k_cache, void* v_cache,
                                               int64_t cache_capacity, int32_t* cache_len,
                                               const int32_t* cache_len_host, float q_descale, float k_descale,
                                               float v_descale, const ism_rope_t* rope, void* o_new, float* lse_new,
                                               void* workspace, size_t workspace_bytes, ism_stream_t stream) {
  ism_status_t r = check_shape(shape, true);
  if (r != ISM_OK) return r;
  if (shape->dtype != ISM_E4M3) return fail(ISM_ERR_INVALID_ARG, "ism_attn_prefill_append_e4m3_rope needs ISM_E4M3");
  if (!valid_descales(q_descale, k_descale, v_descale))
    return fail(ISM_ERR_INVALID_ARG, "descales must be positive finite numbers");
  if (!rope) return fail(ISM_ERR_INVALID_ARG, "rope is NULL");
  if (!tc_available()) return fail(ISM_ERR_UNSUPPORTED, "e4m3 attention needs the sm_103 tensor cores");
  if (batch < 0 || l_new < 0) return fail(ISM_ERR_INVALID_ARG, "batch and l_new must be >= 0");
  if (batch == 0 || l_new == 0) return ISM_OK;
  if (cache_capacity <= 0 || (int64_t)batch * cache_capacity >= (int64_t(1) << 31))
    return fail(ISM_ERR_INVALID_ARG, "batch * cache_capacity must be in (0, 2^31)");
  CacheGeom cg;
  cg.cap = cache_capacity;
  cg.kv_rows = (int64_t)batch * cache_capacity;
  cg.max_keys = cache_capacity;
  cg.pages = KvPages{nullptr, 0, 0};
  return append_impl(shape, batch, q_new, k_new, v_new, l_new, new_seg_end_host, new_seg_type_host, n_new_segs,
                     k_cache, v_cache, cg, cache_len, cache_len_host, o_new, lse_new, workspace, workspace_bytes,
                     reinterpret_cast<cudaStream_t>(stream), q_descale, k_descale, v_descale, rope);
}

}  // extern "C"

namespace {

// Validates a paged cache and describes it: every page a sequence reads or
// writes in this call lies in the pool.
ism_status_t paged_geom(int32_t batch, int32_t l_new, int32_t num_pages, int32_t page_size,
                        const int32_t* block_table, const int32_t* block_table_host, int32_t max_pages,
                        const int32_t* cache_len_host, CacheGeom* cg) {
  if (page_size <= 0 || page_size % kTile != 0)
    return fail(ISM_ERR_INVALID_ARG, "page_size %d must be a positive multiple of %d", page_size, kTile);
  if (num_pages <= 0 || (int64_t)num_pages * page_size >= (int64_t(1) << 31))
    return fail(ISM_ERR_INVALID_ARG, "num_pages * page_size must be in (0, 2^31)");
  if (max_pages <= 0 || !block_table || !block_table_host || !cache_len_host)
    return fail(ISM_ERR_INVALID_ARG, "block_table (device+host), cache_len_host and max_pages > 0 are required");
  for (int b = 0; b < batch; ++b) {
    const int64_t keys = (int64_t)cache_len_host[b] + l_new;
    if (cache_len_host[b] < 0 || keys > (int64_t)max_pages * page_size)
      return fail(ISM_ERR_INVALID_ARG, "sequence %d: cache_len %d + l_new %d exceeds its %d pages", b, cache_len_host[b],
                  l_new, max_pages);
    for (int64_t i = 0; i < (keys + page_size - 1) / page_size; ++i) {
      const int32_t pg = block_table_host[(int64_t)b * max_pages + i];
      if (pg < 0 || pg >= num_pages)
        return fail(ISM_ERR_INVALID_ARG, "sequence %d: page %lld of the block table is %d, outside [0, %d)", b,
                    (long long)i, pg, num_pages);
    }
  }
  cg->cap = 0;
  cg->kv_rows = (int64_t)num_pages * page_size;
  cg->max_keys = (int64_t)max_pages * page_size;
  cg->pages = KvPages{block_table, page_size, max_pages};
  return ISM_OK;
}

}  // namespace

extern "C" {

ism_status_t ism_attn_prefill_append_paged(const ism_attn_shape_t* shape, int32_t batch, const void* q_new,
                                           const void* k_new, const void* v_new, int32_t l_new,
                                           const int32_t* new_seg_end_host, const uint8_t* new_seg_type_host,
                                           int32_t n_new_segs, void* k_pool, void* v_pool, int32_t num_pages,
                                           int32_t page_size, const int32_t* block_table,
                                           const int32_t* block_table_host, int32_t max_pages, int32_t* cache_len,
                                           const int32_t* cache_len_host, void* o_new, float* lse_new,
                                           void* workspace, size_t workspace_bytes, ism_stream_t stream) {
  ism_status_t r = check_shape(shape);
  if (r != ISM_OK) return r;
  if (batch < 0 || l_new < 0) return fail(ISM_ERR_INVALID_ARG, "batch and l_new must be >= 0");
  if (batch == 0 || l_new == 0) return ISM_OK;
  CacheGeom cg;
  if ((r = paged_geom(batch, l_new, num_pages, page_size, block_table, block_table_host, max_pages, cache_len_host,
                      &cg)) != ISM_OK)
    return r;
  return append_impl(shape, batch, q_new, k_new, v_new, l_new, new_seg_end_host, new_seg_type_host, n_new_segs,
                     k_pool, v_pool, cg, cache_len, cache_len_host, o_new, lse_new, workspace, workspace_bytes,
                     reinterpret_cast<cudaStream_t>(stream));
}

ism_status_t ism_attn_prefill_append_paged_rope(const ism_attn_shape_t* shape, int32_t batch, const void* q_new,
                                                const void* k_new, const void* v_new, int32_t l_new,
                                                const int32_t* new_seg_end_host, const uint8_t* new_seg_type_host,
                                                int32_t n_new_segs, void* k_pool, void* v_pool, int32_t num_pages,
                                                int32_t page_size, const int32_t* block_table,
                                                const int32_t* block_table_host, int32_t max_pages,
                                                int32_t* cache_len, const int32_t* cache_len_host,
                                                const ism_rope_t* rope, void* o_new, float* lse_new, void* workspace,
                                                size_t workspace_bytes, ism_stream_t stream) {
  ism_status_t r = check_shape(shape);
  if (r != ISM_OK) return r;
  if (shape->dtype != ISM_BF16)
    return fail(ISM_ERR_INVALID_ARG, "ism_attn_prefill_append_paged_rope needs ISM_BF16");
  if (!rope) return fail(ISM_ERR_INVALID_ARG, "rope is NULL");
  if (batch < 0 || l_new < 0) return fail(ISM_ERR_INVALID_ARG, "batch and l_new must be >= 0");
  if (batch == 0 || l_new == 0) return ISM_OK;
  CacheGeom cg;
  if ((r = paged_geom(batch, l_new, num_pages, page_size, block_table, block_table_host, max_pages, cache_len_host,
                      &cg)) != ISM_OK)
    return r;
  return append_impl(shape, batch, q_new, k_new, v_new, l_new, new_seg_end_host, new_seg_type_host, n_new_segs,
                     k_pool, v_pool, cg, cache_len, cache_len_host, o_new, lse_new, workspace, workspace_bytes,
                     reinterpret_cast<cudaStream_t>(stream), 1.f, 1.f, 1.f, rope);
}

// ---------------------------------------------------------------- status

ism_status_t ism_check_status(ism_stream_t stream) {
  uint32_t* status;
  ism_status_t r = status_ptr(&status);
  if (r != ISM_OK) return r;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  ISM_TRY_CUDA(cudaStreamSynchronize(st), "cudaStreamSynchronize");
  uint32_t word = 0;
  ISM_TRY_CUDA(cudaMemcpy(&word, status, sizeof(word), cudaMemcpyDeviceToHost), "status read");
  if (word) {
    uint32_t zero = 0;
    ISM_TRY_CUDA(cudaMemcpy(status, &zero, sizeof(zero), cudaMemcpyHostToDevice), "status clear");
  }
  if (word & kStatusTimeout) return fail(ISM_ERR_TIMEOUT, "a device-side wait gave up (status word 0x%x)", word);
  if (word & kStatusSmemAlign)
    return fail(ISM_ERR_CUDA, "a kernel found its shared memory misaligned and skipped its work (0x%x)", word);
  return ISM_OK;
}

ism_status_t ism_debug_mma_tile(const void* a, const void* b, float* c, int32_t mode, ism_stream_t stream) {
  if (!a || !b || !c || mode < 0 || mode > 15) return fail(ISM_ERR_INVALID_ARG, "a, b, c non-NULL and mode 0..15");
  if (!tc_available()) return fail(ISM_ERR_UNSUPPORTED, "tensor-core kernels need an sm_103 device");
  uint32_t* status;
  ism_status_t r = status_ptr(&status);
  if (r != ISM_OK) return r;
  ISM_TRY_CUDA(launch_tc_mma_tile(a, b, c, mode, status, reinterpret_cast<cudaStream_t>(stream)), "mma tile launch");
  count_launch(1);
  return ISM_OK;
}

ism_status_t ism_debug_mma_tile_e4m3(const void* a, const void* b, float* c, int32_t mode, ism_stream_t stream) {
  if (!a || !b || !c || mode < 0 || mode > 2) return fail(ISM_ERR_INVALID_ARG, "a, b, c non-NULL and mode 0..2");
  if (!tc_available()) return fail(ISM_ERR_UNSUPPORTED, "tensor-core kernels need an sm_103 device");
  uint32_t* status;
  ism_status_t r = status_ptr(&status);
  if (r != ISM_OK) return r;
  ISM_TRY_CUDA(tc::launch_mma_tile_e4m3(a, b, c, mode, status, reinterpret_cast<cudaStream_t>(stream)),
               "e4m3 mma tile launch");
  count_launch(1);
  return ISM_OK;
}

ism_status_t ism_debug_timeout_probe(uint32_t spin_limit, ism_stream_t stream) {
  uint32_t* status;
  ism_status_t r = status_ptr(&status);
  if (r != ISM_OK) return r;
  if (spin_limit == 0 || spin_limit > (1u << 20)) return fail(ISM_ERR_INVALID_ARG, "spin_limit must be in [1, 2^20]");
  ISM_TRY_CUDA(launch_timeout_probe(spin_limit, status, reinterpret_cast<cudaStream_t>(stream)), "probe launch");
  return ISM_OK;
}

}  // extern "C"
