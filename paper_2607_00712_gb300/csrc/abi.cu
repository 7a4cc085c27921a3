// C-ABI entry points of libispa: argument validation, ring bookkeeping
// (Eq. 7-8 key sets as slot runs), tensor-map encoding and kernel launches.
// See include/ispa.h for the contract of each function.
#include <cuda.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>
#include <string.h>

#include <atomic>
#include <mutex>
#include <set>
#include <utility>
#include <vector>

#include "internal.h"
#include "ptx.cuh"

namespace ispa {

static __device__ int g_status[8];  // device error record (DEVERR_* + location), one per device

namespace {

constexpr uint64_t kDefaultWaitLimitNs = 1000ull * 1000 * 1000;
std::atomic<uint64_t> g_wait_limit{kDefaultWaitLimitNs};

bool aligned16(const void* p) { return p && (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

// The tensor-map encoder below is a driver-API call.  In a host thread that has not yet made a
// CUDA runtime call no context is current, and the encoder fails there (the runtime binds a
// context only for its own calls).  Bind the current device's primary context first, as the
// runtime would: a no-op when a context is already current.
CtxGetCurrentFn ctx_get_current_fn();
CtxGetIdFn ctx_get_id_fn();

void ensure_context() {
  const CtxGetCurrentFn get = ctx_get_current_fn();
  CUcontext c = nullptr;
  if (get && get(&c) == CUDA_SUCCESS && c) return;
  int dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaSetDevice(dev);
}

CtxGetCurrentFn ctx_get_current_fn() {
  static CtxGetCurrentFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<CtxGetCurrentFn>(p);
  });
  return fn;
}

CtxGetIdFn ctx_get_id_fn() {
  static CtxGetIdFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<CtxGetIdFn>(p);
  });
  return fn;
}

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

uint64_t wait_limit_ns() { return g_wait_limit.load(); }

namespace {
uint32_t* g_hb = nullptr;   // host-mapped heartbeat buffer (device address), debug only
int g_hb_slots = 0;
std::atomic<int> g_hb_next{0};
}  // namespace

uint64_t* g_trace = nullptr;
int32_t g_trace_tiles = 0;
int32_t g_drop_k_tile = -1;

uint64_t* trace_buffer(int32_t* n_tiles) {
  *n_tiles = g_trace_tiles;
  return g_trace;
}

uint32_t* next_heartbeat_slot(uint32_t kernel_tag) {
  if (!g_hb || g_hb_slots <= 0) return nullptr;
  uint32_t* slot = g_hb + 4 * (g_hb_next.fetch_add(1, std::memory_order_relaxed) % g_hb_slots);
  (void)kernel_tag;
  return slot;
}

bool current_context_id(uint64_t* id) {
  ensure_context();
  const CtxGetCurrentFn get = ctx_get_current_fn();
  const CtxGetIdFn get_id = ctx_get_id_fn();
  CUcontext c = nullptr;
  unsigned long long v = 0;
  if (!get || !get_id || get(&c) != CUDA_SUCCESS || !c || get_id(c, &v) != CUDA_SUCCESS) return false;
  *id = static_cast<uint64_t>(v);
  return true;
}

// The status record's device address belongs to the context it was looked up in: a
// caller's own (non-primary) context, or the primary context re-created after a
// cudaDeviceReset, gets its own lookup, keyed on the context's process-unique id.
int* device_status_ptr() {
  uint64_t ctx = 0;
  if (!current_context_id(&ctx)) return nullptr;
  thread_local uint64_t t_ctx = 0;
  thread_local int* t_ptr = nullptr;
  if (t_ptr && t_ctx == ctx) return t_ptr;
  static std::mutex mu;
  static std::vector<std::pair<uint64_t, int*>> cache;
  std::lock_guard<std::mutex> lock(mu);
  int* found = nullptr;
  for (const auto& e : cache)
    if (e.first == ctx) found = e.second;
  if (!found) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_status) != cudaSuccess || !p) return nullptr;
    found = static_cast<int*>(p);
    if (cache.size() >= 256) cache.erase(cache.begin());
    cache.emplace_back(ctx, found);
  }
  t_ctx = ctx;
  t_ptr = found;
  return found;
}

cudaError_t set_smem_limit_once(const void* func, int bytes) {
  static std::mutex mu;
  static std::set<std::pair<int, const void*>> done;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  if (done.count({dev, func})) return cudaSuccess;
  e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) done.insert({dev, func});
  return e;
}

bool encode_tmap_3d(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2,
                    uint64_t stride1_bytes, uint64_t stride2_bytes, uint32_t b0, uint32_t b1,
                    uint32_t b2) {
  ensure_context();
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {d0, d1, d2};
  cuuint64_t strides[2] = {stride1_bytes, stride2_bytes};
  cuuint32_t box[3] = {b0, b1, b2};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_tmap_4d(CUtensorMap* m, const void* base, const uint64_t dims4[4], const uint64_t strides3[3],
                    const uint32_t box4[4], bool u8) {
  ensure_context();
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[4] = {dims4[0], dims4[1], dims4[2], dims4[3]};
  cuuint64_t strides[3] = {strides3[0], strides3[1], strides3[2]};
  cuuint32_t box[4] = {box4[0], box4[1], box4[2], box4[3]};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  return fn(m, u8 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_tmap_3d_u8(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2,
                       uint64_t stride1_bytes, uint64_t stride2_bytes, uint32_t b0, uint32_t b1, uint32_t b2) {
  ensure_context();
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {d0, d1, d2};
  cuuint64_t strides[2] = {stride1_bytes, stride2_bytes};
  cuuint32_t box[3] = {b0, b1, b2};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_tmap_2d_u8(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t stride1_bytes,
                       uint32_t b0, uint32_t b1) {
  ensure_context();
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {d0, d1};
  cuuint64_t strides[1] = {stride1_bytes};
  cuuint32_t box[2] = {b0, b1};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_tmap_2d(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1,
                    uint64_t stride1_bytes, uint32_t b0, uint32_t b1) {
  ensure_context();
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {d0, d1};
  cuuint64_t strides[1] = {stride1_bytes};
  cuuint32_t box[2] = {b0, b1};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_tmap_2d_f32(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t stride1_bytes,
                        uint32_t b0, uint32_t b1) {
  ensure_context();
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {d0, d1};
  cuuint64_t strides[1] = {stride1_bytes};
  cuuint32_t box[2] = {b0, b1};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// ------------------------------------------------------------ ring bookkeeping
namespace {

ispa_status check_ring(const ispa_kv_ring* r) {
  if (!r) return ISPA_ERR_INVALID_ARG;
  if (r->num_heads <= 0 || r->tokens_per_frame <= 0 || r->capacity_frames <= 0 ||
      r->n_sink_frames < 0 || r->n_sink_frames >= r->capacity_frames || r->frames_written < 0)
    return ISPA_ERR_INVALID_ARG;
  if (r->head_dim != 64 && r->head_dim != 128) return ISPA_ERR_UNSUPPORTED;
  if (r->k_format != ISPA_KV_BF16 && r->k_format != ISPA_KV_K_E4M3 && r->k_format != ISPA_KV_KV_E4M3)
    return ISPA_ERR_INVALID_ARG;
  if (r->k_format != ISPA_KV_BF16 && r->head_dim != 128) return ISPA_ERR_UNSUPPORTED;
  if (r->k_format == ISPA_KV_KV_E4M3 && r->tokens_per_frame % 4 != 0) return ISPA_ERR_UNSUPPORTED;
  if (static_cast<int64_t>(r->capacity_frames) * r->tokens_per_frame > INT32_MAX)
    return ISPA_ERR_INVALID_ARG;
  return ISPA_OK;
}

bool resident(const ispa_kv_ring* r, int64_t f) {
  if (f < 0 || f >= r->frames_written) return false;
  if (f < r->n_sink_frames) return true;
  return r->frames_written - f <= r->capacity_frames - r->n_sink_frames;
}

int32_t slot_of(const ispa_kv_ring* r, int64_t f) {
  if (f < r->n_sink_frames) return static_cast<int32_t>(f);
  return r->n_sink_frames +
         static_cast<int32_t>((f - r->n_sink_frames) % (r->capacity_frames - r->n_sink_frames));
}

// Maximal runs of set entries of a slot mask.
bool mask_runs(const std::vector<uint8_t>& m, ispa_slot_range* out, int32_t* n) {
  *n = 0;
  const int cap = static_cast<int>(m.size());
  for (int s = 0; s < cap;) {
    if (!m[s]) {
      ++s;
      continue;
    }
    int e = s;
    while (e < cap && m[e]) ++e;
    if (*n >= ISPA_MAX_RANGES) return false;
    out[*n].first_slot = s;
    out[*n].n_slots = e - s;
    ++*n;
    s = e;
  }
  return true;
}

ispa_status resolve(const ispa_kv_ring* r, ispa_window win, ispa_key_sets* ks) {
  if (win.n_sink_frames < 0 || win.n_recent_frames < 0) return ISPA_ERR_INVALID_ARG;
  memset(ks, 0, sizeof(*ks));
  const int64_t F = r->frames_written;
  const int cap = r->capacity_frames;
  std::vector<uint8_t> full(cap, 0), loc(cap, 0), hist(cap, 0);
  for (int64_t f = 0; f < std::min<int64_t>(r->n_sink_frames, F); ++f) full[slot_of(r, f)] = 1;
  for (int64_t f = std::max<int64_t>(r->n_sink_frames, F - (cap - r->n_sink_frames)); f < F; ++f)
    full[slot_of(r, f)] = 1;
  auto mark_local = [&](int64_t f) -> bool {
    if (!resident(r, f)) return false;
    loc[slot_of(r, f)] = 1;
    return true;
  };
  for (int64_t f = 0; f < std::min<int64_t>(win.n_sink_frames, F); ++f)
    if (!mark_local(f)) return ISPA_ERR_CAPACITY;
  for (int64_t f = std::max<int64_t>(0, F - win.n_recent_frames); f < F; ++f)
    if (!mark_local(f)) return ISPA_ERR_CAPACITY;
  for (int s = 0; s < cap; ++s) hist[s] = full[s] && !loc[s];
  if (!mask_runs(full, ks->full, &ks->n_full) || !mask_runs(loc, ks->local, &ks->n_local) ||
      !mask_runs(hist, ks->hist, &ks->n_hist))
    return ISPA_ERR_INVALID_ARG;
  return ISPA_OK;
}

// ------------------------------------------------------------ attention driver
enum Mode { MODE_FULL, MODE_LOCAL, MODE_DUAL, MODE_HIST };

// align16: start every segment on a 16-key boundary (the d-major value tiles of the 8-bit P V
// are TMA boxes whose first key must be a multiple of 16); the keys before the run are masked.
int add_segs(AttnParams& p, int src, const ispa_slot_range* r, int n, int P, int bn, bool align16 = false) {
  int tiles = 0;
  for (int i = 0; i < n; ++i) {
    AttnSeg& s = p.seg[p.n_seg++];
    s.src = src;
    const int first = r[i].first_slot * P;
    s.skip = align16 ? first & 15 : 0;
    s.start = first - s.skip;
    s.count = r[i].n_slots * P + s.skip;
    tiles += (s.count + bn - 1) / bn;
  }
  return tiles;
}

// 8-bit Q K^T: per-head e4m3 code scales of q, of the chunk keys and of the ring keys; with 8-bit
// P V also the values' per-head scale and the row stride of the chunk's d-major value codes.
struct Qk8Scales {
  const float* q;
  const float* k_cur;
  const float* k_ring;
  const float* v = nullptr;
  int64_t vt_ld = 0;
};

ispa_status attn_common(Mode mode, const ispa_kv_ring* ring, ispa_window win, const void* q,
                        const void* k_cur, const void* v_cur, int32_t n_q, float scale, uint32_t flags,
                        void* out, void* out_loc, float* lse, float* lse_loc, float* disc_part,
                        cudaStream_t stream, const Qk8Scales* qk8 = nullptr) {
  ispa_status st = check_ring(ring);
  if (st != ISPA_OK) return st;
  if ((ring->k_format != ISPA_KV_BF16) != (qk8 != nullptr)) return ISPA_ERR_INVALID_ARG;
  if (qk8 && (!qk8->q || !qk8->k_cur || !qk8->k_ring)) return ISPA_ERR_INVALID_ARG;
  const bool kv8 = ring->k_format == ISPA_KV_KV_E4M3;
  if (kv8 && (!qk8->v || qk8->vt_ld < n_q || qk8->vt_ld % 16 != 0)) return ISPA_ERR_INVALID_ARG;
  if (!kv8 && qk8 && qk8->v) return ISPA_ERR_INVALID_ARG;   // 8-bit P V needs a ring with e4m3 values
  if (flags & ~static_cast<uint32_t>(ISPA_ATTN_FRAME_CAUSAL)) return ISPA_ERR_INVALID_ARG;
  if ((flags & ISPA_ATTN_FRAME_CAUSAL) && n_q % ring->tokens_per_frame != 0) return ISPA_ERR_INVALID_ARG;
  if (n_q <= 0 || !aligned16(q) || !aligned16(k_cur) || !aligned16(v_cur) || !aligned16(out) ||
      !aligned16(ring->k) || !aligned16(ring->v))
    return ISPA_ERR_INVALID_ARG;
  if (mode == MODE_DUAL && (!aligned16(out_loc) || !disc_part)) return ISPA_ERR_INVALID_ARG;
  if (!(scale >= 0.f) || !isfinite(scale)) return ISPA_ERR_INVALID_ARG;
  ispa_key_sets ks;
  st = resolve(ring, mode == MODE_FULL ? ispa_window{0, 0} : win, &ks);
  if (st != ISPA_OK) return st;

  const int H = ring->num_heads, HD = ring->head_dim, P = ring->tokens_per_frame;
  const int bn = kAttnBN;   // keys per tile: the TMA box height of K and V and the tile count
  AttnParams p;
  memset(&p, 0, sizeof(p));
  p.n_q = n_q;
  p.num_heads = H;
  const ispa_slot_range chunk{0, 0};
  (void)chunk;
  int tiles = 0;
  const bool al = ring->k_format == ISPA_KV_KV_E4M3;
  if (mode == MODE_HIST) {
    // Eq. 10: the history set alone, no chunk
    tiles = add_segs(p, 0, ks.hist, ks.n_hist, P, bn, al);
    if (tiles == 0) return launch_empty_branch(out, lse, n_q, H, HD, stream) == cudaSuccess ? ISPA_OK : ISPA_ERR_CUDA;
    p.n_local_tiles = tiles;
    p.n_tiles = tiles;
  } else if (mode == MODE_FULL) {
    tiles += add_segs(p, 0, ks.full, ks.n_full, P, bn, al);
  } else {
    tiles += add_segs(p, 0, ks.local, ks.n_local, P, bn, al);
  }
  if (mode != MODE_HIST) {
    AttnSeg& s = p.seg[p.n_seg++];
    s.src = 1;
    s.start = 0;
    s.count = n_q;
    tiles += (n_q + bn - 1) / bn;
  }
  if (mode != MODE_HIST) {
    p.n_local_tiles = tiles;
    if (mode == MODE_DUAL) tiles += add_segs(p, 0, ks.hist, ks.n_hist, P, bn, al);
    p.n_tiles = tiles;
  }
  p.dual = mode == MODE_DUAL ? 1 : 0;
  p.causal_p = (flags & ISPA_ATTN_FRAME_CAUSAL) ? P : 0;
  const float sc = scale == 0.f ? 1.f / sqrtf(static_cast<float>(HD)) : scale;
  p.scale_log2 = sc * 1.4426950408889634f;
  p.wait_limit_ns = g_wait_limit.load();
  p.out = static_cast<__nv_bfloat16*>(out);
  p.out_loc = static_cast<__nv_bfloat16*>(out_loc);
  p.lse = lse;
  p.lse_loc = lse_loc;
  p.disc_part = disc_part;
  p.status = device_status_ptr();
  if (!p.status) return ISPA_ERR_CUDA;
  p.heartbeat = next_heartbeat_slot(1);
  p.trace = trace_buffer(&p.trace_tiles);
  p.drop_k_tile = g_drop_k_tile;

  // Every map views a [rows][d] bf16 operand as (64 columns, rows, d/64 column blocks, heads):
  // the column-block stride (128 B) is smaller than the row stride, so one box of
  // (64, rows, d/64, 1) fetches all of a tile's columns in a single request and lands in
  // shared memory as d/64 consecutive [rows][128 B] swizzled blocks -- the UMMA operand
  // layout.  Fewer, larger requests give the TMA unit about 1.5x the throughput of one
  // request per 64-column block.
  const uint64_t row_b = static_cast<uint64_t>(HD) * 2;
  const uint64_t ring_tok = static_cast<uint64_t>(ring->capacity_frames) * P;
  const uint32_t nb = static_cast<uint32_t>(HD / 64);
  const uint64_t dims_c[4] = {64, static_cast<uint64_t>(n_q), nb, static_cast<uint64_t>(H)};
  const uint64_t str_c[3] = {row_b * H, 128, row_b};
  const uint64_t dims_r[4] = {64, ring_tok, nb, static_cast<uint64_t>(H)};
  const uint64_t str_r[3] = {row_b, 128, row_b * ring_tok};
  const uint32_t box_q[4] = {64, static_cast<uint32_t>(kAttnBM), nb, 1};
  const uint32_t box_k[4] = {64, static_cast<uint32_t>(bn), nb, 1};
  CUtensorMap tq, tkr, tvr, tkc, tvc;
  bool ok;
  if (kv8) {
    // d-major e4m3 values [H][128][keys]: boxes of 128 keys x 128 rows, 128-byte swizzle (the
    // K-major B operand of the 8-bit P V)
    const uint64_t vt_ring = ispa_ring_vt_stride(ring);
    ok = encode_tmap_3d_u8(&tvc, v_cur, static_cast<uint64_t>(n_q), 128, static_cast<uint64_t>(H),
                           static_cast<uint64_t>(qk8->vt_ld), static_cast<uint64_t>(qk8->vt_ld) * 128, 128, 128, 1) &&
         encode_tmap_3d_u8(&tvr, ring->v, ring_tok, 128, static_cast<uint64_t>(H), vt_ring, vt_ring * 128, 128, 128,
                           1);
    p.v_scale = qk8->v;
  } else {
    ok = encode_tmap_4d(&tvc, v_cur, dims_c, str_c, box_k) && encode_tmap_4d(&tvr, ring->v, dims_r, str_r, box_k);
  }
  if (qk8) {
    // e4m3 Q and K: a token's 128 features are one 128-byte row, so the column-block
    // dimension has extent 1
    const uint64_t dims_c8[4] = {128, static_cast<uint64_t>(n_q), 1, static_cast<uint64_t>(H)};
    const uint64_t str_c8[3] = {128ull * H, 128, 128};
    const uint64_t dims_r8[4] = {128, ring_tok, 1, static_cast<uint64_t>(H)};
    const uint64_t str_r8[3] = {128, 128, 128 * ring_tok};
    const uint32_t box_q8[4] = {128, static_cast<uint32_t>(kAttnBM), 1, 1};
    const uint32_t box_k8[4] = {128, static_cast<uint32_t>(kAttnBN), 1, 1};
    ok = ok && encode_tmap_4d(&tq, q, dims_c8, str_c8, box_q8, true) &&
         encode_tmap_4d(&tkc, k_cur, dims_c8, str_c8, box_k8, true) &&
         encode_tmap_4d(&tkr, ring->k, dims_r8, str_r8, box_k8, true);
    p.q_scale = qk8->q;
    p.kc_scale = qk8->k_cur;
    p.kr_scale = qk8->k_ring;
  } else {
    ok = ok && encode_tmap_4d(&tq, q, dims_c, str_c, box_q) && encode_tmap_4d(&tkc, k_cur, dims_c, str_c, box_k) &&
         encode_tmap_4d(&tkr, ring->k, dims_r, str_r, box_k);
  }
  if (!ok) return ISPA_ERR_CUDA;
  if (launch_attention(HD, &tq, &tkr, &tvr, &tkc, &tvc, p, stream) != cudaSuccess) return ISPA_ERR_CUDA;
  return ISPA_OK;
}

__global__ void wait_probe_kernel(uint64_t limit_ns, int* status) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(smem_u32(&bar), 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    WaitCtx w{&abort_flag, status, limit_ns};
    mbar_wait(smem_u32(&bar), 0, w);  // nothing ever arrives: runs out after limit_ns
  }
}

}  // namespace
}  // namespace ispa

using namespace ispa;

extern "C" {

const char* ispa_status_string(ispa_status s) {
  switch (s) {
    case ISPA_OK: return "ok";
    case ISPA_ERR_INVALID_ARG: return "invalid argument";
    case ISPA_ERR_UNSUPPORTED: return "unsupported shape";
    case ISPA_ERR_CAPACITY: return "ring capacity exceeded";
    case ISPA_ERR_NOT_SPD: return "matrix not positive definite";
    case ISPA_ERR_TIMEOUT: return "device wait timed out";
    case ISPA_ERR_CUDA: return "CUDA error";
    case ISPA_ERR_WORKSPACE: return "workspace too small";
  }
  return "unknown status";
}

ispa_status ispa_last_device_error(int32_t* code) {
  int rec[8] = {};
  if (cudaMemcpyFromSymbol(rec, g_status, sizeof(rec)) != cudaSuccess) return ISPA_ERR_CUDA;
  const int zero[8] = {};
  if (cudaMemcpyToSymbol(g_status, zero, sizeof(zero)) != cudaSuccess) return ISPA_ERR_CUDA;
  if (code) *code = rec[0];
  if (rec[0] == DEVERR_TIMEOUT) return ISPA_ERR_TIMEOUT;
  if (rec[0] == DEVERR_LAYOUT) return ISPA_ERR_CUDA;
  return ISPA_OK;
}

ispa_status ispa_debug_error_record(int32_t* rec8) {
  if (!rec8) return ISPA_ERR_INVALID_ARG;
  if (cudaMemcpyFromSymbol(rec8, g_status, 8 * sizeof(int)) != cudaSuccess) return ISPA_ERR_CUDA;
  return ISPA_OK;
}

ispa_status ispa_debug_set_trace(uint64_t* buf, int32_t n_tiles) {
  if ((buf == nullptr) != (n_tiles <= 0)) return ISPA_ERR_INVALID_ARG;
  g_trace = buf;
  g_trace_tiles = n_tiles;
  return ISPA_OK;
}

ispa_status ispa_debug_drop_k_tile(int32_t tile) {
  if (tile < -1) return ISPA_ERR_INVALID_ARG;
  g_drop_k_tile = tile;
  return ISPA_OK;
}

ispa_status ispa_debug_set_heartbeat(uint32_t* counters, int32_t n_slots) {
  if ((counters == nullptr) != (n_slots <= 0)) return ISPA_ERR_INVALID_ARG;
  g_hb = counters;
  g_hb_slots = n_slots;
  g_hb_next.store(0, std::memory_order_relaxed);
  return ISPA_OK;
}

uint64_t ispa_set_wait_limit_ns(uint64_t ns) {
  return g_wait_limit.exchange(ns == 0 ? kDefaultWaitLimitNs : ns);
}

ispa_status ispa_debug_wait_probe(uint64_t limit_ns, ispa_stream stream) {
  int* st = device_status_ptr();
  if (!st) return ISPA_ERR_CUDA;
  wait_probe_kernel<<<1, 32, 0, stream>>>(limit_ns, st);
  return cudaGetLastError() == cudaSuccess ? ISPA_OK : ISPA_ERR_CUDA;
}

size_t ispa_ring_bytes(const ispa_kv_ring* r) {
  if (!r || r->num_heads <= 0 || r->head_dim <= 0 || r->tokens_per_frame <= 0 || r->capacity_frames <= 0)
    return 0;
  const uint64_t elems = 1ull * r->num_heads * r->capacity_frames * r->tokens_per_frame * r->head_dim;
  if (r->k_format == ISPA_KV_KV_E4M3)
    return elems + 1ull * r->num_heads * r->head_dim * static_cast<uint64_t>(ispa_ring_vt_stride(r));
  return elems * (r->k_format == ISPA_KV_K_E4M3 ? 1ull : 2ull) + elems * 2ull;
}

int64_t ispa_ring_vt_stride(const ispa_kv_ring* r) {
  if (!r || r->tokens_per_frame <= 0 || r->capacity_frames <= 0) return 0;
  const int64_t keys = static_cast<int64_t>(r->capacity_frames) * r->tokens_per_frame;
  return (keys + 15) / 16 * 16;
}

int32_t ispa_ring_slot(const ispa_kv_ring* r, int64_t frame) {
  if (check_ring(r) == ISPA_ERR_INVALID_ARG || !resident(r, frame)) return -1;
  return slot_of(r, frame);
}

ispa_status ispa_window_resolve(const ispa_kv_ring* r, ispa_window win, ispa_key_sets* out) {
  if (!out) return ISPA_ERR_INVALID_ARG;
  const ispa_status st = check_ring(r);
  if (st != ISPA_OK) return st;
  return resolve(r, win, out);
}

ispa_status ispa_kv_append_layers(ispa_kv_ring* rings, int32_t n_layers, const void* const* k_new,
                                  const void* const* v_new, int32_t n_frames, ispa_stream stream) {
  if (!rings || !k_new || !v_new || n_layers <= 0 || n_layers > kMaxAppendLayers)
    return ISPA_ERR_INVALID_ARG;
  if (n_frames <= 0) return ISPA_ERR_INVALID_ARG;
  const ispa_kv_ring& r0 = rings[0];
  for (int l = 0; l < n_layers; ++l) {
    const ispa_status st = check_ring(&rings[l]);
    if (st != ISPA_OK) return st;
    const ispa_kv_ring& r = rings[l];
    if (r.k_format != ISPA_KV_BF16) return ISPA_ERR_INVALID_ARG;   // e4m3 keys: ispa_kv_append_qk8
    if (r.num_heads != r0.num_heads || r.head_dim != r0.head_dim || r.tokens_per_frame != r0.tokens_per_frame)
      return ISPA_ERR_INVALID_ARG;
    if (!aligned16(r.k) || !aligned16(r.v) || !aligned16(k_new[l]) || !aligned16(v_new[l]))
      return ISPA_ERR_INVALID_ARG;
    if (n_frames > kMaxAppendFrames || n_frames > r.capacity_frames - r.n_sink_frames) return ISPA_ERR_CAPACITY;
  }
  if (static_cast<int64_t>(n_frames) * r0.tokens_per_frame * r0.num_heads * (r0.head_dim / 8) >
      (int64_t{1} << 30))
    return ISPA_ERR_INVALID_ARG;
  AppendParams p;
  memset(&p, 0, sizeof(p));
  p.n_layers = n_layers;
  p.n_frames = n_frames;
  p.tokens_per_frame = r0.tokens_per_frame;
  p.num_heads = r0.num_heads;
  p.head_dim = r0.head_dim;
  for (int l = 0; l < n_layers; ++l) {
    const ispa_kv_ring& r = rings[l];
    p.capacity_tokens[l] = r.capacity_frames * r.tokens_per_frame;
    for (int i = 0; i < n_frames; ++i) p.slot[l][i] = slot_of(&r, r.frames_written + i);
    p.k_src[l] = k_new[l];
    p.v_src[l] = v_new[l];
    p.k_dst[l] = r.k;
    p.v_dst[l] = r.v;
  }
  if (launch_append(p, stream) != cudaSuccess) return ISPA_ERR_CUDA;
  for (int l = 0; l < n_layers; ++l) rings[l].frames_written += n_frames;
  return ISPA_OK;
}

ispa_status ispa_kv_append(ispa_kv_ring* ring, const void* k_new, const void* v_new,
                           int32_t n_frames, ispa_stream stream) {
  if (!ring) return ISPA_ERR_INVALID_ARG;
  const void* k[1] = {k_new};
  const void* v[1] = {v_new};
  return ispa_kv_append_layers(ring, 1, k, v, n_frames, stream);
}

ispa_status ispa_attn_full_ex(const ispa_kv_ring* ring, const void* q, const void* k_cur,
                              const void* v_cur, int32_t n_q, float scale, uint32_t flags, void* out,
                              float* lse, ispa_stream stream) {
  return attn_common(MODE_FULL, ring, ispa_window{0, 0}, q, k_cur, v_cur, n_q, scale, flags, out, nullptr,
                     lse, nullptr, nullptr, stream);
}

ispa_status ispa_attn_full(const ispa_kv_ring* ring, const void* q, const void* k_cur,
                           const void* v_cur, int32_t n_q, float scale, void* out, float* lse,
                           ispa_stream stream) {
  return ispa_attn_full_ex(ring, q, k_cur, v_cur, n_q, scale, 0u, out, lse, stream);
}

ispa_status ispa_attn_local_ex(const ispa_kv_ring* ring, ispa_window win, const void* q,
                               const void* k_cur, const void* v_cur, int32_t n_q, float scale,
                               uint32_t flags, void* out, float* lse, ispa_stream stream) {
  return attn_common(MODE_LOCAL, ring, win, q, k_cur, v_cur, n_q, scale, flags, out, nullptr, lse, nullptr,
                     nullptr, stream);
}

ispa_status ispa_attn_local(const ispa_kv_ring* ring, ispa_window win, const void* q,
                            const void* k_cur, const void* v_cur, int32_t n_q, float scale,
                            void* out, float* lse, ispa_stream stream) {
  return ispa_attn_local_ex(ring, win, q, k_cur, v_cur, n_q, scale, 0u, out, lse, stream);
}

ispa_status ispa_attn_hist(const ispa_kv_ring* ring, ispa_window win, const void* q, int32_t n_q, float scale,
                           void* out, float* lse, ispa_stream stream) {
  if (!lse) return ISPA_ERR_INVALID_ARG;
  // the chunk tensors are not read in this mode; q stands in for them in the unused maps
  return attn_common(MODE_HIST, ring, win, q, q, q, n_q, scale, 0u, out, nullptr, lse, nullptr, nullptr, stream);
}

size_t ispa_attn_dual_workspace_size(int32_t num_heads, int32_t n_q) {
  if (num_heads <= 0 || n_q <= 0) return 0;
  return static_cast<size_t>(num_heads) * n_q * sizeof(float);
}

ispa_status ispa_attn_dual_ex(const ispa_kv_ring* ring, ispa_window win, const void* q,
                              const void* k_cur, const void* v_cur, int32_t n_q, float scale, uint32_t flags,
                              void* a_full, void* a_loc, float* disc, float* disc_sq_sum,
                              float* lse_full, float* lse_loc, void* workspace, size_t ws_bytes,
                              ispa_stream stream) {
  if (!ring || !disc || !disc_sq_sum) return ISPA_ERR_INVALID_ARG;
  const size_t need = ispa_attn_dual_workspace_size(ring->num_heads, n_q);
  if (need == 0) return ISPA_ERR_INVALID_ARG;
  if (!workspace || ws_bytes < need || !aligned16(workspace)) return ISPA_ERR_WORKSPACE;
  float* part = static_cast<float*>(workspace);
  const ispa_status st = attn_common(MODE_DUAL, ring, win, q, k_cur, v_cur, n_q, scale, flags, a_full,
                                     a_loc, lse_full, lse_loc, part, stream);
  if (st != ISPA_OK) return st;
  if (launch_disc_reduce(part, ring->num_heads, n_q, disc, disc_sq_sum, stream) != cudaSuccess)
    return ISPA_ERR_CUDA;
  return ISPA_OK;
}

ispa_status ispa_attn_dual(const ispa_kv_ring* ring, ispa_window win, const void* q,
                           const void* k_cur, const void* v_cur, int32_t n_q, float scale,
                           void* a_full, void* a_loc, float* disc, float* disc_sq_sum,
                           float* lse_full, float* lse_loc, void* workspace, size_t ws_bytes,
                           ispa_stream stream) {
  return ispa_attn_dual_ex(ring, win, q, k_cur, v_cur, n_q, scale, 0u, a_full, a_loc, disc, disc_sq_sum,
                           lse_full, lse_loc, workspace, ws_bytes, stream);
}

size_t ispa_ls_state_bytes(int32_t dim) {
  if (dim <= 0) return 0;
  return 4ull * dim * dim * sizeof(float);
}

ispa_status ispa_ls_state_reset(ispa_ls_state* st, ispa_stream stream) {
  if (!st || st->dim <= 0 || !aligned16(st->gram)) return ISPA_ERR_INVALID_ARG;
  if (cudaMemsetAsync(st->gram, 0, ispa_ls_state_bytes(st->dim), stream) != cudaSuccess)
    return ISPA_ERR_CUDA;
  st->n_tokens = 0;
  return ISPA_OK;
}

size_t ispa_ls_accumulate_workspace_size(int32_t dim, int64_t T) {
  if (dim <= 0 || T <= 0) return 0;
  return ls_accumulate_ws_bytes(dim, T);
}

ispa_status ispa_ls_accumulate_ex(ispa_ls_state* st, const void* a_loc, const void* a_full, int64_t T,
                                  uint32_t flags, void* workspace, size_t ws_bytes, ispa_stream stream) {
  if (!st || st->dim <= 0 || T <= 0 || T > INT32_MAX || !aligned16(st->gram) || !aligned16(a_loc) ||
      !aligned16(a_full))
    return ISPA_ERR_INVALID_ARG;
  if (flags & ~static_cast<uint32_t>(ISPA_LS_EXACT_DELTA)) return ISPA_ERR_INVALID_ARG;
  if (st->dim % 128 != 0) return ISPA_ERR_UNSUPPORTED;
  const size_t need = ls_accumulate_ws_bytes(st->dim, T);
  if (!workspace || ws_bytes < need || !aligned16(workspace)) return ISPA_ERR_WORKSPACE;
  int* status = device_status_ptr();
  if (!status) return ISPA_ERR_CUDA;
  if (launch_ls_accumulate(st->dim, T, a_loc, a_full, workspace, (flags & ISPA_LS_EXACT_DELTA) != 0, st->gram,
                           status, g_wait_limit.load(), next_heartbeat_slot(2), stream) != cudaSuccess)
    return ISPA_ERR_CUDA;
  st->n_tokens += T;
  return ISPA_OK;
}

ispa_status ispa_ls_accumulate(ispa_ls_state* st, const void* a_loc, const void* a_full, int64_t T,
                               void* workspace, size_t ws_bytes, ispa_stream stream) {
  return ispa_ls_accumulate_ex(st, a_loc, a_full, T, 0u, workspace, ws_bytes, stream);
}

size_t ispa_ls_solve_workspace_size(int32_t dim, int32_t d_out) {
  if (dim <= 0 || d_out <= 0) return 0;
  return ls_solve_ws_bytes(dim, d_out);
}

ispa_status ispa_ls_solve(const ispa_ls_state* st, const float* W, int32_t d_out, double lambda,
                          float* dW, double* eps_out, void* workspace, size_t ws_bytes,
                          ispa_stream stream) {
  if (!st || st->dim <= 0 || d_out <= 0 || !aligned16(st->gram) || !aligned16(W) || !aligned16(dW))
    return ISPA_ERR_INVALID_ARG;
  if (!(lambda >= 0.0) || !isfinite(lambda)) return ISPA_ERR_INVALID_ARG;
  const size_t need = ls_solve_ws_bytes(st->dim, d_out);
  if (!workspace || ws_bytes < need || !aligned16(workspace)) return ISPA_ERR_WORKSPACE;
  return run_ls_solve(st->dim, st->gram, W, d_out, lambda, dW, eps_out, workspace, stream);
}

// ------------------------------------------------------------ W8A8 projection (Sec. 4)

ispa_status ispa_quantize_rows_e4m3(const void* x, int64_t rows, int32_t cols, uint8_t* q, float* scale,
                                    ispa_stream stream) {
  if (!x || !q || !scale || rows <= 0 || cols <= 0 || !aligned16(x) || !aligned16(q)) return ISPA_ERR_INVALID_ARG;
  if (cols % 16 != 0) return ISPA_ERR_UNSUPPORTED;
  if (launch_quant_rows(x, rows, cols, q, scale, stream) != cudaSuccess) return ISPA_ERR_CUDA;
  return ISPA_OK;
}

ispa_status ispa_quantize_weight_e4m3(const float* W, const float* dW, int32_t D, int32_t D_out, uint8_t* q_t,
                                      float* scale, ispa_stream stream) {
  if (!W || !q_t || !scale || D <= 0 || D_out <= 0 || !aligned16(q_t)) return ISPA_ERR_INVALID_ARG;
  if (D % 16 != 0) return ISPA_ERR_UNSUPPORTED;
  if (launch_quant_weight(W, dW, D, D_out, q_t, scale, stream) != cudaSuccess) return ISPA_ERR_CUDA;
  return ISPA_OK;
}

ispa_status ispa_linear_w8a8(const uint8_t* a_q, const float* a_scale, const uint8_t* w_q, const float* w_scale,
                             int64_t T, int32_t D, int32_t D_out, void* out, ispa_stream stream) {
  if (!a_q || !a_scale || !w_q || !w_scale || !out || T <= 0 || T > INT32_MAX || D <= 0 || D_out <= 0 ||
      !aligned16(a_q) || !aligned16(w_q) || !aligned16(w_scale) || !aligned16(out))
    return ISPA_ERR_INVALID_ARG;
  if (D % 128 != 0 || D_out % 128 != 0) return ISPA_ERR_UNSUPPORTED;
  int* status = device_status_ptr();
  if (!status) return ISPA_ERR_CUDA;
  if (launch_w8a8_gemm(a_q, a_scale, w_q, w_scale, static_cast<int32_t>(T), D, D_out, out, status, g_wait_limit.load(),
                       stream) != cudaSuccess)
    return ISPA_ERR_CUDA;
  return ISPA_OK;
}


// ------------------------------------------------------------ 8-bit Q K^T attention

ispa_status ispa_quantize_heads_e4m3(const void* x, int64_t n, int32_t H, int32_t d, uint8_t* q, float* scale,
                                     ispa_stream stream) {
  if (!x || !q || !scale || n <= 0 || H <= 0 || d <= 0 || !aligned16(x) || !aligned16(q))
    return ISPA_ERR_INVALID_ARG;
  if (d % 16 != 0 || H > 256) return ISPA_ERR_UNSUPPORTED;
  if (launch_quant_heads(x, n, H, d, q, scale, stream) != cudaSuccess) return ISPA_ERR_CUDA;
  return ISPA_OK;
}

ispa_status ispa_quantize_q_e4m3(const void* x, int64_t n, int32_t H, int32_t d, uint8_t* q, float* scale,
                                 ispa_stream stream) {
  if (!x || !q || !scale || n <= 0 || H <= 0 || d <= 0 || !aligned16(x) || !aligned16(q))
    return ISPA_ERR_INVALID_ARG;
  if (d % 16 != 0 || d > 256 || H > 65535) return ISPA_ERR_UNSUPPORTED;
  if (launch_quant_q_blocks(x, n, H, d, q, scale, stream) != cudaSuccess) return ISPA_ERR_CUDA;
  return ISPA_OK;
}

ispa_status ispa_quantize_k_e4m3(const void* x, int64_t n, int32_t H, int32_t d, const float* scale, uint8_t* q,
                                 ispa_stream stream) {
  if (!x || !q || !scale || n <= 0 || H <= 0 || d <= 0 || !aligned16(x) || !aligned16(q))
    return ISPA_ERR_INVALID_ARG;
  if (d % 16 != 0) return ISPA_ERR_UNSUPPORTED;
  if (launch_quant_given(x, n, H, d, scale, q, stream) != cudaSuccess) return ISPA_ERR_CUDA;
  return ISPA_OK;
}

ispa_status ispa_kv_append_qk8(ispa_kv_ring* ring, const void* k_new, const void* v_new, int32_t n_frames,
                               const float* k_scale, ispa_stream stream) {
  const ispa_status st = check_ring(ring);
  if (st != ISPA_OK) return st;
  if (ring->k_format != ISPA_KV_K_E4M3 || !k_new || !v_new || !k_scale || n_frames <= 0) return ISPA_ERR_INVALID_ARG;
  if (!aligned16(ring->k) || !aligned16(ring->v) || !aligned16(k_new) || !aligned16(v_new))
    return ISPA_ERR_INVALID_ARG;
  if (n_frames > kMaxAppendFrames || n_frames > ring->capacity_frames - ring->n_sink_frames) return ISPA_ERR_CAPACITY;
  int32_t slots[kMaxAppendFrames];
  for (int i = 0; i < n_frames; ++i) slots[i] = slot_of(ring, ring->frames_written + i);
  const int64_t ring_tok = static_cast<int64_t>(ring->capacity_frames) * ring->tokens_per_frame;
  if (launch_append_qk8(slots, n_frames, ring->tokens_per_frame, ring->num_heads, ring->head_dim, ring_tok, k_new,
                        v_new, ring->k, ring->v, k_scale, stream) != cudaSuccess)
    return ISPA_ERR_CUDA;
  ring->frames_written += n_frames;
  return ISPA_OK;
}

ispa_status ispa_quantize_vt_e4m3(const void* x, int64_t n, int32_t H, int32_t d, const float* scale, uint8_t* qt,
                                  int64_t ld, ispa_stream stream) {
  if (!x || !scale || !qt || n <= 0 || H <= 0 || !aligned16(x) || !aligned16(qt) || ld < n || ld % 16 != 0)
    return ISPA_ERR_INVALID_ARG;
  if (d != 128) return ISPA_ERR_UNSUPPORTED;
  if (launch_quant_vt(x, n, H, d, scale, qt, ld, 0, 0, nullptr, stream) != cudaSuccess) return ISPA_ERR_CUDA;
  return ISPA_OK;
}

ispa_status ispa_kv_append_kv8(ispa_kv_ring* ring, const void* k_new, const void* v_new, int32_t n_frames,
                               const float* k_scale, const float* v_scale, ispa_stream stream) {
  const ispa_status st = check_ring(ring);
  if (st != ISPA_OK) return st;
  if (ring->k_format != ISPA_KV_KV_E4M3 || !k_new || !v_new || !k_scale || !v_scale || n_frames <= 0)
    return ISPA_ERR_INVALID_ARG;
  if (!aligned16(ring->k) || !aligned16(ring->v) || !aligned16(k_new) || !aligned16(v_new))
    return ISPA_ERR_INVALID_ARG;
  if (n_frames > kMaxAppendFrames || n_frames > ring->capacity_frames - ring->n_sink_frames) return ISPA_ERR_CAPACITY;
  int32_t slots[kMaxAppendFrames];
  for (int i = 0; i < n_frames; ++i) slots[i] = slot_of(ring, ring->frames_written + i);
  const int32_t P = ring->tokens_per_frame;
  const int64_t ring_tok = static_cast<int64_t>(ring->capacity_frames) * P;
  if (launch_append_qk8(slots, n_frames, P, ring->num_heads, ring->head_dim, ring_tok, k_new, v_new, ring->k,
                        nullptr, k_scale, stream) != cudaSuccess ||
      launch_quant_vt(v_new, static_cast<int64_t>(n_frames) * P, ring->num_heads, ring->head_dim, v_scale,
                      static_cast<uint8_t*>(ring->v), ispa_ring_vt_stride(ring), P, n_frames, slots,
                      stream) != cudaSuccess)
    return ISPA_ERR_CUDA;
  ring->frames_written += n_frames;
  return ISPA_OK;
}

ispa_status ispa_attn_full_kv8(const ispa_kv_ring* ring, const float* k_ring_scale, const float* v_scale,
                               const void* q8, const float* q_scale, const void* k8_cur, const float* k_cur_scale,
                               const void* vt8_cur, int64_t vt_ld, int32_t n_q, float scale, void* out, float* lse,
                               ispa_stream stream) {
  const Qk8Scales sc{q_scale, k_cur_scale, k_ring_scale, v_scale, vt_ld};
  return attn_common(MODE_FULL, ring, ispa_window{0, 0}, q8, k8_cur, vt8_cur, n_q, scale, 0u, out, nullptr, lse,
                     nullptr, nullptr, stream, &sc);
}

ispa_status ispa_attn_local_kv8(const ispa_kv_ring* ring, const float* k_ring_scale, const float* v_scale,
                                ispa_window win, const void* q8, const float* q_scale, const void* k8_cur,
                                const float* k_cur_scale, const void* vt8_cur, int64_t vt_ld, int32_t n_q, float scale,
                                void* out, float* lse, ispa_stream stream) {
  const Qk8Scales sc{q_scale, k_cur_scale, k_ring_scale, v_scale, vt_ld};
  return attn_common(MODE_LOCAL, ring, win, q8, k8_cur, vt8_cur, n_q, scale, 0u, out, nullptr, lse, nullptr,
                     nullptr, stream, &sc);
}

ispa_status ispa_attn_dual_kv8(const ispa_kv_ring* ring, const float* k_ring_scale, const float* v_scale,
                               ispa_window win, const void* q8, const float* q_scale, const void* k8_cur,
                               const float* k_cur_scale, const void* vt8_cur, int64_t vt_ld, int32_t n_q, float scale,
                               void* a_full, void* a_loc, float* disc, float* disc_sq_sum, float* lse_full,
                               float* lse_loc, void* workspace, size_t ws_bytes, ispa_stream stream) {
  if (!ring || !disc || !disc_sq_sum) return ISPA_ERR_INVALID_ARG;
  const size_t need = ispa_attn_dual_workspace_size(ring->num_heads, n_q);
  if (need == 0) return ISPA_ERR_INVALID_ARG;
  if (!workspace || ws_bytes < need || !aligned16(workspace)) return ISPA_ERR_WORKSPACE;
  float* part = static_cast<float*>(workspace);
  const Qk8Scales sc{q_scale, k_cur_scale, k_ring_scale, v_scale, vt_ld};
  const ispa_status st = attn_common(MODE_DUAL, ring, win, q8, k8_cur, vt8_cur, n_q, scale, 0u, a_full, a_loc,
                                     lse_full, lse_loc, part, stream, &sc);
  if (st != ISPA_OK) return st;
  if (launch_disc_reduce(part, ring->num_heads, n_q, disc, disc_sq_sum, stream) != cudaSuccess)
    return ISPA_ERR_CUDA;
  return ISPA_OK;
}

ispa_status ispa_attn_full_qk8(const ispa_kv_ring* ring, const float* k_ring_scale, const void* q8,
                               const float* q_scale, const void* k8_cur, const float* k_cur_scale, const void* v_cur,
                               int32_t n_q, float scale, void* out, float* lse, ispa_stream stream) {
  const Qk8Scales sc{q_scale, k_cur_scale, k_ring_scale};
  return attn_common(MODE_FULL, ring, ispa_window{0, 0}, q8, k8_cur, v_cur, n_q, scale, 0u, out, nullptr, lse,
                     nullptr, nullptr, stream, &sc);
}

ispa_status ispa_attn_dual_qk8(const ispa_kv_ring* ring, const float* k_ring_scale, ispa_window win, const void* q8,
                               const float* q_scale, const void* k8_cur, const float* k_cur_scale, const void* v_cur,
                               int32_t n_q, float scale, void* a_full, void* a_loc, float* disc, float* disc_sq_sum,
                               float* lse_full, float* lse_loc, void* workspace, size_t ws_bytes, ispa_stream stream) {
  if (!ring || !disc || !disc_sq_sum) return ISPA_ERR_INVALID_ARG;
  const size_t need = ispa_attn_dual_workspace_size(ring->num_heads, n_q);
  if (need == 0) return ISPA_ERR_INVALID_ARG;
  if (!workspace || ws_bytes < need || !aligned16(workspace)) return ISPA_ERR_WORKSPACE;
  float* part = static_cast<float*>(workspace);
  const Qk8Scales sc{q_scale, k_cur_scale, k_ring_scale};
  const ispa_status st = attn_common(MODE_DUAL, ring, win, q8, k8_cur, v_cur, n_q, scale, 0u, a_full, a_loc,
                                     lse_full, lse_loc, part, stream, &sc);
  if (st != ISPA_OK) return st;
  if (launch_disc_reduce(part, ring->num_heads, n_q, disc, disc_sq_sum, stream) != cudaSuccess)
    return ISPA_ERR_CUDA;
  return ISPA_OK;
}

ispa_status ispa_attn_local_qk8(const ispa_kv_ring* ring, const float* k_ring_scale, ispa_window win,
                                const void* q8, const float* q_scale, const void* k8_cur, const float* k_cur_scale,
                                const void* v_cur, int32_t n_q, float scale, void* out, float* lse,
                                ispa_stream stream) {
  const Qk8Scales sc{q_scale, k_cur_scale, k_ring_scale};
  return attn_common(MODE_LOCAL, ring, win, q8, k8_cur, v_cur, n_q, scale, 0u, out, nullptr, lse, nullptr, nullptr,
                     stream, &sc);
}

}  // extern "C"
