// ispa_attn_dual_static: the warmup dual pass for callers that cannot allocate.
//
// ispa_attn_dual needs a small scratch buffer (one fp32 partial sum of the
// discrepancy per head and query).  Some callers have no way to provide one
// at the moment they run the warmup pass: a real-time streaming loop whose
// device memory is planned once at start-up (cudaMalloc would synchronise the
// device and stall the stream), a plug-in living inside a host runtime that
// hands it tensors but no allocator, or code running where allocation is
// forbidden by policy.  This entry point takes that scratch from a fixed array
// in the library's own device memory instead, so the caller passes only its
// inputs and outputs.
//
// The array is a file-scope __device__ variable: every GPU that loads the
// library holds it (ISPA_DUAL_STATIC_MAX_PARTIALS floats) until the process
// exits.  Its device address belongs to one CUDA context.  It is looked up
// once per context -- normally the device's primary context -- on the first
// call made with that context current, and cached under the context's
// process-unique id, so a caller's own context, or the primary context that a
// cudaDeviceReset re-creates, never receives an address from another one.
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <mutex>
#include <utility>
#include <vector>

#include "../../include/ispa.h"
#include "internal.h"

namespace {

static __device__ __align__(256) float g_dual_scratch[ISPA_DUAL_STATIC_MAX_PARTIALS];

std::mutex g_scratch_mu;
std::vector<std::pair<uint64_t, float*>> g_scratch_ptr;   // (context id, device address)
std::atomic<uint32_t> g_scratch_lookups{0};

// Device address of g_dual_scratch in the current context (set-up on first use).
float* scratch_in_current_context(uint64_t* ctx_out = nullptr) {
  uint64_t ctx = 0;
  if (!ispa::current_context_id(&ctx)) return nullptr;
  if (ctx_out) *ctx_out = ctx;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  for (const auto& e : g_scratch_ptr)
    if (e.first == ctx) return e.second;
  float* ptr = nullptr;
  if (cudaGetSymbolAddress(reinterpret_cast<void**>(&ptr), g_dual_scratch) != cudaSuccess || !ptr) return nullptr;
  g_scratch_lookups.fetch_add(1);
  if (g_scratch_ptr.size() >= 256) g_scratch_ptr.erase(g_scratch_ptr.begin());
  g_scratch_ptr.emplace_back(ctx, ptr);
  return ptr;
}

}  // namespace

extern "C" ispa_status ispa_debug_static_scratch(void** addr, uint64_t* context_id, uint32_t* lookups) {
  if (!addr || !context_id || !lookups) return ISPA_ERR_INVALID_ARG;
  uint64_t ctx = 0;
  float* p = scratch_in_current_context(&ctx);
  if (!p) return ISPA_ERR_CUDA;
  *addr = p;
  *context_id = ctx;
  *lookups = g_scratch_lookups.load();
  return ISPA_OK;
}

extern "C" ispa_status ispa_attn_dual_static(const ispa_kv_ring* ring, ispa_window win, const void* q,
                                             const void* k_cur, const void* v_cur, int32_t n_q, float scale,
                                             void* a_full, void* a_loc, float* disc, float* disc_sq_sum,
                                             float* lse_full, float* lse_loc, ispa_stream stream) {
  if (!ring || ring->num_heads <= 0 || n_q <= 0) return ISPA_ERR_INVALID_ARG;
  const size_t need = static_cast<size_t>(ring->num_heads) * static_cast<size_t>(n_q);
  if (need > ISPA_DUAL_STATIC_MAX_PARTIALS) return ISPA_ERR_WORKSPACE;
  float* scratch = scratch_in_current_context();
  if (!scratch) return ISPA_ERR_CUDA;
  // The attention kernel writes every (head, query) partial of this call before the
  // reduction reads it, so nothing left over from an earlier call is ever used.
  return ispa_attn_dual(ring, win, q, k_cur, v_cur, n_q, scale, a_full, a_loc, disc, disc_sq_sum, lse_full,
                        lse_loc, scratch, sizeof(g_dual_scratch), stream);
}
