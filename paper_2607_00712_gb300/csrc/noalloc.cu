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
// exits.  Its device address is looked up once per device, on the first call
// made with that device current.
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>

#include "../../include/ispa.h"

namespace {

static __device__ __align__(256) float g_dual_scratch[ISPA_DUAL_STATIC_MAX_PARTIALS];

constexpr int kMaxDevices = 64;
float* g_scratch_ptr[kMaxDevices] = {};
std::mutex g_scratch_mu;

// Device address of g_dual_scratch on the current device (set-up on first use).
float* scratch_on_current_device() {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_ptr[dev]) {
    float* ptr = nullptr;
    if (cudaGetSymbolAddress(reinterpret_cast<void**>(&ptr), g_dual_scratch) != cudaSuccess || !ptr)
      return nullptr;
    g_scratch_ptr[dev] = ptr;
  }
  return g_scratch_ptr[dev];
}

}  // namespace

extern "C" ispa_status ispa_attn_dual_static(const ispa_kv_ring* ring, ispa_window win, const void* q,
                                             const void* k_cur, const void* v_cur, int32_t n_q, float scale,
                                             void* a_full, void* a_loc, float* disc, float* disc_sq_sum,
                                             float* lse_full, float* lse_loc, ispa_stream stream) {
  if (!ring || ring->num_heads <= 0 || n_q <= 0) return ISPA_ERR_INVALID_ARG;
  const size_t need = static_cast<size_t>(ring->num_heads) * static_cast<size_t>(n_q);
  if (need > ISPA_DUAL_STATIC_MAX_PARTIALS) return ISPA_ERR_WORKSPACE;
  float* scratch = scratch_on_current_device();
  if (!scratch) return ISPA_ERR_CUDA;
  // The attention kernel writes every (head, query) partial of this call before the
  // reduction reads it, so nothing left over from an earlier call is ever used.
  return ispa_attn_dual(ring, win, q, k_cur, v_cur, n_q, scale, a_full, a_loc, disc, disc_sq_sum, lse_full,
                        lse_loc, scratch, sizeof(g_dual_scratch), stream);
}
