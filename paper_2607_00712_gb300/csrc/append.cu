// KV append into the ring cache (Eq. 3: K_past grows by each finished chunk).
//
// Source k_new/v_new is token-major [n_frames*P][H][d]; the ring is head-major
// [H][cap*P][d], so every (token, head) row of d bf16 (256 bytes at d = 128)
// moves as one unit to ring row (slot(frame) * P + t) of its head.  Threads
// copy 16-byte words; 16 consecutive threads cover one row, so both the reads
// and the writes are full 32-byte sectors.  One launch covers K and V of up
// to 64 layers (blockIdx.y = layer * 2 + {K, V}), each with its own ring
// capacity and state; the copy is a pure HBM stream (read + write of the
// same bytes).
#include <cuda_runtime.h>
#include <stdint.h>

#include "internal.h"
#include "pdl.cuh"

namespace ispa {

namespace {
constexpr int kThreads = 256;
constexpr int kUnroll = 4;
}  // namespace

__global__ void __launch_bounds__(kThreads) append_kernel(const AppendParams p) {
  pdl_wait();   // the new K / V may come from the kernel before this one, which may still read the ring
  const int layer = blockIdx.y >> 1;
  const bool is_v = blockIdx.y & 1;
  const uint4* __restrict__ src =
      static_cast<const uint4*>(is_v ? p.v_src[layer] : p.k_src[layer]);
  uint4* __restrict__ dst = static_cast<uint4*>(is_v ? p.v_dst[layer] : p.k_dst[layer]);
  const int words_per_row = p.head_dim / 8;                          // 16-byte words per (token, head)
  const int total = p.n_frames * p.tokens_per_frame * p.num_heads * words_per_row;  // < 2^31 (host check)
  const int stride = gridDim.x * kThreads * kUnroll;
  for (int base = blockIdx.x * kThreads * kUnroll + threadIdx.x; base < total; base += stride) {
    uint4 v[kUnroll];
    int64_t didx[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int i = base + u * kThreads;
      didx[u] = -1;
      if (i < total) {
        const int w = i % words_per_row;
        const int rh = i / words_per_row;                      // (token, head) row
        const int h = rh % p.num_heads;
        const int tok = rh / p.num_heads;                      // token within the append
        const int f = tok / p.tokens_per_frame;
        const int t = tok - f * p.tokens_per_frame;
        const int64_t ring_row = static_cast<int64_t>(h) * p.capacity_tokens[layer] +
                                 static_cast<int64_t>(p.slot[layer][f]) * p.tokens_per_frame + t;
        didx[u] = ring_row * words_per_row + w;
        v[u] = __ldcs(src + i);
      }
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u)
      if (didx[u] >= 0) dst[didx[u]] = v[u];
  }
}

cudaError_t launch_append(const AppendParams& p, cudaStream_t s) {
  const int64_t total = static_cast<int64_t>(p.n_frames) * p.tokens_per_frame * p.num_heads *
                        (p.head_dim / 8);
  int dev = 0, sms = 152;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  // enough CTAs to fill every SM several times over, capped by the work
  const int64_t per_cta = static_cast<int64_t>(kThreads) * kUnroll;
  int64_t blocks = (total + per_cta - 1) / per_cta;
  const int64_t cap = static_cast<int64_t>(sms) * 8;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  dim3 grid(static_cast<unsigned>(blocks), p.n_layers * 2);
  return launch_pdl(append_kernel, grid, dim3(kThreads), 0, s, p);
}

}  // namespace ispa
