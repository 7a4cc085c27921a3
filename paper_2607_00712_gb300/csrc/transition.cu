// Decomposed-dual merge (Eq. 11-12) and the warmup-to-inference transition:
// weight injection W + dW and the permanent eviction of an L-layer's history
// (Sec. 3.1 phase 3, Sec. 3.3).  All HBM-bound elementwise / copy kernels.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <algorithm>
#include <vector>

#include "internal.h"
#include "pdl.cuh"

namespace ispa {

namespace {

// Thread i handles one 16-byte word (8 bf16) of the token-major [n_q][H][d] outputs:
// word w of (token t, head h), elements [8w, 8w+8).
__global__ void __launch_bounds__(256) lse_merge_kernel(const uint4* __restrict__ oa, const float* __restrict__ la,
                                                        const uint4* __restrict__ ob, const float* __restrict__ lb,
                                                        int n_q, int H, int words_per_row, uint4* __restrict__ out,
                                                        float* __restrict__ lse_out) {
  const int64_t total = static_cast<int64_t>(n_q) * H * words_per_row;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int w = static_cast<int>(i % words_per_row);
    const int64_t th = i / words_per_row;           // token-major (t, h)
    const int h = static_cast<int>(th % H);
    const int t = static_cast<int>(th / H);
    const float a = la[static_cast<int64_t>(h) * n_q + t];
    const float b = lb[static_cast<int64_t>(h) * n_q + t];
    const float m = fmaxf(a, b);
    float wa = 0.f, wb = 0.f, lse = -INFINITY;
    if (m != -INFINITY) {
      const float ea = expf(a - m), eb = expf(b - m);
      const float s = ea + eb;
      lse = m + logf(s);
      wa = ea / s;
      wb = eb / s;
    }
    const uint4 va = oa[i], vb = ob[i];
    const uint32_t xa[4] = {va.x, va.y, va.z, va.w}, xb[4] = {vb.x, vb.y, vb.z, vb.w};
    uint32_t r[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float a0 = __uint_as_float(xa[e] << 16), a1 = __uint_as_float(xa[e] & 0xFFFF0000u);
      const float b0 = __uint_as_float(xb[e] << 16), b1 = __uint_as_float(xb[e] & 0xFFFF0000u);
      // an empty branch may hold zeros; its weight is exactly 0
      const float o0 = (wa != 0.f ? wa * a0 : 0.f) + (wb != 0.f ? wb * b0 : 0.f);
      const float o1 = (wa != 0.f ? wa * a1 : 0.f) + (wb != 0.f ? wb * b1 : 0.f);
      __nv_bfloat162 v = __floats2bfloat162_rn(o0, o1);
      r[e] = *reinterpret_cast<uint32_t*>(&v);
    }
    out[i] = make_uint4(r[0], r[1], r[2], r[3]);
    if (lse_out && w == 0) lse_out[static_cast<int64_t>(h) * n_q + t] = lse;
  }
}

// Empty key set: O = 0, LSE = -inf.
__global__ void empty_branch_kernel(uint4* __restrict__ out, int64_t n_words, float* __restrict__ lse, int64_t n_lse) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n_words; i += stride)
    out[i] = make_uint4(0, 0, 0, 0);
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n_lse; i += stride)
    lse[i] = -INFINITY;
}

__global__ void axpy_f32_kernel(float* __restrict__ W, const float* __restrict__ dW, int64_t n) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n; i += stride) W[i] += dW[i];
}

__global__ void axpy_bf16_kernel(__nv_bfloat16* __restrict__ W, const float* __restrict__ dW, int64_t n) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n; i += stride)
    W[i] = __float2bfloat16_rn(__bfloat162float(W[i]) + dW[i]);
}

constexpr int kMaxCompactFrames = 64;
struct CompactParams {
  int32_t n_frames;
  int32_t num_heads;
  int64_t frame_words;       // 16-byte words of one frame of one head (P * d * 2 / 16)
  int64_t src_head_words;    // words of one head's ring in src (cap_src * P * d * 2 / 16)
  int64_t dst_head_words;
  int32_t src_slot[kMaxCompactFrames];
  int32_t dst_slot[kMaxCompactFrames];
  const uint4* src_k;
  const uint4* src_v;
  uint4* dst_k;
  uint4* dst_v;
};

// blockIdx.y = (frame * H + head) * 2 + {K, V}
__global__ void __launch_bounds__(256) compact_kernel(const CompactParams p) {
  const int kv = blockIdx.y & 1;
  const int fh = blockIdx.y >> 1;
  const int h = fh % p.num_heads;
  const int f = fh / p.num_heads;
  const uint4* src = (kv ? p.src_v : p.src_k) + h * p.src_head_words + p.src_slot[f] * p.frame_words;
  uint4* dst = (kv ? p.dst_v : p.dst_k) + h * p.dst_head_words + p.dst_slot[f] * p.frame_words;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < p.frame_words;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x)
    dst[i] = src[i];
}

// Output discrepancy of two stored outputs (Sec. 3.1 phase 1; reading: the L2 norm over all
// D features): disc[t] = || a_full[t] - a_loc[t] ||_2 with bf16 rows, differences and sums in
// fp32, and *disc_sq_sum += sum_t disc[t]^2.  HBM-bound: one warp per token row, each lane
// streaming 16-byte words of both rows with all its loads issued before the arithmetic.
constexpr int DISC_WARPS = 8;
constexpr int DISC_UNROLL = 8;   // 16-byte words per lane in flight per tensor: rows up to 2048 features in one pass

__device__ __forceinline__ float sq_diff8(const uint4 a, const uint4 b) {
  const uint32_t aw[4] = {a.x, a.y, a.z, a.w}, bw[4] = {b.x, b.y, b.z, b.w};
  float s = 0.f;
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float d0 = __uint_as_float(aw[e] << 16) - __uint_as_float(bw[e] << 16);
    const float d1 = __uint_as_float(aw[e] & 0xFFFF0000u) - __uint_as_float(bw[e] & 0xFFFF0000u);
    s = fmaf(d0, d0, s);
    s = fmaf(d1, d1, s);
  }
  return s;
}

__global__ void __launch_bounds__(DISC_WARPS * 32) discrepancy_kernel(const uint4* __restrict__ af,
                                                                     const uint4* __restrict__ al, int32_t n_rows,
                                                                     int32_t words, float* __restrict__ disc,
                                                                     float* __restrict__ disc_sq_sum) {
  __shared__ float red[DISC_WARPS];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float mine = 0.f;   // lane 0: this warp's rows
  for (int64_t r = static_cast<int64_t>(blockIdx.x) * DISC_WARPS + warp; r < n_rows;
       r += static_cast<int64_t>(gridDim.x) * DISC_WARPS) {
    const uint4* f = af + r * words;
    const uint4* l = al + r * words;
    float sq = 0.f;
    for (int w0 = 0; w0 < words; w0 += 32 * DISC_UNROLL) {
      uint4 a[DISC_UNROLL], b[DISC_UNROLL];
#pragma unroll
      for (int u = 0; u < DISC_UNROLL; ++u) {
        const int w = w0 + u * 32 + lane;
        a[u] = w < words ? __ldg(f + w) : make_uint4(0, 0, 0, 0);
        b[u] = w < words ? __ldg(l + w) : make_uint4(0, 0, 0, 0);
      }
#pragma unroll
      for (int u = 0; u < DISC_UNROLL; ++u) sq += sq_diff8(a[u], b[u]);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
    if (lane == 0) {
      disc[r] = sqrtf(sq);
      mine += sq;
    }
  }
  if (lane == 0) red[warp] = mine;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.f;
#pragma unroll
    for (int i = 0; i < DISC_WARPS; ++i) t += red[i];
    atomicAdd(disc_sq_sum, t);
  }
}

int grid_for(int64_t n, int threads) {
  int64_t b = (n + threads - 1) / threads;
  if (b > 152 * 8) b = 152 * 8;
  return static_cast<int>(b < 1 ? 1 : b);
}

bool aligned16(const void* p) { return p && (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }


}  // namespace

cudaError_t launch_empty_branch(void* out, float* lse, int32_t n_q, int32_t H, int32_t d, cudaStream_t s) {
  const int64_t words = static_cast<int64_t>(n_q) * H * d * 2 / 16;
  empty_branch_kernel<<<grid_for(words, 256), 256, 0, s>>>(static_cast<uint4*>(out), words, lse,
                                                           static_cast<int64_t>(n_q) * H);
  return cudaGetLastError();
}


// ------------------------------------------------------------ discrepancy reduction
// disc[t] = sqrt(sum_h part[h][t]);  *disc_sq_sum += sum over the block's tokens.
__global__ void __launch_bounds__(256) disc_reduce_kernel(const float* __restrict__ part, int H,
                                                          int n_q, float* __restrict__ disc,
                                                          float* __restrict__ disc_sq_sum) {
  pdl_wait();   // the partials of the attention launch before this one
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  float v = 0.f;
  if (t < n_q) {
    for (int h = 0; h < H; ++h) v += part[static_cast<size_t>(h) * n_q + t];
    disc[t] = sqrtf(v);
  }
  __shared__ float red[8];
  float w = v;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) w += __shfl_xor_sync(0xffffffffu, w, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = w;
  __syncthreads();
  if (threadIdx.x < 32) {
    w = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) w += __shfl_xor_sync(0xffffffffu, w, o);
    if (threadIdx.x == 0) atomicAdd(disc_sq_sum, w);
  }
}

cudaError_t launch_disc_reduce(const float* part, int32_t H, int32_t n_q, float* disc,
                               float* disc_sq_sum, cudaStream_t s) {
  if (n_q <= 0) return cudaSuccess;
  return launch_pdl(disc_reduce_kernel, dim3(static_cast<unsigned>((n_q + 255) / 256)), dim3(256), 0, s, part, H,
                    n_q, disc, disc_sq_sum);
}

}  // namespace ispa

using namespace ispa;

extern "C" {

ispa_status ispa_lse_merge(const void* o_a, const float* lse_a, const void* o_b, const float* lse_b, int32_t n_q,
                           int32_t num_heads, int32_t head_dim, void* out, float* lse_out, ispa_stream stream) {
  if (n_q <= 0 || num_heads <= 0 || head_dim <= 0 || head_dim % 8 != 0) return ISPA_ERR_INVALID_ARG;
  if (!aligned16(o_a) || !aligned16(o_b) || !aligned16(out) || !lse_a || !lse_b) return ISPA_ERR_INVALID_ARG;
  const int wpr = head_dim / 8;
  const int64_t total = static_cast<int64_t>(n_q) * num_heads * wpr;
  lse_merge_kernel<<<grid_for(total, 256), 256, 0, stream>>>(
      static_cast<const uint4*>(o_a), lse_a, static_cast<const uint4*>(o_b), lse_b, n_q, num_heads, wpr,
      static_cast<uint4*>(out), lse_out);
  return cudaGetLastError() == cudaSuccess ? ISPA_OK : ISPA_ERR_CUDA;
}

ispa_status ispa_discrepancy(const void* a_full, const void* a_loc, int32_t n_q, int32_t dim, float* disc,
                             float* disc_sq_sum, ispa_stream stream) {
  if (n_q <= 0 || dim <= 0 || !disc || !disc_sq_sum) return ISPA_ERR_INVALID_ARG;
  if (!aligned16(a_full) || !aligned16(a_loc)) return ISPA_ERR_INVALID_ARG;
  if (dim % 8 != 0) return ISPA_ERR_UNSUPPORTED;
  int dev = 0, sms = 152;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  // one warp per row; at most 8 CTAs of 256 threads per SM are resident
  int64_t blocks = (static_cast<int64_t>(n_q) + DISC_WARPS - 1) / DISC_WARPS;
  if (blocks > static_cast<int64_t>(sms) * 8) blocks = static_cast<int64_t>(sms) * 8;
  discrepancy_kernel<<<static_cast<unsigned>(blocks), DISC_WARPS * 32, 0, stream>>>(
      static_cast<const uint4*>(a_full), static_cast<const uint4*>(a_loc), n_q, dim / 8, disc, disc_sq_sum);
  return cudaGetLastError() == cudaSuccess ? ISPA_OK : ISPA_ERR_CUDA;
}

ispa_status ispa_select_layers(const double* eps, int32_t n_layers, int32_t k, int32_t* is_l_layer) {
  if (!eps || !is_l_layer || n_layers <= 0 || k < 0 || k > n_layers) return ISPA_ERR_INVALID_ARG;
  std::vector<int32_t> idx(n_layers);
  for (int32_t i = 0; i < n_layers; ++i) idx[i] = i;
  std::stable_sort(idx.begin(), idx.end(), [&](int32_t a, int32_t b) {
    const bool na = std::isnan(eps[a]), nb = std::isnan(eps[b]);
    if (na != nb) return nb;            // NaN ranks last
    if (na) return false;
    return eps[a] < eps[b];             // stable: ties keep the lower index first
  });
  for (int32_t i = 0; i < n_layers; ++i) is_l_layer[i] = 0;
  for (int32_t r = 0; r < k; ++r) is_l_layer[idx[r]] = 1;
  return ISPA_OK;
}

ispa_status ispa_apply_absorption(float* W, const float* dW, int32_t dim, int32_t d_out, ispa_stream stream) {
  if (!W || !dW || dim <= 0 || d_out <= 0) return ISPA_ERR_INVALID_ARG;
  const int64_t n = static_cast<int64_t>(dim) * d_out;
  axpy_f32_kernel<<<grid_for(n, 256), 256, 0, stream>>>(W, dW, n);
  return cudaGetLastError() == cudaSuccess ? ISPA_OK : ISPA_ERR_CUDA;
}

ispa_status ispa_apply_absorption_bf16(void* W, const float* dW, int32_t dim, int32_t d_out, ispa_stream stream) {
  if (!W || !dW || dim <= 0 || d_out <= 0) return ISPA_ERR_INVALID_ARG;
  const int64_t n = static_cast<int64_t>(dim) * d_out;
  axpy_bf16_kernel<<<grid_for(n, 256), 256, 0, stream>>>(static_cast<__nv_bfloat16*>(W), dW, n);
  return cudaGetLastError() == cudaSuccess ? ISPA_OK : ISPA_ERR_CUDA;
}

ispa_status ispa_ring_compact(const ispa_kv_ring* src, ispa_window win, ispa_kv_ring* dst, ispa_stream stream) {
  if (!src || !dst || win.n_sink_frames < 0 || win.n_recent_frames < 0) return ISPA_ERR_INVALID_ARG;
  if (ispa_ring_bytes(src) == 0 || ispa_ring_bytes(dst) == 0) return ISPA_ERR_INVALID_ARG;
  if (src->k_format != ISPA_KV_BF16 || dst->k_format != ISPA_KV_BF16) return ISPA_ERR_UNSUPPORTED;
  if (src->num_heads != dst->num_heads || src->head_dim != dst->head_dim ||
      src->tokens_per_frame != dst->tokens_per_frame || dst->n_sink_frames != win.n_sink_frames ||
      dst->capacity_frames != win.n_sink_frames + win.n_recent_frames || win.n_recent_frames < 1)
    return ISPA_ERR_INVALID_ARG;
  if (!aligned16(src->k) || !aligned16(src->v) || !aligned16(dst->k) || !aligned16(dst->v))
    return ISPA_ERR_INVALID_ARG;
  const int64_t F = src->frames_written;
  ispa_kv_ring probe = *dst;
  probe.frames_written = F;
  CompactParams p{};
  p.num_heads = src->num_heads;
  const int64_t row_words = static_cast<int64_t>(src->head_dim) * 2 / 16;
  p.frame_words = row_words * src->tokens_per_frame;
  p.src_head_words = p.frame_words * src->capacity_frames;
  p.dst_head_words = p.frame_words * dst->capacity_frames;
  p.src_k = static_cast<const uint4*>(src->k);
  p.src_v = static_cast<const uint4*>(src->v);
  p.dst_k = static_cast<uint4*>(dst->k);
  p.dst_v = static_cast<uint4*>(dst->v);
  // frames dst keeps: its sinks and its n_recent newest frames (exactly the window)
  std::vector<int64_t> frames;
  for (int64_t f = 0; f < std::min<int64_t>(win.n_sink_frames, F); ++f) frames.push_back(f);
  for (int64_t f = std::max<int64_t>(win.n_sink_frames, F - win.n_recent_frames); f < F; ++f) frames.push_back(f);
  for (const int64_t f : frames) {
    const int32_t ds = ispa_ring_slot(&probe, f);
    if (ds < 0) continue;
    const int32_t ss = ispa_ring_slot(src, f);
    if (ss < 0) return ISPA_ERR_CAPACITY;
    if (p.n_frames >= kMaxCompactFrames) return ISPA_ERR_CAPACITY;
    p.src_slot[p.n_frames] = ss;
    p.dst_slot[p.n_frames] = ds;
    ++p.n_frames;
  }
  if (p.n_frames > 0) {
    dim3 grid(static_cast<unsigned>(std::min<int64_t>((p.frame_words + 255) / 256, 64)),
              static_cast<unsigned>(p.n_frames * p.num_heads * 2));
    compact_kernel<<<grid, 256, 0, stream>>>(p);
    if (cudaGetLastError() != cudaSuccess) return ISPA_ERR_CUDA;
  }
  dst->frames_written = F;
  return ISPA_OK;
}

}  // extern "C"
