// 8-bit queries and keys for the chunk attention (SageAttention's 8-bit Q K^T with 16-bit
// P V, which the paper cites in Sec. 3.4 for its attention kernels): e4m3 codes with one fp32
// scale per head.
//
//   head_amax_kernel + quant_heads_kernel + head_scale_kernel
//       x bf16 [n][H][d] -> codes [n][H][d], scale[h] = amax_h / 448 (1 for an all-zero head),
//       code = e4m3(x * (1 / scale_h)); the three launches run in stream order, the scale
//       array holding amax (as fp32 bits, reduced with integer atomicMax: non-negative fp32
//       values order like their bit patterns; per block in shared memory first) until the
//       last one converts it.
//   quant_q_blocks_kernel
//       queries: one scale per head and block of 128 tokens (one attention CTA), one pass.
//   quant_given_kernel
//       codes with given per-head scales (the chunk's keys with the ring's key scales).
//   append_qk8_kernel
//       appends frames to a ring whose keys are e4m3: K rows quantised with the ring's given
//       per-head scales into their slots, V rows (bf16) copied (or, for a ring whose values are
//       e4m3 too, left to quant_vt_kernel).
//   quant_vt_kernel
//       values as d-major e4m3 codes [H][d][keys] with given per-head scales (the operand layout
//       of the 8-bit P V): the chunk's values, or appended frames into their ring slots.
#include <cuda.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "internal.h"
#include "ptx.cuh"

namespace ispa {

namespace {

constexpr float kE4M3Max = 448.f;

__device__ __forceinline__ uint16_t e4m3x2(float x0, float x1) {   // x0 in the low byte
  uint16_t r;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(r) : "f"(x1), "f"(x0));
  return r;
}

// 8 bf16 (one 16-byte word) times inv -> 8 codes (8 bytes)
__device__ __forceinline__ uint2 quant8(const uint4 v, float inv) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  uint32_t out[2];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const uint16_t lo = e4m3x2(__fmul_rn(__uint_as_float(w[2 * h] << 16), inv),
                               __fmul_rn(__uint_as_float(w[2 * h] & 0xFFFF0000u), inv));
    const uint16_t hi = e4m3x2(__fmul_rn(__uint_as_float(w[2 * h + 1] << 16), inv),
                               __fmul_rn(__uint_as_float(w[2 * h + 1] & 0xFFFF0000u), inv));
    out[h] = static_cast<uint32_t>(lo) | (static_cast<uint32_t>(hi) << 16);
  }
  return make_uint2(out[0], out[1]);
}

__device__ __forceinline__ float scale_of_amax(float amax) { return amax == 0.f ? 1.f : __fdiv_rn(amax, kE4M3Max); }
__device__ __forceinline__ float inv_of_scale(float s) { return __fdiv_rn(1.f, s); }

// One warp per (token, head) row of d bf16 (d % 8 == 0); amax_bits[h] must start at 0.
// Per-head maxima are gathered in shared memory (H <= kMaxHeadsSmem) and then merged into
// amax_bits with one atomic per head and block.
constexpr int kMaxHeadsSmem = 256;
__global__ void head_amax_kernel(const __nv_bfloat16* __restrict__ x, int64_t rows, int H, int d,
                                 unsigned int* __restrict__ amax_bits) {
  __shared__ unsigned int blk[kMaxHeadsSmem];
  for (int h = threadIdx.x; h < H; h += blockDim.x) blk[h] = 0u;
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int64_t warps = static_cast<int64_t>(gridDim.x) * (blockDim.x >> 5);
  const int nw = d / 8;
  for (int64_t r = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + (threadIdx.x >> 5); r < rows; r += warps) {
    const uint4* xr = reinterpret_cast<const uint4*>(x + r * d);
    float m = 0.f;
    for (int i = lane; i < nw; i += 32) {
      const uint4 v = xr[i];
      const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int e = 0; e < 4; ++e)
        m = fmaxf(m, fmaxf(fabsf(__uint_as_float(w[e] << 16)), fabsf(__uint_as_float(w[e] & 0xFFFF0000u))));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    if (lane == 0) atomicMax(blk + (r % H), __float_as_uint(m));
  }
  __syncthreads();
  for (int h = threadIdx.x; h < H; h += blockDim.x)
    if (blk[h]) atomicMax(amax_bits + h, blk[h]);
}

// Codes of every 16-byte word: grid-stride over n * H * d / 8 words.
__global__ void quant_heads_kernel(const uint4* __restrict__ x, int64_t n_words, int H, int d,
                                   const unsigned int* __restrict__ amax_bits, uint2* __restrict__ q) {
  const int wpr = d / 8;   // words per (token, head) row
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n_words;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int h = static_cast<int>((i / wpr) % H);
    q[i] = quant8(x[i], inv_of_scale(scale_of_amax(__uint_as_float(amax_bits[h]))));
  }
}

__global__ void head_scale_kernel(float* __restrict__ s, int H) {
  const int h = blockIdx.x * blockDim.x + threadIdx.x;
  if (h < H) s[h] = scale_of_amax(s[h]);   // s holds amax until here
}

// Queries: one CTA per (block of 128 tokens, head); the block's rows (d / 8 16-byte words each,
// d <= 256) stay in registers between the max and the quantisation.
constexpr int QB = 128;
constexpr int QW_PER_THREAD = 16;   // 128 rows x 32 words / 256 threads
__global__ void __launch_bounds__(256) quant_q_blocks_kernel(const uint4* __restrict__ x, int64_t n, int H, int d,
                                                             uint2* __restrict__ q, float* __restrict__ scale) {
  __shared__ float red[8];
  const int b = blockIdx.x, h = blockIdx.y;
  const int wpr = d / 8;
  const int64_t t0 = static_cast<int64_t>(b) * QB;
  const int rows = static_cast<int>(n - t0 < QB ? n - t0 : QB);
  const int words = rows * wpr;
  uint4 cache[QW_PER_THREAD];
  float m = 0.f;
#pragma unroll
  for (int c = 0; c < QW_PER_THREAD; ++c) {
    const int w = threadIdx.x + 256 * c;
    cache[c] = make_uint4(0, 0, 0, 0);
    if (w < words) {
      cache[c] = x[((t0 + w / wpr) * H + h) * wpr + w % wpr];
      const uint32_t v[4] = {cache[c].x, cache[c].y, cache[c].z, cache[c].w};
#pragma unroll
      for (int e = 0; e < 4; ++e)
        m = fmaxf(m, fmaxf(fabsf(__uint_as_float(v[e] << 16)), fabsf(__uint_as_float(v[e] & 0xFFFF0000u))));
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = m;
  __syncthreads();
  float amax = 0.f;
#pragma unroll
  for (int i = 0; i < 8; ++i) amax = fmaxf(amax, red[i]);
  const float sc = scale_of_amax(amax);
  const float inv = inv_of_scale(sc);
#pragma unroll
  for (int c = 0; c < QW_PER_THREAD; ++c) {
    const int w = threadIdx.x + 256 * c;
    if (w < words) q[((t0 + w / wpr) * H + h) * wpr + w % wpr] = quant8(cache[c], inv);
  }
  if (threadIdx.x == 0) scale[static_cast<int64_t>(h) * gridDim.x + b] = sc;
}

// Codes with given per-head scales: grid-stride over n * H * d / 8 words.
__global__ void quant_given_kernel(const uint4* __restrict__ x, int64_t n_words, int H, int d,
                                   const float* __restrict__ scale, uint2* __restrict__ q) {
  const int wpr = d / 8;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n_words;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x)
    q[i] = quant8(x[i], inv_of_scale(scale[(i / wpr) % H]));
}

struct AppendQk8Params {
  int32_t n_frames, P, H, d;
  int32_t slot[kMaxAppendFrames];
  int64_t ring_tok;              // capacity_frames * P
  const uint4* k_src;            // bf16 [n_frames * P][H][d]
  const uint4* v_src;
  uint2* k_dst;                  // e4m3 [H][ring_tok][d]
  uint4* v_dst;                  // bf16 [H][ring_tok][d]
  const float* k_scale;          // [H]
};

// One thread per 16-byte word of the source rows (8 bf16): quantise K, copy V.
__global__ void append_qk8_kernel(const AppendQk8Params p) {
  const int wpr = p.d / 8;
  const int64_t total = static_cast<int64_t>(p.n_frames) * p.P * p.H * wpr;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int w = static_cast<int>(i % wpr);
    const int64_t row = i / wpr;                   // token * H + head
    const int h = static_cast<int>(row % p.H);
    const int64_t tok = row / p.H;                 // token of the appended frames
    const int f = static_cast<int>(tok / p.P);
    const int64_t dst_tok = static_cast<int64_t>(p.slot[f]) * p.P + tok % p.P;
    const int64_t dst = (static_cast<int64_t>(h) * p.ring_tok + dst_tok) * wpr + w;
    p.k_dst[dst] = quant8(p.k_src[i], inv_of_scale(p.k_scale[h]));
    if (p.v_dst) p.v_dst[dst] = p.v_src[i];
  }
}

// d-major e4m3 values: out[h][c][key(t)] = e4m3(v[t][h][c] * (1 / scale_h)), key(t) = t, or
// slot[t / P] * P + t % P for appended frames.  One CTA per (block of 64 tokens, head): the block
// is quantised into shared memory as [token][c], then written d-major, four consecutive tokens
// (one 32-bit word: P % 4 == 0 keeps them in one frame and the word aligned) per store.
constexpr int VT_TOK = 64;
struct QuantVtParams {
  const uint4* v;        // bf16 [n][H][d]
  int64_t n;
  int32_t H, d;
  const float* scale;    // [H]
  uint8_t* out;          // [H][d][ld]
  int64_t ld;
  int32_t P, n_frames;   // n_frames == 0: key(t) = t
  int32_t slot[kMaxAppendFrames];
};

__global__ void __launch_bounds__(256) quant_vt_kernel(const QuantVtParams p) {
  __shared__ __align__(16) uint8_t tile[VT_TOK][128 + 16];   // row padding spreads the d-major reads
  const int h = blockIdx.y;
  const int64_t t0 = static_cast<int64_t>(blockIdx.x) * VT_TOK;
  const int rows = static_cast<int>(p.n - t0 < VT_TOK ? p.n - t0 : VT_TOK);
  const float inv = inv_of_scale(p.scale[h]);
  const int wpr = p.d / 8;
  for (int w = threadIdx.x; w < VT_TOK * wpr; w += blockDim.x) {
    const int r = w / wpr, c8 = w % wpr;
    uint2 code = make_uint2(0, 0);
    if (r < rows) code = quant8(p.v[((t0 + r) * p.H + h) * wpr + c8], inv);
    *reinterpret_cast<uint2*>(&tile[r][c8 * 8]) = code;
  }
  __syncthreads();
  const int groups = (rows + 3) / 4;
  for (int w = threadIdx.x; w < p.d * (VT_TOK / 4); w += blockDim.x) {
    const int c = w / (VT_TOK / 4), g = w % (VT_TOK / 4);
    if (g >= groups) continue;
    const int r0 = 4 * g;
    const int64_t t = t0 + r0;
    const int64_t key = p.n_frames > 0 ? static_cast<int64_t>(p.slot[t / p.P]) * p.P + t % p.P : t;
    uint8_t* dst = p.out + (static_cast<int64_t>(h) * p.d + c) * p.ld + key;
    if (r0 + 3 < rows) {
      *reinterpret_cast<uint32_t*>(dst) = static_cast<uint32_t>(tile[r0][c]) | (static_cast<uint32_t>(tile[r0 + 1][c]) << 8) |
                                          (static_cast<uint32_t>(tile[r0 + 2][c]) << 16) |
                                          (static_cast<uint32_t>(tile[r0 + 3][c]) << 24);
    } else {
      for (int i = 0; r0 + i < rows; ++i) dst[i] = tile[r0 + i][c];
    }
  }
}

}  // namespace

cudaError_t launch_quant_heads(const void* x, int64_t n, int32_t H, int32_t d, uint8_t* q, float* scale,
                               cudaStream_t s) {
  cudaError_t e = cudaMemsetAsync(scale, 0, sizeof(float) * H, s);
  if (e != cudaSuccess) return e;
  int dev = 0, sms = 152;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t rows = n * H;
  const int64_t want = (rows + 7) / 8;
  const unsigned blocks = static_cast<unsigned>(want < sms * 16 ? want : sms * 16);
  head_amax_kernel<<<blocks, 256, 0, s>>>(static_cast<const __nv_bfloat16*>(x), rows, H, d,
                                           reinterpret_cast<unsigned int*>(scale));
  const int64_t words = rows * d / 8;
  const int64_t qb = (words + 255) / 256;
  quant_heads_kernel<<<static_cast<unsigned>(qb < sms * 16 ? qb : sms * 16), 256, 0, s>>>(
      static_cast<const uint4*>(x), words, H, d, reinterpret_cast<const unsigned int*>(scale),
      reinterpret_cast<uint2*>(q));
  head_scale_kernel<<<(H + 127) / 128, 128, 0, s>>>(scale, H);
  return cudaGetLastError();
}

cudaError_t launch_append_qk8(const int32_t* slots, int32_t n_frames, int32_t P, int32_t H, int32_t d,
                              int64_t ring_tok, const void* k_src, const void* v_src, void* k_dst, void* v_dst,
                              const float* k_scale, cudaStream_t s) {
  AppendQk8Params p{};
  p.n_frames = n_frames;
  p.P = P;
  p.H = H;
  p.d = d;
  for (int f = 0; f < n_frames; ++f) p.slot[f] = slots[f];
  p.ring_tok = ring_tok;
  p.k_src = static_cast<const uint4*>(k_src);
  p.v_src = static_cast<const uint4*>(v_src);
  p.k_dst = static_cast<uint2*>(k_dst);
  p.v_dst = static_cast<uint4*>(v_dst);
  p.k_scale = k_scale;
  int dev = 0, sms = 152;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t total = static_cast<int64_t>(n_frames) * P * H * d / 8;
  const int64_t b = (total + 255) / 256;
  append_qk8_kernel<<<static_cast<unsigned>(b < sms * 8 ? b : sms * 8), 256, 0, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_quant_vt(const void* x, int64_t n, int32_t H, int32_t d, const float* scale, uint8_t* out,
                            int64_t ld, int32_t P, int32_t n_frames, const int32_t* slots, cudaStream_t s) {
  QuantVtParams p{};
  p.v = static_cast<const uint4*>(x);
  p.n = n;
  p.H = H;
  p.d = d;
  p.scale = scale;
  p.out = out;
  p.ld = ld;
  p.P = P;
  p.n_frames = n_frames;
  for (int f = 0; f < n_frames; ++f) p.slot[f] = slots[f];
  const dim3 grid(static_cast<unsigned>((n + VT_TOK - 1) / VT_TOK), static_cast<unsigned>(H));
  quant_vt_kernel<<<grid, 256, 0, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_quant_q_blocks(const void* x, int64_t n, int32_t H, int32_t d, uint8_t* q, float* scale,
                                  cudaStream_t s) {
  const dim3 grid(static_cast<unsigned>((n + QB - 1) / QB), static_cast<unsigned>(H));
  quant_q_blocks_kernel<<<grid, 256, 0, s>>>(static_cast<const uint4*>(x), n, H, d, reinterpret_cast<uint2*>(q), scale);
  return cudaGetLastError();
}

cudaError_t launch_quant_given(const void* x, int64_t n, int32_t H, int32_t d, const float* scale, uint8_t* q,
                               cudaStream_t s) {
  int dev = 0, sms = 152;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t words = n * H * d / 8;
  const int64_t b = (words + 255) / 256;
  quant_given_kernel<<<static_cast<unsigned>(b < sms * 16 ? b : sms * 16), 256, 0, s>>>(
      static_cast<const uint4*>(x), words, H, d, scale, reinterpret_cast<uint2*>(q));
  return cudaGetLastError();
}

}  // namespace ispa
