// Normal-equation sums of the least-squares absorption (Sec. 3.2, Eq. 5):
//   G += A_loc^T A_loc,  X += A_loc^T Delta,  S += Delta^T Delta,
// with Delta = A_full - A_loc, on the tensor cores (tcgen05, fp32 in TMEM).
//
// Two forms of the operands, both with Delta formed exactly in fp32 from the two bf16 inputs:
//  * scaled (default): amax_kernel takes max |A_loc| and max |Delta| over the call, and
//    convert_kernel writes both as fp16 times a power of two that puts the largest
//    magnitude in [2^14, 2^15) (A_loc's bf16 values convert exactly; Delta rounds once, to
//    2^-11 relative).  One pass per tile: G = a^T a, X = a^T d, S = d^T d on f16 UMMAs,
//    each sum multiplied back by its exact power of two before it reaches the state.
//  * exact (ISPA_LS_EXACT_DELTA): split_kernel stores Delta as the bf16 pair hi = bf16(Delta),
//    lo = bf16(Delta - hi), ~2^-16 relative; G tile: a^T a, X tile: a^T hi + a^T lo, S tile:
//    hi^T hi + hi^T lo + lo^T hi (lo^T lo is below fp32 resolution and dropped) on bf16 UMMAs.
// Every output tile of the upper blocks is a contraction over tokens, the token axis being
// the UMMA K dimension.  Both operands are token-major [T][D] in HBM, i.e. MN-major for the
// UMMA, staged by TMA with 128-byte swizzle, 64 tokens per pipeline stage, one request per
// operand.
//
// gram_wide_kernel (D % 256 == 0): 256 x 256 tiles, two 128 x 256 accumulators
// sharing each B operand, full waves of tiles in a blocked order plus a stream-K
// tail (see the comment above the kernel).
//
// gram_kernel (other D, multiples of 128): 128 x 128 tiles, stream-K over one
// sequence of steps (tile, pass, 64-token block) -- G tiles, X tiles, S tiles with the
// passes of the form -- cut into equal contiguous ranges for a persistent grid of one
// CTA per SM.  A CTA's range covers the tail of one tile, some whole tiles and the
// head of another; each such segment is summed in one of two TMEM accumulators and
// added into the state by the epilogue warps while the UMMA warp already fills the
// other accumulator.
#include <cuda.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "delta.cuh"
#include "internal.h"
#include "pdl.cuh"

#include <cuda_fp16.h>
#include "ptx.cuh"

namespace ispa {

namespace {

constexpr int GM = 128;        // output rows per tile
constexpr int GK = 64;         // tokens per stage
constexpr int GST = 4;         // pipeline stages
constexpr int G_THREADS = 192;  // warp 0 TMA, warp 1 MMA, warps 2-5 epilogue
constexpr uint64_t G_DRAIN_NS = 200ull * 1000 * 1000;

template <int BN>
struct GCfg {
  static constexpr int BOX = GK * 128;            // 64 tokens x 64 features bf16 = 8 KB
  static constexpr int A_BYTES = (GM / 64) * BOX;  // 16 KB
  static constexpr int B_BYTES = (BN / 64) * BOX;
  static constexpr int STAGE = A_BYTES + B_BYTES;
  static constexpr int OFF_BAR = GST * STAGE;
  static constexpr int N_BAR = 2 * GST + 2 + 2 + 1;   // full/empty stages, acc full/empty x2, drain
  static constexpr int OFF_T = (OFF_BAR + N_BAR * 8 + 16 + 15) / 16 * 16;   // epilogue staging, 4 warps x 4 KB
  static constexpr int SMEM = OFF_T + 4 * 32 * 32 * 4;
  static_assert(SMEM <= 232448, "shared memory per CTA");
  static_assert(OFF_T % 16 == 0, "16-byte aligned staging buffers");
  static_assert(STAGE % 1024 == 0 && BOX % 1024 == 0, "swizzle atoms need 1 KB aligned boxes");
  static constexpr uint32_t TMEM_COLS = 2 * BN;  // two accumulators: 256 or 512 columns
};

// Operand sources of the passes of each block type.  Exact form: 0 = A_loc, 1 = hi, 2 = lo;
// scaled form: 0 = A_loc, 1 = Delta (both fp16, scaled).
struct Pass {
  int8_t a, b;
};
__constant__ Pass kPasses[2][3][3] = {
    {
        {{0, 0}, {0, 0}, {0, 0}},  // G: one pass
        {{0, 1}, {0, 2}, {0, 0}},  // X: two passes
        {{1, 1}, {1, 2}, {2, 1}},  // S: three passes
    },
    {
        {{0, 0}, {0, 0}, {0, 0}},  // G
        {{0, 1}, {0, 0}, {0, 0}},  // X
        {{1, 1}, {0, 0}, {0, 0}},  // S
    },
};
constexpr int kPassesExact[3] = {1, 2, 3};
constexpr int kPassesScaled[3] = {1, 1, 1};

// The bf16 descriptor with the A and B format fields (bits 7-9, 10-12) set to f16 (0).
__host__ __device__ constexpr uint32_t idesc_f16(int M, int N, bool a_mn_major, bool b_mn_major) {
  return idesc_bf16(M, N, a_mn_major, b_mn_major) & ~((7u << 7) | (7u << 10));
}

struct GramParams {
  int32_t D;
  int32_t T;
  int32_t n_ktiles;   // ceil(T / GK)
  int32_t n_upper;    // upper-block tiles of G (and of S)
  int32_t n_full;     // tiles of X
  int32_t total;      // steps over all tiles
  int32_t form;       // 0 exact (bf16 hi / lo), 1 scaled (fp16)
  int32_t passes[3];  // passes per tile of G, X, S
  uint32_t idesc;     // UMMA instruction descriptor of the form
  const float* unscale;   // scaled form: the factor of G, X, S sums; null: 1
  float* gram;        // [2D][2D]
  int* status;
  uint64_t wait_limit_ns;
  uint32_t* heartbeat;
};

// Kernel parameters indexed by a run-time kind without a local copy of the arrays.
__device__ __forceinline__ int32_t pick3(const int32_t (&a)[3], int k) {
  return k == 0 ? a[0] : (k == 1 ? a[1] : a[2]);
}

// Step g of the global sequence -> tile (item, numbered as decode_tile expects) and its
// first step.  Tiles: n_upper G tiles, n_full X tiles, n_upper S tiles, each of
// passes[kind] * n_kt steps.
__device__ __forceinline__ void step_item(const GramParams& p, int g, int& item, int& first) {
  const int n_kt = p.n_ktiles;
  const int lg = p.passes[0] * n_kt, lx = p.passes[1] * n_kt, ls = p.passes[2] * n_kt;
  const int g_end = p.n_upper * lg;
  const int x_end = g_end + p.n_full * lx;
  if (g < g_end) {
    item = g / lg;
    first = item * lg;
  } else if (g < x_end) {
    const int i = (g - g_end) / lx;
    item = p.n_upper + i;
    first = g_end + i * lx;
  } else {
    const int i = (g - x_end) / ls;
    item = p.n_upper + p.n_full + i;
    first = x_end + i * ls;
  }
}

// Decode blockIdx.x into (kind, row block, col block).  Items: upper G tiles,
// then all X tiles, then upper S tiles.
template <int BN>
__device__ __forceinline__ void decode_tile(int item, int D, int& kind, int& bi, int& bj) {
  const int RB = D / GM, CB = D / BN;
  int n_upper = 0;
  for (int r = 0; r < RB; ++r) n_upper += CB - (r * GM) / BN;
  kind = 0;
  if (item >= n_upper) {
    item -= n_upper;
    if (item < RB * CB) {
      kind = 1;
      bi = item / CB;
      bj = item % CB;
      return;
    }
    item -= RB * CB;
    kind = 2;
  }
  for (int r = 0; r < RB; ++r) {
    const int c0 = (r * GM) / BN;
    const int n = CB - c0;
    if (item < n) {
      bi = r;
      bj = c0 + item;
      return;
    }
    item -= n;
  }
  bi = bj = 0;
}

}  // namespace

// Add one warp's 32 x 32 block of fp32 sums (TMEM lanes = rows, 32 columns from `taddr`)
// into the row-major state at `dst` (row stride `ld` floats) with vector atomics.  The
// block goes through shared memory first (16-byte chunk q of row t stored at chunk
// q ^ (t & 7): no bank conflicts on the write or the read) so that each atomic
// instruction of the warp covers 4 rows x 128 contiguous bytes instead of 32 rows x
// 16 bytes; measured on GB300 this made the whole accumulate 23-36 % faster.
__device__ __forceinline__ void flush_block32(uint32_t taddr, float4* tbuf, float* dst, size_t ld, int lane,
                                              float scale) {
  uint32_t v[32];
  tmem_ld32(taddr, v);
  tmem_wait_ld32(v);
#pragma unroll
  for (int q = 0; q < 8; ++q)
    tbuf[lane * 8 + (q ^ (lane & 7))] =
        make_float4(__uint_as_float(v[4 * q]) * scale, __uint_as_float(v[4 * q + 1]) * scale,
                    __uint_as_float(v[4 * q + 2]) * scale, __uint_as_float(v[4 * q + 3]) * scale);
  __syncwarp();
  const int rr = lane >> 3, qq = lane & 7;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int row = 4 * i + rr;
    atomicAdd(reinterpret_cast<float4*>(dst + static_cast<size_t>(row) * ld) + qq, tbuf[row * 8 + (qq ^ (row & 7))]);
  }
  __syncwarp();   // the buffer is rewritten by the next block
}

// Delta = a_full - a_loc (exact in fp32), hi = bf16(Delta), lo = bf16(Delta - hi).
__global__ void __launch_bounds__(256) split_kernel(const uint4* __restrict__ a_loc,
                                                    const uint4* __restrict__ a_full,
                                                    uint4* __restrict__ hi, uint4* __restrict__ lo,
                                                    int64_t n_words) {
  pdl_wait();      // the inputs may come from the kernel before this one
  pdl_trigger();   // the Gram kernel after this one may set itself up meanwhile
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n_words; i += stride)
    split_delta8(a_loc[i], a_full[i], hi[i], lo[i]);
}

// Largest |value| of a block's 256 threads (all threads call it; the result is in every thread).
__device__ __forceinline__ float block_max256(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  __syncthreads();   // red may still be read by a previous call
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
  __syncthreads();
  v = red[0];
#pragma unroll
  for (int w = 1; w < 8; ++w) v = fmaxf(v, red[w]);
  return v;
}

// Scaled form, pass 1: max |A_loc| and max |Delta| of each block's words -> part[b], part[nb + b].
__global__ void __launch_bounds__(256) amax_kernel(const uint4* __restrict__ a_loc, const uint4* __restrict__ a_full,
                                                   int64_t n_words, float* __restrict__ part) {
  pdl_wait();      // the inputs may come from the kernel before this one
  pdl_trigger();   // convert_kernel may set itself up meanwhile
  __shared__ float red[8];
  float ma = 0.f, md = 0.f;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  // four words per thread and round, all loaded before any is used
  for (int64_t i0 = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i0 < n_words; i0 += 4 * stride) {
    uint4 a[4], f[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int64_t i = i0 + u * stride;
      a[u] = i < n_words ? a_loc[i] : make_uint4(0, 0, 0, 0);
      f[u] = i < n_words ? a_full[i] : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const uint32_t aw[4] = {a[u].x, a[u].y, a[u].z, a[u].w}, fw[4] = {f[u].x, f[u].y, f[u].z, f[u].w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float a0 = __uint_as_float(aw[e] << 16), a1 = __uint_as_float(aw[e] & 0xFFFF0000u);
        const float f0 = __uint_as_float(fw[e] << 16), f1 = __uint_as_float(fw[e] & 0xFFFF0000u);
        ma = fmaxf(ma, fmaxf(fabsf(a0), fabsf(a1)));
        md = fmaxf(md, fmaxf(fabsf(f0 - a0), fabsf(f1 - a1)));
      }
    }
  }
  ma = block_max256(ma, red);
  md = block_max256(md, red);
  if (threadIdx.x == 0) {
    part[blockIdx.x] = ma;
    part[gridDim.x + blockIdx.x] = md;
  }
}

// Exponent s with amax * 2^s in [2^14, 2^15) (0 for amax = 0), kept in [-60, 60] so that
// 2^s and 2^-2s are normal fp32 numbers.
__device__ __forceinline__ int scale_exp(float amax) {
  if (!(amax > 0.f)) return 0;
  const int e = static_cast<int>((__float_as_uint(amax) >> 23) & 0xFF) - 127;
  return max(-60, min(60, 14 - e));
}
__device__ __forceinline__ float pow2f(int s) { return __uint_as_float(static_cast<uint32_t>(127 + s) << 23); }

// Scaled form, pass 2: the call's maxima from amax_kernel's nb partials, then
// a16 = fp16(A_loc * 2^sa) (exact) and d16 = fp16(Delta * 2^sd) (one rounding), eight
// features per thread and step; block 0 stores the factors 2^-2sa, 2^-(sa+sd), 2^-2sd that
// take the G, X and S sums back to the inputs' scale.
__global__ void __launch_bounds__(256) convert_kernel(const uint4* __restrict__ a_loc,
                                                      const uint4* __restrict__ a_full, int64_t n_words,
                                                      const float* __restrict__ part, int nb,
                                                      uint4* __restrict__ a16, uint4* __restrict__ d16,
                                                      float* __restrict__ unscale) {
  pdl_wait();   // amax_kernel's partials
  __shared__ float red[8];
  float ma = 0.f, md = 0.f;
  for (int b = threadIdx.x; b < nb; b += blockDim.x) {
    ma = fmaxf(ma, part[b]);
    md = fmaxf(md, part[nb + b]);
  }
  ma = block_max256(ma, red);
  md = block_max256(md, red);
  const int sa = scale_exp(ma), sd = scale_exp(md);
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    unscale[0] = pow2f(-2 * sa);
    unscale[1] = pow2f(-(sa + sd));
    unscale[2] = pow2f(-2 * sd);
  }
  pdl_trigger();   // the Gram kernel may set itself up meanwhile
  const float ka = pow2f(sa), kd = pow2f(sd);
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  // four words per thread and round, all loaded before any is converted
  for (int64_t i0 = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i0 < n_words; i0 += 4 * stride) {
    uint4 a[4], f[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int64_t i = i0 + u * stride;
      if (i < n_words) {
        a[u] = a_loc[i];
        f[u] = a_full[i];
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int64_t i = i0 + u * stride;
      if (i >= n_words) break;
      const uint32_t aw[4] = {a[u].x, a[u].y, a[u].z, a[u].w}, fw[4] = {f[u].x, f[u].y, f[u].z, f[u].w};
      uint32_t ow[4], dw[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float a0 = __uint_as_float(aw[e] << 16), a1 = __uint_as_float(aw[e] & 0xFFFF0000u);
        const float f0 = __uint_as_float(fw[e] << 16), f1 = __uint_as_float(fw[e] & 0xFFFF0000u);
        __half2 h = __floats2half2_rn(a0 * ka, a1 * ka);
        ow[e] = *reinterpret_cast<uint32_t*>(&h);
        h = __floats2half2_rn((f0 - a0) * kd, (f1 - a1) * kd);
        dw[e] = *reinterpret_cast<uint32_t*>(&h);
      }
      a16[i] = make_uint4(ow[0], ow[1], ow[2], ow[3]);
      d16[i] = make_uint4(dw[0], dw[1], dw[2], dw[3]);
    }
  }
}

template <int BN>
__global__ void __launch_bounds__(G_THREADS, 1)
    gram_kernel(const __grid_constant__ CUtensorMap tm_a_r, const __grid_constant__ CUtensorMap tm_hi_r,
                const __grid_constant__ CUtensorMap tm_lo_r, const __grid_constant__ CUtensorMap tm_a_c,
                const __grid_constant__ CUtensorMap tm_hi_c, const __grid_constant__ CUtensorMap tm_lo_c,
                const GramParams p) {
  using C = GCfg<BN>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = smem_raw;
  const uint32_t sbase = smem_u32(smem);
  if (sbase & 1023u) {  // uniform over the CTA; nothing is initialised yet
    if (threadIdx.x == 0) record_error(p.status, DEVERR_LAYOUT, 0, sbase, 0, 1);
    return;
  }
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + C::N_BAR);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8 * GST, accf0 = empty0 + 8 * GST,
                 acce0 = accf0 + 16, drain_bar = acce0 + 16;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // this CTA's contiguous step range
  const int g0 = static_cast<int>(static_cast<int64_t>(p.total) * blockIdx.x / gridDim.x);
  const int g1 = static_cast<int>(static_cast<int64_t>(p.total) * (blockIdx.x + 1) / gridDim.x);
  const int n_kt = p.n_ktiles;

  if (threadIdx.x == 0) {
    for (int i = 0; i < GST; ++i) {
      mbar_init(full0 + 8 * i, 1);
      mbar_init(empty0 + 8 * i, 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(accf0 + 8 * i, 1);
      mbar_init(acce0 + 8 * i, 128);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (threadIdx.x == 0) heartbeat(p.heartbeat, 0);
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), C::TMEM_COLS);
    tmem_relinquish();
    if (lane == 0) heartbeat(p.heartbeat, 1);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();   // the operands and the state may come from the kernel before this one
  const WaitCtx wc{abort_flag, p.status, p.wait_limit_ns};

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0 && g1 > g0) {
      // _r maps fetch a tile's GM row features, _c maps its BN column features
      auto map_r = [&](int w) { return w == 0 ? &tm_a_r : (w == 1 ? &tm_hi_r : &tm_lo_r); };
      auto map_c = [&](int w) { return w == 0 ? &tm_a_c : (w == 1 ? &tm_hi_c : &tm_lo_c); };
      int issued = 0;
      int item = -1, first = 0, kind = 0, bi = 0, bj = 0;
      for (int g = g0; g < g1; ++g) {
        const int i = g - g0;
        if (item < 0 || g >= first + pick3(p.passes, kind) * n_kt) {
          step_item(p, g, item, first);
          decode_tile<BN>(item, p.D, kind, bi, bj);
        }
        const int local = g - first;
        const int pass = local / n_kt;
        const int tok = (local % n_kt) * GK;
        const int st = i % GST;
        if (!mbar_wait(empty0 + 8 * st, ((i / GST) & 1) ^ 1, wc, 21, i)) break;
        mbar_arrive_expect_tx(full0 + 8 * st, C::STAGE);
        const uint32_t sa = sbase + st * C::STAGE, sb = sa + C::A_BYTES;
        const CUtensorMap* ma = map_r(kPasses[p.form][kind][pass].a);
        const CUtensorMap* mb = map_c(kPasses[p.form][kind][pass].b);
        // one request per operand: (64 features, GK tokens, GM/64 or BN/64 feature blocks)
        tma_load_3d(sa, ma, full0 + 8 * st, 0, tok, bi * (GM / 64));
        tma_load_3d(sb, mb, full0 + 8 * st, 0, tok, bj * (BN / 64));
        issued = i + 1;
      }
      for (int i = issued > GST ? issued - GST : 0; i < issued; ++i)
        mbar_wait_drain(full0 + 8 * (i % GST), (i / GST) & 1, G_DRAIN_NS);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ UMMA issuer
    if (lane == 0 && g1 > g0) {
      bool ok = true;
      int seg = 0, item = -1, first = 0, last = 0;
      for (int g = g0; ok && g < g1; ++g) {
        const int i = g - g0;
        if (g == g0 || g >= last) {   // a new segment starts: claim accumulator seg & 1
          if (g > g0) ++seg;
          step_item(p, g, item, first);
          int kind, bi, bj;
          decode_tile<BN>(item, p.D, kind, bi, bj);
          last = first + pick3(p.passes, kind) * n_kt;
          const int b = seg & 1;
          if (!mbar_wait(acce0 + 8 * b, ((seg >> 1) & 1) ^ 1, wc, 24, seg)) {
            ok = false;
            break;
          }
          tc_fence_after();
        }
        const int st = i % GST;
        if (!mbar_wait(full0 + 8 * st, (i / GST) & 1, wc, 22, i)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t sa = sbase + st * C::STAGE, sb = sa + C::A_BYTES;
        const uint32_t acc = tmem + (seg & 1) * BN;
        const bool seg_first = (g == g0) || (g == first);
#pragma unroll
        for (int k = 0; k < GK / 16; ++k)
          umma_ss(acc, sw128_desc(sa + k * 2048, C::BOX, 1024), sw128_desc(sb + k * 2048, C::BOX, 1024), p.idesc,
                  (!seg_first || k > 0) ? 1u : 0u);
        tc_commit(empty0 + 8 * st);
        if (g + 1 == g1 || g + 1 == last) tc_commit(accf0 + 8 * (seg & 1));
      }
      tc_commit(drain_bar);
      mbar_wait_drain(drain_bar, 0, G_DRAIN_NS);
    }
    __syncwarp();
  } else if (g1 > g0) {
    // ------------------------------------------------------------ epilogue (warps 2-5)
    // warp w reads TMEM lanes 32*(w%4) .. +31 = output rows of the tile
    const int quarter = warp & 3;
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
    float4* tbuf = reinterpret_cast<float4*>(smem + C::OFF_T) + (warp - 2) * 32 * 8;
    int item_a, first_a, item_b, first_b;
    step_item(p, g0, item_a, first_a);
    step_item(p, g1 - 1, item_b, first_b);
    bool ok = true;
    for (int seg = 0; seg <= item_b - item_a; ++seg) {
      const int b = seg & 1;
      ok = ok && __all_sync(0xffffffffu, mbar_wait(accf0 + 8 * b, (seg >> 1) & 1, wc, 23, seg));
      if (!ok) break;
      tc_fence_after();
      int kind, bi, bj;
      decode_tile<BN>(item_a + seg, p.D, kind, bi, bj);
      const int D = p.D;
      const int row0 = (kind == 2 ? D : 0) + bi * GM;
      const int col0 = (kind == 0 ? 0 : D) + bj * BN;
      float* gblk = p.gram + static_cast<size_t>(row0 + quarter * 32) * (2 * D) + col0;
      const float scale = p.unscale ? p.unscale[kind] : 1.f;
#pragma unroll 1
      for (int c = 0; c < BN / 32; ++c)
        flush_block32(lane_base + b * BN + 32 * c, tbuf, gblk + 32 * c, 2 * static_cast<size_t>(D), lane, scale);
      tc_fence_before();
      mbar_arrive(acce0 + 8 * b);   // accumulator b may be overwritten
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
    if (lane == 0) heartbeat(p.heartbeat, 2);
  }
}

// ---------------------------------------------------------------- 256 x 256 tiles
// For hidden sizes that are multiples of 256 the work unit is a 256 x 256 output tile,
// summed as two 128 x 256 accumulators (its upper and lower 128 rows) that share every
// B operand: 64 KB of operands per 64-token step feed 8 UMMAs, against 48 KB for 4 with
// 128 x 256 tiles.  TMEM holds exactly the two accumulators, so the epilogue of a tile
// (warps 2-5 drain the upper accumulator, warps 6-9 the lower one, in parallel) is not
// overlapped with the next tile's UMMAs.
//
// Schedule.  Per kind (G, X, S) the tiles are numbered in a blocked order -- bands of
// 8 tile columns, row by row inside a band -- so that consecutive tiles share operand
// panels.  Every CTA first takes one whole tile (all its passes) in each full wave of
// its kind: tile w * grid + cta in wave w.  The CTAs of a wave run the same number of
// steps on tiles that share panels, in step with one another, so each panel's token
// slices are read from DRAM about once per wave and then served from L2.  The tiles
// left over (fewer than one wave per kind) form one shared tail of steps, cut into
// equal contiguous ranges (stream-K), which balances the load exactly.
namespace {

constexpr int W_ST = 3;                 // pipeline stages
constexpr int W_THREADS = 320;          // warp 0 TMA, warp 1 MMA, warps 2-9 epilogue
constexpr int W_BOX = GK * 128;         // 64 tokens x 64 features bf16 = 8 KB
constexpr int W_OPER = 4 * W_BOX;       // one operand: 64 tokens x 256 features = 32 KB
constexpr int W_STAGE = 2 * W_OPER;
constexpr int W_OFF_BAR = W_ST * W_STAGE;
constexpr int W_N_BAR = 2 * W_ST + 1 + 2 + 1;   // full/empty stages, acc full, acc empty x2, drain
constexpr int W_OFF_T = (W_OFF_BAR + W_N_BAR * 8 + 16 + 1023) / 1024 * 1024;   // epilogue staging, 8 warps x 4 KB
constexpr int W_SMEM = W_OFF_T + 8 * 32 * 32 * 4;
constexpr int W_BAND = 8;               // tile columns per band of the blocked order
static_assert(W_SMEM <= 232448, "shared memory per CTA");
static_assert(W_OFF_T % 1024 == 0, "staging blocks on the 1 KB period of the 128-byte swizzle");
static_assert(W_STAGE % 1024 == 0, "swizzle atoms need 1 KB aligned boxes");

struct WideParams {
  int32_t D;
  int32_t NB;          // D / 256
  int32_t n_ktiles;    // ceil(T / GK)
  int32_t U[3];        // tiles per kind: G (upper, diagonal included), X (all), S (upper)
  int32_t waves[3];    // full waves per kind
  int64_t tail_total;  // steps of the shared tail
  int32_t form;        // 0 exact (bf16 hi / lo), 1 scaled (fp16)
  int32_t passes[3];   // passes per tile of G, X, S
  uint32_t idesc;      // UMMA instruction descriptor of the form
  const float* unscale;   // scaled form: the factor of G, X, S sums; null: 1
  float* gram;
  int* status;
  uint64_t wait_limit_ns;
  uint32_t* heartbeat;
};

// t-th tile of a kind in the blocked order -> (row block, column block), 256-feature units.
__device__ __forceinline__ void wide_tile(int kind, int t, int NB, int& bi, int& bj) {
  const bool upper = kind != 1;
  for (int c0 = 0; c0 < NB; c0 += W_BAND) {
    const int c1 = min(c0 + W_BAND, NB);
    for (int r = 0; r < NB; ++r) {
      const int lo = upper ? max(c0, r) : c0;
      const int n = c1 > lo ? c1 - lo : 0;
      if (t < n) {
        bi = r;
        bj = lo + t;
        return;
      }
      t -= n;
    }
  }
  bi = bj = 0;
}

struct WSeg {
  int kind, bi, bj;
  int s0, s1;   // steps [s0, s1) of the tile; step = pass * n_ktiles + token block
};

struct WIter {
  int k, w;
  int64_t g, ge;   // this CTA's range of the tail
};

__device__ __forceinline__ void wit_init(const WideParams& p, WIter& it) {
  it.k = 0;
  it.w = 0;
  it.g = p.tail_total * blockIdx.x / gridDim.x;
  it.ge = p.tail_total * (blockIdx.x + 1) / gridDim.x;
}

// Next segment of this CTA's work (the same sequence for all its roles).
__device__ __forceinline__ bool wit_next(const WideParams& p, WIter& it, WSeg& s) {
  const int G = gridDim.x;
  while (it.k < 3) {
    if (it.w < pick3(p.waves, it.k)) {
      s.kind = it.k;
      wide_tile(it.k, it.w * G + static_cast<int>(blockIdx.x), p.NB, s.bi, s.bj);
      s.s0 = 0;
      s.s1 = pick3(p.passes, it.k) * p.n_ktiles;
      ++it.w;
      return true;
    }
    ++it.k;
    it.w = 0;
  }
  if (it.g >= it.ge) return false;
  int64_t g = it.g;
  int k = 0;
  for (; k < 3; ++k) {
    const int64_t n = static_cast<int64_t>(pick3(p.U, k) - pick3(p.waves, k) * G) * pick3(p.passes, k) * p.n_ktiles;
    if (g < n) break;
    g -= n;
  }
  if (k >= 3) return false;
  const int64_t L = static_cast<int64_t>(pick3(p.passes, k)) * p.n_ktiles;
  s.kind = k;
  wide_tile(k, pick3(p.waves, k) * G + static_cast<int>(g / L), p.NB, s.bi, s.bj);
  s.s0 = static_cast<int>(g % L);
  const int64_t rest = it.ge - it.g;
  s.s1 = static_cast<int>(L < s.s0 + rest ? L : s.s0 + rest);
  it.g += s.s1 - s.s0;
  return true;
}

}  // namespace

__global__ void __launch_bounds__(W_THREADS, 1)
    gram_wide_kernel(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_hi,
                     const __grid_constant__ CUtensorMap tm_lo, const __grid_constant__ CUtensorMap tm_state,
                     const WideParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = smem_raw;
  const uint32_t sbase = smem_u32(smem);
  if (sbase & 1023u) {  // uniform over the CTA; nothing is initialised yet
    if (threadIdx.x == 0) record_error(p.status, DEVERR_LAYOUT, 0, sbase, 0, 2);
    return;
  }
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + W_OFF_BAR);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + W_N_BAR);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8 * W_ST, accf = empty0 + 8 * W_ST,
                 acce0 = accf + 8, drain_bar = acce0 + 16;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_kt = p.n_ktiles;

  if (threadIdx.x == 0) {
    for (int i = 0; i < W_ST; ++i) {
      mbar_init(full0 + 8 * i, 1);
      mbar_init(empty0 + 8 * i, 1);
    }
    mbar_init(accf, 1);
    mbar_init(acce0, 128);
    mbar_init(acce0 + 8, 128);
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (threadIdx.x == 0) heartbeat(p.heartbeat, 0);
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), 512);
    tmem_relinquish();
    if (lane == 0) heartbeat(p.heartbeat, 1);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();   // the operands and the state may come from the kernel before this one
  const WaitCtx wc{abort_flag, p.status, p.wait_limit_ns};

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      auto map = [&](int w) { return w == 0 ? &tm_a : (w == 1 ? &tm_hi : &tm_lo); };
      WIter it;
      wit_init(p, it);
      WSeg sg;
      int i = 0;
      bool ok = true;
      while (ok && wit_next(p, it, sg)) {
        for (int st = sg.s0; st < sg.s1; ++st, ++i) {
          const int pass = st / n_kt;
          const int tok = (st % n_kt) * GK;
          const int sl = i % W_ST;
          if (!mbar_wait(empty0 + 8 * sl, ((i / W_ST) & 1) ^ 1, wc, 31, i)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(full0 + 8 * sl, W_STAGE);
          const uint32_t sa = sbase + sl * W_STAGE, sb = sa + W_OPER;
          // one request per operand: (64 features, GK tokens, 4 feature blocks)
          tma_load_3d(sa, map(kPasses[p.form][sg.kind][pass].a), full0 + 8 * sl, 0, tok, sg.bi * 4);
          tma_load_3d(sb, map(kPasses[p.form][sg.kind][pass].b), full0 + 8 * sl, 0, tok, sg.bj * 4);
        }
      }
      for (int k = i > W_ST ? i - W_ST : 0; k < i; ++k)
        mbar_wait_drain(full0 + 8 * (k % W_ST), (k / W_ST) & 1, G_DRAIN_NS);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ UMMA issuer
    if (lane == 0) {
      WIter it;
      wit_init(p, it);
      WSeg sg;
      int i = 0, m = 0;
      bool ok = true;
      while (ok && wit_next(p, it, sg)) {
        // both accumulators drained by the epilogue of segment m - 1
        if (!mbar_wait(acce0, (m & 1) ^ 1, wc, 34, m) || !mbar_wait(acce0 + 8, (m & 1) ^ 1, wc, 35, m)) break;
        tc_fence_after();
        for (int st = sg.s0; st < sg.s1; ++st, ++i) {
          const int sl = i % W_ST;
          if (!mbar_wait(full0 + 8 * sl, (i / W_ST) & 1, wc, 32, i)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = sbase + sl * W_STAGE, sb = sa + W_OPER;
#pragma unroll
          for (int k = 0; k < GK / 16; ++k) {
            const uint32_t acc = (st != sg.s0 || k > 0) ? 1u : 0u;
            const uint64_t db = sw128_desc(sb + k * 2048, W_BOX, 1024);
            umma_ss(tmem, sw128_desc(sa + k * 2048, W_BOX, 1024), db, p.idesc, acc);
            umma_ss(tmem + 256, sw128_desc(sa + 2 * W_BOX + k * 2048, W_BOX, 1024), db, p.idesc, acc);
          }
          tc_commit(empty0 + 8 * sl);
        }
        if (!ok) break;
        tc_commit(accf);
        ++m;
      }
      tc_commit(drain_bar);
      mbar_wait_drain(drain_bar, 0, G_DRAIN_NS);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue (warps 2-9)
    // warps 2-5 drain the upper accumulator, 6-9 the lower one; warp w reads TMEM lanes
    // 32 (w % 4) .. + 31
    // Each 32 x 32 block goes TMEM -> registers -> this warp's 4 KB staging block (16-byte
    // chunk q of row r at chunk q ^ (r & 7), the 128-byte swizzle of the state's tensor map) ->
    // one bulk tensor reduce-add into the fp32 state, performed by the memory system.  The
    // accumulator is handed back to the UMMA thread as soon as the warp's last TMEM load has
    // completed, so the next tile's UMMAs overlap the staging and reduction of the last block.
    const int half = (warp - 2) >> 2;
    const int quarter = warp & 3;
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(quarter * 32) << 16) + half * 256;
    const int D = p.D;
    float4* tbuf = reinterpret_cast<float4*>(smem + W_OFF_T) + (warp - 2) * 32 * 8;
    const uint32_t tbuf_s = smem_u32(tbuf);
    WIter it;
    wit_init(p, it);
    WSeg sg;
    int m = 0;
    while (wit_next(p, it, sg)) {
      if (!__all_sync(0xffffffffu, mbar_wait(accf, m & 1, wc, 33, m))) break;
      tc_fence_after();
      const int row0 = (sg.kind == 2 ? D : 0) + sg.bi * 256 + half * 128 + quarter * 32;
      const int col0 = (sg.kind == 0 ? 0 : D) + sg.bj * 256;
      const float scale = p.unscale ? p.unscale[sg.kind] : 1.f;
      // Two batches of four 32-column chunks: a batch's TMEM loads go out together, and the
      // accumulator is handed back after the second batch's loads, waiting on the staging of
      // three blocks instead of seven.
#pragma unroll 1
      for (int hb = 0; hb < 2; ++hb) {
        uint32_t v[4][32];
#pragma unroll
        for (int cc = 0; cc < 4; ++cc) tmem_ld32(lane_base + 32 * (4 * hb + cc), v[cc]);
#pragma unroll
        for (int cc = 0; cc < 4; ++cc) tmem_wait_ld32(v[cc]);
        if (hb == 1) {
          tc_fence_before();
          mbar_arrive(acce0 + 8 * half);   // accumulator may be overwritten
        }
#pragma unroll
        for (int cc = 0; cc < 4; ++cc) {
          const int c = 4 * hb + cc;
          if (lane == 0) bulk_wait_read_all();   // the previous block's reduce has read the staging block
          __syncwarp();
#pragma unroll
          for (int q = 0; q < 8; ++q)
            tbuf[lane * 8 + (q ^ (lane & 7))] =
                make_float4(__uint_as_float(v[cc][4 * q]) * scale, __uint_as_float(v[cc][4 * q + 1]) * scale,
                            __uint_as_float(v[cc][4 * q + 2]) * scale, __uint_as_float(v[cc][4 * q + 3]) * scale);
          fence_proxy_async_smem();   // these generic-proxy writes before the bulk copy reads them
          __syncwarp();
          if (lane == 0) {
            tma_reduce_add_2d(&tm_state, tbuf_s, col0 + 32 * c, row0);
            bulk_commit_group();
          }
        }
      }
      ++m;
    }
    if (lane == 0) bulk_wait_all();   // every reduce done before the CTA exits
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
    if (lane == 0) heartbeat(p.heartbeat, 2);
  }
}

static cudaError_t launch_gram_wide(int32_t D, int64_t T, int form, const void* op0, const void* op1,
                                    const void* op2, const float* unscale, float* gram, int* status,
                                    uint64_t wait_limit_ns, uint32_t* hb, cudaStream_t s) {
  int dev = 0, sms = 152;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  {
    const cudaError_t e = set_smem_limit_once(reinterpret_cast<const void*>(gram_wide_kernel), W_SMEM);
    if (e != cudaSuccess) return e;
  }
  // [T][D] operands viewed as (64 features, T tokens, D/64 feature blocks); one box
  // (64, GK, 4) is a 256-feature slice of GK tokens as 4 swizzled [GK][128 B] blocks
  // (the maps' bf16 element type only sets the 2-byte element size and the zero fill: the
  // scaled form's fp16 operands go through the same maps)
  CUtensorMap tm[3], tm_state;
  const void* srcs[3] = {op0, op1, op2};
  for (int i = 0; i < 3; ++i)
    if (!encode_tmap_3d(&tm[i], srcs[i], 64, T, D / 64, static_cast<uint64_t>(D) * 2, 128, 64, GK, 4))
      return cudaErrorInvalidValue;
  // the fp32 [2D][2D] state, 32 x 32 boxes of 128-byte rows
  if (!encode_tmap_2d_f32(&tm_state, gram, 2 * static_cast<uint64_t>(D), 2 * static_cast<uint64_t>(D),
                          2 * static_cast<uint64_t>(D) * 4, 32, 32))
    return cudaErrorInvalidValue;
  WideParams p;
  p.D = D;
  p.NB = D / 256;
  p.n_ktiles = static_cast<int32_t>((T + GK - 1) / GK);
  const int32_t n_upper = p.NB * (p.NB + 1) / 2;
  p.U[0] = n_upper;
  p.U[1] = p.NB * p.NB;
  p.U[2] = n_upper;
  const int* passes = form ? kPassesScaled : kPassesExact;
  p.form = form;
  for (int k = 0; k < 3; ++k) p.passes[k] = passes[k];
  p.idesc = form ? idesc_f16(128, 256, true, true) : idesc_bf16(128, 256, true, true);
  p.unscale = unscale;
  int64_t total = 0;
  for (int k = 0; k < 3; ++k) total += static_cast<int64_t>(p.U[k]) * passes[k] * p.n_ktiles;
  if (total > INT32_MAX) return cudaErrorInvalidValue;
  // one CTA per SM, each with at least 16 steps (a 1024-token run of one tile)
  const int64_t want = (total + 15) / 16;
  const int grid = static_cast<int>(want < sms ? (want > 0 ? want : 1) : sms);
  p.tail_total = 0;
  for (int k = 0; k < 3; ++k) {
    p.waves[k] = p.U[k] / grid;
    p.tail_total += static_cast<int64_t>(p.U[k] - p.waves[k] * grid) * passes[k] * p.n_ktiles;
  }
  p.gram = gram;
  p.status = status;
  p.wait_limit_ns = wait_limit_ns;
  p.heartbeat = hb;
  return launch_pdl(gram_wide_kernel, grid, dim3(W_THREADS), W_SMEM, s, tm[0], tm[1], tm[2], tm_state, p);
}

// The workspace of one call: two 2-byte [T][D] operands (hi and lo, or the scaled A_loc and
// Delta), 256-byte aligned, then the scaled form's block maxima and its three factors.
constexpr int kAmaxBlocks = 1024;   // at most this many amax_kernel blocks
constexpr size_t kAmaxBytes = (2 * kAmaxBlocks + 4) * sizeof(float);

static size_t ls_operand_bytes(int32_t D, int64_t T) {
  return (static_cast<size_t>(T) * D * 2 + 255) & ~static_cast<size_t>(255);
}

size_t ls_accumulate_ws_bytes(int32_t D, int64_t T) { return 2 * ls_operand_bytes(D, T) + kAmaxBytes; }

template <int BN>
static cudaError_t launch_gram(int32_t D, int64_t T, int form, const void* op0, const void* op1, const void* op2,
                               const float* unscale, float* gram, int* status, uint64_t wait_limit_ns, uint32_t* hb,
                               cudaStream_t s) {
  using C = GCfg<BN>;
  int dev = 0, sms = 152;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  {
    const cudaError_t e = set_smem_limit_once(reinterpret_cast<const void*>(gram_kernel<BN>), C::SMEM);
    if (e != cudaSuccess) return e;
  }
  // [T][D] operands viewed as (64 features, T tokens, D/64 feature blocks): the block
  // stride (128 B) is below the token stride, so one box (64, GK, n) fetches n adjacent
  // 64-feature blocks as n consecutive [GK][128 B] swizzled blocks in a single request.
  // (measured on GB300: 11 % faster than one 2-D request per 64-feature block at hidden
  // 1536, 1 % at hidden 5120)
  CUtensorMap tr[3], tc[3];
  const void* srcs[3] = {op0, op1, op2};
  for (int i = 0; i < 3; ++i)
    if (!encode_tmap_3d(&tr[i], srcs[i], 64, T, D / 64, static_cast<uint64_t>(D) * 2, 128, 64, GK, GM / 64) ||
        !encode_tmap_3d(&tc[i], srcs[i], 64, T, D / 64, static_cast<uint64_t>(D) * 2, 128, 64, GK, BN / 64))
      return cudaErrorInvalidValue;
  const int RB = D / GM, CB = D / BN;
  int n_upper = 0;
  for (int r = 0; r < RB; ++r) n_upper += CB - (r * GM) / BN;
  GramParams p;
  p.D = D;
  p.T = static_cast<int32_t>(T);
  p.n_ktiles = static_cast<int32_t>((T + GK - 1) / GK);
  p.n_upper = n_upper;
  p.n_full = RB * CB;
  const int* passes = form ? kPassesScaled : kPassesExact;
  p.form = form;
  for (int k = 0; k < 3; ++k) p.passes[k] = passes[k];
  p.idesc = form ? idesc_f16(GM, BN, true, true) : idesc_bf16(GM, BN, true, true);
  p.unscale = unscale;
  const int64_t total =
      static_cast<int64_t>(p.n_ktiles) * (n_upper * passes[0] + p.n_full * passes[1] + n_upper * passes[2]);
  if (total > INT32_MAX) return cudaErrorInvalidValue;
  p.total = static_cast<int32_t>(total);
  p.gram = gram;
  p.status = status;
  p.wait_limit_ns = wait_limit_ns;
  p.heartbeat = hb;
  // one CTA per SM, each with at least 16 steps (a 1024-token run of one tile)
  const int64_t want = (total + 15) / 16;
  const dim3 grid(static_cast<unsigned>(want < sms ? (want > 0 ? want : 1) : sms));
  return launch_pdl(gram_kernel<BN>, grid, dim3(G_THREADS), C::SMEM, s, tr[0], tr[1], tr[2], tc[0], tc[1], tc[2],
                    p);
}

cudaError_t launch_ls_accumulate(int32_t D, int64_t T, const void* a_loc, const void* a_full, void* ws,
                                 bool exact, float* gram, int* status, uint64_t wait_limit_ns, uint32_t* hb,
                                 cudaStream_t s) {
  const size_t one = ls_operand_bytes(D, T);
  uint8_t* op1 = static_cast<uint8_t*>(ws);
  uint8_t* op2 = op1 + one;
  float* part = reinterpret_cast<float*>(op2 + one);
  float* unscale = part + 2 * kAmaxBlocks;
  const int64_t n_words = static_cast<int64_t>(T) * D / 8;
  int dev = 0, sms = 152;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int64_t blocks = (n_words + 255) / 256;
  if (blocks > static_cast<int64_t>(sms) * 8) blocks = static_cast<int64_t>(sms) * 8;
  if (exact) {
    // hi, lo of Delta; the Gram kernel reads A_loc itself
    const cudaError_t e = launch_pdl(split_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, s,
                                     static_cast<const uint4*>(a_loc), static_cast<const uint4*>(a_full),
                                     reinterpret_cast<uint4*>(op1), reinterpret_cast<uint4*>(op2), n_words);
    if (e != cudaSuccess) return e;
    if (D % 256 == 0) return launch_gram_wide(D, T, 0, a_loc, op1, op2, nullptr, gram, status, wait_limit_ns, hb, s);
    return launch_gram<128>(D, T, 0, a_loc, op1, op2, nullptr, gram, status, wait_limit_ns, hb, s);
  }
  // scaled A_loc (op1) and Delta (op2) in fp16
  int nb = static_cast<int>(blocks < kAmaxBlocks ? blocks : kAmaxBlocks);
  cudaError_t e = launch_pdl(amax_kernel, dim3(static_cast<unsigned>(nb)), dim3(256), 0, s,
                             static_cast<const uint4*>(a_loc), static_cast<const uint4*>(a_full), n_words, part);
  if (e != cudaSuccess) return e;
  e = launch_pdl(convert_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, s,
                 static_cast<const uint4*>(a_loc), static_cast<const uint4*>(a_full), n_words,
                 static_cast<const float*>(part), nb, reinterpret_cast<uint4*>(op1), reinterpret_cast<uint4*>(op2),
                 unscale);
  if (e != cudaSuccess) return e;
  if (D % 256 == 0) return launch_gram_wide(D, T, 1, op1, op2, op2, unscale, gram, status, wait_limit_ns, hb, s);
  return launch_gram<128>(D, T, 1, op1, op2, op2, unscale, gram, status, wait_limit_ns, hb, s);
}

}  // namespace ispa
