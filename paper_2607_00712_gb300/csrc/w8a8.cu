// W8A8 output projection on W + dW (Sec. 4, post-training quantisation; Sec. 3.2 for the
// injected weight): 8-bit e4m3 activations and weights on the tensor cores
// (tcgen05 kind::f8f6f4, fp32 accumulators in TMEM).
//
//   quant_rows_kernel    activations [T][D] bf16 -> e4m3 codes [T][D] + one fp32 scale per token
//   col_amax_kernel,     W (+ dW) fp32 [D][D_out] -> e4m3 codes [D_out][D] (K-major, i.e. the
//   quant_wt_kernel,     layout of a torch Linear weight) + one fp32 scale per output channel
//   col_scale_kernel
//   w8a8_gemm_kernel     out[t][n] = bf16(a_scale[t] * w_scale[n] * sum_k a[t][k] w[n][k])
//
// Quantisation arithmetic (fp32, rounded to nearest at every step, identical to the
// oracle's): amax = max |x|; inv = 448 / amax, scale = amax / 448 (both 1 for an all-zero
// group); code = e4m3(x * inv), round to nearest even with saturation at +-448.
//
// GEMM: persistent, one CTA per SM looping over 128 x BN output tiles (BN = 256, 192 or 128,
// whichever gives the shortest estimated run: waves of tiles x their cost); both operands
// K-major with 128-byte swizzle (one 128-byte row = 128 codes = four K=32 UMMA steps), a
// 4-stage TMA ring that runs on across tile boundaries, two accumulator sets in TMEM so that
// the epilogue of one tile (both scales, bf16 store) overlaps the UMMAs of the next; with
// 128-column tiles each set has two accumulation chains that the k-steps alternate between.
// Warp 0 issues TMA, warp 1 allocates TMEM and issues UMMAs, warps 2-5 drain TMEM (warp w
// reads lanes 32 (w % 4) .. +31).  Every wait is bounded.
#include <cuda.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include <algorithm>

#include "internal.h"
#include "ptx.cuh"

namespace ispa {

namespace {

constexpr float kE4M3Max = 448.f;

// Two fp32 values -> two e4m3 codes (round to nearest even, saturating), x0 in the low byte.
__device__ __forceinline__ uint16_t e4m3x2(float x0, float x1) {
  uint16_t r;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(r) : "f"(x1), "f"(x0));
  return r;
}

// One warp per row (grid-stride over rows); cols % 8 == 0.  Rows of up to 32 * CACHE
// 16-byte words (8 bf16 each) stay in registers between the max and the quantisation pass;
// longer rows are read twice.
constexpr int CACHE = 12;
__global__ void __launch_bounds__(256) quant_rows_kernel(const __nv_bfloat16* __restrict__ x, int64_t rows,
                                                         int cols, uint8_t* __restrict__ q,
                                                         float* __restrict__ scale) {
  const int lane = threadIdx.x & 31;
  const int nw = cols / 8;   // 16-byte words of bf16 per row
  const int64_t warps = static_cast<int64_t>(gridDim.x) * (blockDim.x >> 5);
  for (int64_t r = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + (threadIdx.x >> 5); r < rows; r += warps) {
    const uint4* xr = reinterpret_cast<const uint4*>(x + r * cols);
    uint4 cache[CACHE];
    float amax = 0.f;
#pragma unroll
    for (int c = 0; c < CACHE; ++c) {
      const int i = lane + 32 * c;
      cache[c] = i < nw ? xr[i] : make_uint4(0, 0, 0, 0);
    }
    for (int i = lane + 32 * CACHE; i < nw; i += 32) {
      const uint4 v = xr[i];
      const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int e = 0; e < 4; ++e)
        amax = fmaxf(amax, fmaxf(fabsf(__uint_as_float(w[e] << 16)), fabsf(__uint_as_float(w[e] & 0xFFFF0000u))));
    }
#pragma unroll
    for (int c = 0; c < CACHE; ++c) {
      const uint32_t w[4] = {cache[c].x, cache[c].y, cache[c].z, cache[c].w};
#pragma unroll
      for (int e = 0; e < 4; ++e)
        amax = fmaxf(amax, fmaxf(fabsf(__uint_as_float(w[e] << 16)), fabsf(__uint_as_float(w[e] & 0xFFFF0000u))));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
    const float inv = amax == 0.f ? 1.f : __fdiv_rn(kE4M3Max, amax);
    uint2* qr = reinterpret_cast<uint2*>(q + r * cols);
    auto quant8 = [&](const uint4& v) {
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
    };
#pragma unroll
    for (int c = 0; c < CACHE; ++c) {
      const int i = lane + 32 * c;
      if (i < nw) qr[i] = quant8(cache[c]);
    }
    for (int i = lane + 32 * CACHE; i < nw; i += 32) qr[i] = quant8(xr[i]);
    if (lane == 0) scale[r] = amax == 0.f ? 1.f : __fdiv_rn(amax, kE4M3Max);
  }
}

__device__ __forceinline__ float w_plus_dw(const float* W, const float* dW, int64_t i) {
  return dW ? __fadd_rn(W[i], dW[i]) : W[i];
}

// Per-column max |W + dW| into amax[D_out].  Block (32, 8) per 32 columns.
__global__ void col_amax_kernel(const float* __restrict__ W, const float* __restrict__ dW, int D, int Dout,
                                float* __restrict__ amax) {
  __shared__ float red[8][33];
  const int n = blockIdx.x * 32 + threadIdx.x;
  float m = 0.f;
  if (n < Dout)
    for (int k = threadIdx.y; k < D; k += 8) m = fmaxf(m, fabsf(w_plus_dw(W, dW, static_cast<int64_t>(k) * Dout + n)));
  red[threadIdx.y][threadIdx.x] = m;
  __syncthreads();
  if (threadIdx.y == 0 && n < Dout) {
#pragma unroll
    for (int i = 1; i < 8; ++i) m = fmaxf(m, red[i][threadIdx.x]);
    amax[n] = m;
  }
}

// codes[n][k] = e4m3((W + dW)[k][n] * inv_n) through a 32 x 32 shared-memory transpose.
// Block (32, 8); grid (ceil(D / 32), ceil(Dout / 32)).
__global__ void quant_wt_kernel(const float* __restrict__ W, const float* __restrict__ dW, int D, int Dout,
                                const float* __restrict__ amax, uint8_t* __restrict__ q_t) {
  __shared__ uint8_t tile[32][36];
  const int k0 = blockIdx.x * 32, n0 = blockIdx.y * 32;
  const int n = n0 + threadIdx.x;
  const float am = n < Dout ? amax[n] : 0.f;
  const float inv = am == 0.f ? 1.f : __fdiv_rn(kE4M3Max, am);
  for (int j = threadIdx.y; j < 32; j += 8) {
    const int k = k0 + j;
    uint8_t c = 0;
    if (k < D && n < Dout) {
      const float v = __fmul_rn(w_plus_dw(W, dW, static_cast<int64_t>(k) * Dout + n), inv);
      c = static_cast<uint8_t>(e4m3x2(v, 0.f) & 0xFF);
    }
    tile[j][threadIdx.x] = c;   // [k][n]
  }
  __syncthreads();
  for (int j = threadIdx.y; j < 32; j += 8) {
    const int nn = n0 + j, k = k0 + threadIdx.x;
    if (nn < Dout && k < D) q_t[static_cast<int64_t>(nn) * D + k] = tile[threadIdx.x][j];
  }
}

__global__ void col_scale_kernel(float* __restrict__ s, int Dout) {
  const int n = blockIdx.x * blockDim.x + threadIdx.x;
  if (n < Dout) s[n] = s[n] == 0.f ? 1.f : __fdiv_rn(s[n], kE4M3Max);
}

// ------------------------------------------------------------ GEMM
constexpr int QM = 128;        // output rows (tokens) per tile
constexpr int QK = 128;        // K (bytes = codes) per stage: one 128-byte swizzled row
constexpr int Q_THREADS = 192;
constexpr uint64_t Q_DRAIN_NS = 200ull * 1000 * 1000;

template <int BN>
struct QCfg {
  // Persistent: one CTA per SM loops over output tiles.  Two accumulator sets in TMEM let the
  // epilogue of one tile overlap the UMMAs of the next; with 128-column tiles each set holds
  // two accumulation chains (k-steps alternate between them), with 192- and 256-column tiles one.
  static_assert(BN == 128 || BN == 192 || BN == 256, "tile width");
  static constexpr int CHAINS = BN == 128 ? 2 : 1;
  static constexpr int SET = CHAINS * BN;         // TMEM columns per accumulator set
  static constexpr int QST = 4;
  static constexpr int A_BYTES = QM * QK;         // 16 KB
  static constexpr int B_BYTES = BN * QK;         // 32, 24 or 16 KB
  static constexpr int STAGE = A_BYTES + B_BYTES;
  static constexpr int OFF_BAR = QST * STAGE;
  static constexpr int N_BAR = 2 * QST + 4 + 1;   // full/empty per stage, set full/empty x2, drain
  static constexpr int SMEM = OFF_BAR + N_BAR * 8 + 16;
  // more than half of an SM's shared memory: one CTA per SM, so the 512-column TMEM
  // allocation never waits for another CTA
  static_assert(SMEM > 116 * 1024 && SMEM <= 232448 && STAGE % 1024 == 0, "shared memory layout");
  static constexpr uint32_t IDESC = idesc_e4m3(QM, BN);
  static constexpr uint32_t TMEM_COLS = 512;      // the allocation (a power of two)
  static_assert(2 * SET <= 512, "two accumulator sets fit in TMEM");
};

struct GemmParams {
  int32_t T, D, Dout, n_kb;
  int32_t n_mt, n_tiles;   // row tiles; all tiles (tile t: rows (t % n_mt), columns (t / n_mt))
  const float* a_scale;
  const float* w_scale;
  __nv_bfloat16* out;
  int* status;
  uint64_t wait_limit_ns;
};

template <int BN>
__global__ void __launch_bounds__(Q_THREADS, 1)
    w8a8_gemm_kernel(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_w,
                     const GemmParams p) {
  using C = QCfg<BN>;
  constexpr int QST = C::QST;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = smem_raw;
  const uint32_t sbase = smem_u32(smem);
  if (sbase & 1023u) {
    if (threadIdx.x == 0) record_error(p.status, DEVERR_LAYOUT, 0, sbase, 0, 2);
    return;
  }
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + C::N_BAR);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8 * QST, accf0 = empty0 + 8 * QST,
                 acce0 = accf0 + 16, drain_bar = acce0 + 16;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_kb = p.n_kb;

  if (threadIdx.x == 0) {
    for (int i = 0; i < QST; ++i) {
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
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const WaitCtx wc{abort_flag, p.status, p.wait_limit_ns};

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      int g = 0;   // k-blocks issued over all tiles of this CTA
      bool ok = true;
      for (int t = blockIdx.x; ok && t < p.n_tiles; t += gridDim.x) {
        const int m0 = (t % p.n_mt) * QM, n0 = (t / p.n_mt) * BN;
        for (int kb = 0; kb < n_kb; ++kb, ++g) {
          const int st = g % QST;
          if (!mbar_wait(empty0 + 8 * st, ((g / QST) & 1) ^ 1, wc, 31, g)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(full0 + 8 * st, C::STAGE);
          const uint32_t sa = sbase + st * C::STAGE;
          tma_load_2d(sa, &tm_a, full0 + 8 * st, kb * QK, m0);
          tma_load_2d(sa + C::A_BYTES, &tm_w, full0 + 8 * st, kb * QK, n0);
        }
      }
      for (int i = g > QST ? g - QST : 0; i < g; ++i)
        mbar_wait_drain(full0 + 8 * (i % QST), (i / QST) & 1, Q_DRAIN_NS);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ UMMA issuer
    if (lane == 0) {
      int g = 0, i = 0;
      bool ok = true;
      for (int t = blockIdx.x; ok && t < p.n_tiles; t += gridDim.x, ++i) {
        const int set = i & 1;
        // the epilogue has drained this set's previous tile (tile i - 2)
        if (!mbar_wait(acce0 + 8 * set, ((i >> 1) & 1) ^ 1, wc, 34, i)) break;
        tc_fence_after();
        const uint32_t acc = tmem + set * C::SET;
        for (int kb = 0; kb < n_kb; ++kb, ++g) {
          const int st = g % QST;
          if (!mbar_wait(full0 + 8 * st, (g / QST) & 1, wc, 32, g)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = sbase + st * C::STAGE, sb = sa + C::A_BYTES;
          // four K=32 steps inside the 128-byte swizzle row (alternating chains for BN 128)
#pragma unroll
          for (int k = 0; k < QK / 32; ++k)
            umma_f8(acc + (C::CHAINS == 2 ? (k & 1) * BN : 0), sw128_desc(sa + 32 * k, 16, 1024),
                    sw128_desc(sb + 32 * k, 16, 1024), C::IDESC, (kb > 0 || k >= C::CHAINS) ? 1u : 0u);
          tc_commit(empty0 + 8 * st);
        }
        if (!ok) break;
        tc_commit(accf0 + 8 * set);
      }
      tc_commit(drain_bar);
      mbar_wait_drain(drain_bar, 0, Q_DRAIN_NS);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue (warps 2-5)
    const int quarter = warp & 3;
    int i = 0;
    for (int t = blockIdx.x; t < p.n_tiles; t += gridDim.x, ++i) {
      const int set = i & 1;
      if (!__all_sync(0xffffffffu, mbar_wait(accf0 + 8 * set, (i >> 1) & 1, wc, 33, i))) break;
      tc_fence_after();
      const int m0 = (t % p.n_mt) * QM, n0 = (t / p.n_mt) * BN;
      const int row = m0 + quarter * 32 + lane;
      const uint32_t taddr = tmem + (static_cast<uint32_t>(quarter * 32) << 16) + set * C::SET;
      const float sa = row < p.T ? p.a_scale[row] : 0.f;
      __nv_bfloat16* orow = p.out + static_cast<size_t>(row) * p.Dout + n0;
#pragma unroll 1
      for (int c = 0; c < BN / 32; ++c) {
        // the 32 columns' weight scales (the same for every lane), loaded before the TMEM wait
        float sw[32];
        const float4* sw4 = reinterpret_cast<const float4*>(p.w_scale + n0 + 32 * c);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const float4 t = sw4[q];
          sw[4 * q] = t.x;
          sw[4 * q + 1] = t.y;
          sw[4 * q + 2] = t.z;
          sw[4 * q + 3] = t.w;
        }
        uint32_t v0[32], v1[32];
        tmem_ld32(taddr + 32 * c, v0);
        tmem_wait_ld32(v0);
        if constexpr (C::CHAINS == 2) {
          tmem_ld32(taddr + BN + 32 * c, v1);
          tmem_wait_ld32(v1);
        }
        if (row < p.T) {
          uint32_t pk[16];
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            float s0 = __uint_as_float(v0[2 * e]), s1 = __uint_as_float(v0[2 * e + 1]);
            if constexpr (C::CHAINS == 2) {
              s0 += __uint_as_float(v1[2 * e]);
              s1 += __uint_as_float(v1[2 * e + 1]);
            }
            pk[e] = pack_bf16x2(__fmul_rn(__fmul_rn(s0, sa), sw[2 * e]), __fmul_rn(__fmul_rn(s1, sa), sw[2 * e + 1]));
          }
          uint4* d4 = reinterpret_cast<uint4*>(orow + 32 * c);
#pragma unroll
          for (int q = 0; q < 4; ++q) d4[q] = make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
        }
      }
      tc_fence_before();
      mbar_arrive(acce0 + 8 * set);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

template <int BN>
cudaError_t launch_gemm_bn(const uint8_t* a_q, const float* a_scale, const uint8_t* w_q, const float* w_scale,
                           int32_t T, int32_t D, int32_t Dout, __nv_bfloat16* out, int* status,
                           uint64_t wait_limit_ns, cudaStream_t s) {
  using C = QCfg<BN>;
  int dev = 0;
  cudaGetDevice(&dev);
  {
    const cudaError_t e = set_smem_limit_once(reinterpret_cast<const void*>(w8a8_gemm_kernel<BN>), C::SMEM);
    if (e != cudaSuccess) return e;
  }
  CUtensorMap ta, tw;
  if (!encode_tmap_2d_u8(&ta, a_q, D, T, D, QK, QM) || !encode_tmap_2d_u8(&tw, w_q, D, Dout, D, QK, BN))
    return cudaErrorInvalidValue;
  GemmParams p;
  p.T = T;
  p.D = D;
  p.Dout = Dout;
  p.n_kb = D / QK;
  p.n_mt = (T + QM - 1) / QM;
  p.n_tiles = p.n_mt * (Dout / BN);
  p.a_scale = a_scale;
  p.w_scale = w_scale;
  p.out = out;
  p.status = status;
  p.wait_limit_ns = wait_limit_ns;
  int dev_sms = 152;
  cudaDeviceGetAttribute(&dev_sms, cudaDevAttrMultiProcessorCount, dev);
  const int grid = p.n_tiles < dev_sms ? p.n_tiles : dev_sms;
  w8a8_gemm_kernel<BN><<<grid, Q_THREADS, C::SMEM, s>>>(ta, tw, p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_quant_rows(const void* x, int64_t rows, int32_t cols, uint8_t* q, float* scale, cudaStream_t s) {
  int dev = 0, sms = 152;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t want = (rows + 7) / 8;   // one warp per row, 8 warps per block
  const int64_t blocks = want < static_cast<int64_t>(sms) * 16 ? want : static_cast<int64_t>(sms) * 16;
  quant_rows_kernel<<<static_cast<unsigned>(blocks), 256, 0, s>>>(static_cast<const __nv_bfloat16*>(x), rows, cols,
                                                                    q, scale);
  return cudaGetLastError();
}

cudaError_t launch_quant_weight(const float* W, const float* dW, int32_t D, int32_t Dout, uint8_t* q_t, float* scale,
                                cudaStream_t s) {
  col_amax_kernel<<<(Dout + 31) / 32, dim3(32, 8), 0, s>>>(W, dW, D, Dout, scale);
  quant_wt_kernel<<<dim3((D + 31) / 32, (Dout + 31) / 32), dim3(32, 8), 0, s>>>(W, dW, D, Dout, scale, q_t);
  col_scale_kernel<<<(Dout + 255) / 256, 256, 0, s>>>(scale, Dout);
  return cudaGetLastError();
}

cudaError_t launch_w8a8_gemm(const uint8_t* a_q, const float* a_scale, const uint8_t* w_q, const float* w_scale,
                             int32_t T, int32_t D, int32_t Dout, void* out, int* status, uint64_t wait_limit_ns,
                             cudaStream_t s) {
  __nv_bfloat16* o = static_cast<__nv_bfloat16*>(out);
  int dev = 0, sms = 152;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  // Estimated run: waves of tiles (one tile per SM per wave) x the time of one tile.  A
  // k-block of a 128 x BN tile moves (128 + BN) x 128 bytes through shared memory twice (TMA
  // write, UMMA read) for 128 x BN x 128 MACs, so wider tiles need fewer bytes per MAC: relative
  // time per tile at the shared-memory limit ~ (128 + BN), with a floor at the tensor rate.
  const int64_t m_tiles = (T + QM - 1) / QM;
  int best = 128;
  double best_cost = 0.0;
  for (const int bn : {256, 192, 128}) {
    if (Dout % bn != 0) continue;
    const int64_t tiles = m_tiles * (Dout / bn);
    const double waves = static_cast<double>((tiles + sms - 1) / sms);
    const double per_tile = std::max(static_cast<double>(128 + bn), 1.5 * bn);
    const double cost = waves * per_tile;
    if (best_cost == 0.0 || cost < best_cost) {
      best = bn;
      best_cost = cost;
    }
  }
  if (best == 256)
    return launch_gemm_bn<256>(a_q, a_scale, w_q, w_scale, T, D, Dout, o, status, wait_limit_ns, s);
  if (best == 192)
    return launch_gemm_bn<192>(a_q, a_scale, w_q, w_scale, T, D, Dout, o, status, wait_limit_ns, s);
  return launch_gemm_bn<128>(a_q, a_scale, w_q, w_scale, T, D, Dout, o, status, wait_limit_ns, s);
}

}  // namespace ispa
