// Tensor-pipe cost of tcgen05 UMMA issue patterns on sm_103a (bf16 operands, fp32 accumulators
// in TMEM, M = 128, K = 16 per instruction).  One CTA per SM on every SM; thread 0 issues
// `iters` iterations of a pattern back to back and waits on one commit at the end; the cycle
// count (clock64) per UMMA and the MAC rate per SM are printed.  Optional background work on
// the other warps of the CTA shows what does and does not slow the stream down.
//
//   umma_stream            all patterns, each with and without background work
//
// Operands are whatever the CTA wrote into shared memory (small bf16 values) and whatever
// TMEM holds: the timing of a UMMA does not depend on the values.  Every wait is bounded.
#include <cstdio>
#include <cstdlib>
#include <vector>

#include "ptx.cuh"

using namespace ispa;

namespace {

constexpr int SMEM = 224 * 1024 + 1024;   // operand area + barriers
constexpr int AREA = 224 * 1024;
constexpr uint32_t KB = 1024;
constexpr int ROT_STAGE = 64 * 1024;      // pattern "rotating": K 32 KB + V 32 KB per stage

enum Pattern {
  P_PAIRS,        // PV_A S_A PV_B S_B: 8 TS N=128 + 8 SS N=128 per pair (two accumulator pairs)
  P_INTERLEAVED,  // the same instructions, the two pairs interleaved instruction by instruction
  P_TILE192,      // 12 TS N=128 + 8 SS N=192: the attention kernel's 192-key tile
  P_N256_1,       // one chain of SS N=256
  P_N256_2,       // two interleaved chains of SS N=256
  P_PVT,          // O^T = V^T P^T as SS N=256 (two query tiles) + two S chains of SS N=128
  P_ROTATING,     // P_PAIRS with K and V rotating over three stages
  P_COMMITS,      // P_PAIRS with two tcgen05.commit after every group of 8
  P_PAIRS_PLAIN,  // P_PAIRS in a code path of its own (no per-group pattern selects)
  P_PAIRS_DESC,   // the same with every descriptor precomputed (one add per UMMA)
  P_KERNEL,       // the attention kernel's issue code for one 192-key tile: PV_j (12 TS N=128) from
                  // V stage j%2 then S_j+2 (8 SS N=192) from K stage j%2, commit after each group
  P_KERNEL_NC,    // the same without the commits
  P_KERNEL_U2,    // P_KERNEL with the tile loop unrolled by two (stage and buffer parity known at
                  // compile time) and every descriptor built before the loop
  P_COUNT
};
const char* kName[P_COUNT] = {"8 TS N128 + 8 SS N128, two pairs", "same, pairs interleaved",
                              "12 TS N128 + 8 SS N192 (192-key tile)", "one chain SS N256",
                              "two interleaved chains SS N256", "O^T PV SS N256 + two S chains N128",
                              "two pairs, K/V rotating over 3 stages", "two pairs + 2 commits per group",
                              "two pairs, own code path", "two pairs, precomputed descriptors",
                              "kernel issue code, 192-key tile", "kernel issue code, no commits",
                              "kernel issue code, unrolled by 2, hoisted"};
const int kUmmas[P_COUNT] = {32, 32, 20, 8, 16, 24, 32, 32, 32, 32, 20, 20, 20};
const double kMacs[P_COUNT] = {2.0 * 256 * 128 * 128, 2.0 * 256 * 128 * 128, 2.0 * 128 * 192 * 128,
                               128.0 * 256 * 128,     2.0 * 128 * 256 * 128, 2.0 * 256 * 128 * 128,
                               2.0 * 256 * 128 * 128, 2.0 * 256 * 128 * 128, 2.0 * 256 * 128 * 128,
                               2.0 * 256 * 128 * 128, 2.0 * 128 * 192 * 128, 2.0 * 128 * 192 * 128,
                               2.0 * 128 * 192 * 128};

// background work (bit flags) on warps other than the issuing one
enum { BG_COPY = 1, BG_TMEM_LOAD = 2, BG_MUFU = 4 };

__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
               ::"r"(dst), "l"(src), "r"(bytes), "r"(bar)
               : "memory");
}
__device__ __forceinline__ bool wait_bounded(uint32_t bar, uint32_t parity, uint64_t limit_ns) {
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity))
    if (globaltimer_ns() - t0 > limit_ns) return false;
  return true;
}

__global__ void __launch_bounds__(256, 1)
    umma_kernel(int pattern, int iters, int bg, const uint8_t* src, long long src_bytes, long long* cycles,
                int* timeouts) {
  extern __shared__ __align__(1024) uint8_t sm[];
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + AREA);   // [0] end of stream, [1] copies
  uint32_t* tslot = reinterpret_cast<uint32_t*>(sm + AREA + 64);
  volatile int* done = reinterpret_cast<volatile int*>(sm + AREA + 68);
  const uint32_t sb = smem_u32(sm);
  const int warp = threadIdx.x >> 5;
  if (sb & 1023u) {   // the swizzle atoms need a 1 KB aligned window
    if (threadIdx.x == 0) atomicAdd(timeouts, 1000);
    return;
  }
  for (int i = threadIdx.x; i < AREA / 4; i += blockDim.x) {
    const uint32_t h = (static_cast<uint32_t>(i) * 2654435761u) ^ (blockIdx.x * 40503u);
    reinterpret_cast<uint32_t*>(sm)[i] = (0x3C00u | (h & 0x7Fu)) | ((0x3C00u | ((h >> 16) & 0x7Fu)) << 16);
  }
  if (threadIdx.x == 0) {
    mbar_init(smem_u32(bars), 1);
    mbar_init(smem_u32(bars + 1), 1);
    mbar_init(smem_u32(bars + 2), 1);
    *done = 0;
    fence_mbar_init();
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  if (warp == 0) {
    tmem_alloc(smem_u32(tslot), 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tm = *tslot;

  if (threadIdx.x == 0) {
    // layouts (bytes): Q_A [0,32K); Q_B 32K; K 64K; V 96K (32 KB tiles = two [128 rows][128 B]
    // boxes); the 192-key tile uses K 64K and V 112K (48 KB); N=256 B operands live at 128K
    // ([256 rows][128 B] x 2 boxes); the rotating pattern uses stages of K + V at 32K + 64K s.
    const uint32_t sQA = sb, sQB = sb + 32 * KB, sK = sb + 64 * KB, sV = sb + 96 * KB, sB256 = sb + 128 * KB;
    const uint32_t I_S128 = idesc_bf16(128, 128, false, false), I_S192 = idesc_bf16(128, 192, false, false);
    const uint32_t I_PV = idesc_bf16(128, 128, false, true), I_N256 = idesc_bf16(128, 256, false, false);
    const uint32_t I_T256 = idesc_bf16(128, 256, true, false);   // A = V^T (MN-major), B = P^T
    auto qdesc = [](uint32_t q, int k) { return sw128_desc(q + (k >> 2) * 16 * KB + (k & 3) * 32, 16, 1024); };
    auto s_chain = [&](uint32_t d, uint32_t q, uint32_t k, int kbox, uint32_t idesc) {
#pragma unroll
      for (int kk = 0; kk < 8; ++kk)
        umma_ss(d, qdesc(q, kk), sw128_desc(k + (kk >> 2) * kbox + (kk & 3) * 32, 16, 1024), idesc, kk > 0);
    };
    auto pv_chain = [&](uint32_t d, uint32_t a, uint32_t v, int nk, int kbox) {
      for (int kk = 0; kk < nk; ++kk) umma_ts(d, a + 8 * kk, sw128_desc(v + kk * 2048, kbox, 1024), I_PV, 1);
    };
    // P_KERNEL_U2: descriptors of both stages, built once
    uint64_t dq[8], dk[2][8], dv[2][12];
#pragma unroll
    for (int k = 0; k < 8; ++k) dq[k] = sw128_desc(sQA + (k >> 2) * 16 * KB + (k & 3) * 32, 16, 1024);
#pragma unroll
    for (int st = 0; st < 2; ++st) {
#pragma unroll
      for (int k = 0; k < 8; ++k)
        dk[st][k] = sw128_desc(sb + 32 * KB + st * 48 * KB + (k >> 2) * 24 * KB + (k & 3) * 32, 16, 1024);
#pragma unroll
      for (int k = 0; k < 12; ++k) dv[st][k] = sw128_desc(sb + 128 * KB + st * 48 * KB + k * 2048, 24 * KB, 1024);
    }
    const long long t0 = clock64();
    if (pattern == P_KERNEL_U2) {
      for (int it = 0; it < iters; it += 2) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {   // tile j = it + h: V stage h, S buffer h, S_j+2 into buffer h, K stage h
          const int j = it + h;
#pragma unroll
          for (int k = 0; k < 12; ++k)
            umma_ts(tm + 384, tm + h * 192 + 8 * k, dv[h][k], I_PV, (j > 0 || k > 0) ? 1u : 0u);
          tc_commit(smem_u32(bars + 2));
#pragma unroll
          for (int k = 0; k < 8; ++k) umma_ss(tm + h * 192, dq[k], dk[h][k], I_S192, k > 0 ? 1u : 0u);
          tc_commit(smem_u32(bars + 2));
        }
      }
    }
    for (int it = 0; pattern != P_KERNEL_U2 && it < iters; ++it) {
      switch (pattern) {
        case P_PAIRS:
        case P_COMMITS:
        case P_ROTATING:
          for (int g = 0; g < 2; ++g) {
            const int st = pattern == P_ROTATING ? (2 * it + g) % 3 : 0;
            const uint32_t k = pattern == P_ROTATING ? sb + 32 * KB + st * ROT_STAGE : sK;
            const uint32_t v = pattern == P_ROTATING ? sb + 64 * KB + st * ROT_STAGE : sV;
            const uint32_t q = pattern == P_ROTATING ? sQA : (g ? sQB : sQA);
            pv_chain(tm + 256 + 128 * g, tm + 128 * g, v, 8, 16 * KB);
            if (pattern == P_COMMITS) {
              tc_commit(smem_u32(bars + 2));
              tc_commit(smem_u32(bars + 2));
            }
            s_chain(tm + 128 * g, q, k, 16 * KB, I_S128);
            if (pattern == P_COMMITS) {
              tc_commit(smem_u32(bars + 2));
              tc_commit(smem_u32(bars + 2));
            }
          }
          break;
        case P_PAIRS_PLAIN:
          pv_chain(tm + 256, tm, sV, 8, 16 * KB);
          s_chain(tm, sQA, sK, 16 * KB, I_S128);
          pv_chain(tm + 384, tm + 128, sV, 8, 16 * KB);
          s_chain(tm + 128, sQB, sK, 16 * KB, I_S128);
          break;
        case P_PAIRS_DESC: {
          const uint64_t dv = sw128_desc(sV, 16 * KB, 1024), dk = sw128_desc(sK, 16, 1024);
          const uint64_t dqa = sw128_desc(sQA, 16, 1024), dqb = sw128_desc(sQB, 16, 1024);
#pragma unroll
          for (int g = 0; g < 2; ++g) {
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) umma_ts(tm + 256 + 128 * g, tm + 128 * g + 8 * kk, dv + ((kk * 2048) >> 4), I_PV, 1);
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
              const uint32_t o = ((kk >> 2) * 16 * KB + (kk & 3) * 32) >> 4;
              umma_ss(tm + 128 * g, (g ? dqb : dqa) + o, dk + o, I_S128, kk > 0);
            }
          }
          break;
        }
        case P_KERNEL:
        case P_KERNEL_NC: {
          // shared memory: Q [0,32K), K stages of 48 KB at 32K, V stages of 48 KB at 128K
          const int j = it, vs = j & 1, ks = (j + 2) & 1;
          const uint32_t sVs = sb + 128 * KB + vs * 48 * KB, sKs = sb + 32 * KB + ks * 48 * KB;
          const uint32_t a = tm + (j & 1) * 192;
#pragma unroll
          for (int k = 0; k < 12; ++k)
            umma_ts(tm + 384, a + 8 * k, sw128_desc(sVs + k * 2048, 24 * KB, 1024), I_PV, (j > 0 || k > 0) ? 1u : 0u);
          if (pattern == P_KERNEL) tc_commit(smem_u32(bars + 2));
          const uint32_t d = tm + ((j + 2) & 1) * 192;
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const uint32_t kin = (k & 3) * 32;
            umma_ss(d, sw128_desc(sQA + (k >> 2) * 16 * KB + kin, 16, 1024), sw128_desc(sKs + (k >> 2) * 24 * KB + kin, 16, 1024),
                    I_S192, k > 0 ? 1u : 0u);
          }
          if (pattern == P_KERNEL) tc_commit(smem_u32(bars + 2));
          break;
        }
        case P_INTERLEAVED:
          for (int kk = 0; kk < 8; ++kk) {
            umma_ts(tm + 256, tm + 8 * kk, sw128_desc(sV + kk * 2048, 16 * KB, 1024), I_PV, 1);
            umma_ts(tm + 384, tm + 128 + 8 * kk, sw128_desc(sV + kk * 2048, 16 * KB, 1024), I_PV, 1);
          }
          for (int kk = 0; kk < 8; ++kk) {
            const uint64_t bk = sw128_desc(sK + (kk >> 2) * 16 * KB + (kk & 3) * 32, 16, 1024);
            umma_ss(tm, qdesc(sQA, kk), bk, I_S128, kk > 0);
            umma_ss(tm + 128, qdesc(sQB, kk), bk, I_S128, kk > 0);
          }
          break;
        case P_TILE192: {
          const uint32_t s = tm + (it & 1) * 192;
          pv_chain(tm + 384, s, sb + 112 * KB, 12, 24 * KB);
          s_chain(s, sQA, sK, 24 * KB, I_S192);
          break;
        }
        case P_N256_1:
          for (int kk = 0; kk < 8; ++kk)
            umma_ss(tm, qdesc(sQA, kk), sw128_desc(sB256 + (kk >> 2) * 32 * KB + (kk & 3) * 32, 16, 1024), I_N256,
                    kk > 0);
          break;
        case P_N256_2:
          for (int kk = 0; kk < 8; ++kk) {
            const uint64_t bp = sw128_desc(sB256 + (kk >> 2) * 32 * KB + (kk & 3) * 32, 16, 1024);
            umma_ss(tm, qdesc(sQA, kk), bp, I_N256, kk > 0);
            umma_ss(tm + 256, qdesc(sQB, kk), bp, I_N256, kk > 0);
          }
          break;
        case P_PVT:
          for (int kk = 0; kk < 8; ++kk)
            umma_ss(tm + 256, sw128_desc(sV + kk * 2048, 16 * KB, 1024),
                    sw128_desc(sB256 + (kk >> 2) * 32 * KB + (kk & 3) * 32, 16, 1024), I_T256, 1);
          s_chain(tm, sQA, sK, 16 * KB, I_S128);
          s_chain(tm + 128, sQB, sK, 16 * KB, I_S128);
          break;
      }
    }
    tc_commit(smem_u32(bars));
    const bool ok = wait_bounded(smem_u32(bars), 0, 2000000000ull);
    cycles[blockIdx.x] = clock64() - t0;
    if (!ok) {
      atomicAdd(timeouts, 1);
      wait_bounded(smem_u32(bars), 0, 2000000000ull);   // let the stream finish before TMEM goes
    }
    *done = 1;
  }
  if (warp == 1 && (threadIdx.x & 31) == 0 && (bg & BG_COPY)) {
    // bulk copies of fresh data from a global buffer over the K and V tiles (64 KB a round)
    long long off = static_cast<long long>(blockIdx.x) * 65536, n = 0;
    const uint64_t t0 = globaltimer_ns();
    while (!*done && globaltimer_ns() - t0 < 1000000000ull) {
      const uint32_t k = pattern == P_ROTATING ? sb + 32 * KB + (n % 3) * ROT_STAGE : sb + 64 * KB;
      mbar_arrive_expect_tx(smem_u32(bars + 1), 65536);
      bulk_g2s(k, src + off, 32768, smem_u32(bars + 1));
      bulk_g2s(k + 32 * KB, src + off + 32768, 32768, smem_u32(bars + 1));
      if (!wait_bounded(smem_u32(bars + 1), n & 1, 100000000ull)) {
        atomicAdd(timeouts, 1);
        break;
      }
      off += 65536ll * gridDim.x;
      if (off + 65536 > src_bytes) off = static_cast<long long>(blockIdx.x) * 65536;
      ++n;
    }
  }
  if (warp >= 4 && (bg & BG_TMEM_LOAD)) {
    // tcgen05.ld of this warp's lane quarter, 128 columns at a time, as fast as they go
    const uint32_t ta = tm + (static_cast<uint32_t>((warp & 3) * 32) << 16);
    uint32_t acc = 0;
    const uint64_t t0 = globaltimer_ns();
    while (!*done && globaltimer_ns() - t0 < 1000000000ull) {
      uint32_t r[32];
      for (int c = 0; c < 4; ++c) {
        tmem_ld32(ta + 32 * c, r);
        tmem_wait_ld32(r);
        acc ^= r[c];
      }
    }
    if (acc == 0x9e3779b9u) atomicAdd(timeouts, 0);   // keeps the loads
  }
  if (warp >= 2 && warp < 4 && (bg & BG_MUFU)) {
    float x[8];
    for (int k = 0; k < 8; ++k) x[k] = -0.001f * (threadIdx.x + k);
    const uint64_t t0 = globaltimer_ns();
    while (!*done && globaltimer_ns() - t0 < 1000000000ull) {
#pragma unroll
      for (int r = 0; r < 16; ++r)
#pragma unroll
        for (int k = 0; k < 8; ++k) x[k] = ex2_approx(fmaf(x[k], 0.5f, -0.25f));
    }
    float s = 0.f;
    for (int k = 0; k < 8; ++k) s += x[k];
    if (s == 1234.5f) atomicAdd(timeouts, 0);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 0) tmem_dealloc(tm, 512);
}

}  // namespace

int main() {
  int nsm = 0;
  cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, 0);
  const long long src_bytes = 64ll << 20;
  uint8_t* src = nullptr;
  long long* d_cycles = nullptr;
  int* d_timeouts = nullptr;
  cudaMalloc(&src, src_bytes);
  std::vector<uint16_t> h(src_bytes / 2);
  uint32_t x = 12345;
  for (auto& v : h) {
    x = x * 1664525u + 1013904223u;
    v = static_cast<uint16_t>(0x3C00u | ((x >> 9) & 0x7Fu) | ((x >> 16) & 0x8000u));
  }
  cudaMemcpy(src, h.data(), src_bytes, cudaMemcpyHostToDevice);
  cudaMalloc(&d_cycles, nsm * sizeof(long long));
  cudaMalloc(&d_timeouts, sizeof(int));
  cudaMemset(d_timeouts, 0, sizeof(int));
  cudaFuncSetAttribute(umma_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM);
  const int iters = 512;
  const int bgs[4] = {0, BG_COPY, BG_TMEM_LOAD, BG_MUFU};
  const char* bg_name[4] = {"", " + bulk copies", " + TMEM loads", " + MUFU loops"};
  printf("%-44s %-15s %9s %8s\n", "pattern", "background", "clk/UMMA", "MAC/clk");
  for (int p = 0; p < P_COUNT; ++p)
    for (int b = 0; b < 4; ++b) {
      if (b > 0 && p != P_PAIRS && p != P_PAIRS_PLAIN && !(p == P_ROTATING && bgs[b] == BG_COPY)) continue;
      umma_kernel<<<nsm, 256, SMEM>>>(p, 8, bgs[b], src, src_bytes, d_cycles, d_timeouts);   // warm-up
      umma_kernel<<<nsm, 256, SMEM>>>(p, iters, bgs[b], src, src_bytes, d_cycles, d_timeouts);
      const cudaError_t e = cudaDeviceSynchronize();
      if (e != cudaSuccess) {
        printf("CUDA error %s\n", cudaGetErrorString(e));
        return 1;
      }
      std::vector<long long> c(nsm);
      cudaMemcpy(c.data(), d_cycles, nsm * sizeof(long long), cudaMemcpyDeviceToHost);
      double avg = 0;
      for (long long v : c) avg += static_cast<double>(v);
      avg /= nsm;
      const double per_iter = avg / iters;
      printf("%-44s %-15s %9.1f %8.0f\n", kName[p], bg_name[b] + (b ? 3 : 0), per_iter / kUmmas[p],
             kMacs[p] / per_iter);
    }
  int to = 0;
  cudaMemcpy(&to, d_timeouts, sizeof(int), cudaMemcpyDeviceToHost);
  if (to) printf("bounded waits that ran out: %d\n", to);
  return to ? 1 : 0;
}
