// Chunk-step attention against the KV ring on sm_103a (tcgen05 + TMEM + TMA).
//
// One kernel serves the three modes of ISPA's attention:
//   * F-layer (Eq. 3): keys = every resident past frame plus the chunk (dense, or
//     optionally frame-causal: a query sees the chunk's frames up to its own);
//   * L-layer (Sec. 3.3, Eq. 7): keys = sink + recent window + chunk;
//   * dual warmup (Sec. 3.1 phase 1, Sec. 3.4): the local segments are visited
//     first; after the last local tile the running online-softmax state
//     (O, m, l) is snapshotted as A_loc, and the same state keeps absorbing the
//     history tiles to give A_full.  This is the LSE fusion of Eq. 11-12
//     carried out inside one pass: the history branch's (O, LSE) is never
//     materialised, every key is visited once, and the fusion costs one
//     extra read of O from TMEM per row.
//
// Tensor maps: every operand as (64 columns, rows, d/64 column blocks, heads), the
// ring with rows = cap*P slots and the chunk tensors q/k_cur/v_cur with rows = n_q;
// one box (64, tile rows, d/64, 1) with 128-byte swizzle fetches a whole Q, K or V
// tile in one request as d/64 consecutive [rows][128 B] blocks, which is the
// K-major (Q, K) and MN-major (V) UMMA operand layout.
// CTA = one head x one tile of 128 queries, key tiles of 192 keys; 320 threads:
//   warps 0-7  softmax: warp w owns query rows 32(w%4)..+31 (its TMEM lane
//              quarter) and the score columns 96(w/4)..+95 of every key tile,
//              so each row's 192 scores are split over a warp pair (w, w+4) on
//              one SM sub-partition;
//   warp 8     TMA producer (Q once, then K/V tiles into staged rings);
//   warp 9     TMEM allocator and UMMA issuer.
// TMEM columns: S0 [0,192) S1 [192,384) O [384,384+d).
// Shared memory (d = 128): Q 32 KB, two K and two V stages of 48 KB, 2 KB of
// exchange arrays, the pair status words and barriers: 231,568 bytes.
// Per key tile j: S_j = Q K_j^T (SS-UMMA, M=128 N=192, fp32 in TMEM), one commit
// (S_j done, which also tells the TMA thread that K_j has been read) -> the softmax
// warps read S_j, take the tile max of their half-row, and meet their partner at one
// 64-thread reducing barrier (bar.red.or) that orders both halves' score reads
// before either half's P stores and carries the rescale decision (lazy: O is
// rescaled only when the max grows by more than 2^8, rarely) and the pair's abort
// status; they write P_j = exp2(.) as bf16 over the first 96 columns of S_j's own
// buffer -> O += P_j V_j (TS-UMMA: A operand read from TMEM), one commit (V_j's
// stage free, O holds tiles 0..j).  S is double buffered so S_{j+1} runs on the
// tensor cores while the softmax warps work on S_j; S_{j+2} overwrites P_j only
// after PV_j, which the in-order execution of one thread's UMMAs guarantees.
// The tensor pipe runs a continuous UMMA stream at full rate; what a tile costs
// beyond that is per-tile latency (barrier hand-offs, the TMA latency of K, the
// softmax warps' TMEM loads), which long tiles amortise: 192-key tiles measured
// ahead of 176 (F-layer even, L-layer and dual 0.7-0.8 %, 8-bit Q K^T 4 %), and
// every 128-key structure tried measured 15-22 % slower.
//
// Every wait is bounded; after a timeout the softmax warps skip their TMEM work but
// keep walking the tiles through the same barriers, so no warp is left behind.
#include <cuda.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "internal.h"
#include "ptx.cuh"

namespace ispa {

namespace {

constexpr int BM = kAttnBM;    // queries per CTA
constexpr int BN = kAttnBN;    // keys per tile
constexpr int N_SOFT_WARPS = 8;
constexpr int N_SOFT = N_SOFT_WARPS * 32;
constexpr int NTHREADS = N_SOFT + 64;
constexpr int WARP_TMA = 8;
constexpr int WARP_MMA = 9;
constexpr uint32_t TMEM_COLS = 512;
constexpr float RESCALE_THRESHOLD = 8.0f;  // log2 units
constexpr uint64_t DRAIN_LIMIT_NS = 200ull * 1000 * 1000;
constexpr int HALF_COLS = BN / 2;          // score columns per softmax warp
constexpr int P_HALF = HALF_COLS / 2;      // packed bf16 P columns per softmax warp
static_assert(BN % 16 == 0 && BN <= 256 && HALF_COLS % 8 == 0 && P_HALF % 4 == 0, "key tile shape");

// QK8: Q and K as e4m3 codes (one 128-byte swizzled row = the 128 features of a token), S by
// kind::f8f6f4 UMMAs with K = 32; V, P and O as in the bf16 path.
template <int HD, bool QK8 = false>
struct Cfg {
  static_assert(!QK8 || HD == 128, "8-bit Q K^T is built for head_dim 128");
  static constexpr int NBOX = HD / 64;          // 64-column (128-byte) TMA boxes per bf16 tile row
  static constexpr int QBOX = BM * 128;         // [128 rows][64 bf16] = 16 KB
  static constexpr int KBOX = BN * 128;         // [192 rows][64 bf16] = 24 KB
  static constexpr int Q_TILE = QK8 ? BM * HD : NBOX * QBOX;
  static constexpr int K_TILE = QK8 ? BN * HD : NBOX * KBOX;
  static constexpr int V_TILE = NBOX * KBOX;
  static constexpr int KST = (HD == 128 && !QK8) ? 2 : 4;  // K stages
  static constexpr int VST = HD == 128 ? 2 : 4;            // V stages
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K = Q_TILE;
  static constexpr int OFF_V = OFF_K + KST * K_TILE;
  static constexpr int OFF_X = OFF_V + VST * V_TILE;          // exchange arrays (fp32)
  static constexpr int X_FLOATS = 2 * 2 * BM;  // [block][half][BM]: pair exchanges and the epilogue
  static constexpr int OFF_FLAG = OFF_X + X_FLOATS * 4;  // pair status [half][quarter] (int)
  static constexpr int OFF_BAR = OFF_FLAG + 32;
  static constexpr int N_BAR = 1 + KST + 2 * VST + 4 + 1;
  static constexpr int SMEM = OFF_BAR + N_BAR * 8 + 16;  // + tmem slot / abort flag / spare
  static_assert(SMEM <= 232448, "shared memory per CTA");
  static constexpr uint32_t COL_S0 = 0, COL_O = 2 * BN;
  static constexpr int O_HALF = HD / 2;             // O columns per softmax warp
  static constexpr uint32_t IDESC_QK = QK8 ? idesc_e4m3(BM, BN) : idesc_bf16(BM, BN, false, false);
  static constexpr uint32_t IDESC_PV = idesc_bf16(BM, HD, false, true);
  static_assert(COL_O + HD <= 512, "TMEM columns");
  static_assert(KBOX % 1024 == 0 && QBOX % 1024 == 0, "swizzle atoms need 1 KB aligned boxes");
};

struct Bars {
  uint32_t q_full, k_full0, v_full0, v_empty0, s_full0, p_full0, drain;
};

__device__ __forceinline__ void next_tile(const AttnParams& p, int& seg, int& off) {
  off += BN;
  if (off >= p.seg[seg].count) {
    ++seg;
    off = 0;
  }
}

__device__ __forceinline__ void soft_barrier() {
  asm volatile("bar.sync 1, %0;" ::"n"(N_SOFT) : "memory");
}
// Barriers of one softmax warp pair (the two warps of a TMEM lane quarter, 64 threads), ids
// 2..5; pair_or also ORs a predicate over the pair.
__device__ __forceinline__ void pair_sync(int id) {
  asm volatile("bar.sync %0, 64;" ::"r"(id) : "memory");
}
__device__ __forceinline__ bool pair_or(int id, bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.or.pred q, %2, 64, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(v)), "r"(id)
      : "memory");
  return r != 0;
}

// Round 32 consecutive fp32 values (times inv) to bf16 pairs.
__device__ __forceinline__ void pack_row32(const uint32_t* r, float inv, uint32_t* pk) {
#pragma unroll
  for (int k = 0; k < 16; ++k)
    pk[k] = pack_bf16x2(__uint_as_float(r[2 * k]) * inv, __uint_as_float(r[2 * k + 1]) * inv);
}

__device__ __forceinline__ void store_pk16(__nv_bfloat16* dst, const uint32_t* pk) {
  uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll
  for (int q = 0; q < 4; ++q) d4[q] = make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
}

__device__ __forceinline__ uint64_t f2_pack(float a, float b) {
  return static_cast<uint64_t>(__float_as_uint(a)) | (static_cast<uint64_t>(__float_as_uint(b)) << 32);
}

// (x0, x1) * c + (d, d) with one packed fp32x2 FMA
__device__ __forceinline__ uint64_t f2_fma(uint64_t x, uint64_t c, uint64_t d) {
  uint64_t r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(x), "l"(c), "l"(d));
  return r;
}

__device__ __forceinline__ uint64_t f2_add(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}

__device__ __forceinline__ float max3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

}  // namespace

// TRACE: the instance launched while a trace buffer is set records the per-tile events of
// ispa_debug_set_trace; the production instances contain no trace code at all (even an
// untaken clock64 read constrains instruction scheduling: it cost 6 % here).
template <int HD, bool QK8, bool TRACE>
__global__ void __launch_bounds__(NTHREADS, 1)
    attn_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_kr,
                const __grid_constant__ CUtensorMap tm_vr, const __grid_constant__ CUtensorMap tm_kc,
                const __grid_constant__ CUtensorMap tm_vc, const AttnParams p) {
  using C = Cfg<HD, QK8>;
  // The dynamic shared window must start on a 1 KB boundary (the swizzle atoms of the
  // TMA boxes); the declaration asks for it and the check below enforces it.
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = smem_raw;
  const uint32_t sbase = smem_u32(smem);
  if (sbase & 1023u) {  // uniform over the CTA; nothing is initialised yet
    if (threadIdx.x == 0) record_error(p.status, DEVERR_LAYOUT, 0, sbase, 0, 0);
    return;
  }
  uint64_t t_start = 0;
  if constexpr (TRACE) t_start = clock64();
  float* x_max = reinterpret_cast<float*>(smem + C::OFF_X);  // [block][half][row]
  volatile int* x_flag = reinterpret_cast<volatile int*>(smem + C::OFF_FLAG);   // [half][quarter]
  uint64_t* bar_mem = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bar_mem + C::N_BAR);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int q_tile = blockIdx.x;
  const int head = blockIdx.y;
  const int q0 = q_tile * BM;

  Bars b;
  {
    const uint32_t b0 = smem_u32(bar_mem);
    b.q_full = b0;
    b.k_full0 = b0 + 8 * 1;
    b.v_full0 = b.k_full0 + 8 * C::KST;
    b.v_empty0 = b.v_full0 + 8 * C::VST;
    b.s_full0 = b.v_empty0 + 8 * C::VST;
    b.p_full0 = b.s_full0 + 16;
    b.drain = b.p_full0 + 16;
  }

  if (threadIdx.x == 0) {
    mbar_init(b.q_full, 1);
    for (int i = 0; i < C::KST; ++i) {
      mbar_init(b.k_full0 + 8 * i, 1);
    }
    for (int i = 0; i < C::VST; ++i) {
      mbar_init(b.v_full0 + 8 * i, 1);
      mbar_init(b.v_empty0 + 8 * i, 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(b.s_full0 + 8 * i, 1);
      mbar_init(b.p_full0 + 8 * i, N_SOFT);
    }
    mbar_init(b.drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (threadIdx.x == 0) heartbeat(p.heartbeat, 0);
  if (warp == WARP_MMA) {
    tmem_alloc(smem_u32(tmem_slot), TMEM_COLS);
    tmem_relinquish();
    if (lane == 0) heartbeat(p.heartbeat, 1);
  }
  if (warp == WARP_TMA && lane == 0) {
    tma_prefetch_desc(&tm_q);
    tma_prefetch_desc(&tm_kr);
    tma_prefetch_desc(&tm_vr);
    tma_prefetch_desc(&tm_kc);
    tma_prefetch_desc(&tm_vc);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const WaitCtx wc{abort_flag, p.status, p.wait_limit_ns};
  const int n_tiles = p.n_tiles;
  auto tr = [&](int tile, int ev) {
    if constexpr (TRACE) trace_event(p.trace, p.trace_tiles, tile, ev);
  };
  if constexpr (TRACE) {
    // once per CTA, in tile 0's spare slots: 12 kernel entry, 13 TMEM allocated
    if (threadIdx.x == 0 && p.trace && p.trace_tiles > 0 && blockIdx.x == 0 && blockIdx.y == 0) p.trace[12] = t_start;
    if (threadIdx.x == 0) tr(0, 13);
  }

  if (warp == WARP_TMA) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint32_t sQ = sbase + C::OFF_Q;
      mbar_arrive_expect_tx(b.q_full, C::Q_TILE);
      tma_load_4d(sQ, &tm_q, b.q_full, 0, q0, 0, head);
      // Loads are issued in the order their stages free up: the UMMA stream is
      // S_0 S_1 PV_0 S_2 PV_1 S_3 ..., so K_t goes out once S_t-2 has completed and
      // V_{t-1} once PV_{t-1-VST} has; V therefore trails K by one tile.
      int kseg = 0, koff = 0, vseg = 0, voff = 0;
      int nk = 0, nv = 0;  // K and V tiles issued
      for (int t = 0; t <= n_tiles; ++t) {
        if (t == p.drop_k_tile) break;   // debug: this load never goes out (timeout-path test)
        if (t < n_tiles) {
          const bool chunk = p.seg[kseg].src != 0;
          const int row = p.seg[kseg].start + koff;
          const int ks = t % C::KST;
          // K_t's stage held K_t-KST; S_t-2 complete means K_t-2 (and every older K) has been
          // read.  S_t cannot complete before K_t lands, so this barrier is never a phase ahead.
          if (t >= 2 && !mbar_wait(b.s_full0 + 8 * ((t - 2) & 1), ((t - 2) >> 1) & 1, wc, 1, t)) break;
          mbar_arrive_expect_tx(b.k_full0 + 8 * ks, C::K_TILE);
          const uint32_t sK = sbase + C::OFF_K + ks * C::K_TILE;
          tma_load_4d(sK, chunk ? &tm_kc : &tm_kr, b.k_full0 + 8 * ks, 0, row, 0, head);
          nk = t + 1;
          tr(t, 6);
          next_tile(p, kseg, koff);
        }
        if (t >= 1) {
          const int j = t - 1;
          const bool chunk = p.seg[vseg].src != 0;
          const int row = p.seg[vseg].start + voff;
          const int vs = j % C::VST;
          if (!mbar_wait(b.v_empty0 + 8 * vs, ((j / C::VST) & 1) ^ 1, wc, 2, j)) break;
          mbar_arrive_expect_tx(b.v_full0 + 8 * vs, C::V_TILE);
          const uint32_t sV = sbase + C::OFF_V + vs * C::V_TILE;
          tma_load_4d(sV, chunk ? &tm_vc : &tm_vr, b.v_full0 + 8 * vs, 0, row, 0, head);
          nv = j + 1;
          tr(j, 7);
          next_tile(p, vseg, voff);
        }
      }
      // Every load issued must have landed before the CTA may exit.  Older tiles of
      // a stage completed before the stage was refilled, so the last KST (VST) suffice.
      mbar_wait_drain(b.q_full, 0, DRAIN_LIMIT_NS);
      for (int t = nk > C::KST ? nk - C::KST : 0; t < nk; ++t)
        mbar_wait_drain(b.k_full0 + 8 * (t % C::KST), (t / C::KST) & 1, DRAIN_LIMIT_NS);
      for (int t = nv > C::VST ? nv - C::VST : 0; t < nv; ++t)
        mbar_wait_drain(b.v_full0 + 8 * (t % C::VST), (t / C::VST) & 1, DRAIN_LIMIT_NS);
    }
    __syncwarp();
  } else if (warp == WARP_MMA) {
    // ------------------------------------------------------------ UMMA issuer
    if (lane == 0) {
      const uint32_t sQ = sbase + C::OFF_Q;
      bool ok = mbar_wait(b.q_full, 0, wc, 3, 0);
      tr(0, 14);   // Q tile landed
      tc_fence_after();
      auto issue_s = [&](int j) -> bool {
        const int ks = j % C::KST;
        if (!mbar_wait(b.k_full0 + 8 * ks, (j / C::KST) & 1, wc, 4, j)) return false;
        if (j > 0) tr(j, 15);   // K_j landed (seen by the UMMA thread); tile 0's slot 15 is the CTA's
        tc_fence_after();
        const uint32_t sK = sbase + C::OFF_K + ks * C::K_TILE;
        const uint32_t d = tmem + C::COL_S0 + (j & 1) * BN;
        if constexpr (QK8) {
#pragma unroll
          for (int k = 0; k < HD / 32; ++k)   // K = 32 codes per step inside the 128-byte row
            umma_f8(d, sw128_desc(sQ + 32 * k, 16, 1024), sw128_desc(sK + 32 * k, 16, 1024), C::IDESC_QK,
                    k > 0 ? 1u : 0u);
        } else {
#pragma unroll
          for (int k = 0; k < HD / 16; ++k) {
            const uint32_t kin = (k & 3) * 32;
            umma_ss(d, sw128_desc(sQ + (k >> 2) * C::QBOX + kin, 16, 1024),
                    sw128_desc(sK + (k >> 2) * C::KBOX + kin, 16, 1024), C::IDESC_QK, k > 0 ? 1u : 0u);
          }
        }
        tc_commit(b.s_full0 + 8 * (j & 1));   // also tells the TMA thread that K_j has been read
        return true;
      };
      if constexpr (!QK8 && C::KST == 2 && C::VST == 2) {
        // The production shape.  A UMMA stream issues at the full tensor rate only when the
        // issuing thread has nothing but the instructions themselves to execute between them:
        // with the loop unrolled by two, the K/V stage and S buffer of each half are known at
        // compile time and every descriptor is built once, before the loop (measured in
        // isolation: 77 cycles per UMMA of this tile mix, the pipe's own rate, against 94-108
        // with the descriptors rebuilt per tile).
        uint64_t dq[HD / 16], dk[2][HD / 16], dv[2][BN / 16];
#pragma unroll
        for (int k = 0; k < HD / 16; ++k) dq[k] = sw128_desc(sQ + (k >> 2) * C::QBOX + (k & 3) * 32, 16, 1024);
#pragma unroll
        for (int h = 0; h < 2; ++h) {
#pragma unroll
          for (int k = 0; k < HD / 16; ++k)
            dk[h][k] = sw128_desc(sbase + C::OFF_K + h * C::K_TILE + (k >> 2) * C::KBOX + (k & 3) * 32, 16, 1024);
#pragma unroll
          for (int k = 0; k < BN / 16; ++k)
            dv[h][k] = sw128_desc(sbase + C::OFF_V + h * C::V_TILE + k * 2048, C::KBOX, 1024);
        }
        auto s_tile = [&](int j, int h) -> bool {   // S_j into buffer h = j & 1 from K stage h
          if (!mbar_wait(b.k_full0 + 8 * h, (j >> 1) & 1, wc, 4, j)) return false;
          if (j > 0) tr(j, 15);   // K_j landed (seen by the UMMA thread); tile 0's slot 15 is the CTA's
          tc_fence_after();
          const uint32_t d = tmem + C::COL_S0 + h * BN;
#pragma unroll
          for (int k = 0; k < HD / 16; ++k) umma_ss(d, dq[k], dk[h][k], C::IDESC_QK, k > 0 ? 1u : 0u);
          tc_commit(b.s_full0 + 8 * h);   // also tells the TMA thread that K_j has been read
          return true;
        };
        if (ok) ok = s_tile(0, 0);
        if (ok && n_tiles > 1) ok = s_tile(1, 1);
        for (int j0 = 0; ok && j0 < n_tiles; j0 += 2) {
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const int j = j0 + h;
            if (!ok || j >= n_tiles) break;
            if (!mbar_wait(b.p_full0 + 8 * h, (j >> 1) & 1, wc, 5, j)) {
              ok = false;
              break;
            }
            tr(j, 3);
            if (!mbar_wait(b.v_full0 + 8 * h, (j >> 1) & 1, wc, 6, j)) {
              ok = false;
              break;
            }
            tr(j, 11);
            tc_fence_after();
            const uint32_t a = tmem + C::COL_S0 + h * BN;   // P_j, packed bf16, aliases S_j
#pragma unroll
            for (int k = 0; k < BN / 16; ++k)
              umma_ts(tmem + C::COL_O, a + 8 * k, dv[h][k], C::IDESC_PV, (j > 0 || k > 0) ? 1u : 0u);
            tc_commit(b.v_empty0 + 8 * h);   // V_j read, and O holds tiles 0..j
            tr(j, 4);
            if (j + 2 < n_tiles) ok = s_tile(j + 2, h);
            tr(j, 5);
          }
        }
      } else {
        if (ok) ok = issue_s(0);
        if (ok && n_tiles > 1) ok = issue_s(1);
        for (int j = 0; ok && j < n_tiles; ++j) {
          const int vs = j % C::VST;
          if (!mbar_wait(b.p_full0 + 8 * (j & 1), (j >> 1) & 1, wc, 5, j)) break;
          tr(j, 3);
          if (!mbar_wait(b.v_full0 + 8 * vs, (j / C::VST) & 1, wc, 6, j)) break;
          tr(j, 11);
          tc_fence_after();
          const uint32_t sV = sbase + C::OFF_V + vs * C::V_TILE;
          const uint32_t a = tmem + C::COL_S0 + (j & 1) * BN;   // P_j, packed bf16, aliases S_j
#pragma unroll
          for (int k = 0; k < BN / 16; ++k) {
            umma_ts(tmem + C::COL_O, a + 8 * k, sw128_desc(sV + k * 2048, C::KBOX, 1024), C::IDESC_PV,
                    (j > 0 || k > 0) ? 1u : 0u);
          }
          tc_commit(b.v_empty0 + 8 * vs);   // V_j read, and O holds tiles 0..j
          tr(j, 4);
          if (j + 2 < n_tiles) ok = issue_s(j + 2);
          tr(j, 5);
        }
      }
      // All UMMAs must have finished before TMEM is released.
      tc_commit(b.drain);
      mbar_wait_drain(b.drain, 0, DRAIN_LIMIT_NS);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ softmax warps
    const int quarter = warp & 3;          // TMEM lane quarter = row block
    const int half = warp >> 2;            // score / output column half
    const int row = quarter * 32 + lane;
    const int qrow = q0 + row;
    const bool row_ok = qrow < p.n_q;
    const uint32_t trow = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
    const int D = p.num_heads * HD;
    // log2-domain score scale; with 8-bit Q and K it also carries the per-head code scales,
    // which differ between ring keys and chunk keys
    float sl2_ring = p.scale_log2, sl2_chunk = p.scale_log2;
    if constexpr (QK8) {
      const float qs = p.q_scale[static_cast<int64_t>(head) * gridDim.x + q_tile];   // [H][query blocks]
      sl2_ring = p.scale_log2 * qs * p.kr_scale[head];
      sl2_chunk = p.scale_log2 * qs * p.kc_scale[head];
    }
    float m_run = -INFINITY, l_run = 0.f;  // l_run: this warp's column half only
    int seg = 0, off = 0;
    bool ok = true;

    auto warp_ok = [&](bool v) { return __all_sync(0xffffffffu, v); };

    // Normalise O by the full-row l and store this warp's half of the row (bf16); optional
    // LSE; optional discrepancy partial sum_d (A_full - A_loc)^2 of this head on the stored
    // bf16 values.  Executes the same two named barriers whether or not `live`.  Block 0 of
    // the exchange area (also used by the pair exchanges, which are complete on both sides of
    // the pair before either warp gets here) holds l, block 1 the squared sums.
    auto emit = [&](bool live, __nv_bfloat16* dst, float* lse_dst, bool with_disc) {
      float* x_l = x_max;             // [half][row]
      float* x_sq = x_max + 2 * BM;   // [half][row]
      x_l[half * BM + row] = l_run;
      soft_barrier();
      const float l_row = l_run + x_l[(half ^ 1) * BM + row];
      float sq = 0.f;
      if (live) {
        const float inv = 1.f / l_row;
        const int c0 = half * C::O_HALF;
        __nv_bfloat16* drow = dst + static_cast<size_t>(qrow) * D + head * HD + c0;
        const __nv_bfloat16* lrow = p.out_loc + static_cast<size_t>(qrow) * D + head * HD + c0;
#pragma unroll 1
        for (int c = 0; c < C::O_HALF / 32; ++c) {
          uint32_t r[32];
          tmem_ld32(trow + C::COL_O + c0 + 32 * c, r);
          tmem_wait_ld32(r);
          if (row_ok) {
            uint32_t pk[16];
            pack_row32(r, inv, pk);
            store_pk16(drow + 32 * c, pk);
            if (with_disc) {
              const uint4* l4 = reinterpret_cast<const uint4*>(lrow + 32 * c);
#pragma unroll
              for (int q = 0; q < 4; ++q) {
                const uint4 v = l4[q];
                const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                  const uint32_t f = pk[4 * q + e];
                  const float d0 = __uint_as_float(f << 16) - __uint_as_float(w[e] << 16);
                  const float d1 = __uint_as_float(f & 0xFFFF0000u) - __uint_as_float(w[e] & 0xFFFF0000u);
                  sq = fmaf(d0, d0, sq);
                  sq = fmaf(d1, d1, sq);
                }
              }
            }
          }
        }
      }
      // A warp that left through the abort path contributes NaN, so a row whose partial sum
      // is incomplete reaches disc (and the running sum of disc^2) as NaN, never as a value.
      x_sq[half * BM + row] = live ? sq : __int_as_float(0x7fc00000);
      soft_barrier();
      if (row_ok && half == 0) {
        if (live && lse_dst)
          lse_dst[static_cast<size_t>(head) * p.n_q + qrow] = (m_run + __log2f(l_row)) * 0.69314718055994531f;
        if (with_disc)
          p.disc_part[static_cast<size_t>(head) * p.n_q + qrow] = x_sq[row] + x_sq[BM + row];
      }
    };

    const int pair_id = 2 + quarter;   // named barrier of the warp pair (quarter, quarter + 4)
    // O holds tiles 0..j once PV_j has completed: the commit that frees V_j's stage.
    auto wait_o = [&](int j, int site) {
      return warp_ok(mbar_wait(b.v_empty0 + 8 * (j % C::VST), (j / C::VST) & 1, wc, site, j));
    };
    // Exchange a value and the status within the warp pair; returns the partner's value and
    // whether both warps are ok.  Two pair barriers: the slots are free again on return.
    auto pair_exchange = [&](float v, float& other) {
      x_max[half * BM + row] = v;
      if (lane == 0) x_flag[half * 4 + quarter] = ok ? 1 : 0;
      pair_sync(pair_id);
      other = x_max[(half ^ 1) * BM + row];
      const bool both = ok && x_flag[(half ^ 1) * 4 + quarter] != 0;
      pair_sync(pair_id);
      return both;
    };
    // P = exp2(s * sl2 - m) for this thread's HALF_COLS scores, stored packed (bf16 pairs) at
    // pcol as it is computed; returns the row-sum share.
    auto exps_store = [&](const uint32_t* s, float sl2, float m, uint32_t pcol) {
      const float mm = m == -INFINITY ? 0.f : m;   // no visible key yet: every P is 0
      const uint64_t negm = f2_pack(-mm, -mm);
      const uint64_t sl2x2 = f2_pack(sl2, sl2);
      uint64_t acc0 = 0, acc1 = 0;
#pragma unroll
      for (int c = 0; c < P_HALF / 4; ++c) {
        uint32_t pk[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int e = 8 * c + 2 * k;
          const uint64_t x = f2_fma(f2_pack(__uint_as_float(s[e]), __uint_as_float(s[e + 1])), sl2x2, negm);
          const float e0 = ex2_approx(__uint_as_float(static_cast<uint32_t>(x)));
          const float e1 = ex2_approx(__uint_as_float(static_cast<uint32_t>(x >> 32)));
          if (k & 1) acc1 = f2_add(acc1, f2_pack(e0, e1));
          else acc0 = f2_add(acc0, f2_pack(e0, e1));
          pk[k] = pack_bf16x2(e0, e1);
        }
        tmem_st4(pcol + 4 * c, pk);
      }
      const uint64_t acc = f2_add(acc0, acc1);
      return __uint_as_float(static_cast<uint32_t>(acc)) + __uint_as_float(static_cast<uint32_t>(acc >> 32));
    };
    // maximum of this thread's scores: eight independent chains (the max is on the critical path)
    auto raw_max = [&](const uint32_t* s) {
      float m[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) m[k] = -INFINITY;
#pragma unroll
      for (int i = 0; i < HALF_COLS; i += 2) {
        const int k = (i / 2) & 7;
        m[k] = max3(m[k], __uint_as_float(s[i]), __uint_as_float(s[i + 1]));
      }
      return fmaxf(fmaxf(fmaxf(m[0], m[1]), fmaxf(m[2], m[3])), fmaxf(fmaxf(m[4], m[5]), fmaxf(m[6], m[7])));
    };

    // Every warp walks every tile and executes the same barriers whether or not it is ok:
    // the pair barriers of each tile, the snapshot and the epilogue.
    for (int j = 0; j < n_tiles; ++j) {
      const int sb = j & 1;
      if (p.dual && j == p.n_local_tiles && j > 0) {
        // A_loc snapshot: O and l hold exactly the local tiles 0..j-1.
        if (ok) ok = wait_o(j - 1, 7);
        if (ok) tc_fence_after();
        emit(ok, p.out_loc, p.lse_loc, false);
      }
      if (ok) ok = warp_ok(mbar_wait(b.s_full0 + 8 * sb, (j >> 1) & 1, wc, 8, j));
      if (threadIdx.x == 0) tr(j, 0);
      if (lane == 0) tr(j, 24 + warp);
      int vloc = min(BN, p.seg[seg].count - off) - half * HALF_COLS;   // valid columns of this half
      if (p.causal_p != 0 && p.seg[seg].src != 0) {
        // frame-causal chunk: this row sees chunk keys below the end of its own frame
        const int kc0 = p.seg[seg].start + off + half * HALF_COLS;   // chunk index of column 0
        vloc = min(vloc, (qrow / p.causal_p + 1) * p.causal_p - kc0);
      }
      const float sl2 = p.seg[seg].src != 0 ? sl2_chunk : sl2_ring;
      const uint32_t scol = trow + C::COL_S0 + sb * BN + half * HALF_COLS;
      // load this half's scores (masked columns -inf)
      auto load_s = [&](uint32_t* s) {
        tc_fence_after();
#pragma unroll
        for (int i = 0; i < HALF_COLS / 8; ++i) tmem_ld8(scol + 8 * i, s + 8 * i);
#pragma unroll
        for (int i = 0; i < HALF_COLS / 8; ++i) tmem_wait_ld8(s + 8 * i);
        if (vloc < HALF_COLS) {
#pragma unroll
          for (int i = 0; i < HALF_COLS; ++i)
            if (i >= vloc) s[i] = __float_as_uint(-INFINITY);
        }
      };
      // P_j overwrites the first 96 columns of S_j (this half's 48 packed columns), so both
      // halves of the pair must have read their scores first: the pair barrier below orders it.
      const uint32_t pcol = trow + C::COL_S0 + sb * BN + half * P_HALF;
      uint32_t s[HALF_COLS];
      float mx = -INFINITY;
      if (ok) {
        load_s(s);
        if (threadIdx.x == 0) tr(j, 8);
        mx = raw_max(s);
      }
      if (threadIdx.x == 0) tr(j, 9);
      if (j == 0) {
        // first tile: the row max comes from both halves
        float mo;
        ok = pair_exchange(mx, mo);
        m_run = fmaxf(mx, mo) * sl2;
      } else {
        // the running max stands unless the tile's max exceeds it by more than 2^8 somewhere in
        // the pair's rows (rare); then O is rescaled first
        const bool need = ok && mx * sl2 > m_run + RESCALE_THRESHOLD;
        if (pair_or(pair_id, need || !ok)) {
          float mo;
          ok = pair_exchange(mx, mo);
          // O holds PV of tiles 0..j-1 once PV_j-1 has completed; lanes whose max did not grow
          // keep alpha = 1.
          if (ok) ok = wait_o(j - 1, 9);
          if (ok) {
            tc_fence_after();
            const float m_new = fmaxf(m_run, fmaxf(mx, mo) * sl2);
            const float alpha = m_new == m_run ? 1.f : ex2_approx(m_run - m_new);
            l_run *= alpha;
#pragma unroll 1
            for (int c = 0; c < C::O_HALF / 8; ++c) {
              uint32_t r[8];
              const uint32_t ocol = trow + C::COL_O + half * C::O_HALF + 8 * c;
              tmem_ld8(ocol, r);
              tmem_wait_ld8(r);
#pragma unroll
              for (int i = 0; i < 8; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * alpha);
              tmem_st4(ocol, r);
              tmem_st4(ocol + 4, r + 4);
            }
            tmem_wait_st();
            m_run = m_new;
          }
        }
      }
      if (threadIdx.x == 0) tr(j, 1);
      if (ok) {
        l_run += exps_store(s, sl2, m_run, pcol);
        if (threadIdx.x == 0) tr(j, 10);
        tmem_wait_st();
        tc_fence_before();
        mbar_arrive(b.p_full0 + 8 * sb);
        if (threadIdx.x == 0) tr(j, 2);
        if (lane == 0) tr(j, 16 + warp);
      }
      next_tile(p, seg, off);
    }
    {
      if (ok) ok = wait_o(n_tiles - 1, 11);
      if (ok) tc_fence_after();
      if (p.dual && p.n_local_tiles >= n_tiles) emit(ok, p.out_loc, p.lse_loc, false);
      emit(ok, p.out, p.lse, p.dual != 0);
      if (threadIdx.x == 0) tr(0, 15);   // epilogue stored
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == WARP_MMA) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
    if (lane == 0) heartbeat(p.heartbeat, 2);
  }
}

template <int HD, bool QK8, bool TRACE = false>
static cudaError_t launch_hd(const CUtensorMap* tq, const CUtensorMap* tkr, const CUtensorMap* tvr,
                             const CUtensorMap* tkc, const CUtensorMap* tvc, const AttnParams& p,
                             cudaStream_t s) {
  using C = Cfg<HD, QK8>;
  int dev = 0;
  cudaGetDevice(&dev);
  {
    const cudaError_t e = set_smem_limit_once(reinterpret_cast<const void*>(attn_kernel<HD, QK8, TRACE>), C::SMEM);
    if (e != cudaSuccess) return e;
  }
  dim3 grid((p.n_q + BM - 1) / BM, p.num_heads);
  attn_kernel<HD, QK8, TRACE><<<grid, NTHREADS, C::SMEM, s>>>(*tq, *tkr, *tvr, *tkc, *tvc, p);
  return cudaGetLastError();
}

cudaError_t launch_attention(int head_dim, const CUtensorMap* tq, const CUtensorMap* tkr,
                             const CUtensorMap* tvr, const CUtensorMap* tkc,
                             const CUtensorMap* tvc, const AttnParams& p, cudaStream_t s) {
  if (p.q_scale) {
    if (head_dim == 128) return launch_hd<128, true>(tq, tkr, tvr, tkc, tvc, p, s);
    return cudaErrorInvalidValue;
  }
  if (head_dim == 128 && p.trace) return launch_hd<128, false, true>(tq, tkr, tvr, tkc, tvc, p, s);
  if (head_dim == 128) return launch_hd<128, false>(tq, tkr, tvr, tkc, tvc, p, s);
  if (head_dim == 64) return launch_hd<64, false>(tq, tkr, tvr, tkc, tvc, p, s);
  return cudaErrorInvalidValue;
}

// ------------------------------------------------------------ discrepancy reduction
// disc[t] = sqrt(sum_h part[h][t]);  *disc_sq_sum += sum over the block's tokens.
__global__ void __launch_bounds__(256) disc_reduce_kernel(const float* __restrict__ part, int H,
                                                          int n_q, float* __restrict__ disc,
                                                          float* __restrict__ disc_sq_sum) {
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
  disc_reduce_kernel<<<(n_q + 255) / 256, 256, 0, s>>>(part, H, n_q, disc, disc_sq_sum);
  return cudaGetLastError();
}

}  // namespace ispa
