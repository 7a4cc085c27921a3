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

// PV8 (with QK8): V as e4m3 codes too, from d-major ("transposed") tiles [128 d rows][keys]: the
// K-major B operand of a kind::f8f6f4 P V with P as e4m3 in TMEM (four keys per column).  A TMA
// box must start on a 16-byte boundary, so every ring segment of this instance starts on a
// 16-key boundary: the host moves its start back by up to 15 keys (`skip`), whose scores are
// masked; a tile's V window is two 128-key boxes with 128-byte swizzle, and P V is 6 UMMAs of
// K = 32.  P is scaled by 2^4 before its e4m3 rounding (the running max is kept within 2^4 of
// every tile's max, so P' <= 2^8 < 448), which keeps values down to 2^-10 of the row maximum
// in e4m3's normal range.
// QK8: Q and K as e4m3 codes (one 128-byte swizzled row = the 128 features of a token), S by
// kind::f8f6f4 UMMAs with K = 32; V, P and O as in the bf16 path.
template <int HD, bool QK8 = false, bool PV8 = false>
struct Cfg {
  static_assert(!QK8 || HD == 128, "8-bit Q K^T is built for head_dim 128");
  static_assert(!PV8 || QK8, "8-bit P V comes with 8-bit Q K^T");
  static constexpr int NBOX = HD / 64;          // 64-column (128-byte) TMA boxes per bf16 tile row
  static constexpr int QBOX = BM * 128;         // [128 rows][64 bf16] = 16 KB
  static constexpr int KBOX = BN * 128;         // [192 rows][64 bf16] = 24 KB
  static constexpr int Q_TILE = QK8 ? BM * HD : NBOX * QBOX;
  static constexpr int K_TILE = QK8 ? BN * HD : NBOX * KBOX;
  static constexpr int V_BOX8 = 128 * HD;                  // [HD rows][128 keys] e4m3 = 16 KB
  static constexpr int V_TILE = PV8 ? 2 * V_BOX8 : NBOX * KBOX;
  static constexpr int PV_STEPS = PV8 ? BN / 32 : BN / 16;   // UMMAs of one P V
  static constexpr float RESCALE = PV8 ? 4.0f : RESCALE_THRESHOLD;   // lazy rescale bound (log2)
  static constexpr float P_SHIFT = PV8 ? 4.0f : 0.0f;      // log2 of the scale P gets before rounding
  static constexpr int KST = (HD == 128 && !QK8) ? 2 : 4;  // K stages
  static constexpr int VST = HD == 128 ? 2 : 4;            // V stages
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K = Q_TILE;
  static constexpr int OFF_V = OFF_K + KST * K_TILE;
  static constexpr int OFF_X = OFF_V + VST * V_TILE;          // exchange arrays (fp32)
  static constexpr int X_FLOATS = 2 * 2 * BM;  // [block][half][BM]: pair exchanges and the epilogue
  static constexpr int OFF_FLAG = OFF_X + X_FLOATS * 4;  // pair status [half][quarter] (int)
  static constexpr int OFF_BAR = OFF_FLAG + 32;
  // q, K stages, V full/empty, S x2, P x2, drain, try_cancel, item mailbox full/empty x2
  static constexpr int N_BAR = 1 + KST + 2 * VST + 4 + 1 + 1 + 4;
  static constexpr int OFF_MISC = (OFF_BAR + N_BAR * 8 + 15) / 16 * 16;   // tmem slot, abort flag, spare
  static constexpr int OFF_CLC = OFF_MISC + 16;          // try_cancel response (16 B)
  static constexpr int OFF_ITEMS = OFF_CLC + 16;         // item mailbox: 2 slots of (q tile, head)
  static constexpr int SMEM = OFF_ITEMS + 16;
  static_assert(OFF_CLC % 16 == 0, "try_cancel response alignment");
  static_assert(SMEM <= 232448, "shared memory per CTA");
  static constexpr uint32_t COL_S0 = 0, COL_O = 2 * BN;
  static constexpr int O_HALF = HD / 2;             // O columns per softmax warp
  static constexpr uint32_t IDESC_QK = QK8 ? idesc_e4m3(BM, BN) : idesc_bf16(BM, BN, false, false);
  static constexpr uint32_t IDESC_PV = PV8 ? idesc_e4m3(BM, HD) : idesc_bf16(BM, HD, false, true);
  static_assert(COL_O + HD <= 512, "TMEM columns");
  static_assert(KBOX % 1024 == 0 && QBOX % 1024 == 0, "swizzle atoms need 1 KB aligned boxes");
};

struct Bars {
  uint32_t q_full, k_full0, v_full0, v_empty0, s_full0, p_full0, drain, clc, item_full0, item_empty0;
};

__device__ __forceinline__ void next_tile(const AttnParams& p, int& seg, int& off) {
  off += BN;
  if (off >= p.seg[seg].count) {
    ++seg;
    off = 0;
  }
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
// ispa_debug_set_trace (first work item of CTA (0, 0)); the production instances contain no
// trace code at all (even an untaken clock64 read constrains instruction scheduling: it cost 6 %
// here).
//
// Work items.  A work item is one (query tile, head); the grid has one CTA per item.  A running
// CTA takes further items from the CTAs of the grid that have not started yet (cluster launch
// control try_cancel: a cancelled CTA never runs and its item is done here), so the CTAs that
// hold the SMs stay resident until no item is left and the SMs that finish first take more
// items.  Item k of a CTA covers its key tiles g = k * n_tiles + j (j = 0 .. n_tiles - 1): stage
// rings, S buffers and barrier phases count g, so the TMA and UMMA pipelines run on across item
// boundaries and the next item's Q, first K/V tiles and first two S tiles overlap this item's
// last tile and epilogue.  At a boundary the UMMA stream is ... S_n-1 PV_n-2 PV_n-1 S'_0 S'_1
// PV'_0 ...: the next item's first S tiles reuse the buffers of P_n-2 and P_n-1 after both PVs,
// and PV'_0 (which overwrites O) follows P'_0, which the softmax warps publish after the
// epilogue's reads of O.
// The TMA thread asks for the next item a few tiles before the end of the current one and
// publishes it (or "none") to the UMMA thread and the softmax warps through a two-slot mailbox.
template <int HD, bool QK8, bool PV8, bool TRACE>
__global__ void __launch_bounds__(NTHREADS, 1)
    attn_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_kr,
                const __grid_constant__ CUtensorMap tm_vr, const __grid_constant__ CUtensorMap tm_kc,
                const __grid_constant__ CUtensorMap tm_vc, const AttnParams p) {
  using C = Cfg<HD, QK8, PV8>;
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
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int* mailbox = reinterpret_cast<volatile int*>(smem + C::OFF_ITEMS);   // [slot][q tile, head]
  const uint32_t clc_resp = sbase + C::OFF_CLC;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

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
    b.clc = b.drain + 8;
    b.item_full0 = b.clc + 8;
    b.item_empty0 = b.item_full0 + 16;
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
      mbar_init(b.item_full0 + 8 * i, 1);
      mbar_init(b.item_empty0 + 8 * i, 1 + N_SOFT_WARPS);   // the UMMA thread + one lane per softmax warp
    }
    mbar_init(b.drain, 1);
    mbar_init(b.clc, 1);
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
  // tile events of the CTA's first item (global tile index = item tile index there)
  auto tr = [&](int g, int ev) {
    if constexpr (TRACE) {
      if (g < n_tiles) trace_event(p.trace, p.trace_tiles, g, ev);
    }
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
      // item (q tile, head) of the K cursor, and the head of the item before it: V trails K by
      // at most one tile, so it is on one of the two
      int kq = static_cast<int>(blockIdx.x), kh = static_cast<int>(blockIdx.y), prev_h = kh;
      bool can_steal = true;     // no try_cancel has failed yet
      int n_req = 0, n_resp = 0;  // try_cancel requests issued / responses consumed
      int nq = 0;                 // Q tiles issued
      auto request = [&]() {
        if (!can_steal) return;
        fence_proxy_async_smem();
        mbar_arrive_expect_tx(b.clc, 16);
        clc_try_cancel(clc_resp, b.clc);
        ++n_req;
      };
      auto load_q = [&]() {   // Q of the K cursor's item
        mbar_arrive_expect_tx(b.q_full, C::Q_TILE);
        tma_load_4d(sQ, &tm_q, b.q_full, 0, kq * BM, 0, kh);
        ++nq;
      };
      // the request for the item after item k goes out this many K tiles before its end
      const int req_at = n_tiles > 4 ? n_tiles - 4 : 0;
      int kk = 0, kj = 0, kseg = 0, koff = 0;   // K cursor: item, tile of the item, segment walk
      int vk = 0, vj = 0, vseg = 0, voff = 0;   // V cursor
      int t = 0, tv = 0;                        // global K and V tiles issued
      bool k_live = true, ok = true;
      load_q();
      if (req_at == 0) request();
      // Loads are issued in the order their stages free up: inside an item the UMMA stream is
      // S_0 S_1 PV_0 S_2 PV_1 S_3 ..., so K_t goes out once S_t-2 has completed and V_t-1 once
      // PV_t-1-VST has; V therefore trails K by one tile.
      auto issue_v = [&]() -> bool {
        const int vs = tv % C::VST;
        if (!mbar_wait(b.v_empty0 + 8 * vs, ((tv / C::VST) & 1) ^ 1, wc, 2, tv)) return false;
        const bool chunk = p.seg[vseg].src != 0;
        mbar_arrive_expect_tx(b.v_full0 + 8 * vs, C::V_TILE);
        const uint32_t sV = sbase + C::OFF_V + vs * C::V_TILE;
        const int vhead = vk == kk ? kh : prev_h;
        if constexpr (PV8) {
          // d-major e4m3 V: the tile's first key is a multiple of 16 (segments start aligned)
          const int x0 = p.seg[vseg].start + voff;
          tma_load_3d(sV, chunk ? &tm_vc : &tm_vr, b.v_full0 + 8 * vs, x0, 0, vhead);
          tma_load_3d(sV + C::V_BOX8, chunk ? &tm_vc : &tm_vr, b.v_full0 + 8 * vs, x0 + 128, 0, vhead);
        } else {
          tma_load_4d(sV, chunk ? &tm_vc : &tm_vr, b.v_full0 + 8 * vs, 0, p.seg[vseg].start + voff, 0, vhead);
        }
        tr(tv, 7);
        ++tv;
        if (++vj == n_tiles) {
          vj = vseg = voff = 0;
          ++vk;
        } else {
          next_tile(p, vseg, voff);
        }
        return true;
      };
      while (ok) {
        if (k_live) {
          if (kj == 0 && kk > 0) {
            // item boundary: the previous item's last V first (its PV comes next in the UMMA
            // stream), then the next item's Q once the previous item's last S has read Q
            if (tv < t && !issue_v()) break;
            if (!mbar_wait(b.s_full0 + 8 * ((t - 1) & 1), ((t - 1) >> 1) & 1, wc, 1, t)) break;
            load_q();
            if (req_at == 0) request();
          }
          if (kj == p.drop_k_tile) break;   // debug: this load never goes out (timeout-path test)
          const int ks = t % C::KST;
          // K_t's stage held K_t-KST; S_t-2 complete means K_t-2 (and every older K) has been
          // read.  S_t cannot complete before K_t lands, so this barrier is never a phase ahead.
          if (t >= 2 && !mbar_wait(b.s_full0 + 8 * ((t - 2) & 1), ((t - 2) >> 1) & 1, wc, 1, t)) break;
          const bool chunk = p.seg[kseg].src != 0;
          mbar_arrive_expect_tx(b.k_full0 + 8 * ks, C::K_TILE);
          tma_load_4d(sbase + C::OFF_K + ks * C::K_TILE, chunk ? &tm_kc : &tm_kr, b.k_full0 + 8 * ks, 0,
                      p.seg[kseg].start + koff, 0, kh);
          tr(t, 6);
          ++t;
          if (++kj == req_at && req_at > 0) request();
          if (kj == n_tiles) {
            // end of item kk: learn item kk + 1 (a cancelled CTA's item, or none) and post it
            int nx = -1, ny = -1;
            if (n_req > n_resp) {
              if (!mbar_wait(b.clc, n_resp & 1, wc, 12, kk)) break;
              ++n_resp;
              int cx, cy;
              if (clc_query(clc_resp, cx, cy)) {
                nx = cx;
                ny = cy;
              } else {
                can_steal = false;
              }
            }
            const int sl = kk & 1;
            if (!mbar_wait(b.item_empty0 + 8 * sl, ((kk >> 1) & 1) ^ 1, wc, 13, kk)) break;
            mailbox[2 * sl] = nx;
            mailbox[2 * sl + 1] = ny;
            mbar_arrive(b.item_full0 + 8 * sl);   // release: orders the mailbox writes before it
            if (ny < 0) {
              k_live = false;
            } else {
              ++kk;
              kj = kseg = koff = 0;
              prev_h = kh;
              kq = nx;
              kh = ny;
            }
          } else {
            next_tile(p, kseg, koff);
          }
        }
        if (tv < t - (k_live ? 1 : 0)) {
          if (!issue_v()) break;
        } else if (!k_live) {
          break;
        }
      }
      // Every load issued must have landed before the CTA may exit.  Older tiles of a stage
      // completed before the stage was refilled, so the last KST (VST) suffice; likewise the
      // last Q tile and an unconsumed try_cancel response.
      if (nq > 0) mbar_wait_drain(b.q_full, (nq - 1) & 1, DRAIN_LIMIT_NS);
      for (int g = t > C::KST ? t - C::KST : 0; g < t; ++g)
        mbar_wait_drain(b.k_full0 + 8 * (g % C::KST), (g / C::KST) & 1, DRAIN_LIMIT_NS);
      for (int g = tv > C::VST ? tv - C::VST : 0; g < tv; ++g)
        mbar_wait_drain(b.v_full0 + 8 * (g % C::VST), (g / C::VST) & 1, DRAIN_LIMIT_NS);
      if (n_req > n_resp) mbar_wait_drain(b.clc, n_resp & 1, DRAIN_LIMIT_NS);
    }
    __syncwarp();
  } else if (warp == WARP_MMA) {
    // ------------------------------------------------------------ UMMA issuer
    if (lane == 0) {
      const uint32_t sQ = sbase + C::OFF_Q;
      bool ok = mbar_wait(b.q_full, 0, wc, 3, 0);
      tr(0, 14);   // Q tile landed
      tc_fence_after();
      auto issue_s = [&](int g) -> bool {
        const int ks = g % C::KST;
        if (!mbar_wait(b.k_full0 + 8 * ks, (g / C::KST) & 1, wc, 4, g)) return false;
        if (g > 0) tr(g, 15);   // K_g landed (seen by the UMMA thread); tile 0's slot 15 is the CTA's
        tc_fence_after();
        const uint32_t sK = sbase + C::OFF_K + ks * C::K_TILE;
        const uint32_t d = tmem + C::COL_S0 + (g & 1) * BN;
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
        tc_commit(b.s_full0 + 8 * (g & 1));   // also tells the TMA thread that K_g has been read
        return true;
      };
      // End of item k: read the next item from the mailbox; if there is one, wait for its Q and
      // issue its first two S tiles (after this item's last PV in the stream).
      auto next_item = [&](int k, int g_next, auto&& s_any) -> bool {
        const int sl = k & 1;
        if (!mbar_wait(b.item_full0 + 8 * sl, (k >> 1) & 1, wc, 14, k)) return false;
        const int head = mailbox[2 * sl + 1];
        mbar_arrive(b.item_empty0 + 8 * sl);
        if (head < 0) return false;
        if (!mbar_wait(b.q_full, (k + 1) & 1, wc, 3, k + 1)) return false;
        tc_fence_after();
        if (!s_any(g_next)) return false;
        return n_tiles < 2 || s_any(g_next + 1);
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
        auto s_tile = [&](int g, int h) -> bool {   // S_g into buffer h = g & 1 from K stage h
          if (!mbar_wait(b.k_full0 + 8 * h, (g >> 1) & 1, wc, 4, g)) return false;
          if (g > 0) tr(g, 15);   // K_g landed (seen by the UMMA thread); tile 0's slot 15 is the CTA's
          tc_fence_after();
          const uint32_t d = tmem + C::COL_S0 + h * BN;
#pragma unroll
          for (int k = 0; k < HD / 16; ++k) umma_ss(d, dq[k], dk[h][k], C::IDESC_QK, k > 0 ? 1u : 0u);
          tc_commit(b.s_full0 + 8 * h);   // also tells the TMA thread that K_g has been read
          return true;
        };
        auto s_any = [&](int g) -> bool { return (g & 1) ? s_tile(g, 1) : s_tile(g, 0); };
        if (ok) ok = s_tile(0, 0);
        if (ok && n_tiles > 1) ok = s_tile(1, 1);
        for (int k = 0; ok; ++k) {
          const int base = k * n_tiles, end = base + n_tiles;
          for (int g0 = base & ~1; ok && g0 < end; g0 += 2) {
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const int g = g0 + h;
              if (g < base) continue;
              if (!ok || g >= end) break;
              if (!mbar_wait(b.p_full0 + 8 * h, (g >> 1) & 1, wc, 5, g)) {
                ok = false;
                break;
              }
              tr(g, 3);
              if (!mbar_wait(b.v_full0 + 8 * h, (g >> 1) & 1, wc, 6, g)) {
                ok = false;
                break;
              }
              tr(g, 11);
              tc_fence_after();
              const uint32_t a = tmem + C::COL_S0 + h * BN;   // P_g, packed bf16, aliases S_g
#pragma unroll
              for (int kk = 0; kk < BN / 16; ++kk)
                umma_ts(tmem + C::COL_O, a + 8 * kk, dv[h][kk], C::IDESC_PV, (g > base || kk > 0) ? 1u : 0u);
              tc_commit(b.v_empty0 + 8 * h);   // V_g read, and O holds the item's tiles up to g
              tr(g, 4);
              if (g + 2 < end) ok = s_tile(g + 2, h);
              tr(g, 5);
            }
          }
          if (ok) ok = next_item(k, end, s_any);
        }
      } else {
        if (ok) ok = issue_s(0);
        if (ok && n_tiles > 1) ok = issue_s(1);
        for (int k = 0; ok; ++k) {
          const int base = k * n_tiles, end = base + n_tiles;
          for (int g = base; ok && g < end; ++g) {
            const int vs = g % C::VST;
            if (!mbar_wait(b.p_full0 + 8 * (g & 1), (g >> 1) & 1, wc, 5, g)) {
              ok = false;
              break;
            }
            tr(g, 3);
            if (!mbar_wait(b.v_full0 + 8 * vs, (g / C::VST) & 1, wc, 6, g)) {
              ok = false;
              break;
            }
            tr(g, 11);
            tc_fence_after();
            const uint32_t sV = sbase + C::OFF_V + vs * C::V_TILE;
            const uint32_t a = tmem + C::COL_S0 + (g & 1) * BN;   // P_g, packed bf16 or e4m3, aliases S_g
            if constexpr (PV8) {
#pragma unroll
              for (int kk = 0; kk < C::PV_STEPS; ++kk)   // K = 32 keys (8 TMEM columns, 32 bytes of a V row)
                umma_f8_ts(tmem + C::COL_O, a + 8 * kk,
                           sw128_desc(sV + (kk >> 2) * C::V_BOX8 + (kk & 3) * 32, 16, 1024), C::IDESC_PV,
                           (g > base || kk > 0) ? 1u : 0u);
            } else {
#pragma unroll
              for (int kk = 0; kk < BN / 16; ++kk) {
                umma_ts(tmem + C::COL_O, a + 8 * kk, sw128_desc(sV + kk * 2048, C::KBOX, 1024), C::IDESC_PV,
                        (g > base || kk > 0) ? 1u : 0u);
              }
            }
            tc_commit(b.v_empty0 + 8 * vs);   // V_g read, and O holds the item's tiles up to g
            tr(g, 4);
            if (g + 2 < end) ok = issue_s(g + 2);
            tr(g, 5);
          }
          if (ok) ok = next_item(k, end, issue_s);
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
    const uint32_t trow = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
    const int D = p.num_heads * HD;
    int q_tile = blockIdx.x, head = blockIdx.y;   // the current item
    int qrow = 0;
    bool row_ok = false;
    float sl2_ring = p.scale_log2, sl2_chunk = p.scale_log2;
    float m_run = -INFINITY, l_run = 0.f;  // l_run: this warp's column half only
    int seg = 0, off = 0;
    bool ok = true;

    auto warp_ok = [&](bool v) { return __all_sync(0xffffffffu, v); };

    const int pair_id = 2 + quarter;   // named barrier of the warp pair (quarter, quarter + 4)
    // The full row's l from the two column halves of the warp pair (block 0 of the exchange
    // area, also used by the pair exchanges, which are complete on both sides of the pair
    // before either warp gets here).  It does not depend on O, so the epilogue takes it before
    // waiting for the last P V.  One pair barrier.
    auto row_l = [&]() {
      x_max[half * BM + row] = l_run;
      pair_sync(pair_id);
      return l_run + x_max[(half ^ 1) * BM + row];
    };
    // Normalise O by the full-row l and store this warp's half of the row (bf16); optional
    // LSE; optional discrepancy partial sum_d (A_full - A_loc)^2 of this head on the stored
    // bf16 values.  Executes the same pair barrier whether or not `live`; after it both warps
    // have read the l slots of row_l (block 0) and may reuse them.  Block 1 holds the squared sums.
    auto emit = [&](bool live, float l_row, __nv_bfloat16* dst, float* lse_dst, bool with_disc) {
      float* x_sq = x_max + 2 * BM;   // [half][row]
      float sq = 0.f;
      if (live) {
        const float inv = (PV8 ? p.v_scale[head] : 1.f) / l_row;
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
      pair_sync(pair_id);
      if (row_ok && half == 0) {
        if (live && lse_dst)
          lse_dst[static_cast<size_t>(head) * p.n_q + qrow] =
              (m_run - C::P_SHIFT + __log2f(l_row)) * 0.69314718055994531f;
        if (with_disc)
          p.disc_part[static_cast<size_t>(head) * p.n_q + qrow] = x_sq[row] + x_sq[BM + row];
      }
    };

    // O holds the item's tiles up to g once PV_g has completed: the commit that frees V_g's stage.
    auto wait_o = [&](int g, int site) {
      return warp_ok(mbar_wait(b.v_empty0 + 8 * (g % C::VST), (g / C::VST) & 1, wc, site, g));
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
    // PV8: P' = exp2(s * sl2 - m + P_SHIFT) as e4m3, four keys per TMEM column, this half's 96
    // keys at key offset r + 96 * half of the tile's V window; returns the row-sum share of P'.
    auto exps_store8 = [&](const uint32_t* s, float sl2, float m, uint32_t pcol) {
      const float mm = m == -INFINITY ? 0.f : m;
      const uint64_t negm = f2_pack(C::P_SHIFT - mm, C::P_SHIFT - mm);
      const uint64_t sl2x2 = f2_pack(sl2, sl2);
      uint64_t acc0 = 0, acc1 = 0;
#pragma unroll
      for (int c = 0; c < HALF_COLS / 16; ++c) {
        uint32_t pk[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          float e[4];
#pragma unroll
          for (int h2 = 0; h2 < 2; ++h2) {
            const int i = 16 * c + 4 * k + 2 * h2;
            const uint64_t x = f2_fma(f2_pack(__uint_as_float(s[i]), __uint_as_float(s[i + 1])), sl2x2, negm);
            e[2 * h2] = ex2_approx(__uint_as_float(static_cast<uint32_t>(x)));
            e[2 * h2 + 1] = ex2_approx(__uint_as_float(static_cast<uint32_t>(x >> 32)));
            if (h2) acc1 = f2_add(acc1, f2_pack(e[2], e[3]));
            else acc0 = f2_add(acc0, f2_pack(e[0], e[1]));
          }
          pk[k] = pack_e4m3x4(e[0], e[1], e[2], e[3]);
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

    // Every warp walks every tile of its items and executes the same barriers whether or not it
    // is ok: the pair barriers of each tile, the snapshot and the epilogue.
    for (int k = 0;; ++k) {
      const int base = k * n_tiles;
      qrow = q_tile * BM + row;
      row_ok = qrow < p.n_q;
      // log2-domain score scale; with 8-bit Q and K it also carries the per-head code scales,
      // which differ between ring keys and chunk keys
      if constexpr (QK8) {
        const int n_qt = (p.n_q + BM - 1) / BM;
        const float qs = p.q_scale[static_cast<int64_t>(head) * n_qt + q_tile];   // [H][query blocks]
        sl2_ring = p.scale_log2 * qs * p.kr_scale[head];
        sl2_chunk = p.scale_log2 * qs * p.kc_scale[head];
      }
      m_run = -INFINITY;
      l_run = 0.f;
      seg = off = 0;
      for (int j = 0; j < n_tiles; ++j) {
        const int g = base + j;
        const int sb = g & 1;
        if (p.dual && j == p.n_local_tiles && j > 0) {
          // A_loc snapshot: O and l hold exactly the local tiles 0..j-1.
          const float l_loc = row_l();
          if (ok) ok = wait_o(g - 1, 7);
          if (ok) tc_fence_after();
          emit(ok, l_loc, p.out_loc, p.lse_loc, false);
        }
        if (ok) ok = warp_ok(mbar_wait(b.s_full0 + 8 * sb, (g >> 1) & 1, wc, 8, g));
        if (threadIdx.x == 0) tr(g, 0);
        if (lane == 0) tr(g, 24 + warp);
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
          if constexpr (PV8) {
            // keys before the run at the start of an aligned segment
            const int vfirst = (off == 0 ? p.seg[seg].skip : 0) - half * HALF_COLS;
            if (vfirst > 0) {
#pragma unroll
              for (int i = 0; i < 16; ++i)
                if (i < vfirst) s[i] = __float_as_uint(-INFINITY);
            }
          }
        };
        // P_j overwrites the first 96 columns of S_j (this half's 48 packed columns), so both
        // halves of the pair must have read their scores first: the pair barrier below orders it.
        const uint32_t pcol = trow + C::COL_S0 + sb * BN + half * P_HALF;
        uint32_t s[HALF_COLS];
        float mx = -INFINITY;
        if (ok) {
          load_s(s);
          if (threadIdx.x == 0) tr(g, 8);
          mx = raw_max(s);
        }
        if (threadIdx.x == 0) tr(g, 9);
        if (j == 0) {
          // first tile: the row max comes from both halves
          float mo;
          ok = pair_exchange(mx, mo);
          m_run = fmaxf(mx, mo) * sl2;
        } else {
          // the running max stands unless the tile's max exceeds it by more than 2^8 somewhere in
          // the pair's rows (rare); then O is rescaled first
          const bool need = ok && mx * sl2 > m_run + C::RESCALE;
          if (pair_or(pair_id, need || !ok)) {
            float mo;
            ok = pair_exchange(mx, mo);
            // O holds PV of tiles 0..j-1 once PV_j-1 has completed; lanes whose max did not grow
            // keep alpha = 1.
            if (ok) ok = wait_o(g - 1, 9);
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
        if (threadIdx.x == 0) tr(g, 1);
        if (ok) {
          if constexpr (PV8) {
            // e4m3 P: this half's 96 keys are 24 columns of S_j's buffer
            l_run += exps_store8(s, sl2, m_run, trow + C::COL_S0 + sb * BN + 24 * half);
          } else {
            l_run += exps_store(s, sl2, m_run, pcol);
          }
          if (threadIdx.x == 0) tr(g, 10);
          tmem_wait_st();
          tc_fence_before();
          mbar_arrive(b.p_full0 + 8 * sb);
          if (threadIdx.x == 0) tr(g, 2);
          if (lane == 0) tr(g, 16 + warp);
        }
        next_tile(p, seg, off);
      }
      {
        const float l_row = row_l();   // overlaps the last P V
        if (ok) ok = wait_o(base + n_tiles - 1, 11);
        if (ok) tc_fence_after();
        if (p.dual && p.n_local_tiles >= n_tiles) emit(ok, l_row, p.out_loc, p.lse_loc, false);
        emit(ok, l_row, p.out, p.lse, p.dual != 0);
        if (threadIdx.x == 0 && k == 0) tr(0, 15);   // epilogue stored
      }
      // The next item's first PV (which overwrites O) waits for P'_0, which every softmax thread
      // publishes only after its epilogue's TMEM loads of O have completed.
      if (!ok) break;
      const int sl = k & 1;
      ok = warp_ok(mbar_wait(b.item_full0 + 8 * sl, (k >> 1) & 1, wc, 15, k));
      if (!ok) break;
      const int nx = mailbox[2 * sl], ny = mailbox[2 * sl + 1];
      __syncwarp();
      if (lane == 0) mbar_arrive(b.item_empty0 + 8 * sl);
      if (ny < 0) break;
      q_tile = nx;
      head = ny;
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

template <int HD, bool QK8, bool TRACE = false, bool PV8 = false>
static cudaError_t launch_hd(const CUtensorMap* tq, const CUtensorMap* tkr, const CUtensorMap* tvr,
                             const CUtensorMap* tkc, const CUtensorMap* tvc, const AttnParams& p,
                             cudaStream_t s) {
  using C = Cfg<HD, QK8, PV8>;
  int dev = 0;
  cudaGetDevice(&dev);
  {
    const cudaError_t e =
        set_smem_limit_once(reinterpret_cast<const void*>(attn_kernel<HD, QK8, PV8, TRACE>), C::SMEM);
    if (e != cudaSuccess) return e;
  }
  dim3 grid((p.n_q + BM - 1) / BM, p.num_heads);
  attn_kernel<HD, QK8, PV8, TRACE><<<grid, NTHREADS, C::SMEM, s>>>(*tq, *tkr, *tvr, *tkc, *tvc, p);
  return cudaGetLastError();
}

cudaError_t launch_attention(int head_dim, const CUtensorMap* tq, const CUtensorMap* tkr,
                             const CUtensorMap* tvr, const CUtensorMap* tkc,
                             const CUtensorMap* tvc, const AttnParams& p, cudaStream_t s) {
  if (p.q_scale) {
    if (head_dim == 128 && p.v_scale) return launch_hd<128, true, false, true>(tq, tkr, tvr, tkc, tvc, p, s);
    if (head_dim == 128) return launch_hd<128, true>(tq, tkr, tvr, tkc, tvc, p, s);
    return cudaErrorInvalidValue;
  }
  if (head_dim == 128 && p.trace) return launch_hd<128, false, true>(tq, tkr, tvr, tkc, tvc, p, s);
  if (head_dim == 128) return launch_hd<128, false>(tq, tkr, tvr, tkc, tvc, p, s);
  if (head_dim == 64) return launch_hd<64, false>(tq, tkr, tvr, tkc, tvc, p, s);
  return cudaErrorInvalidValue;
}

}  // namespace ispa
