/*
 * libispa -- the data-parallel hot path of ISPA (Instance-Specific Parametric
 * Absorption, arxiv 2607.00712) on one GB300 (sm_103a).
 *
 * The library computes, for one transformer layer of an autoregressive video
 * DiT and one chunk step:
 *   - F-layer attention over the whole KV cache (Sec. 2, Eq. 3);
 *   - L-layer attention over a sink + recent-frame window (Sec. 3.3, Eq. 7);
 *   - the dual warmup pass returning both outputs from one sweep over the key
 *     tiles, with their per-token discrepancy (Sec. 3.1, Sec. 3.4, Eq. 9-12);
 *   - the running sums of the least-squares absorption (Sec. 3.2, Eq. 5) and
 *     the closed-form solve with its feasibility score (Eq. 5-6);
 *   - appending a finished chunk's K/V into a ring-buffer cache.
 *
 * Conventions (all entry points)
 *   - Every tensor argument is a DEVICE pointer owned by the caller, unless
 *     the argument says "host".  The library allocates no device memory;
 *     calls that need scratch take a caller workspace and have a size query.
 *   - bf16 = IEEE bfloat16 stored as 16-bit words.  Layouts are row-major,
 *     dense, innermost index last.  Device pointers must be 16-byte aligned.
 *   - Work is enqueued asynchronously on `stream` (a cudaStream_t; NULL is the
 *     legacy default stream) except where a function says it synchronises.
 *   - Errors are returned as ispa_status; no exception crosses the ABI.  On a
 *     non-OK return of argument validation nothing has been enqueued.
 *   - Kernels never spin without bound: a wait that runs out records a device
 *     error, which ispa_last_device_error() reports as ISPA_ERR_TIMEOUT.
 *   - The attention kernels launch one CTA per (query tile, head); the CTAs
 *     that start first take the items of CTAs that have not started yet
 *     (cluster launch control), so each SM works through a run of items.
 *   - Head dims supported: 64 and 128.  Tokens per frame P >= 1.
 *   - Counts (queries n_q, tokens T, frames n_frames, rows) must be at least
 *     1: an empty call is an argument error (ISPA_ERR_INVALID_ARG) and
 *     enqueues nothing, so callers skip empty work themselves.
 *   - CUDA graphs: after one eager call on a device, the attention, append, LS
 *     accumulate / reset, quantisation and W8A8 entry points enqueue only
 *     kernel launches and memsets on `stream` and can be captured.  A replay reuses what the call
 *     saw at capture time: pointers, and the ring's frames_written and hence its
 *     key sets (an append advances frames_written on the host when it is
 *     captured, not when it is replayed).  ispa_ls_solve and the functions that
 *     read the device error record synchronise and cannot be captured.
 *   - Threads: entry points may be called from several host threads for
 *     different rings, states and streams.  ispa_set_wait_limit_ns and the
 *     ispa_debug_* setters change process-wide settings without locking; set
 *     them before work is issued from other threads.  The device error record
 *     is one per device and shared by every call on it.
 */
#ifndef ISPA_H_
#define ISPA_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define ISPA_API __attribute__((visibility("default")))
#else
#define ISPA_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* ispa_stream; /* == cudaStream_t */

typedef enum {
  ISPA_OK = 0,
  ISPA_ERR_INVALID_ARG = 1, /* null/misaligned pointer, bad size or layout */
  ISPA_ERR_UNSUPPORTED = 2, /* head_dim or hidden size the kernels do not handle */
  ISPA_ERR_CAPACITY = 3,    /* window or append does not fit the ring */
  ISPA_ERR_NOT_SPD = 4,     /* Gram matrix + lambda I not positive definite */
  ISPA_ERR_TIMEOUT = 5,     /* a device-side bounded wait ran out */
  ISPA_ERR_CUDA = 6,        /* a CUDA runtime/driver call failed */
  ISPA_ERR_WORKSPACE = 7    /* workspace missing or smaller than the size query */
} ispa_status;

/*
 * Per-layer KV cache as a frame-granular ring (Sec. 2: the cache keeps only
 * the latest frames' keys and values; Sec. 3.4: the sink frame K_1 is kept).
 *   k, v : bf16 [num_heads][capacity_frames * tokens_per_frame][head_dim],
 *          caller-owned device memory of ispa_ring_bytes()/2 bytes each.
 *   Logical frame f (0, 1, 2, ... in generation order) lives in slot
 *     f                                              if f <  n_sink_frames,
 *     n_sink_frames + (f - n_sink_frames) mod (capacity_frames - n_sink_frames)
 *                                                    otherwise,
 *   so the first n_sink_frames frames are pinned and every later frame
 *   overwrites the oldest non-sink frame.  frames_written counts the frames
 *   appended so far; it is advanced on the host by ispa_kv_append when the
 *   copy is enqueued.  The struct is plain data: copying it (and the two
 *   buffers) checkpoints the cache.  With k_format = ISPA_KV_K_E4M3, k holds
 *   e4m3 codes [H][capacity_frames * P][head_dim] (one byte each; head_dim 128)
 *   written by ispa_kv_append_qk8 with one fp32 scale per head that the caller
 *   keeps for the ring's life.  With k_format = ISPA_KV_KV_E4M3 (head_dim 128,
 *   P % 4 == 0), k holds those key codes and v holds the values as e4m3 codes
 *   d-major, [H][head_dim][ispa_ring_vt_stride(ring)] (key index slot * P + t
 *   within a row), written by ispa_kv_append_kv8 with the caller's per-head key
 *   and value scales.  Slots never written must still hold
 *   finite values (zero-fill the buffers at creation): a key tile that ends
 *   inside a run reads the rows after it with weight zero, and 0 * NaN is NaN.
 */
#define ISPA_KV_BF16 0     /* k_format: keys bf16 (every entry point except *_qk8) */
#define ISPA_KV_K_E4M3 1   /* k_format: keys e4m3 codes, 1 byte each (the *_qk8 entry points) */
#define ISPA_KV_KV_E4M3 2  /* k_format: keys and d-major values as e4m3 codes (the *_kv8 entry points) */

typedef struct {
  int32_t num_heads;
  int32_t head_dim;
  int32_t tokens_per_frame;
  int32_t capacity_frames;
  int32_t n_sink_frames;
  int32_t k_format;       /* ISPA_KV_BF16, ISPA_KV_K_E4M3 (values bf16) or ISPA_KV_KV_E4M3 */
  int64_t frames_written;
  void* k;
  void* v;
} ispa_kv_ring;

/*
 * Local window of an L-layer (Eq. 7, read as a parameterised window): the
 * n_sink_frames oldest past frames plus the n_recent_frames newest past
 * frames; the chunk itself is always local.  The paper-literal set is
 * {n_sink_frames = 1, n_recent_frames = 0}.
 */
typedef struct {
  int32_t n_sink_frames;
  int32_t n_recent_frames;
} ispa_window;

typedef struct {
  int32_t first_slot;
  int32_t n_slots;
} ispa_slot_range;

#define ISPA_MAX_RANGES 4

/* Slot runs of the full, local and history key sets of a ring (Eq. 7-8). */
typedef struct {
  int32_t n_full, n_local, n_hist, reserved;
  ispa_slot_range full[ISPA_MAX_RANGES];
  ispa_slot_range local[ISPA_MAX_RANGES];
  ispa_slot_range hist[ISPA_MAX_RANGES];
} ispa_key_sets;

/*
 * Least-squares accumulators (Sec. 3.2: "summing the outer products of
 * activations").  gram: caller-owned fp32 [2*dim][2*dim], row-major, holding
 * the blocks of [A_loc | Delta]^T [A_loc | Delta] with Delta = A_full - A_loc:
 *   G = A_loc^T A_loc   rows [0,dim)     cols [0,dim)
 *   X = A_loc^T Delta   rows [0,dim)     cols [dim,2dim)
 *   S = Delta^T Delta   rows [dim,2dim)  cols [dim,2dim)
 * All of X is maintained, and of G and S every 128x128 tile on or above the
 * diagonal (tile (i, j), j >= i, diagonal tiles in full); with dim a multiple
 * of 256 the tiles (2k+1, 2k) just below the diagonal hold their sums too.
 * No other part of the buffer is written.  The paper's
 * A_loc^T R equals X W and is formed by the solve.  n_tokens counts the rows
 * accumulated (host side).  Plain data: copying it checkpoints the warmup.
 */
typedef struct {
  int32_t dim;
  int32_t reserved;
  int64_t n_tokens;
  float* gram;
} ispa_ls_state;

/* ------------------------------------------------------------ misc / host */

/* Static English name of a status code. */
ISPA_API const char* ispa_status_string(ispa_status s);

/* Device error recorded by a kernel on the current device since the last
 * call (then cleared): ISPA_OK, ISPA_ERR_TIMEOUT (raw code 1), or ISPA_ERR_CUDA
 * (raw code 3: a CTA of a tcgen05 kernel -- attention, Gram, W8A8 -- found its
 * shared-memory window off a 1 KB boundary and wrote nothing).  Synchronises the device with a blocking copy
 * of one word.  *code (nullable, host) gets the raw code. */
ISPA_API ispa_status ispa_last_device_error(int32_t* code);

/* Bound of every device-side wait, in nanoseconds (default 1e9).  Applies to
 * launches enqueued after the call.  Returns the previous value.  Meant for
 * tests of the timeout path; 0 restores the default. */
ISPA_API uint64_t ispa_set_wait_limit_ns(uint64_t ns);

/* Enqueue one CTA that waits on an mbarrier nobody arrives at, with the given
 * bound; it records ISPA_ERR_TIMEOUT and exits.  Exercises the bounded-wait
 * and status path without touching any other state. */
ISPA_API ispa_status ispa_debug_wait_probe(uint64_t limit_ns, ispa_stream stream);

/* Copy (without clearing) the device error record of the current device:
 * rec8[0] = code (0 none, 1 timeout, 3 layout), then the first failing wait: [1] wait
 * site, [2] blockIdx.x, [3] blockIdx.y, [4] threadIdx.x, [5] barrier shared
 * address, [6] parity, [7] tile index.  rec8: host array of 8 int32.
 * Synchronises like ispa_last_device_error. */
ISPA_API ispa_status ispa_debug_error_record(int32_t* rec8);

/* Debug aid: counters (a device-accessible pointer to host-mapped memory,
 * n_slots * 4 uint32) that the tcgen05 kernels bump per CTA: [0] started,
 * [1] TMEM allocated, [2] finished.  Each launch takes the next slot in turn.
 * NULL / 0 turns it off (the default). */
ISPA_API ispa_status ispa_debug_set_heartbeat(uint32_t* counters, int32_t n_slots);

/* Debug aid: per-key-tile cycle trace of CTA (0, 0) of the bf16, head_dim 128
 * attention kernel (a separate instance of it, launched while a buffer is set;
 * it computes the same results).
 * buf: device-accessible uint64 [n_tiles][32], clock64 values, zero where an
 * event is not recorded.  The counters of an SM's four sub-partitions are not
 * aligned with one another: compare stamps of warps on different sub-partitions
 * (warp index mod 4) only through intervals each warp measures on its own.
 * Events of key tile j:
 *   0, 8, 9, 1, 10, 2  softmax warp 0: S_j seen, S_j loaded from TMEM, tile max
 *                      of its half-row done, rescale decided (warp-pair barrier),
 *                      exp loop done, P_j arrived;
 *   3, 11, 4, 5        UMMA thread: P_j seen, V_j seen, PV_j issued, S_{j+2} issued;
 *   15 (j >= 1)        UMMA thread: K_j landed;
 *   6, 7               TMA thread: K_j issued, V_j issued;
 *   16 + w, 24 + w     softmax warp w (0-7): P_j arrived, S_j seen;
 *   12-15 of tile 0    once per CTA: kernel entry, TMEM allocated, Q tile landed,
 *                      epilogue stored.
 * NULL / 0 turns it off (the default). */
ISPA_API ispa_status ispa_debug_set_trace(uint64_t* buf, int32_t n_tiles);

/* Debug aid for the timeout path: while tile >= 0, the TMA thread of every attention CTA
 * stops before loading key tile `tile` (it issues nothing more and drains what it issued),
 * so the UMMA thread's wait for that tile runs out after the wait limit and the CTA leaves
 * through its abort path, recording ISPA_ERR_TIMEOUT.  CTAs with fewer tiles run normally.
 * Nothing faults: the missing load simply never arrives.  -1 turns it off (the default). */
ISPA_API ispa_status ispa_debug_drop_k_tile(int32_t tile);

/* Debug aid for ispa_attn_dual_static: the device address of its scratch array in the
 * calling thread's current CUDA context (looked up and cached exactly as that entry point
 * does), the context's process-unique id, and how many address lookups the library has
 * made so far.  Launches nothing and allocates nothing.  The paper has no counterpart. */
ISPA_API ispa_status ispa_debug_static_scratch(void** addr, uint64_t* context_id, uint32_t* lookups);

/* Bytes of one ring's K and V buffers together: H * cap * P * d * (2 + 2), or
 * * (1 + 2) with e4m3 keys. */
ISPA_API size_t ispa_ring_bytes(const ispa_kv_ring* ring);

/* Host-only: ring slot of logical frame `frame` (see ispa_kv_ring), or -1 if
 * the frame is not resident. */
ISPA_API int32_t ispa_ring_slot(const ispa_kv_ring* ring, int64_t frame);

/*
 * Host-only (Eq. 7-8): resolve the key sets of the ring's current state.
 * With F = frames_written, local past frames are {f < win.n_sink_frames}
 * united with {F - win.n_recent_frames <= f < F}; full = every resident
 * frame; hist = full minus local.  Each set is returned as increasing runs of
 * ring slots.  Errors: ISPA_ERR_CAPACITY if a local frame has been evicted,
 * ISPA_ERR_INVALID_ARG on a bad ring or window.
 */
ISPA_API ispa_status ispa_window_resolve(const ispa_kv_ring* ring, ispa_window win, ispa_key_sets* out);

/* ------------------------------------------------------------ KV append */

/*
 * Write a finished chunk's keys and values into the ring (Eq. 3's K_past
 * grows by the chunk) and advance ring->frames_written by n_frames.
 *   k_new, v_new : bf16 [n_frames * P][num_heads][head_dim] (token-major, as
 *                  produced by the QKV projection).
 * Frame frames_written + i goes to its ring slot, evicting the oldest non-sink
 * frame.  Errors: ISPA_ERR_CAPACITY if n_frames > capacity - n_sink (a frame
 * of this append would overwrite another one of it) or n_frames > 16.
 */
ISPA_API ispa_status ispa_kv_append(ispa_kv_ring* ring, const void* k_new, const void* v_new,
                           int32_t n_frames, ispa_stream stream);

/* Same for n_layers rings in ONE launch.  The rings share num_heads,
 * head_dim and tokens_per_frame; capacity, sinks and frames_written may differ.
 * rings: host array of n_layers ring structs (each advanced); k_new/v_new:
 * host arrays of n_layers device pointers.  n_layers <= 64. */
ISPA_API ispa_status ispa_kv_append_layers(ispa_kv_ring* rings, int32_t n_layers,
                                  const void* const* k_new, const void* const* v_new,
                                  int32_t n_frames, ispa_stream stream);

/* ------------------------------------------------------------ attention */

/* Option bits of the *_ex attention entry points. */
#define ISPA_ATTN_FRAME_CAUSAL 1u
/*   ISPA_ATTN_FRAME_CAUSAL: block-causal at frame granularity inside the chunk.
 *   Eq. 3 leaves the chunk dense (every chunk query sees every chunk key); with
 *   this bit a query of the chunk's frame a (rows a*P .. a*P+P-1) sees the
 *   chunk's frames 0..a only.  Past frames stay fully visible.  n_q must be a
 *   multiple of tokens_per_frame (else ISPA_ERR_INVALID_ARG).  Unknown bits are
 *   ISPA_ERR_INVALID_ARG.  flags = 0 is the plain entry point. */

/*
 * F-layer chunk attention (Eq. 3): Q = Q_cur, K = [K_past; K_cur],
 * V = [V_past; V_cur], with K_past/V_past every resident frame of the ring.
 * The chunk is dense inside itself (no intra-chunk mask).
 *   q, k_cur, v_cur : bf16 [n_q][num_heads][head_dim]
 *   out             : bf16 [n_q][num_heads * head_dim]  (heads concatenated)
 *   lse             : fp32 [num_heads][n_q], natural-log LSE, or NULL
 *   scale           : softmax scale; 0 means 1/sqrt(head_dim)
 * Computation: bf16 inputs, fp32 accumulation, bf16 output (round to nearest).
 */
ISPA_API ispa_status ispa_attn_full(const ispa_kv_ring* ring, const void* q, const void* k_cur,
                           const void* v_cur, int32_t n_q, float scale, void* out, float* lse,
                           ispa_stream stream);
/* ispa_attn_full with option bits (ISPA_ATTN_FRAME_CAUSAL). */
ISPA_API ispa_status ispa_attn_full_ex(const ispa_kv_ring* ring, const void* q, const void* k_cur,
                              const void* v_cur, int32_t n_q, float scale, uint32_t flags, void* out,
                              float* lse, ispa_stream stream);

/*
 * L-layer chunk attention (Sec. 3.3, Eq. 7): the same over the local set
 * only -- the window's sink and recent frames plus the chunk.  Arguments as
 * for ispa_attn_full.  Errors: ISPA_ERR_CAPACITY if a window frame has been
 * evicted from the ring.
 */
ISPA_API ispa_status ispa_attn_local(const ispa_kv_ring* ring, ispa_window win, const void* q,
                            const void* k_cur, const void* v_cur, int32_t n_q, float scale,
                            void* out, float* lse, ispa_stream stream);
/* ispa_attn_local with option bits (ISPA_ATTN_FRAME_CAUSAL). */
ISPA_API ispa_status ispa_attn_local_ex(const ispa_kv_ring* ring, ispa_window win, const void* q,
                               const void* k_cur, const void* v_cur, int32_t n_q, float scale,
                               uint32_t flags, void* out, float* lse, ispa_stream stream);

/* Workspace bytes of ispa_attn_dual (fp32 [num_heads][n_q] partial sums). */
ISPA_API size_t ispa_attn_dual_workspace_size(int32_t num_heads, int32_t n_q);

/*
 * Warmup dual pass (Sec. 3.1 phase 1, Sec. 3.4): A_loc (local set) and A_full
 * (full set) of the same queries from one sweep over the key tiles -- the
 * local tiles first, then the history tiles, fusing the two online-softmax
 * states as Eq. 11-12 do.
 *   a_full, a_loc  : bf16 [n_q][num_heads * head_dim]
 *   disc           : fp32 [n_q], disc_t = || A_full,t - A_loc,t ||_2 over all
 *                    num_heads*head_dim features, taken on the stored bf16
 *                    outputs (Sec. 3.1 leaves the discrepancy undefined; read as this norm)
 *   disc_sq_sum    : fp32 device scalar, += sum_t disc_t^2 (not reset)
 *   lse_full, lse_loc : fp32 [num_heads][n_q] or NULL
 *   workspace      : >= ispa_attn_dual_workspace_size bytes
 * An empty history set gives a_full == a_loc bit for bit and disc == 0.
 * If a device wait runs out (ISPA_ERR_TIMEOUT), the outputs of the call are
 * undefined and disc_sq_sum becomes NaN: an aborted row contributes a NaN
 * partial, so a running sum never silently absorbs a partial or stale value.
 */
ISPA_API ispa_status ispa_attn_dual(const ispa_kv_ring* ring, ispa_window win, const void* q,
                           const void* k_cur, const void* v_cur, int32_t n_q, float scale,
                           void* a_full, void* a_loc, float* disc, float* disc_sq_sum,
                           float* lse_full, float* lse_loc, void* workspace, size_t ws_bytes,
                           ispa_stream stream);
/* ispa_attn_dual with option bits (ISPA_ATTN_FRAME_CAUSAL: the chunk part of both
 * A_loc and A_full is frame-causal). */
ISPA_API ispa_status ispa_attn_dual_ex(const ispa_kv_ring* ring, ispa_window win, const void* q,
                              const void* k_cur, const void* v_cur, int32_t n_q, float scale,
                              uint32_t flags, void* a_full, void* a_loc, float* disc,
                              float* disc_sq_sum, float* lse_full, float* lse_loc, void* workspace,
                              size_t ws_bytes, ispa_stream stream);

/* Largest num_heads * n_q that ispa_attn_dual_static accepts (4 MiB of fp32). */
#define ISPA_DUAL_STATIC_MAX_PARTIALS (1u << 20)

/*
 * ispa_attn_dual without a workspace argument, for callers that cannot
 * allocate device memory when they run the warmup pass -- e.g. a real-time
 * streaming loop whose memory is planned once at start-up (cudaMalloc would
 * synchronise the device mid-stream), or a plug-in whose host runtime gives it
 * tensors but no allocator.  The paper has no counterpart; this is a library
 * convenience.  Arguments and results are those of ispa_attn_dual.
 *   - Scratch comes from a fixed array inside the library, present on every
 *     GPU that loads it until the process exits; num_heads * n_q must not
 *     exceed ISPA_DUAL_STATIC_MAX_PARTIALS, else ISPA_ERR_WORKSPACE is returned
 *     and nothing is enqueued.
 *   - The array's device address belongs to one CUDA context.  The first call
 *     made with a context current (normally the device's primary context)
 *     looks it up and caches it under that context's process-unique id, so a
 *     caller's own context, or the primary context re-created after a
 *     cudaDeviceReset, gets its own lookup.  Make that first call before any
 *     stream capture.
 *   - Allocates nothing: no cudaMalloc / cudaFree, no allocating library call.
 *   - All calls share the one array, so calls that overlap on the GPU (e.g.
 *     on two streams) race; serialise them.  Each call overwrites every entry
 *     it reads, so nothing needs clearing between calls.
 */
ISPA_API ispa_status ispa_attn_dual_static(const ispa_kv_ring* ring, ispa_window win, const void* q,
                                           const void* k_cur, const void* v_cur, int32_t n_q, float scale,
                                           void* a_full, void* a_loc, float* disc, float* disc_sq_sum,
                                           float* lse_full, float* lse_loc, ispa_stream stream);

/*
 * History branch of the decomposed dual pass (Eq. 10): attention of the chunk's
 * queries over the history set only -- the resident past frames outside the
 * window, without the chunk.  Together with ispa_attn_local (Eq. 9) and
 * ispa_lse_merge (Eq. 11-12) it is the paper's two-call form of the dual pass;
 * ispa_attn_dual computes the same in one sweep.  Arguments as for
 * ispa_attn_local; lse must not be NULL here.  An empty history set gives
 * out = 0 and lse = -inf (a branch that contributes nothing to the merge).
 */
ISPA_API ispa_status ispa_attn_hist(const ispa_kv_ring* ring, ispa_window win, const void* q, int32_t n_q,
                                    float scale, void* out, float* lse, ispa_stream stream);

/*
 * Eq. 11-12: merge two attention branches over disjoint key sets.
 *   o_a, o_b   : bf16 [n_q][num_heads * head_dim]; lse_a, lse_b : fp32 [num_heads][n_q]
 *   out        : bf16 [n_q][num_heads * head_dim]; lse_out : fp32 [num_heads][n_q] or NULL
 * LSE = log(exp(lse_a) + exp(lse_b)); out = exp(lse_a - LSE) o_a + exp(lse_b - LSE) o_b,
 * in fp32, rounded to bf16.  A branch with lse = -inf has weight 0.  out may alias o_a or o_b.
 */
ISPA_API ispa_status ispa_lse_merge(const void* o_a, const float* lse_a, const void* o_b, const float* lse_b,
                                    int32_t n_q, int32_t num_heads, int32_t head_dim, void* out, float* lse_out,
                                    ispa_stream stream);

/*
 * Output discrepancy of the warmup pass (Sec. 3.1 phase 1, which monitors the
 * discrepancy between the global and the local output; the paper gives no formula,
 * the reading is disc_t = ||A_full,t - A_loc,t||_2 over all D features) from two
 * stored outputs -- the discrepancy of the decomposed dual pass (ispa_attn_local +
 * ispa_attn_hist + ispa_lse_merge); ispa_attn_dual takes it inside its own sweep.
 *   a_full, a_loc : bf16 [n_q][dim], 16-byte aligned, dim a multiple of 8
 *                   (else ISPA_ERR_UNSUPPORTED)
 *   disc          : fp32 [n_q] (overwritten)
 *   disc_sq_sum   : fp32 device scalar, += sum_t disc_t^2 (not reset)
 * Differences and sums in fp32.  Asynchronous on `stream`.
 */
ISPA_API ispa_status ispa_discrepancy(const void* a_full, const void* a_loc, int32_t n_q, int32_t dim, float* disc,
                                      float* disc_sq_sum, ispa_stream stream);

/* ------------------------------------------------------------ transition */

/*
 * Host-only dynamic layer selection (Sec. 3.3): rank the n_layers layers by
 * ascending feasibility score eps (host array) and mark the k lowest as
 * L-layers (is_l_layer[i] = 1, else 0; host array of n_layers).  Ties go to
 * the lower layer index; NaN scores rank last.  0 <= k <= n_layers.
 */
ISPA_API ispa_status ispa_select_layers(const double* eps, int32_t n_layers, int32_t k, int32_t* is_l_layer);

/*
 * Weight injection W_new = W + dW (Sec. 3.1 phase 3, Sec. 3.3), in place, on
 * the output projection in row-vector convention.
 *   W  : fp32 [dim][d_out] (ispa_apply_absorption) or bf16 (..._bf16: the sum is
 *        taken in fp32 and rounded to bf16);  dW : fp32 [dim][d_out].
 */
ISPA_API ispa_status ispa_apply_absorption(float* W, const float* dW, int32_t dim, int32_t d_out,
                                           ispa_stream stream);
ISPA_API ispa_status ispa_apply_absorption_bf16(void* W, const float* dW, int32_t dim, int32_t d_out,
                                                ispa_stream stream);

/*
 * Permanent eviction of an L-layer's history (Sec. 3.1 phase 3: "completely
 * discard their historical KV cache, retaining only the local context"): copy
 * the window's frames of `src` into the smaller caller-allocated ring `dst`
 * and make dst the layer's cache.  dst must have src's head shape,
 * n_sink_frames == win.n_sink_frames and capacity_frames == win.n_sink_frames +
 * win.n_recent_frames; on success dst->frames_written = src->frames_written and
 * every frame of the window sits in its dst slot (so later appends keep the
 * window sliding).  Errors: ISPA_ERR_CAPACITY if a window frame is not resident
 * in src, ISPA_ERR_INVALID_ARG on mismatched shapes.
 */
ISPA_API ispa_status ispa_ring_compact(const ispa_kv_ring* src, ispa_window win, ispa_kv_ring* dst,
                                       ispa_stream stream);

/* ------------------------------------------------------------ least squares */

/* Bytes of the fp32 [2*dim][2*dim] gram buffer. */
ISPA_API size_t ispa_ls_state_bytes(int32_t dim);

/* Zero state->gram (async) and state->n_tokens. */
ISPA_API ispa_status ispa_ls_state_reset(ispa_ls_state* state, ispa_stream stream);

/* Workspace bytes of ispa_ls_accumulate for T tokens of width dim. */
ISPA_API size_t ispa_ls_accumulate_workspace_size(int32_t dim, int64_t T);

/*
 * Add T tokens to the normal-equation sums (Sec. 3.2, "summing the outer
 * products ... during the standard forward pass"):
 *   G += A_loc^T A_loc,  X += A_loc^T Delta,  S += Delta^T Delta,  n += T,
 * Delta = A_full - A_loc taken exactly in fp32, products on the tensor cores
 * with fp32 accumulation.  A_loc and Delta enter as fp16, each multiplied by
 * the power of two that puts its largest magnitude over the call in
 * [2^14, 2^15); the factors are undone exactly when the sums are added to the
 * state.  A_loc's bf16 values convert exactly (down to 2^-29 of its largest
 * magnitude); Delta is rounded once, to 2^-11 relative, which leaves X and S
 * within about 1e-4 (Frobenius-relative) of the exact sums on typical inputs
 * and within 2 x 2^-11 in the worst case; the trace form of eps (Eq. 6) and
 * dW (Eq. 5) are affected far less, because independent roundings cancel in
 * them.  ISPA_LS_EXACT_DELTA (ispa_ls_accumulate_ex) carries Delta instead as
 * a bf16 hi + lo pair (2^-16 relative) at twice the tensor work for X and three
 * times for S.
 *   a_loc, a_full : bf16 [T][dim], dim a multiple of 128 (else UNSUPPORTED).
 *   workspace     : >= ispa_ls_accumulate_workspace_size(dim, T) bytes.
 */
ISPA_API ispa_status ispa_ls_accumulate(ispa_ls_state* state, const void* a_loc, const void* a_full,
                               int64_t T, void* workspace, size_t ws_bytes, ispa_stream stream);

/* Option bits of ispa_ls_accumulate_ex. */
#define ISPA_LS_EXACT_DELTA 1u

/* ispa_ls_accumulate with option bits (unknown bits: ISPA_ERR_INVALID_ARG). */
ISPA_API ispa_status ispa_ls_accumulate_ex(ispa_ls_state* state, const void* a_loc, const void* a_full,
                                  int64_t T, uint32_t flags, void* workspace, size_t ws_bytes,
                                  ispa_stream stream);

/* Workspace bytes of ispa_ls_solve. */
ISPA_API size_t ispa_ls_solve_workspace_size(int32_t dim, int32_t d_out);

/*
 * Closed-form absorption (Eq. 5) and feasibility score (Eq. 6), fp64:
 *   dW  = (G + lambda I)^{-1} X W          (Cholesky solve, Eq. 5 with R = Delta W)
 *   eps = || A_loc (W + dW) - A_full W ||_F^2
 *       = tr(W^T S W) - ||L^{-1} X W||_F^2 - lambda ||dW||_F^2,  L L^T = G + lambda I.
 *   W       : fp32 [dim][d_out], row-vector convention (out = A @ W; a torch
 *             nn.Linear weight is W^T)
 *   dW      : fp32 [dim][d_out] output
 *   eps_out : HOST double (nullable)
 *   lambda  : ridge weight on the unnormalised sums (paper default 1e-3)
 * Synchronises `stream`.  Errors: ISPA_ERR_NOT_SPD if a Cholesky pivot is not
 * positive.
 */
ISPA_API ispa_status ispa_ls_solve(const ispa_ls_state* state, const float* W, int32_t d_out,
                          double lambda, float* dW, double* eps_out, void* workspace,
                          size_t ws_bytes, ispa_stream stream);

/* ------------------------------------------------------------ 8-bit Q K^T attention */
/*
 * The chunk attention with queries and keys as fp8 e4m3 codes and values,
 * probabilities and output as in the bf16 path -- the 8-bit Q K^T / 16-bit P V
 * split of SageAttention, which the paper cites for its attention (Sec. 3.4).
 * One fp32 scale per head: x ~ code * scale.  The result is the attention of
 * the dequantised q and k (Eq. 3 / Eq. 7 on them), computed like the bf16 path.
 * Head dim 128 only.
 */

/* x: bf16 [n][H][d] -> codes q: uint8 [n][H][d] and scale: fp32 [H] (written),
 * scale_h = max |x_h| / 448 (1 for an all-zero head), code = e4m3(x * (1 / scale_h))
 * (each step in fp32, rounded to nearest even), saturating.  d % 16 == 0, H <= 256. */
ISPA_API ispa_status ispa_quantize_heads_e4m3(const void* x, int64_t n, int32_t H, int32_t d, uint8_t* q,
                                              float* scale, ispa_stream stream);

/* Queries for the *_qk8 attention: x bf16 [n][H][d] -> codes q [n][H][d] and
 * scale fp32 [H][ceil(n / 128)] (written): one scale per head and block of 128
 * consecutive tokens (the attention's query tile), computed like
 * ispa_quantize_heads_e4m3 within each block.  d % 16 == 0, d <= 256. */
ISPA_API ispa_status ispa_quantize_q_e4m3(const void* x, int64_t n, int32_t H, int32_t d, uint8_t* q,
                                          float* scale, ispa_stream stream);

/* Codes with given per-head scales: x bf16 [n][H][d], scale fp32 [H] (device)
 * -> q [n][H][d], code = e4m3(x * (1 / scale_h)).  For the chunk's keys, with
 * the ring's key scales.  d % 16 == 0. */
ISPA_API ispa_status ispa_quantize_k_e4m3(const void* x, int64_t n, int32_t H, int32_t d, const float* scale,
                                          uint8_t* q, ispa_stream stream);

/* ispa_kv_append for a ring with k_format = ISPA_KV_K_E4M3: keys are coded
 * with the ring's per-head scales k_scale[H] (device fp32, chosen by the caller
 * once for the ring's life, e.g. from the first chunk's ispa_quantize_heads_e4m3;
 * code = e4m3(k * (1 / scale)) as there; larger magnitudes saturate at
 * +-448 * scale), values are copied as bf16. */
ISPA_API ispa_status ispa_kv_append_qk8(ispa_kv_ring* ring, const void* k_new, const void* v_new,
                                        int32_t n_frames, const float* k_scale, ispa_stream stream);

/* ispa_attn_full / ispa_attn_local over a ring with e4m3 keys:
 *   q8     : uint8 [n_q][H][128] codes, q_scale fp32 [H][ceil(n_q / 128)] (from
 *            ispa_quantize_q_e4m3)
 *   k8_cur : uint8 [n_q][H][128] codes, k_cur_scale fp32 [H] (e.g. the ring's)
 *   k_ring_scale : the ring's key scales (as given to ispa_kv_append_qk8)
 *   v_cur : bf16 [n_q][H][128]; out, lse, scale as in ispa_attn_full.
 * Scale arrays live in device memory.  Errors as ispa_attn_full; a bf16 ring
 * (or an e4m3 ring given to the bf16 entry points) is ISPA_ERR_INVALID_ARG. */
ISPA_API ispa_status ispa_attn_full_qk8(const ispa_kv_ring* ring, const float* k_ring_scale, const void* q8,
                                        const float* q_scale, const void* k8_cur, const float* k_cur_scale,
                                        const void* v_cur, int32_t n_q, float scale, void* out, float* lse,
                                        ispa_stream stream);
ISPA_API ispa_status ispa_attn_local_qk8(const ispa_kv_ring* ring, const float* k_ring_scale, ispa_window win,
                                         const void* q8, const float* q_scale, const void* k8_cur,
                                         const float* k_cur_scale, const void* v_cur, int32_t n_q, float scale,
                                         void* out, float* lse, ispa_stream stream);
/* ispa_attn_dual over a ring with e4m3 keys (scales as above; other arguments
 * and the workspace as in ispa_attn_dual). */
ISPA_API ispa_status ispa_attn_dual_qk8(const ispa_kv_ring* ring, const float* k_ring_scale, ispa_window win,
                                        const void* q8, const float* q_scale, const void* k8_cur,
                                        const float* k_cur_scale, const void* v_cur, int32_t n_q, float scale,
                                        void* a_full, void* a_loc, float* disc, float* disc_sq_sum,
                                        float* lse_full, float* lse_loc, void* workspace, size_t ws_bytes,
                                        ispa_stream stream);

/* ------------------------------------------------------------ 8-bit Q K^T and P V attention */
/*
 * SageAttention's second form, which the paper cites for its attention kernels
 * (Sec. 3.4): Q K^T as above and P V in fp8 too -- the values as e4m3 codes with
 * one fp32 scale per head, the probabilities rounded to e4m3 in the kernel.  V is
 * stored d-major ([H][128][keys]), the operand layout of the 8-bit P V.  The result
 * approximates the attention of the dequantised q, k and v; the difference comes
 * from the e4m3 rounding of P only.  P_i = 2^(s_i - m) against a running maximum m
 * that stays within 2^4 of the row's maximum score, scaled by 2^4 before rounding:
 * each weight p_i = P_i / l (l = sum_i P_i >= 1, exact in fp32) is used with relative
 * error <= 2^-4, or absolute error <= 2^-14 / l where e4m3 is subnormal, so an
 * output element differs by at most 2^-4 sum_i p_i |v_i| + 2^-14 sum_i |v_i| / L,
 * L = sum_i exp(s_i - max_j s_j) <= l, plus the bf16 path's own rounding.  Head dim
 * 128; tokens per frame a multiple of 4.
 */

/* Row stride in bytes of a ISPA_KV_KV_E4M3 ring's d-major value codes:
 * capacity_frames * P rounded up to a multiple of 16. */
ISPA_API int64_t ispa_ring_vt_stride(const ispa_kv_ring* ring);

/* Values as d-major codes with given per-head scales: x bf16 [n][H][d] (d = 128),
 * scale fp32 [H] (device) -> qt uint8 [H][d][ld] with qt[h][c][t] =
 * e4m3(x[t][h][c] * (1 / scale_h)) as in ispa_quantize_k_e4m3; entries t >= n of a
 * row are left as they are.  ld >= n, ld % 16 == 0.  For the chunk's values,
 * with the ring's value scales. */
ISPA_API ispa_status ispa_quantize_vt_e4m3(const void* x, int64_t n, int32_t H, int32_t d, const float* scale,
                                           uint8_t* qt, int64_t ld, ispa_stream stream);

/* ispa_kv_append for a ring with k_format = ISPA_KV_KV_E4M3: keys coded with the
 * ring's key scales k_scale[H] as ispa_kv_append_qk8 does, values coded with the
 * ring's value scales v_scale[H] (device fp32, fixed for the ring's life, e.g. from
 * ispa_quantize_heads_e4m3 of the first values) into their d-major slots. */
ISPA_API ispa_status ispa_kv_append_kv8(ispa_kv_ring* ring, const void* k_new, const void* v_new,
                                        int32_t n_frames, const float* k_scale, const float* v_scale,
                                        ispa_stream stream);

/* ispa_attn_full_qk8 / ispa_attn_local_qk8 / ispa_attn_dual_qk8 with 8-bit P V over a
 * ISPA_KV_KV_E4M3 ring:
 *   v_scale : the ring's value scales (as given to ispa_kv_append_kv8), device fp32 [H]
 *   vt8_cur : the chunk's values as d-major codes [H][128][vt_ld] with v_scale (from
 *             ispa_quantize_vt_e4m3), vt_ld >= n_q, vt_ld % 16 == 0
 * Other arguments and errors as the *_qk8 calls; any other ring is
 * ISPA_ERR_INVALID_ARG. */
ISPA_API ispa_status ispa_attn_full_kv8(const ispa_kv_ring* ring, const float* k_ring_scale, const float* v_scale,
                                        const void* q8, const float* q_scale, const void* k8_cur,
                                        const float* k_cur_scale, const void* vt8_cur, int64_t vt_ld, int32_t n_q,
                                        float scale, void* out, float* lse, ispa_stream stream);
ISPA_API ispa_status ispa_attn_local_kv8(const ispa_kv_ring* ring, const float* k_ring_scale, const float* v_scale,
                                         ispa_window win, const void* q8, const float* q_scale, const void* k8_cur,
                                         const float* k_cur_scale, const void* vt8_cur, int64_t vt_ld, int32_t n_q,
                                         float scale, void* out, float* lse, ispa_stream stream);
ISPA_API ispa_status ispa_attn_dual_kv8(const ispa_kv_ring* ring, const float* k_ring_scale, const float* v_scale,
                                        ispa_window win, const void* q8, const float* q_scale, const void* k8_cur,
                                        const float* k_cur_scale, const void* vt8_cur, int64_t vt_ld, int32_t n_q,
                                        float scale, void* a_full, void* a_loc, float* disc, float* disc_sq_sum,
                                        float* lse_full, float* lse_loc, void* workspace, size_t ws_bytes,
                                        ispa_stream stream);

/* ------------------------------------------------------------ W8A8 projection */
/*
 * 8-bit weights and activations for the attention output projection on the
 * injected weight W + dW (Sec. 4 runs ISPA with W8A8 linear layers; Sec. 3.2
 * gives W_new = W + dW).  The paper fixes no 8-bit format; here it is fp8 e4m3
 * ("fn": largest magnitude 448, no infinities) with one fp32 scale per token
 * for activations and one per output channel for weights:
 *   amax = max |x| over the group; inv = 448 / amax and scale = amax / 448 in
 *   fp32 (both 1 for an all-zero group); code = e4m3(x * inv), rounded to
 *   nearest even and saturated at +-448.
 */

/* Activations x: bf16 [rows][cols] -> codes q: uint8 [rows][cols], scale: fp32
 * [rows].  cols % 16 == 0 (else ISPA_ERR_UNSUPPORTED); x and q 16-byte aligned. */
ISPA_API ispa_status ispa_quantize_rows_e4m3(const void* x, int64_t rows, int32_t cols, uint8_t* q,
                                             float* scale, ispa_stream stream);

/* Weight W (+ dW, nullable): fp32 [D][D_out] (row-vector convention y = a W) ->
 * codes q_t: uint8 [D_out][D] (K-major, the layout of a Linear weight) and
 * scale: fp32 [D_out], one per output channel of W + dW (summed in fp32).
 * D % 16 == 0.  Three launches; once per weight update, not per step. */
ISPA_API ispa_status ispa_quantize_weight_e4m3(const float* W, const float* dW, int32_t D, int32_t D_out,
                                               uint8_t* q_t, float* scale, ispa_stream stream);

/* out: bf16 [T][D_out] = a_scale[t] * w_scale[n] * sum_k dec(a_q[t][k]) * dec(w_q[n][k]),
 * with a_q [T][D] and w_q [D_out][D] e4m3 codes from the two calls above, fp32
 * accumulation on the tensor cores, bf16 output (round to nearest).
 * D % 128 == 0 and D_out % 128 == 0 (else ISPA_ERR_UNSUPPORTED); a_q, w_q, w_scale
 * and out 16-byte aligned. */
ISPA_API ispa_status ispa_linear_w8a8(const uint8_t* a_q, const float* a_scale, const uint8_t* w_q,
                                      const float* w_scale, int64_t T, int32_t D, int32_t D_out, void* out,
                                      ispa_stream stream);

#ifdef __cplusplus
}
#endif

#endif /* ISPA_H_ */
