// Internal declarations shared by the translation units of libispa (host side).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/ispa.h"

namespace ispa {

// ------------------------------------------------------------ attention
// One contiguous run of keys.  src 0 = the KV ring ([H][cap*P][d]), src 1 = the
// chunk's own k_cur/v_cur ([n_q][H][d]).  start/count are token rows.
struct AttnSeg {
  int32_t src;
  int32_t start;
  int32_t count;
  int32_t skip;   // leading keys of the segment that are not in the key set (masked): 0, or the
                  // alignment a segment of the 8-bit P V instance starts with
};

constexpr int kMaxSegs = 8;
constexpr int kAttnBM = 128;  // queries per attention CTA
constexpr int kAttnBN = 192;  // keys per attention tile (TMA box rows of the K/V maps)

struct AttnParams {
  int32_t n_q;
  int32_t num_heads;
  int32_t n_seg;           // segments in seg[]
  int32_t n_tiles;         // total key tiles over all segments
  int32_t n_local_tiles;   // dual: tiles of the local set (they come first)
  int32_t dual;            // 1 = emit A_loc snapshot and discrepancy partials
  float scale_log2;        // softmax scale * log2(e)
  int32_t causal_p;        // frame-causal chunk: tokens per frame (query row r sees chunk keys
                           // < (r / causal_p + 1) * causal_p); 0 = the chunk is dense
  uint64_t wait_limit_ns;  // bounded-wait limit
  AttnSeg seg[kMaxSegs];
  __nv_bfloat16* out;      // [n_q][H*d]  (A_full in dual mode)
  __nv_bfloat16* out_loc;  // [n_q][H*d]  dual only
  float* lse;              // [H][n_q] or null
  float* lse_loc;          // [H][n_q] or null (dual)
  float* disc_part;        // [H][n_q] per-head sum of squared discrepancy (dual)
  int* status;             // library status record
  uint32_t* heartbeat;     // debug counters (host-mapped) or null
  uint64_t* trace;         // debug per-tile cycle trace of CTA (0,0) or null: [tile][8]
  int32_t trace_tiles;
  int32_t drop_k_tile;     // debug: key tile the TMA thread never loads (-1: none)
  // 8-bit Q K^T (null for bf16 Q and K): per-head e4m3 code scales of q, chunk keys, ring keys
  const float* q_scale;
  const float* kc_scale;
  const float* kr_scale;
  // 8-bit P V (null for bf16 V): per-head e4m3 code scale of V (ring and chunk alike)
  const float* v_scale;
};

// Raise the dynamic shared-memory limit of `func` to `bytes` on the current device, once
// per (device, kernel); safe to call from several host threads.
cudaError_t set_smem_limit_once(const void* func, int bytes);

// Launch the attention kernel.  tensor maps are encoded by the caller.
cudaError_t launch_attention(int head_dim, const CUtensorMap* tm_q, const CUtensorMap* tm_kr,
                             const CUtensorMap* tm_vr, const CUtensorMap* tm_kc,
                             const CUtensorMap* tm_vc, const AttnParams& p, cudaStream_t s);
// disc[t] = sqrt(sum_h part[h][t]); *disc_sq_sum += sum_t sum_h part[h][t]
cudaError_t launch_disc_reduce(const float* part, int32_t H, int32_t n_q, float* disc,
                               float* disc_sq_sum, cudaStream_t s);

// O = 0 and LSE = -inf for an empty key set (the history branch with no history).
cudaError_t launch_empty_branch(void* out, float* lse, int32_t n_q, int32_t H, int32_t d, cudaStream_t s);

// ------------------------------------------------------------ KV append
constexpr int kMaxAppendFrames = 16;
constexpr int kMaxAppendLayers = 64;

struct AppendParams {
  int32_t n_layers;
  int32_t n_frames;
  int32_t tokens_per_frame;
  int32_t num_heads;
  int32_t head_dim;
  int32_t pad;
  int32_t capacity_tokens[kMaxAppendLayers];           // capacity_frames * P of each layer's ring
  int32_t slot[kMaxAppendLayers][kMaxAppendFrames];    // ring slot of each appended frame
  const void* k_src[kMaxAppendLayers];
  const void* v_src[kMaxAppendLayers];
  void* k_dst[kMaxAppendLayers];
  void* v_dst[kMaxAppendLayers];
};
cudaError_t launch_append(const AppendParams& p, cudaStream_t s);

// ------------------------------------------------------------ least squares
// Accumulate the upper blocks of [A | dlt]^T [A | dlt] into the fp32 state; exact: Delta as a
// bf16 hi / lo pair, else A_loc and Delta as scaled fp16.
cudaError_t launch_ls_accumulate(int32_t D, int64_t T, const void* a_loc, const void* a_full, void* ws,
                                 bool exact, float* gram, int* status, uint64_t wait_limit_ns,
                                 uint32_t* heartbeat, cudaStream_t s);
size_t ls_accumulate_ws_bytes(int32_t D, int64_t T);

size_t ls_solve_ws_bytes(int32_t D, int32_t d_out);
// Returns ISPA_OK, ISPA_ERR_NOT_SPD or ISPA_ERR_CUDA; synchronises the stream.
ispa_status run_ls_solve(int32_t D, const float* gram, const float* W, int32_t d_out,
                         double lambda, float* dW, double* eps_out, void* ws, cudaStream_t s);

// ------------------------------------------------------------ W8A8 projection
cudaError_t launch_quant_rows(const void* x, int64_t rows, int32_t cols, uint8_t* q, float* scale, cudaStream_t s);
cudaError_t launch_quant_weight(const float* W, const float* dW, int32_t D, int32_t Dout, uint8_t* q_t, float* scale,
                                cudaStream_t s);
cudaError_t launch_w8a8_gemm(const uint8_t* a_q, const float* a_scale, const uint8_t* w_q, const float* w_scale,
                             int32_t T, int32_t D, int32_t Dout, void* out, int* status, uint64_t wait_limit_ns,
                             cudaStream_t s);

// ------------------------------------------------------------ 8-bit Q K^T
cudaError_t launch_quant_heads(const void* x, int64_t n, int32_t H, int32_t d, uint8_t* q, float* scale,
                               cudaStream_t s);
cudaError_t launch_quant_q_blocks(const void* x, int64_t n, int32_t H, int32_t d, uint8_t* q, float* scale,
                                  cudaStream_t s);
cudaError_t launch_quant_given(const void* x, int64_t n, int32_t H, int32_t d, const float* scale, uint8_t* q,
                               cudaStream_t s);
// d-major e4m3 values: out[h][c][key] (key = t, or slots[t / P] * P + t % P when n_frames > 0);
// d = 128, ld % 16 == 0, P % 4 == 0.
cudaError_t launch_quant_vt(const void* x, int64_t n, int32_t H, int32_t d, const float* scale, uint8_t* out,
                            int64_t ld, int32_t P, int32_t n_frames, const int32_t* slots, cudaStream_t s);
cudaError_t launch_append_qk8(const int32_t* slots, int32_t n_frames, int32_t P, int32_t H, int32_t d,
                              int64_t ring_tok, const void* k_src, const void* v_src, void* k_dst, void* v_dst,
                              const float* k_scale, cudaStream_t s);

// ------------------------------------------------------------ misc
int* device_status_ptr();  // library status word in the current context (nullptr on error)
// Process-unique id of the calling thread's current CUDA context (the device's primary
// context is bound first when none is current); false if the driver cannot report it.
bool current_context_id(uint64_t* id);
bool encode_tmap_3d(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2,
                    uint64_t stride1_bytes, uint64_t stride2_bytes, uint32_t b0, uint32_t b1,
                    uint32_t b2);
// 128-byte swizzle, rank 4 (dims / strides in bytes for dims 1-3 / box).
bool encode_tmap_4d(CUtensorMap* m, const void* base, const uint64_t dims4[4], const uint64_t strides3[3],
                    const uint32_t box4[4], bool u8 = false);   // u8: uint8 elements instead of bf16
bool encode_tmap_2d(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1,
                    uint64_t stride1_bytes, uint32_t b0, uint32_t b1);
// uint8 elements, 128-byte swizzle, rank 2.
// fp32 [d1][d0] with 128-byte swizzle (the Gram state, for bulk reduce-adds)
bool encode_tmap_2d_f32(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t stride1_bytes,
                        uint32_t b0, uint32_t b1);
// uint8 (d0 inner, d1, d2) with 128-byte swizzle
bool encode_tmap_3d_u8(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2,
                       uint64_t stride1_bytes, uint64_t stride2_bytes, uint32_t b0, uint32_t b1, uint32_t b2);
bool encode_tmap_2d_u8(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t stride1_bytes,
                       uint32_t b0, uint32_t b1);
uint64_t wait_limit_ns();
uint32_t* next_heartbeat_slot(uint32_t kernel_tag);  // null unless a heartbeat buffer is set
uint64_t* trace_buffer(int32_t* n_tiles);            // null unless a trace buffer is set

}  // namespace ispa
