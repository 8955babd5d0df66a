// Host-side launchers of the CUDA kernels (one translation unit each).
#pragma once

#include <cuda_runtime.h>
#include <cuda.h>
#include <stdint.h>

#include "epilogue.cuh"

// Launch options shared by every launcher: stream and whether to request
// programmatic dependent launch (overlap with the previous kernel's tail).
struct LaunchCtx {
  cudaStream_t stream;
  bool pdl;
  int num_sms;
  bool f16 = false;  // 16-bit operands are fp16 (else bf16); ignored in fp32 mode
};

// ---- decode projections (k_gemv.cu): out[b][n] = act[b] . W[n], B <= 64
// tokens, 16 weight rows per CTA, fused epilogue `kind`. Projections with
// few row tiles split K over CTAs; the partial tiles go to `part` and the
// per-tile tickets (zeroed, re-armed by the kernel) pick the CTA that sums.
struct SplitKWork {
  float* part;     // [max_ctas][16][64]
  int* ticket;     // [max_tiles]
  int max_tiles;
  int max_ctas;
};
struct SplitK {
  int count;
  float* part;
  int* ticket;
};
// act_lo (optional, fp16 mode): second term
// of a split activation operand, same layout and stride as act.
cudaError_t launch_gemv(const LaunchCtx& lc, int kind, bool fp32, const void* W, int N, int K, const void* act,
                        long long act_stride, int B, const EpiArgs& ep, const SplitKWork& wk,
                        const void* act_lo = nullptr);
// Query occupancy of the projection kernels (once, before launches).
cudaError_t prepare_gemv_kernels();


// ---- embedding gather producing x, a = x * g and the row sum of squares.
// rinv (optional): 1 / sqrt(mean(x^2) + eps) per row.
cudaError_t launch_embed(const LaunchCtx& lc, bool fp32, const void* E, int V, int D, const int* ids, int M, float* x,
                         void* a, const float* g, float* ss, int ss_stride, float* rinv, float eps, int* err,
                         void* a_lo = nullptr);

// ---- greedy token from argmax keys; clears the keys; optionally advances
// context lengths.
cudaError_t launch_finalize(const LaunchCtx& lc, unsigned long long* keys, int n_keys, int key_stride,
                            int key_offset, int B, int* next, int* ctx);

// ---- variable-length batches (k_varlen.cu)
// Row map of a packed batch: rowmap[m] = (sequence b, position past[b] + m -
// cu[b]) for the T rows; checks cu (cu[0] = 0, non-decreasing, cu[B] = T,
// chunks of 1 .. max_chunk rows) and past (>= 0, past + chunk <= max_pos),
// setting DEVERR_SEQ / DEVERR_POS; a row it cannot place gets (0, -1).
cudaError_t launch_varlen_rows(const LaunchCtx& lc, const int* cu, const int* past, int B, int T, int max_chunk,
                               int max_pos, int2* rowmap, int* err);
// Last row of each sequence's chunk gathered into dense [B] rows: the 16-bit
// (or fp32) operand a (and its second term a_lo, fp16 mode) and the row's
// inverse RMS, from either reduced rinv[row] or `parts` partial sums of
// squares ss[row * ss_stride + i].
cudaError_t launch_gather_last(const LaunchCtx& lc, const int* cu, int B, int T, const void* a, const void* a_lo,
                               int row_bytes, const float* rinv, const float* ss, int ss_stride, int parts,
                               float inv_D, float eps, void* a_out, void* a_lo_out, float* rinv_out);
// Greedy token of each sequence from argmax keys (keys[b] when last_rows is
// 0, else keys[cu[b+1]-1]), context lengths advanced by the chunk lengths
// (optional), and the first n_keys keys cleared.
cudaError_t launch_finalize_varlen(const LaunchCtx& lc, unsigned long long* keys, int n_keys, const int* cu,
                                   int last_rows, int B, int* next, int* ctx);

// ---- qk-norm (k_varlen.cu): q and k of `rows` rows from e.qk_raw,
// normalised per head, scaled by the gains, rotated and stored (q, its second
// term when e.q_lo_out is set, k into the cache slot of the row's position);
// e is the QKV launch's epilogue argument block.
cudaError_t launch_qk_norm_rope(const LaunchCtx& lc, bool fp32, const EpiArgs& e, int rows);

// ---- mixture of experts (k_moe.cu): routing, the stable sort of
// (token, expert) slots into 128-row expert segments, the sorted operand
// rows and the combine into the residual; the expert products run on the
// grouped tcgen05 GEMM (GemmGroup).
constexpr int MOE_MAX_EXPERTS = 256;
struct MoeArgs {
  int D, E, k, norm_topk;
  const void* act;     // normed operand a = x * g [T][act_stride] (16-bit)
  const void* act_lo;  // its second term (fp16 mode), or null
  long long act_stride;
  const float* logits;  // [T][E] router logits (fp32, norm scale applied)
  int* topk_idx;        // [T * k]
  float* topk_w;        // [T * k]
  int* slot_row;        // [T * k] sorted row of each (token, j) slot
  int* row_tok;         // [rows] token of each sorted row, -1 for padding
  float* row_w;         // [rows] routing weight of each sorted row
  int* mb_expert;       // [rows / 128] expert of each 128-row block
  int* n_mblocks;       // [1] blocks laid out
  void* a_sorted;       // [rows][D] sorted operand rows (normalised, 16-bit)
  float* y_sorted;      // [rows][D] expert outputs times routing weight
  int* record;          // optional [record_rows][k]: copy of the chosen experts (inspection)
  int record_rows;
  int* err;
};
cudaError_t prepare_moe_kernels(int D, int E);
// Routing of T tokens from a.logits and the sorted layout (one or two launches).
cudaError_t launch_moe_route_plan(const LaunchCtx& lc, const MoeArgs& a, int T);
// ns: the norm state of `act` (row_rinv).
cudaError_t launch_moe_gather(const LaunchCtx& lc, const MoeArgs& a, int T, const EpiArgs& ns);
// ep: residual x (ep.x, ep.N = D) and, when ep.a_out is set, the residual
// epilogue's outputs (a_out, a_lo_out, gain, ss_out / ss_out_stride).
cudaError_t launch_moe_combine(const LaunchCtx& lc, const MoeArgs& a, int T, const EpiArgs& ep);

// ---- attention (k_attn.cu)
struct AttnArgs {
  const void* q;  // [rows][H*d]
  const void* k;  // layer pool [num_blocks][G][16][d]
  const void* v;
  void* o;        // [rows][H*d]
  const int* ctx;  // decode: [B] tokens cached before the step
  const int* block_table;
  int bt_stride;
  int blocks_per_seq;
  int num_blocks;
  int H, G, d;
  int S;        // prefill prompt length
  int splits;   // decode split-KV factor
  int window;   // sliding window: a query at position p sees keys p-window+1 .. p (0: no window)
  float scale_log2;
  float* part;  // decode partials
  void* o_lo;   // optional [rows][H*d]: o minus its 16-bit rounding (decode, fp16 mode)
  const void* q_lo;  // optional [rows][H*d]: q minus its 16-bit rounding (decode)
  int* counter;  // decode [B][G] tickets
  int* err;
};
// Variable-length prefill: sequence b's chunk is rows cu[b] .. cu[b+1]-1 of
// q / o at positions past[b] + i; `rows` bounds the row offsets and the
// AttnArgs' S is the longest chunk (grid height). Kept out of AttnArgs: the
// decode kernels take AttnArgs by value and their register allocation
// (measured 147 vs 128 per thread at head_dim 128) depends on its size.
struct AttnVarlen {
  const int* cu;
  const int* past;
  int rows;
  const int2* rowmap;  // fp32 debug path: (sequence, position) per row
};
cudaError_t launch_attn_decode(const LaunchCtx& lc, bool fp32, const AttnArgs& a, int B);
// vl: variable-length batch, or null (B sequences of a.S tokens from position 0)
cudaError_t launch_attn_prefill(const LaunchCtx& lc, bool fp32, const AttnArgs& a, int B,
                                const AttnVarlen* vl = nullptr);
// Key splits of the decode attention (1 .. min(max_blocks, 64)): the count
// with the smallest estimated makespan over num_sms SMs, or, with
// target_ctas > 0, as many as keep B x G x splits within that many CTAs.
int attn_decode_splits(int B, int G, int max_blocks, int num_sms, int target_ctas);
// Set kernel attributes (dynamic shared memory limits) once, before any
// launch or graph capture.
cudaError_t prepare_attn_kernels();
cudaError_t prepare_gemm_kernels();

// ---- prefill projections (k_gemm.cu): tcgen05 + TMA persistent GEMM,
// out[m][n] = A[m] . W[n], M x N x K with K % 64 == 0.
struct GemmMaps {
  CUtensorMap a;     // activations [rows][K], box 64 x 128
  CUtensorMap w;     // weights [N][K], box 64 x 256 (64 x 128 in the n128 set)
  CUtensorMap a_lo;  // second term of a split activation operand (used when split)
  // the same activation operand (and second term) in boxes of 16 and of 64
  // rows: at most 16 (64) rows (decode), the ring stages hold only those
  CUtensorMap a16;
  CUtensorMap a_lo16;
  CUtensorMap a64;
  CUtensorMap a_lo64;
  bool has16 = false;
  bool has64 = false;
  bool split = false;
  const GemmMaps* n128 = nullptr;  // the same operands with 128-row weight boxes (128-wide tiles), or null
};
bool make_tma_2d_16(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows, bool f16);
// Row-major [rows][cols] 16-bit matrix, box box_cols x box_rows, no swizzle
// (dense rows in shared memory); out-of-range elements read as zero.
bool make_tma_2d_plain(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_cols,
                       uint32_t box_rows, bool f16);
// Split-K mode of the GEMM for M <= 128 rows (decode): the K blocks are cut
// into ks parts; each (256-wide tile, part) unit leaves its fp32 partial
// tile in ws ([unit][128][256], rows < M written) and the last unit of a
// tile to finish (ticket per tile, zero between launches, reset by that
// unit; nobody waits) sums the parts in order and runs the epilogue.
constexpr int GEMM_MAX_UNITS = 320;
struct GemmSplitK {
  int ks = 1;
  float* ws = nullptr;       // GEMM_MAX_UNITS * 128 * 256 floats
  int* tickets = nullptr;    // [max_tiles]
  int max_tiles = 0;
};
// Grouped mode (mixture of experts, stacked experts): the activation rows
// are sorted by expert, each expert's rows padded to whole 128-row blocks;
// m-block b belongs to expert mb_expert[b], and *n_mblocks blocks exist
// (both written on the device by the routing plan). The weight operand is
// the experts' matrices stacked as one [E * N][K] tensor: block b's tiles
// read rows mb_expert[b] * N + n. Rows whose row_valid entry is negative
// are padding and get no epilogue. M bounds the sorted rows.
struct GemmGroup {
  const int* mb_expert = nullptr;  // null: ordinary GEMM
  const int* n_mblocks = nullptr;
  const int* row_valid = nullptr;
};
// tile_n: 256 or 128 (from gemm_tile_n); the residual epilogue writes one
// norm partial per row and tile, i.e. ceil(N / tile_n) of them.
cudaError_t launch_gemm_tc(const LaunchCtx& lc, int kind, const GemmMaps& maps, int M, int N, int K, const EpiArgs& ep,
                           int tile_n = 256, const GemmSplitK* split = nullptr, const GemmGroup* group = nullptr);
int gemm_tile_n(const LaunchCtx& lc, const GemmMaps& maps, int M, int N);
// K split (1 = none) for a decode-sized M x N x K product whose 256-wide
// tiles cannot fill half the GPU.
int gemm_split_k(const LaunchCtx& lc, int M, int N, int K);

// ---- fp32 debug projections (k_simt.cu): plain tiled CUDA-core GEMM with
// the same epilogues, any M.
cudaError_t launch_gemm_simt(const LaunchCtx& lc, int kind, const float* A, long long a_stride, const float* W, int M,
                             int N, int K, const EpiArgs& ep);

// ---- persistent decode step (k_persist.cu): one cooperative launch of one
// CTA per SM runs a whole decode step for B <= PERSIST_MAX_B sequences.
constexpr int PERSIST_MAX_B = 8;
constexpr int PERSIST_BOX_COLS = 256;
struct PersistLayer {
  const void* wqkv;
  const float* bqkv;  // or null
  const void* wo;
  const void* wgu;
  const void* wd;
  const float* g1;     // input norm gain
  const float* g2;     // post-attention norm gain
  const float* gnext;  // gain of the norm after this layer (next layer's g1, or the final norm)
  void* kc;            // this layer's K pool
  void* vc;            // this layer's V pool
};
// Grid barrier state: zero before a launch; the launch leaves it zero.
struct PersistGrid {
  unsigned count;
  unsigned exit;
  unsigned abort;
  unsigned pad;
};
struct PersistArgs {
  int L, D, H, G, d, F, V, Nqkv, Pmax, B;
  int max_pos, blocks_per_seq, num_blocks, splits, window, act;
  float eps, inv_D, scale_log2;
  const PersistLayer* layers;  // device [L]
  // device [4L + 1]: per layer the QKV, O, gate/up and down weights, then the
  // LM head; box PERSIST_BOX_COLS x 16 rows, no swizzle
  const CUtensorMap* wmaps;
  const void* embed;
  const void* head;
  const float* gf;
  const float2* rope;
  float* x;
  void* a;
  void* a_lo;  // fp16 mode: second term of a
  float* ss;   // norm partials [B][Pmax]
  void* q;
  void* q_lo;  // second term of q (16-bit modes)
  void* o;
  void* u;
  void* o_lo;  // fp16 mode: second terms of o and u
  void* u_lo;
  unsigned long long* keys;
  float* attn_part;
  int* attn_cnt;
  int* err;
  PersistGrid* grid;
  const int* tokens;
  int* ctx;
  const int* block_table;
  float* logits;
  int* next;
};
// Resident CTAs per SM of the kernel for this head_dim / type (0: not
// available); also sets its shared-memory limit. Call before any launch.
int persist_ctas_per_sm(int head_dim, bool use_f16);
// Whether B sequences of width D (widest projection input kmax) suit the
// kernel (their activations stage in shared memory); else the decode step
// takes the launch chain.
bool persist_fits(int head_dim, bool use_f16, int B, int D, int kmax);
cudaError_t launch_persist_decode(const PersistArgs& a, int head_dim, bool use_f16, int nctas, cudaStream_t st);
