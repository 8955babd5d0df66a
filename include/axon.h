/*
 * axon.h -- C ABI of the GB300 (sm_103a) Llama-family decoder forward.
 *
 * The operation behind these calls is the forward pass that the Axon paper
 * (arxiv 2608.19889) compiles to its backends: a model definition plus a
 * safetensors checkpoint go in (Fig. 1; Sec. "The Axon Compiler", Phase 3:
 * backends implement `forward` and `generate` with static-cache scaffolding),
 * logits and greedy next tokens come out (Sec. "Results", Measures). The
 * per-layer math is the pre-norm block of Sec. "The Axon Language" (RMSNorm,
 * grouped-query causal attention with rotary positions and a KV cache,
 * residual add, SwiGLU MLP) built from the library of Sec. "Built-In
 * Libraries"; the model skeleton follows the appendix causal_lm listing
 * (embedding, layer loop threading the cache, final norm, tied or untied
 * LM head).
 *
 * Conventions for every call
 *   - Return value: AXON_OK (0) or one AXON_ERR_* code. Nothing aborts or
 *     throws across the ABI. axon_status_string() names a code.
 *   - Pointers named d_* are DEVICE pointers (CUDA global memory of the
 *     device current when the model was created). The caller owns them.
 *   - Work is enqueued asynchronously on `stream` (a cudaStream_t; NULL =
 *     the legacy default stream). Argument errors are reported
 *     synchronously; device-side range checks (token ids, block-table
 *     entries, positions) set a device error word that
 *     axon_check_device() reads, and the offending access is skipped.
 *   - Token ids, context lengths and block tables are int32.
 *   - Floating point: weights bf16 (or fp32 widened in AXON_FP32_DEBUG),
 *     fp32 accumulation everywhere, fp32 residual stream and logits.
 */
#ifndef AXON_H
#define AXON_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Status codes. */
enum {
  AXON_OK = 0,
  AXON_ERR_INVALID_ARG = 1,    /* null pointer, bad enum, B or S out of range */
  AXON_ERR_SHAPE_MISMATCH = 2, /* a weight's shape disagrees with the config */
  AXON_ERR_MISSING_WEIGHT = 3, /* a required weight name is absent */
  AXON_ERR_UNSUPPORTED = 4,    /* config outside what the kernels implement */
  AXON_ERR_OOM = 5,            /* device allocation failed */
  AXON_ERR_CUDA = 6,           /* a CUDA runtime call failed */
  AXON_ERR_TIMEOUT = 7,        /* a bounded device wait expired */
  AXON_ERR_DEVICE_CHECK = 8    /* a device-side range check fired */
};

/* KV cache layouts (Sec. Built-In Libraries: a static, preallocated cache
 * overlay; vLLM's PagedAttention manager, Sec. Related Work). */
enum { AXON_KV_CONTIGUOUS = 0, AXON_KV_PAGED = 1 };

/* Arithmetic mode (Sec. Results: bf16 primary, fp32 fallback):
 *   AXON_BF16        bf16 weights, bf16 GEMM operands and KV cache, fp32
 *                    accumulation, fp32 residual stream and logits;
 *   AXON_FP32_DEBUG  everything fp32 (CUDA-core GEMMs), for checking;
 *   AXON_FP16        the bf16 checkpoint converted exactly to fp16 (every
 *                    bf16 value of magnitude 2^-14 .. 65504 is an fp16
 *                    value), fp16 GEMM operands and KV cache, fp32
 *                    accumulation and residual: same speed as AXON_BF16, 8x
 *                    smaller operand rounding (10- vs 7-bit mantissa).
 *                    Operands saturate at +-65504; a weight beyond that
 *                    range makes axon_model_create return
 *                    AXON_ERR_UNSUPPORTED. */
enum { AXON_BF16 = 0, AXON_FP32_DEBUG = 1, AXON_FP16 = 2 };

/* Gate activation of the gated MLP (Activations built-ins, Sec. Built-In
 * Libraries): silu (SwiGLU, Llama / Qwen / Mistral) or the tanh form of
 * GELU, gelu_new of the appendix GPT-2 listing (gated GELU). */
enum { AXON_ACT_SILU = 0, AXON_ACT_GELU_TANH = 1 };

/* Element types of weight tensors handed to axon_model_create. */
enum { AXON_DTYPE_BF16 = 0, AXON_DTYPE_F32 = 1 };

/* Which positions of a prefill get logits written. */
enum { AXON_LOGITS_LAST = 0, AXON_LOGITS_ALL = 1 };

/* Model configuration: HF config.json equivalents (the appendix causal_lm
 * listing reads hidden size, layer and head counts and vocabulary size
 * through `Config.dim @@key`), plus capacity and layout fields. */
typedef struct axon_config {
  int32_t num_hidden_layers;   /* L */
  int32_t hidden_size;         /* D, multiple of 64 */
  int32_t num_attention_heads; /* H, multiple of num_key_value_heads */
  int32_t num_key_value_heads; /* G */
  int32_t head_dim;            /* d: 64 or 128 */
  int32_t intermediate_size;   /* F, multiple of 64 */
  int32_t vocab_size;          /* V */
  int32_t tie_word_embeddings; /* 1: LM head = embedding matrix */
  int32_t attention_bias;      /* 1: q, k, v projections carry biases */
  float rope_theta;            /* rotary base */
  float rms_norm_eps;          /* RMSNorm epsilon */
  int32_t max_batch;           /* sequences (contiguous cache slots) */
  int32_t max_context;         /* tokens per sequence, multiple of 16 */
  int32_t max_prefill_tokens;  /* largest B*S per axon_prefill; 0 = max_batch*max_context */
  int32_t kv_layout;           /* AXON_KV_CONTIGUOUS or AXON_KV_PAGED */
  int32_t kv_block_size;       /* tokens per block: must be 16 */
  int32_t kv_num_blocks;       /* paged pool size in blocks (ignored if contiguous) */
  int32_t precision;           /* AXON_BF16, AXON_FP16 or AXON_FP32_DEBUG */
  int32_t sliding_window;      /* W > 0: a query at position p attends only to
                                  keys p-W+1 .. p (the `window=` argument of
                                  causal_mask_for_input, appendix GPT-2
                                  listing); 0: full causal attention */
  /* RoPE frequency scaling of Llama-3.1-family checkpoints (HF
   * rope_scaling {"rope_type": "llama3", ...}); rope_scaling_factor 0 =
   * none. A rotary frequency f with wavelength w = 2 pi / f is kept when
   * w < original / high_freq_factor, divided by the factor when
   * w > original / low_freq_factor, and blended linearly in
   * t = (original / w - low) / (high - low) between: (1-t) f / factor + t f. */
  float rope_scaling_factor;
  float rope_low_freq_factor;
  float rope_high_freq_factor;
  int32_t rope_original_max_position;
  int32_t hidden_act;          /* AXON_ACT_SILU or AXON_ACT_GELU_TANH: u = act(h W_gate^T) * (h W_up^T) */
  int32_t qk_norm;             /* 1: each head's q and k (after the projection and its bias) go
                                  through RMSNorm over their head_dim values, with rms_norm_eps and
                                  the gains model.layers.{i}.self_attn.{q,k}_norm.weight [head_dim],
                                  before RoPE (Qwen3-family layers); 0: none. Decode then always
                                  takes the launch chain. */
  /* Mixture of experts (the MoE built-ins: softmax top-k router, grouped
   * experts; DeepSeek-MoE layout). n_routed_experts E > 0: layers from
   * first_k_dense_replace on replace the MLP by
   *   p = softmax(h W_router^T) over the E experts (fp32 router),
   *   the num_experts_per_tok experts with the largest p (lowest index on
   *   ties), weights p (divided by their sum when norm_topk_prob),
   *   y = sum_j w_j * SwiGLU-MLP_j(h) + SwiGLU-MLP_shared(h),
   * with experts of width moe_intermediate_size and, when
   * n_shared_experts > 0, one shared MLP of width n_shared_experts *
   * moe_intermediate_size. E <= 256, 1 <= num_experts_per_tok <= min(8, E),
   * 16-bit modes only; decode takes the launch chain. */
  int32_t n_routed_experts;
  int32_t num_experts_per_tok;
  int32_t moe_intermediate_size;
  int32_t n_shared_experts;
  int32_t first_k_dense_replace;
  int32_t norm_topk_prob;
} axon_config;

/* One named checkpoint tensor, HF Llama naming and [out, in] matrices, as a
 * safetensors file stores them (Fig. 1; weights looked up by flat dotted
 * path, appendix "Python Overhead"):
 *   model.embed_tokens.weight                       [V, D]
 *   model.layers.{i}.input_layernorm.weight         [D]
 *   model.layers.{i}.self_attn.{q,k,v}_proj.weight  [H*d | G*d | G*d, D]
 *   model.layers.{i}.self_attn.{q,k,v}_proj.bias    (if attention_bias)
 *   model.layers.{i}.self_attn.o_proj.weight        [D, H*d]
 *   model.layers.{i}.post_attention_layernorm.weight[D]
 *   model.layers.{i}.mlp.{gate,up}_proj.weight      [F, D]
 *   model.layers.{i}.mlp.down_proj.weight           [D, F]
 *   model.layers.{i}.self_attn.{q,k}_norm.weight    [d] (if qk_norm)
 *   mixture-of-experts layers (i >= first_k_dense_replace when
 *   n_routed_experts > 0) carry instead of mlp.{gate,up,down}_proj:
 *   model.layers.{i}.mlp.gate.weight                [E, D] (router)
 *   model.layers.{i}.mlp.experts.{e}.{gate,up}_proj.weight [Fe, D]
 *   model.layers.{i}.mlp.experts.{e}.down_proj.weight      [D, Fe]
 *   model.layers.{i}.mlp.shared_experts.{gate,up}_proj.weight [Fs, D]
 *   model.layers.{i}.mlp.shared_experts.down_proj.weight   [D, Fs]
 *     (Fe = moe_intermediate_size, Fs = n_shared_experts * Fe; shared only
 *     when n_shared_experts > 0)
 *   model.norm.weight                               [D]
 *   lm_head.weight                                  [V, D] (absent if tied)
 * `data` may be a host or a device pointer (unified addressing); it is
 * only read during axon_model_create. Row-major, contiguous. */
typedef struct axon_tensor {
  const char* name;
  const void* data;
  int32_t dtype; /* AXON_DTYPE_BF16 or AXON_DTYPE_F32 */
  int32_t ndim;  /* 1 or 2 */
  int64_t shape[4];
} axon_tensor;

typedef struct axon_model axon_model;

/* Build a model: validate the config against the named weights (symbolic
 * dimensions, Sec. The Axon Language, Types), allocate and repack weights
 * into the kernels' layout (fused QKV, interleaved gate/up), allocate the KV
 * cache and workspace. The weight table is copied; the caller may free it
 * on return. Work is done on `stream` and synchronised before returning.
 * *out receives the model, or NULL on error. */
int axon_model_create(const axon_config* cfg, const axon_tensor* weights, int32_t n_weights,
                      void* stream, axon_model** out);

/* Prompt pass (Positions.position_ids with past_length 0; Cache.update of
 * every prompt token; Sec. Built-In Libraries).
 *   d_ids          [B, S] token ids.
 *   B              1 .. max_batch; sequence b uses contiguous slot b, or the
 *                  blocks named by row b of d_block_table.
 *   S              1 .. max_context, B*S <= max_prefill_tokens.
 *   d_block_table  paged layout: [B, ceil(max_context/16)] pool block ids,
 *                  row b for sequence b (entries past the prompt unused);
 *                  must be NULL for the contiguous layout.
 *   logits_mode    AXON_LOGITS_LAST: d_logits is [B, V], the last position;
 *                  AXON_LOGITS_ALL: d_logits is [B, S, V].
 *   d_logits       fp32 output, or NULL to skip storing logits.
 *   d_next         [B] greedy next token (argmax of the last position's
 *                  logits, lowest index on ties), or NULL.
 * Previous contents of the used cache slots are overwritten. */
int axon_prefill(axon_model* m, const int32_t* d_ids, int32_t B, int32_t S,
                 const int32_t* d_block_table, int32_t logits_mode, float* d_logits,
                 int32_t* d_next, void* stream);

/* Variable-length batch: B sequences each append one chunk of new tokens
 * after the tokens they already hold in the cache -- a whole prompt, the
 * next piece of a long prompt (chunked prefill), or a single decode token
 * -- packed row after row into one forward pass (Positions.position_ids
 * with a per-sequence past_length and Cache.update, Sec. Built-In
 * Libraries; the continuous batching of vLLM's PagedAttention manager,
 * Sec. Related Work). Every chunk attends causally to its own sequence's
 * cached tokens and to the earlier tokens of the chunk.
 *   d_ids           [T] token ids, sequence b's chunk at rows
 *                   cu_seqlens[b] .. cu_seqlens[b+1]-1.
 *   B               1 .. max_batch; sequence b uses contiguous slot b, or
 *                   the blocks named by row b of d_block_table.
 *   T               total new tokens, B .. max_prefill_tokens.
 *   d_cu_seqlens    [B+1] row offsets: cu[0] = 0, cu[B] = T, every chunk
 *                   1 .. max_chunk tokens long.
 *   d_context_lens  [B] IN/OUT: tokens already cached for sequence b (0 for
 *                   a new prompt); chunk token i takes position
 *                   context_lens[b] + i, which must stay below
 *                   max_context. The call adds each chunk's length (in
 *                   stream order, after all reads), so the next call --
 *                   another chunk or axon_decode_step -- can follow
 *                   without host work.
 *   max_chunk       host bound on the longest chunk, 1 .. min(T,
 *                   max_context); it sizes the attention grid.
 *   d_block_table   paged layout: [B, ceil(max_context/16)], else NULL.
 *   logits_mode     AXON_LOGITS_LAST: d_logits is [B, V], the last token of
 *                   each chunk; AXON_LOGITS_ALL: d_logits is [T, V].
 *   d_logits        fp32 output, or NULL.
 *   d_next          [B] greedy next token after each chunk's last token
 *                   (lowest index on ties), or NULL.
 * Offsets and lengths are read on the device: inconsistent ones (cu not
 * starting at 0, not ending at T, a chunk outside 1 .. max_chunk) or
 * positions past max_context set the device error word
 * (AXON_ERR_DEVICE_CHECK from axon_check_device) and the rows they affect
 * are skipped. Cache slots at the chunk's positions are overwritten. */
int axon_prefill_varlen(axon_model* m, const int32_t* d_ids, int32_t B, int32_t T, const int32_t* d_cu_seqlens,
                        int32_t* d_context_lens, int32_t max_chunk, const int32_t* d_block_table,
                        int32_t logits_mode, float* d_logits, int32_t* d_next, void* stream);

/* One KV-cached greedy decode step for B sequences (generate loop, Sec.
 * Results; Cache.append in the appendix causal_lm listing).
 *   d_tokens        [B] the newest token of each sequence.
 *   d_context_lens  [B] IN/OUT: tokens already cached for sequence b; the
 *                   new token takes position context_lens[b]. The step adds
 *                   1 to every entry (in stream order, after all reads), so
 *                   consecutive steps can be replayed without host work.
 *   d_block_table   paged layout: [B, ceil(max_context/16)], else NULL.
 *   d_logits        [B, V] fp32 output, or NULL.
 *   d_next          [B] greedy next token; may alias d_tokens.
 * With B <= 8 (16-bit modes, head_dim 64 or 128) the whole step is one
 * cooperative launch with one CTA per SM (the persistent decode step); if
 * the device cannot hold that grid co-resident, or with AXON_NO_PERSIST=1
 * set when the model was created, the step is a chain of 5L+3 kernels,
 * recorded once per (B, pointer set) into a CUDA graph and replayed
 * afterwards (AXON_NO_GRAPH=1: launched directly). Both paths compute the
 * same operations; their fp32 summation orders differ. */
int axon_decode_step(axon_model* m, const int32_t* d_tokens, int32_t B, int32_t* d_context_lens,
                     const int32_t* d_block_table, float* d_logits, int32_t* d_next, void* stream);

/* Forget cached sequences: zero the KV cache and clear the device error
 * word. Synchronous. */
int axon_reset(axon_model* m);

/* Synchronise `stream` and read the device error word. Returns AXON_OK,
 * AXON_ERR_DEVICE_CHECK (a range check fired) or AXON_ERR_TIMEOUT (a
 * bounded wait expired). *bits (optional) receives the raw word; the word
 * is cleared. */
int axon_check_device(axon_model* m, void* stream, int32_t* bits);

/* Read-only view of the KV pools for inspection (tests check cache
 * placement through it). Layout of either pool: [L][num_blocks][G][16][d],
 * element type bf16 (fp32 in AXON_FP32_DEBUG). In the contiguous layout,
 * sequence b's logical block j is pool block b*blocks_per_seq + j. */
typedef struct axon_kv_view {
  void* k_pool;
  void* v_pool;
  int64_t num_blocks;
  int32_t blocks_per_seq;
  int32_t block_size;
  int32_t elem_bytes;
} axon_kv_view;
int axon_kv_view_get(const axon_model* m, axon_kv_view* out);

/* Per-kernel timing of one pass (tracing hook; the paper profiles its
 * generate loop's GPU kernels, appendix "Python Overhead", Table 5).
 * The pass runs exactly as axon_prefill / axon_decode_step would (same
 * kernels, same side effects on the cache and, for decode, on
 * d_context_lens), but launched one kernel at a time with a CUDA event pair
 * around each launch and no CUDA graph or programmatic overlap, then
 * synchronised. Entries aggregate launches of one kind:
 *   name       kernel kind ("decode_gateup", "prefill_qkv", ...)
 *   launches   number of launches in the pass
 *   total_ms   summed event time of those launches
 *   bytes      algorithmic HBM bytes of those launches (weights once, KV
 *              cache reads/writes, activations in/out)
 *   flops      algorithmic floating-point operations
 * `out` receives at most max_out entries (16 suffice); *n_out their count.
 * Prefill logits are not stored (LAST mode, next tokens only). */
typedef struct axon_kernel_time {
  char name[32];
  int32_t launches;
  float total_ms;
  double bytes;
  double flops;
} axon_kernel_time;
int axon_profile_decode_step(axon_model* m, const int32_t* d_tokens, int32_t B, int32_t* d_context_lens,
                             const int32_t* d_block_table, int32_t* d_next, void* stream, axon_kernel_time* out,
                             int32_t max_out, int32_t* n_out);
int axon_profile_prefill(axon_model* m, const int32_t* d_ids, int32_t B, int32_t S, const int32_t* d_block_table,
                         int32_t* d_next, void* stream, axon_kernel_time* out, int32_t max_out, int32_t* n_out);

/* Decode step that allocates nothing (no counterpart in the paper; a
 * deployment affordance of this library). Same arguments, results and
 * side effects as axon_decode_step, for callers that must not allocate on
 * the call path -- for example a serving loop running while another
 * component owns the device memory pool, or a caller whose allocator is
 * locked after start-up: axon_decode_step instantiates a CUDA graph the
 * first time it meets a new (B, pointer set), and instantiation allocates.
 * This entry point instead launches the step's kernels directly, and the
 * split-KV attention takes its merge scratch from a fixed, library-owned
 * device array (256 merge slots, about 2.1 MB, resident on every device
 * that loads the library until the process exits) instead of from memory
 * allocated per call. It calls no cudaMalloc, cudaFree or graph
 * instantiation.
 *   Limits: B * num_key_value_heads <= 256 and head_dim <= 128, else
 *   AXON_ERR_UNSUPPORTED; the 16-bit modes AXON_BF16 and AXON_FP16 only
 *   (AXON_ERR_UNSUPPORTED in AXON_FP32_DEBUG). The attention keeps at most
 *   256 / (B * num_key_value_heads) key splits per sequence and kv head.
 *   First call on a device (and the first after the device's context was
 *   torn down, e.g. by cudaDeviceReset): resolves the array's device address
 *   in the current context, with that device current -- make that first
 *   call before any stream capture.
 *   Every call shares the one array and clears the parts that must start
 *   at zero: calls that overlap on the GPU (different streams, or several
 *   models at once) race on it and must be serialised by the caller.
 * The key-split count may differ from axon_decode_step's, so logits can
 * differ from it by floating-point rounding of the merge. */
int axon_decode_step_noalloc(axon_model* m, const int32_t* d_tokens, int32_t B, int32_t* d_context_lens,
                             const int32_t* d_block_table, float* d_logits, int32_t* d_next, void* stream);

/* Inspection hook for mixture-of-experts models (the routing is decided on
 * the device; tests compare it with the oracle's). With d_experts non-NULL,
 * every later prefill or decode pass writes, for each MoE layer l and each
 * of its first `rows` token rows t (in the pass's row order: b * S + s for
 * axon_prefill, b for axon_decode_step, packed rows for
 * axon_prefill_varlen), the chosen experts in rank order into
 * d_experts[(l * rows + t) * num_experts_per_tok + j] (int32, device
 * memory owned by the caller, L * rows * num_experts_per_tok entries;
 * rows of dense layers are not written). NULL turns recording off.
 * AXON_ERR_UNSUPPORTED for models without experts. Decode graphs recorded
 * before the call are dropped. */
int axon_moe_routing_record(axon_model* m, int32_t* d_experts, int32_t rows);

/* Release everything the model owns. NULL is a no-op. */
void axon_free(axon_model* m);

/* Static string naming a status code. */
const char* axon_status_string(int status);

#ifdef __cplusplus
}
#endif

#endif /* AXON_H */
