// C ABI of the decoder forward: model creation (config validation, weight
// repack, KV cache and workspace), prefill and decode launch plans, and the
// per-(B, pointer set) CUDA-graph cache of the decode step.
//
// The launch plans are the layer loop of the paper's causal_lm listing
// (`for@h i <- [0..NUM_LAYERS) carry (x, work_kv)`), with every block of the
// pre-norm layer turned into one fused kernel:
//   QKV projection (+norm scale, bias, RoPE, KV store) -> attention ->
//   O projection (+residual, next norm's operand) -> gate/up (+SwiGLU) ->
//   down projection (+residual, next norm's operand),
// then final norm + LM head (+argmax) and the greedy-token finaliser.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <map>
#include <string>
#include <tuple>
#include <vector>

#include "../../include/axon.h"
#include "kernels.h"

namespace {

struct LayerW {
  void* wqkv = nullptr;
  float* bqkv = nullptr;
  void* wo = nullptr;
  void* wgu = nullptr;
  void* wd = nullptr;
  float* g1 = nullptr;
  float* g2 = nullptr;
  float* qn = nullptr;  // qk-norm gains [d] (null when off)
  float* kn = nullptr;
  int Fl = 0;  // width of the layer's dense SwiGLU MLP (the shared experts' in a MoE layer; 0: none)
  // mixture of experts: router [E][D]; the experts stacked as one
  // [E * 2Fe][D] gate/up tensor (each expert's rows interleaved in 16-row
  // chunks like the dense one) and one [E * D][Fe] down tensor
  bool moe = false;
  void* router = nullptr;  // [E][D] in the model's 16-bit type (the checkpoint's bf16 values)
  GemmMaps m_router{}, m_router128{};
  void* wgu_e = nullptr;
  void* wd_e = nullptr;
  GemmMaps m_gu_e{}, m_d_e{}, m_gu_e128{}, m_d_e128{};
  GemmMaps m_qkv{}, m_o{}, m_gu{}, m_d{};
  GemmMaps m_qkv128{}, m_o128{}, m_gu128{}, m_d128{};  // the same with 128-row weight boxes
  CUtensorMap v_qkv{}, v_o{}, v_gu{}, v_d{};  // weight maps for the decode projections (box 64 x 128)
};

using GraphKey = std::tuple<int, const void*, const void*, const void*, const void*, const void*>;

bool env_flag(const char* name) {
  const char* v = getenv(name);
  return v && v[0] && v[0] != '0';
}

}  // namespace

struct axon_model {
  axon_config cfg{};
  int L = 0, D = 0, H = 0, G = 0, d = 0, F = 0, V = 0, Nqkv = 0;
  bool fp32 = false;
  bool f16 = false;  // 16-bit operands are fp16 (AXON_FP16) rather than bf16
  size_t esz = 2;
  int device = 0;
  int num_sms = 148;
  // weights
  std::vector<void*> allocs;
  void* embed = nullptr;
  void* head = nullptr;
  float* gf = nullptr;
  std::vector<LayerW> layers;
  GemmMaps m_head{}, m_head128{};
  CUtensorMap v_head{};
  // KV cache
  void* kpool = nullptr;
  void* vpool = nullptr;
  long long num_blocks = 0;
  int blocks_per_seq = 0;
  size_t layer_kv_elems = 0;
  float2* rope = nullptr;
  // workspace
  int Mcap = 0;
  int Pmax = 0;
  float* x = nullptr;
  void* a = nullptr;
  void* a_lo = nullptr;  // fp16 mode: second term of the normed operand (x*g - a), same layout as a
  void* q_lo = nullptr;  // 16-bit modes, decode: second term of q (rows 8..15 of the attention tiles)
  void* o_lo = nullptr;  // fp16 mode, decode: second terms of the attention output and the SwiGLU output
  void* u_lo = nullptr;
  float* ss = nullptr;
  void* q = nullptr;
  void* o = nullptr;
  void* u = nullptr;
  unsigned long long* keys = nullptr;
  float* rinv = nullptr;   // [Mcap] per-row inverse RMS from decode producers
  float* qk_raw = nullptr;  // qk-norm: [Mcap][H + G][d] fp32 q and k before the norm
  // variable-length batches: (sequence, position) per row, and each chunk's
  // last row of a (and a_lo) with its inverse RMS, gathered for the LM head
  int2* rowmap = nullptr;     // [Mcap]
  void* a_last = nullptr;     // [max_batch][D]
  void* a_lo_last = nullptr;  // fp16 mode
  float* rinv_last = nullptr;  // [max_batch]
  SplitKWork splitk{};     // decode projections' cross-CTA split-K workspace
  int* ticket = nullptr;   // last-CTA counter of the residual producers
  float* attn_part = nullptr;
  int* attn_cnt = nullptr;
  int max_splits = 1;
  int* err = nullptr;
  CUtensorMap t_a{}, t_o{}, t_alo{};
  CUtensorMap t_a16{}, t_o16{}, t_alo16{};  // the same in boxes of 16 rows (decode GEMMs)
  CUtensorMap t_a64{}, t_o64{}, t_alo64{};  // and of 64 rows
  // decode graphs
  cudaStream_t cap_stream = nullptr;
  std::map<GraphKey, cudaGraphExec_t> graphs;
  bool use_graphs = true;
  bool use_pdl = true;
  // persistent decode step (B <= PERSIST_MAX_B): device layer table, grid
  // barrier state, CTAs per launch (0: not available)
  PersistLayer* players = nullptr;
  CUtensorMap* pmaps = nullptr;  // [4L + 1] weight maps, box 256 x 16
  PersistGrid* pgrid = nullptr;
  int persist_ctas = 0;
  int decode_gemv_max = 32;  // decode projections with more tokens take the tcgen05 GEMM (AXON_DECODE_GEMV_MAX)
  bool qkv_split = true;     // decode QKV of 9-16 tokens on the split-K GEMM (AXON_QKV_SPLITK=0: the GEMV)
  int persist_split_blocks = 16;  // persistent step: key blocks per split-KV item (AXON_PERSIST_SPLIT_BLOCKS)
  // decode attention grid budget in CTAs (AXON_ATTN_TARGET_CTAS; 0: the
  // split count with the smallest estimated makespan)
  int attn_target_ctas = 0;
  GemmSplitK gemm_sk{};      // split-K workspace of the decode-sized tensor-core GEMMs
  // mixture of experts: routing and sorted-row workspace for up to Mcap
  // tokens (R_cap sorted rows)
  bool moe = false;
  int E = 0, topk = 0, Fe = 0;
  long long R_cap = 0;
  int* moe_topk_idx = nullptr;
  float* moe_topk_w = nullptr;
  int* moe_slot_row = nullptr;
  int* moe_row_tok = nullptr;
  float* moe_row_w = nullptr;
  int* moe_mb_expert = nullptr;
  int* moe_nmb = nullptr;
  float* moe_logits = nullptr;  // [Mcap][E] router logits
  unsigned long long* moe_keys = nullptr;  // [Mcap] argmax keys of the router projection (unused)
  float* moe_ones = nullptr;  // [1] = 1.0: the sorted operand is already normalised
  void* moe_a_sorted = nullptr;
  void* moe_u_sorted = nullptr;
  float* moe_y_sorted = nullptr;
  CUtensorMap t_asorted{}, t_usorted{};
  int32_t* moe_record = nullptr;  // axon_moe_routing_record: [L][record_rows][k], or null
  int moe_record_rows = 0;
};

namespace {

#define CK(call)                                                                    \
  do {                                                                              \
    cudaError_t e_ = (call);                                                        \
    if (e_ != cudaSuccess) {                                                        \
      if (env_flag("AXON_DEBUG"))                                                   \
        fprintf(stderr, "axon: %s failed: %s (%s:%d)\n", #call, cudaGetErrorString(e_), __FILE__, __LINE__); \
      return AXON_ERR_CUDA;                                                         \
    }                                                                               \
  } while (0)

#define CK_RC(expr)        \
  do {                     \
    const int rc_ = (expr); \
    if (rc_) return rc_;    \
  } while (0)

int dev_alloc(axon_model* m, void** p, size_t bytes) {
  if (bytes == 0) bytes = 16;
  if (cudaMalloc(p, bytes) != cudaSuccess) {
    cudaGetLastError();
    *p = nullptr;
    return AXON_ERR_OOM;
  }
  m->allocs.push_back(*p);
  return AXON_OK;
}

// Element types of repacked tensors.
enum : int { DT_BF16 = 0, DT_F32 = 1, DT_F16 = 2 };

// dst[p][:] = src[rowmap[p]][:] with dtype conversion (bf16/f32 -> bf16/f32/f16).
// Values outside the finite fp16 range raise *overflow (fp16 destinations).
__global__ void gather_rows_kernel(void* dst, int dst_dt, const void* src, int src_f32, const int* rowmap,
                                   const int* dstmap, int rows, int cols, int* overflow) {
  const int p0 = blockIdx.x;
  if (p0 >= rows) return;
  const long long sr = rowmap ? rowmap[p0] : p0;
  const int p = dstmap ? dstmap[p0] : p0;
  for (int c = threadIdx.x; c < cols; c += blockDim.x) {
    const float v = src_f32 ? static_cast<const float*>(src)[sr * cols + c]
                            : __bfloat162float(static_cast<const bf16*>(src)[sr * cols + c]);
    const long long o = static_cast<long long>(p) * cols + c;
    if (dst_dt == DT_F32) {
      static_cast<float*>(dst)[o] = v;
    } else if (dst_dt == DT_F16) {
      if (!(fabsf(v) <= 65504.f)) atomicOr(overflow, 1);
      static_cast<f16*>(dst)[o] = __float2half_rn(v);
    } else {
      static_cast<bf16*>(dst)[o] = __float2bfloat16_rn(v);
    }
  }
}

struct Builder {
  axon_model* m;
  const axon_tensor* w;
  int n;
  cudaStream_t st;
  void* staging = nullptr;
  size_t staging_bytes = 0;
  int* d_rowmap = nullptr;
  size_t rowmap_cap = 0;
  int* d_overflow = nullptr;
  int* d_dstmap = nullptr;
  size_t dstmap_cap = 0;

  const axon_tensor* find(const std::string& name) const {
    for (int i = 0; i < n; ++i)
      if (w[i].name && name == w[i].name) return &w[i];
    return nullptr;
  }
  int check(const axon_tensor* t, int64_t d0, int64_t d1) const {
    if (!t) return AXON_ERR_MISSING_WEIGHT;
    if (!t->data || (t->dtype != AXON_DTYPE_BF16 && t->dtype != AXON_DTYPE_F32)) return AXON_ERR_INVALID_ARG;
    if (d1 < 0) {
      if (t->ndim != 1 || t->shape[0] != d0) return AXON_ERR_SHAPE_MISMATCH;
    } else {
      if (t->ndim != 2 || t->shape[0] != d0 || t->shape[1] != d1) return AXON_ERR_SHAPE_MISMATCH;
    }
    return AXON_OK;
  }
  // Copy a checkpoint tensor (host or device) into device staging.
  int stage(const axon_tensor* t, size_t elems) {
    const size_t bytes = elems * (t->dtype == AXON_DTYPE_F32 ? 4 : 2);
    if (bytes > staging_bytes) {
      if (staging) cudaFree(staging);
      staging = nullptr;
      if (cudaMalloc(&staging, bytes) != cudaSuccess) {
        cudaGetLastError();
        return AXON_ERR_OOM;
      }
      staging_bytes = bytes;
    }
    CK(cudaMemcpyAsync(staging, t->data, bytes, cudaMemcpyDefault, st));
    return AXON_OK;
  }
  // dst_f32: fp32 destination; otherwise the model's 16-bit operand type.
  // dstmap (optional): destination row of each gathered row.
  int gather(void* dst, bool dst_f32, const axon_tensor* t, const std::vector<int>* rowmap, int rows, int cols,
             const std::vector<int>* dstmap = nullptr) {
    int rc = stage(t, static_cast<size_t>(t->ndim == 2 ? t->shape[0] : 1) * cols);
    if (rc) return rc;
    if (!d_overflow) {
      if (cudaMalloc(&d_overflow, sizeof(int)) != cudaSuccess) {
        cudaGetLastError();
        return AXON_ERR_OOM;
      }
      CK(cudaMemsetAsync(d_overflow, 0, sizeof(int), st));
    }
    const int* dm = nullptr;
    if (rowmap) {
      if (rowmap->size() > rowmap_cap) {
        if (d_rowmap) cudaFree(d_rowmap);
        if (cudaMalloc(&d_rowmap, rowmap->size() * sizeof(int)) != cudaSuccess) {
          cudaGetLastError();
          return AXON_ERR_OOM;
        }
        rowmap_cap = rowmap->size();
      }
      CK(cudaMemcpyAsync(d_rowmap, rowmap->data(), rowmap->size() * sizeof(int), cudaMemcpyHostToDevice, st));
      dm = d_rowmap;
    }
    const int* ddm = nullptr;
    if (dstmap) {
      if (dstmap->size() > dstmap_cap) {
        if (d_dstmap) cudaFree(d_dstmap);
        if (cudaMalloc(&d_dstmap, dstmap->size() * sizeof(int)) != cudaSuccess) {
          cudaGetLastError();
          return AXON_ERR_OOM;
        }
        dstmap_cap = dstmap->size();
      }
      CK(cudaMemcpyAsync(d_dstmap, dstmap->data(), dstmap->size() * sizeof(int), cudaMemcpyHostToDevice, st));
      ddm = d_dstmap;
    }
    const int dt = dst_f32 ? DT_F32 : (m->f16 ? DT_F16 : DT_BF16);
    gather_rows_kernel<<<rows, 256, 0, st>>>(dst, dt, staging, t->dtype == AXON_DTYPE_F32 ? 1 : 0, dm, ddm, rows,
                                             cols, d_overflow);
    CK(cudaGetLastError());
    // staging and rowmap are reused by the next call
    CK(cudaStreamSynchronize(st));
    int ovf = 0;
    CK(cudaMemcpy(&ovf, d_overflow, sizeof(int), cudaMemcpyDeviceToHost));
    return ovf ? AXON_ERR_UNSUPPORTED : AXON_OK;
  }
  ~Builder() {
    if (staging) cudaFree(staging);
    if (d_rowmap) cudaFree(d_rowmap);
    if (d_overflow) cudaFree(d_overflow);
    if (d_dstmap) cudaFree(d_dstmap);
  }
};

int validate_config(const axon_config* c) {
  if (c->num_hidden_layers < 0 || c->hidden_size <= 0 || c->num_attention_heads <= 0 ||
      c->num_key_value_heads <= 0 || c->intermediate_size <= 0 || c->vocab_size <= 0 || c->max_batch <= 0 ||
      c->max_context <= 0)
    return AXON_ERR_INVALID_ARG;
  if (c->kv_layout != AXON_KV_CONTIGUOUS && c->kv_layout != AXON_KV_PAGED) return AXON_ERR_INVALID_ARG;
  if (c->precision != AXON_BF16 && c->precision != AXON_FP32_DEBUG && c->precision != AXON_FP16)
    return AXON_ERR_INVALID_ARG;
  if (c->kv_block_size != 16) return AXON_ERR_UNSUPPORTED;
  if (c->sliding_window < 0) return AXON_ERR_INVALID_ARG;
  if (c->rope_scaling_factor < 0.f) return AXON_ERR_INVALID_ARG;
  if (c->hidden_act != AXON_ACT_SILU && c->hidden_act != AXON_ACT_GELU_TANH) return AXON_ERR_INVALID_ARG;
  if (c->qk_norm != 0 && c->qk_norm != 1) return AXON_ERR_INVALID_ARG;
  if (c->n_routed_experts < 0 || c->n_shared_experts < 0 || c->first_k_dense_replace < 0 ||
      (c->norm_topk_prob != 0 && c->norm_topk_prob != 1))
    return AXON_ERR_INVALID_ARG;
  if (c->n_routed_experts > 0) {
    if (c->num_experts_per_tok < 1 || c->num_experts_per_tok > 8 || c->num_experts_per_tok > c->n_routed_experts ||
        c->moe_intermediate_size <= 0 || c->first_k_dense_replace > c->num_hidden_layers)
      return AXON_ERR_INVALID_ARG;
    if (c->n_routed_experts > MOE_MAX_EXPERTS || c->moe_intermediate_size % 64 || c->hidden_size % 128 ||
        c->precision == AXON_FP32_DEBUG)
      return AXON_ERR_UNSUPPORTED;
  }
  if (c->rope_scaling_factor > 0.f &&
      (c->rope_original_max_position <= 0 || c->rope_low_freq_factor <= 0.f ||
       c->rope_high_freq_factor <= c->rope_low_freq_factor))
    return AXON_ERR_INVALID_ARG;
  if (c->kv_layout == AXON_KV_PAGED && c->kv_num_blocks <= 0) return AXON_ERR_INVALID_ARG;
  if (c->num_attention_heads % c->num_key_value_heads) return AXON_ERR_UNSUPPORTED;
  if (c->num_attention_heads / c->num_key_value_heads > 16) return AXON_ERR_UNSUPPORTED;
  if (c->head_dim != 64 && c->head_dim != 128) return AXON_ERR_UNSUPPORTED;
  if (c->hidden_size % 64 || c->intermediate_size % 64 || (c->num_attention_heads * c->head_dim) % 64)
    return AXON_ERR_UNSUPPORTED;
  if (c->max_context % 16) return AXON_ERR_UNSUPPORTED;
  if (c->max_batch > 64 && c->max_prefill_tokens == 0) return AXON_ERR_UNSUPPORTED;
  return AXON_OK;
}

// Packed row p of one head (QKV): chunk c = p / 16 holds natural dims
// c*8 + i (slots 0..7) and c*8 + i + d/2 (slots 8..15).
int qkv_natural(int p, int d) {
  const int c = p >> 4, i = p & 15;
  return i < 8 ? c * 8 + i : c * 8 + (i - 8) + d / 2;
}

void kv_layout_args(const axon_model* m, int layer, const int* block_table, EpiArgs& e) {
  e.k_cache = static_cast<char*>(m->kpool) + static_cast<size_t>(layer) * m->layer_kv_elems * m->esz;
  e.v_cache = static_cast<char*>(m->vpool) + static_cast<size_t>(layer) * m->layer_kv_elems * m->esz;
  e.block_table = block_table;
  e.bt_stride = m->blocks_per_seq;
  e.blocks_per_seq = m->blocks_per_seq;
  e.num_blocks = static_cast<int>(m->num_blocks);
}

EpiArgs base_epi(const axon_model* m) {
  EpiArgs e;
  memset(&e, 0, sizeof(e));
  e.max_pos = m->cfg.max_context;
  e.inv_D = 1.0f / static_cast<float>(m->D);
  e.eps = m->cfg.rms_norm_eps;
  e.act = m->cfg.hidden_act;
  e.H = m->H;
  e.G = m->G;
  e.d = m->d;
  e.rope = m->rope;
  e.err = m->err;
  return e;
}

AttnArgs base_attn(const axon_model* m, int layer, const int* block_table) {
  AttnArgs a;
  memset(&a, 0, sizeof(a));
  a.q = m->q;
  a.o = m->o;
  a.k = static_cast<char*>(m->kpool) + static_cast<size_t>(layer) * m->layer_kv_elems * m->esz;
  a.v = static_cast<char*>(m->vpool) + static_cast<size_t>(layer) * m->layer_kv_elems * m->esz;
  a.block_table = block_table;
  a.bt_stride = m->blocks_per_seq;
  a.blocks_per_seq = m->blocks_per_seq;
  a.num_blocks = static_cast<int>(m->num_blocks);
  a.H = m->H;
  a.G = m->G;
  a.d = m->d;
  a.scale_log2 = static_cast<float>(1.0 / std::sqrt(static_cast<double>(m->d)) * 1.4426950408889634);
  a.window = m->cfg.sliding_window;
  a.err = m->err;
  return a;
}

// qk-norm inputs of a QKV epilogue (left null when the model has none).
void set_qk_norm(const axon_model* m, const LayerW& w, EpiArgs& e) {
  if (!m->cfg.qk_norm) return;
  e.qk_raw = m->qk_raw;
  e.qn_gain = w.qn;
  e.kn_gain = w.kn;
}

// Which form the next norm's scale is available in after a producer: the
// reduced per-row inverse RMS (`rinv` buffer) or `parts` partial sums of
// squares per row in `ss`.
struct NormState {
  bool rinv = false;
  int parts = 1;
};

void set_norm(const axon_model* m, const NormState& ns, EpiArgs& e, int row_offset = 0, int row_stride = 1) {
  if (ns.rinv) {
    e.rinv = m->rinv + row_offset;
    e.rinv_stride = row_stride;
  } else {
    e.ss = m->ss + static_cast<size_t>(row_offset) * m->Pmax;
    e.ss_stride = row_stride * m->Pmax;
    e.ss_parts = ns.parts;
  }
}

// Optional per-launch timing (axon_profile_*): an event pair around every
// kernel, with the launch's algorithmic bytes and FLOPs.
struct Prof {
  struct Entry {
    std::string name;
    cudaEvent_t a, b;
    double bytes, flops;
  };
  cudaStream_t st;
  std::vector<Entry> entries;
  void begin(const char* name) {
    Entry e{name, nullptr, nullptr, 0, 0};
    cudaEventCreate(&e.a);
    cudaEventCreate(&e.b);
    cudaEventRecord(e.a, st);
    entries.push_back(e);
  }
  void end(double bytes, double flops) {
    Entry& e = entries.back();
    cudaEventRecord(e.b, st);
    e.bytes = bytes;
    e.flops = flops;
  }
  ~Prof() {
    for (auto& e : entries) {
      cudaEventDestroy(e.a);
      cudaEventDestroy(e.b);
    }
  }
};
// AXON_TRACE=1: name every launch on stderr and wait for it (debugging aid;
// ignored while a stream is being captured).
bool g_trace = false;
cudaStream_t g_trace_stream = nullptr;
const char* g_trace_name = "";
inline void pbeg(Prof* p, const char* n) {
  if (p) p->begin(n);
  if (g_trace) {
    g_trace_name = n;
    fprintf(stderr, "axon: launch %s\n", n);
    fflush(stderr);
  }
}
inline void pend(Prof* p, double bytes, double flops) {
  if (p) p->end(bytes, flops);
  if (g_trace && g_trace_stream) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    cudaStreamIsCapturing(g_trace_stream, &cs);
    if (cs == cudaStreamCaptureStatusNone) {
      const cudaError_t e = cudaStreamSynchronize(g_trace_stream);
      fprintf(stderr, "axon: done %s (%s)\n", g_trace_name, cudaGetErrorString(e));
      fflush(stderr);
    }
  }
}

// One projection: picks the kernel for the mode and row count.
struct Proj {
  const axon_model* m;
  LaunchCtx lc;
  bool decode = false;  // o_lo / u_lo were written by this step's producers
  int gemv_max = 64;    // rows up to which the register-streaming GEMV runs (else the tcgen05 GEMM)
  cudaError_t rc = cudaSuccess;
  // act: activation rows (row stride act_stride elements), M rows. Returns
  // the norm state a RESID producer leaves behind.
  NormState run(int kind, const void* W, const GemmMaps* maps, int N, int K, const void* act, long long act_stride,
                int M, EpiArgs& ep) {
    ep.M = M;
    ep.N = N;
    NormState ns;
    // Decode (gemv_max < 64) above 8 tokens, measured choices:
    //  * the tcgen05 GEMM where its 128-wide tiles cover every SM (gate/up,
    //    LM head);
    //  * the residual projections (O, down) on the split-K GEMM where the
    //    parts stay cheap to sum: a long K (>= 8192) or at most 16 tokens;
    //    QKV too at most 16 tokens (qkv_split);
    //  * otherwise the GEMV up to gemv_max tokens, the plain GEMM above.
    const bool dec = gemv_max < 64 && maps != nullptr && !m->fp32 && M > 8;
    const bool wide = dec && static_cast<long long>((N + 127) / 128) * ((M + 127) / 128) >= m->num_sms;
    const bool split_kind =
        (kind == EPI_RESID && (K >= 8192 || M <= 16)) || (kind == EPI_QKV && m->qkv_split && M <= 16);
    const bool resid_split =
        dec && !wide && split_kind && gemm_split_k(lc, M, N, K) > 1 && m->gemm_sk.ws != nullptr;
    const bool gemv = (M <= gemv_max && !wide && !resid_split) || (!m->fp32 && maps == nullptr);
    if (gemv && kind == EPI_RESID) {
      ep.rinv_out = m->rinv;
      ep.ticket = m->ticket;
      ns.rinv = true;
    }
    if (gemv) {
      // fp16 mode: consumers of the normed operand `a` also read its
      // second term a_lo
      const void* lo = nullptr;
      if (m->f16) {
        if (act == m->a) lo = m->a_lo;
        else if (decode && act == m->o) lo = m->o_lo;
        else if (decode && act == m->u) lo = m->u_lo;
      }
      rc = launch_gemv(lc, kind, m->fp32, W, N, K, act, act_stride, M, ep, m->splitk, lo);
      ns.parts = N / 16;
    } else if (m->fp32) {
      rc = launch_gemm_simt(lc, kind, static_cast<const float*>(act), act_stride, static_cast<const float*>(W), M, N,
                            K, ep);
      ns.parts = N / 16;
    } else {
      int tn = gemm_tile_n(lc, *maps, M, N);
      GemmSplitK sk = m->gemm_sk;
      sk.ks = resid_split ? gemm_split_k(lc, M, N, K) : 1;
      if (sk.ks > 1) tn = 256;
      rc = launch_gemm_tc(lc, kind, *maps, M, N, K, ep, tn, &sk);
      ns.parts = (N + tn - 1) / tn;
    }
    return ns;
  }
};

// Expected number of distinct experts that T tokens route to when each
// picks k of E experts uniformly: E * (1 - (1 - k/E)^T). The algorithmic
// expert-weight bytes of a mixture-of-experts step (the routing itself is
// known only on the device).
double expected_active_experts(int E, int k, int T) {
  return E * (1.0 - std::pow(1.0 - static_cast<double>(k) / E, static_cast<double>(T)));
}

MoeArgs moe_args(const axon_model* m, const LayerW& w) {
  MoeArgs a;
  memset(&a, 0, sizeof(a));
  a.D = m->D;
  a.E = m->E;
  a.k = m->topk;
  a.norm_topk = m->cfg.norm_topk_prob;
  a.act = m->a;
  a.act_lo = m->a_lo;
  a.act_stride = m->D;
  a.logits = m->moe_logits;
  a.topk_idx = m->moe_topk_idx;
  a.topk_w = m->moe_topk_w;
  a.slot_row = m->moe_slot_row;
  a.row_tok = m->moe_row_tok;
  a.row_w = m->moe_row_w;
  a.mb_expert = m->moe_mb_expert;
  a.n_mblocks = m->moe_nmb;
  a.a_sorted = m->moe_a_sorted;
  a.y_sorted = m->moe_y_sorted;
  a.err = m->err;
  return a;
}

// The MLP half of layer l, after the O projection left the operand
// a = x * g2 with norm state ns: the dense SwiGLU MLP, or the mixture of
// experts -- routing, the stable sort into expert segments, the grouped
// expert GEMMs (gate/up + SwiGLU, down scaled by the routing weight), the
// combine into the residual -- followed by the shared experts' MLP when the
// layer has one. `row` carries the row -> (sequence, position) map of the
// pass (S, rowmap or ctx); `decode` selects the decode projections' second
// SwiGLU term and the profiler names. Updates ns to the next operand's
// norm state.
int enqueue_mlp(axon_model* m, int l, Proj& pj, const LaunchCtx& lc, Prof* pf, const EpiArgs& row, int M,
                bool decode, NormState& ns) {
  const LayerW& w = m->layers[l];
  const int D = m->D;
  const double es = static_cast<double>(m->esz);
  const float* gnext = (l + 1 < m->L) ? m->layers[l + 1].g1 : m->gf;
  if (w.moe) {
    const int E = m->E, k = m->topk, Fe = m->Fe;
    const int R = static_cast<int>(m->R_cap);
    const double act = expected_active_experts(E, k, M);
    // router logits [M][E] on the projection kernels (norm scale applied)
    EpiArgs rl = row;
    set_norm(m, ns, rl);
    rl.logits = m->moe_logits;
    rl.logits_stride = E;
    rl.keys = m->moe_keys;
    pbeg(pf, decode ? "decode_moe_router" : "prefill_moe_router");
    pj.run(EPI_LOGITS, w.router, &w.m_router, E, D, m->a, D, M, rl);
    CK(pj.rc);
    pend(pf, static_cast<double>(E) * D * es + M * (D * es + E * 4.0), 2.0 * M * E * D);
    MoeArgs ma = moe_args(m, w);
    if (m->moe_record) {
      ma.record = m->moe_record + static_cast<size_t>(l) * m->moe_record_rows * k;
      ma.record_rows = m->moe_record_rows;
    }
    EpiArgs nx = base_epi(m);
    set_norm(m, ns, nx);
    pbeg(pf, decode ? "decode_moe_route" : "prefill_moe_route");
    CK(launch_moe_route_plan(lc, ma, M));
    CK(launch_moe_gather(lc, ma, M, nx));
    pend(pf, M * (E * 4.0 + D * (2 * es + es * k)), 0);
    // tile width: 128 when the experts' blocks alone leave most SMs idle
    const int tn = (static_cast<long long>(M) * k * ((D + 255) / 256) < m->num_sms) ? 128 : 256;
    GemmGroup grp;
    grp.mb_expert = m->moe_mb_expert;
    grp.n_mblocks = m->moe_nmb;
    grp.row_valid = m->moe_row_tok;
    EpiArgs g = base_epi(m);
    g.M = R;
    g.N = 2 * Fe;
    g.u_out = m->moe_u_sorted;
    g.rinv = m->moe_ones;  // the sorted rows are normalised already
    g.rinv_stride = 0;
    pbeg(pf, decode ? "decode_moe_gateup" : "prefill_moe_gateup");
    CK(launch_gemm_tc(lc, EPI_SWIGLU, w.m_gu_e, R, 2 * Fe, D, g, tn, nullptr, &grp));
    pend(pf, act * 2.0 * Fe * D * es + M * k * (D + Fe) * es, 2.0 * M * k * 2 * Fe * D);
    EpiArgs dn = base_epi(m);
    dn.M = R;
    dn.N = D;
    dn.y_out = m->moe_y_sorted;
    dn.row_w = m->moe_row_w;
    pbeg(pf, decode ? "decode_moe_down" : "prefill_moe_down");
    CK(launch_gemm_tc(lc, EPI_ROWSCALE, w.m_d_e, R, D, Fe, dn, tn, nullptr, &grp));
    pend(pf, act * static_cast<double>(D) * Fe * es + M * k * (Fe * es + D * 4.0), 2.0 * M * k * D * Fe);
    EpiArgs cb = base_epi(m);
    cb.M = M;
    cb.N = D;
    cb.x = m->x;
    if (!w.Fl) {  // no shared experts: the combine is the layer's residual producer
      cb.a_out = m->a;
      cb.a_lo_out = m->a_lo;
      cb.gain = gnext;
      cb.ss_out = m->ss;
      cb.ss_out_stride = m->Pmax;
    }
    pbeg(pf, decode ? "decode_moe_combine" : "prefill_moe_combine");
    CK(launch_moe_combine(lc, ma, M, cb));
    pend(pf, M * (k * D * 4.0 + D * (8.0 + (w.Fl ? 0 : es))), 0);
    if (!w.Fl) {
      ns.rinv = false;
      ns.parts = D / 16;
      return AXON_OK;
    }
  }
  const int Fl = w.Fl;
  EpiArgs g = row;
  set_norm(m, ns, g);
  g.u_out = m->u;
  if (decode) g.u_lo_out = m->u_lo;
  pbeg(pf, decode ? "decode_gateup" : "prefill_gateup");
  pj.run(EPI_SWIGLU, w.wgu, &w.m_gu, 2 * Fl, D, m->a, D, M, g);
  CK(pj.rc);
  pend(pf, 2.0 * Fl * D * es + M * (D + Fl) * es, 2.0 * M * 2 * Fl * D);

  EpiArgs dn = row;
  dn.x = m->x;
  dn.a_out = m->a;
  dn.gain = gnext;
  dn.a_lo_out = m->a_lo;
  dn.ss_out = m->ss;
  dn.ss_out_stride = m->Pmax;
  pbeg(pf, decode ? "decode_down" : "prefill_down");
  ns = pj.run(EPI_RESID, w.wd, &w.m_d, D, Fl, m->u, Fl, M, dn);
  CK(pj.rc);
  pend(pf, static_cast<double>(D) * Fl * es + M * (Fl * es + D * (8 + es)), 2.0 * M * D * Fl);
  return AXON_OK;
}

// A variable-length batch (axon_prefill_varlen): sequence b's chunk is rows
// cu[b] .. cu[b+1]-1 of the T packed rows, after ctx[b] cached tokens; ctx is
// advanced by the chunk lengths at the end.
struct VarlenBatch {
  const int* cu;
  int* ctx;
  int T;
  int max_chunk;
};

int enqueue_prefill(axon_model* m, const int32_t* ids, int B, int S, const int32_t* bt, int logits_mode, float* logits,
                    int32_t* next, cudaStream_t st, Prof* pf = nullptr, const VarlenBatch* vl = nullptr) {
  const int M = vl ? vl->T : B * S;
  LaunchCtx lc{st, m->use_pdl && !pf, m->num_sms, m->f16};
  const int2* rowmap = vl ? m->rowmap : nullptr;
  if (vl) CK(launch_varlen_rows(lc, vl->cu, vl->ctx, B, M, vl->max_chunk, m->cfg.max_context, m->rowmap, m->err));
  g_trace_stream = st;
  const double es = static_cast<double>(m->esz);
  const double wq = static_cast<double>(m->Nqkv) * m->D * es, wo = static_cast<double>(m->D) * m->H * m->d * es,
               whd = static_cast<double>(m->V) * m->D * es;
  Proj pj{m, lc};
  const int D = m->D, Hd = m->H * m->d;
  pbeg(pf, "embed");
  CK(launch_embed(lc, m->fp32, m->embed, m->V, D, ids, M, m->x, m->a, m->L > 0 ? m->layers[0].g1 : m->gf, m->ss,
                  m->Pmax, m->rinv, m->cfg.rms_norm_eps, m->err, m->a_lo));
  pend(pf, static_cast<double>(M) * D * (es + 4 + es), 0);
  NormState ns;
  ns.rinv = true;
  for (int l = 0; l < m->L; ++l) {
    const LayerW& w = m->layers[l];
    EpiArgs e = base_epi(m);
    e.S = S;
    e.rowmap = rowmap;
    set_norm(m, ns, e);
    e.bias = w.bqkv;
    e.q_out = m->q;
    kv_layout_args(m, l, bt, e);
    set_qk_norm(m, w, e);
    pbeg(pf, "prefill_qkv");
    pj.run(EPI_QKV, w.wqkv, &w.m_qkv, m->Nqkv, D, m->a, D, M, e);
    CK(pj.rc);
    pend(pf, wq + M * (D + m->Nqkv) * es, 2.0 * M * m->Nqkv * D);
    if (e.qk_raw) {
      pbeg(pf, "prefill_qk_norm");
      CK(launch_qk_norm_rope(lc, m->fp32, e, M));
      pend(pf, static_cast<double>(M) * (m->H + m->G) * m->d * (4 + es), 0);
    }

    AttnArgs at = base_attn(m, l, bt);
    at.S = vl ? vl->max_chunk : S;
    const AttnVarlen avl{vl ? vl->cu : nullptr, vl ? vl->ctx : nullptr, M, rowmap};
    pbeg(pf, "prefill_attention");
    CK(launch_attn_prefill(lc, m->fp32, at, B, vl ? &avl : nullptr));
    pend(pf, static_cast<double>(M) * (m->H + 2 * m->G) * m->d * es + static_cast<double>(M) * Hd * es,
         4.0 * B * m->H * m->d * (static_cast<double>(S) * (S + 1) / 2));

    EpiArgs r = base_epi(m);
    r.S = S;
    r.rowmap = rowmap;
    r.x = m->x;
    r.a_out = m->a;
    r.gain = w.g2;
    r.a_lo_out = m->a_lo;
    r.ss_out = m->ss;
    r.ss_out_stride = m->Pmax;
    pbeg(pf, "prefill_o");
    ns = pj.run(EPI_RESID, w.wo, &w.m_o, D, Hd, m->o, Hd, M, r);
    CK(pj.rc);
    pend(pf, wo + M * (Hd * es + D * (8 + es)), 2.0 * M * D * Hd);

    EpiArgs row = base_epi(m);
    row.S = S;
    row.rowmap = rowmap;
    CK_RC(enqueue_mlp(m, l, pj, lc, pf, row, M, false, ns));
  }
  EpiArgs h = base_epi(m);
  h.S = S;
  h.rowmap = rowmap;
  h.keys = m->keys;
  h.logits = logits;
  h.logits_stride = m->V;
  if (vl && logits_mode == AXON_LOGITS_ALL) {
    set_norm(m, ns, h);
    pj.run(EPI_LOGITS, m->head, &m->m_head, m->V, D, m->a, D, M, h);
    CK(pj.rc);
    CK(launch_finalize_varlen(lc, m->keys, M, vl->cu, 1, B, next, vl->ctx));
  } else if (vl) {
    // Last row of every chunk, gathered into B dense rows, then a GEMV of at
    // most 64 rows at a time over the LM head.
    const float* rv = ns.rinv ? m->rinv : nullptr;
    CK(launch_gather_last(lc, vl->cu, B, M, m->a, m->a_lo, D * static_cast<int>(m->esz), rv, m->ss, m->Pmax,
                          ns.parts, 1.0f / static_cast<float>(D), m->cfg.rms_norm_eps, m->a_last, m->a_lo_last,
                          m->rinv_last));
    for (int b0 = 0; b0 < B; b0 += 64) {
      const int nb = std::min(64, B - b0);
      EpiArgs hg = h;
      hg.rowmap = nullptr;
      hg.rinv = m->rinv_last + b0;
      hg.rinv_stride = 1;
      hg.M = nb;
      hg.N = m->V;
      hg.keys = m->keys + b0;
      hg.logits = logits ? logits + static_cast<size_t>(b0) * m->V : nullptr;
      const size_t off = static_cast<size_t>(b0) * D * m->esz;
      CK(launch_gemv(lc, EPI_LOGITS, m->fp32, m->head, m->V, D, static_cast<char*>(m->a_last) + off, D, nb, hg,
                     m->splitk, m->a_lo_last ? static_cast<char*>(m->a_lo_last) + off : nullptr));
    }
    CK(launch_finalize_varlen(lc, m->keys, B, vl->cu, 0, B, next, vl->ctx));
  } else if (logits_mode == AXON_LOGITS_ALL) {
    set_norm(m, ns, h);
    pbeg(pf, "prefill_lm_head");
    pj.run(EPI_LOGITS, m->head, &m->m_head, m->V, D, m->a, D, M, h);
    CK(pj.rc);
    pend(pf, whd + M * (D * es + (logits ? 4.0 * m->V : 0.0)), 2.0 * M * m->V * D);
    pbeg(pf, "finalize");
    CK(launch_finalize(lc, m->keys, M, S, S - 1, B, next, nullptr));
    pend(pf, 8.0 * M, 0);
  } else {
    // Last position of each sequence: rows S-1, 2S-1, ... as a B-row GEMV.
    const size_t off = static_cast<size_t>(S - 1) * D * m->esz;
    set_norm(m, ns, h, S - 1, S);
    h.M = B;
    h.N = m->V;
    pbeg(pf, "prefill_lm_head");
    CK(launch_gemv(lc, EPI_LOGITS, m->fp32, m->head, m->V, D, static_cast<char*>(m->a) + off,
                   static_cast<long long>(S) * D, B, h, m->splitk,
                   m->a_lo ? static_cast<char*>(m->a_lo) + off : nullptr));
    pend(pf, whd + B * (D * es + (logits ? 4.0 * m->V : 0.0)), 2.0 * B * m->V * D);
    pbeg(pf, "finalize");
    CK(launch_finalize(lc, m->keys, B, 1, 0, B, next, nullptr));
    pend(pf, 8.0 * B, 0);
  }
  return AXON_OK;
}

// The persistent step's attention always pairs q's two terms in one MMA
// tile, which needs at most 8 query heads per kv head; qk-norm needs a
// kernel of its own between QKV and attention and mixture-of-experts layers
// their routing kernels, so those models decode on the launch chain.
bool persist_eligible(const axon_model* m, int B) {
  return m->persist_ctas > 0 && !m->fp32 && !m->cfg.qk_norm && !m->moe && m->H / m->G <= 8 &&
         persist_fits(m->d, m->f16, B, m->D, std::max(std::max(m->D, m->H * m->d), m->F));
}

PersistArgs persist_args(const axon_model* m, const int32_t* tokens, int B, int32_t* ctx, const int32_t* bt,
                         float* logits, int32_t* next, int splits, float* attn_part, int* attn_cnt) {
  PersistArgs a;
  memset(&a, 0, sizeof(a));
  a.L = m->L;
  a.D = m->D;
  a.H = m->H;
  a.G = m->G;
  a.d = m->d;
  a.F = m->F;
  a.V = m->V;
  a.Nqkv = m->Nqkv;
  a.Pmax = m->Pmax;
  a.B = B;
  a.max_pos = m->cfg.max_context;
  a.blocks_per_seq = m->blocks_per_seq;
  a.num_blocks = static_cast<int>(m->num_blocks);
  a.splits = splits;
  a.window = m->cfg.sliding_window;
  a.eps = m->cfg.rms_norm_eps;
  a.act = m->cfg.hidden_act;
  a.inv_D = 1.0f / static_cast<float>(m->D);
  a.scale_log2 = static_cast<float>(1.0 / std::sqrt(static_cast<double>(m->d)) * 1.4426950408889634);
  a.layers = m->players;
  a.wmaps = m->pmaps;
  a.embed = m->embed;
  a.head = m->head;
  a.gf = m->gf;
  a.rope = m->rope;
  a.x = m->x;
  a.a = m->a;
  a.a_lo = m->a_lo;
  a.ss = m->ss;
  a.q = m->q;
  a.q_lo = m->q_lo;
  a.o = m->o;
  a.u = m->u;
  a.o_lo = m->o_lo;
  a.u_lo = m->u_lo;
  a.keys = m->keys;
  a.attn_part = attn_part;
  a.attn_cnt = attn_cnt;
  a.err = m->err;
  a.grid = m->pgrid;
  a.tokens = tokens;
  a.ctx = ctx;
  a.block_table = bt;
  a.logits = logits;
  a.next = next;
  return a;
}

int enqueue_decode(axon_model* m, const int32_t* tokens, int B, int32_t* ctx, const int32_t* bt, float* logits,
                   int32_t* next, cudaStream_t st, Prof* pf = nullptr, double kv_tokens = 0,
                   float* attn_part = nullptr, int* attn_cnt = nullptr, int attn_rows_cap = 0) {
  LaunchCtx lc{st, m->use_pdl && !pf, m->num_sms, m->f16};
  g_trace_stream = st;
  Proj pj{m, lc};
  pj.decode = true;
  // Above 32 tokens the GEMV's per-CTA re-reads of every activation row from
  // L2 cost more than the weights; the tensor-core GEMM takes the 33..64
  // tokens as one M tile and streams each weight tile once through TMA.
  pj.gemv_max = m->decode_gemv_max;
  const int D = m->D, Hd = m->H * m->d;
  const double es = static_cast<double>(m->esz);
  const double wq = static_cast<double>(m->Nqkv) * m->D * es, wo = static_cast<double>(m->D) * Hd * es,
               wgu = 2.0 * m->F * m->D * es, wdn = static_cast<double>(m->D) * m->F * es,
               whd = static_cast<double>(m->V) * m->D * es;
  // merge slots per (sequence, kv head): the model's partial buffer, or the
  // caller-supplied scratch of attn_rows_cap (sequence, kv head, split) slots
  int cap = m->max_splits;
  if (attn_rows_cap > 0) {
    const int c = attn_rows_cap / (B * m->G);
    cap = c < 1 ? 1 : (c < cap ? c : cap);
  }
  int splits = m->fp32 ? 1 : attn_decode_splits(B, m->G, m->blocks_per_seq, m->num_sms, m->attn_target_ctas);
  if (splits > cap) splits = cap;
  if (persist_eligible(m, B)) {
    // Inside one launch a cross-CTA merge costs more than it saves up to 64
    // key blocks (8 per warp; measured at 40 blocks, head_dim 64: 0.743 ms
    // per step unsplit, 0.775-0.790 ms split). Beyond that the keys split
    // into items of persist_split_blocks blocks (80 blocks, head_dim 128:
    // 3.170 ms per step in items of 16, 3.239 ms in items of 64). Head_dim
    // 128 stages one block per warp: items of 8 blocks, one round.
    const int sblocks = m->d == 128 ? 8 : m->persist_split_blocks;
    int psplits = (m->blocks_per_seq > 64 || sblocks == 8) ? (m->blocks_per_seq + sblocks - 1) / sblocks : 1;
    if (psplits > cap) psplits = cap;
    PersistArgs pa = persist_args(m, tokens, B, ctx, bt, logits, next, psplits, attn_part ? attn_part : m->attn_part,
                                  attn_cnt ? attn_cnt : m->attn_cnt);
    pbeg(pf, "decode_persistent");
    const cudaError_t pe = launch_persist_decode(pa, m->d, m->f16, m->persist_ctas, st);
    if (pe == cudaErrorCooperativeLaunchTooLarge) {
      // not every SM is free for a co-resident grid: take the launch chain
      cudaGetLastError();
      if (pf) {
        cudaEventDestroy(pf->entries.back().a);
        cudaEventDestroy(pf->entries.back().b);
        pf->entries.pop_back();
      }
      goto launch_chain;
    }
    CK(pe);
    const double kvb = kv_tokens * 2.0 * m->G * m->d * es * m->L;
    pend(pf, m->L * (wq + wo + wgu + wdn) + whd + kvb + B * (logits ? 4.0 * m->V : 0.0),
         2.0 * B * (m->L * (static_cast<double>(m->Nqkv) * D + static_cast<double>(D) * Hd + 3.0 * m->F * D) +
                    static_cast<double>(m->V) * D) +
             4.0 * kv_tokens * m->H * m->d * m->L);
    return AXON_OK;
  }
launch_chain:
  pbeg(pf, "embed");
  CK(launch_embed(lc, m->fp32, m->embed, m->V, D, tokens, B, m->x, m->a, m->L > 0 ? m->layers[0].g1 : m->gf, m->ss,
                  m->Pmax, m->rinv, m->cfg.rms_norm_eps, m->err, m->a_lo));
  pend(pf, static_cast<double>(B) * D * (es + 4 + es), 0);
  NormState ns;
  ns.rinv = true;
  for (int l = 0; l < m->L; ++l) {
    const LayerW& w = m->layers[l];
    EpiArgs e = base_epi(m);
    e.S = 1;
    e.ctx = ctx;
    set_norm(m, ns, e);
    e.bias = w.bqkv;
    e.q_out = m->q;
    e.q_lo_out = m->q_lo;
    kv_layout_args(m, l, bt, e);
    set_qk_norm(m, w, e);
    pbeg(pf, "decode_qkv");
    pj.run(EPI_QKV, w.wqkv, &w.m_qkv, m->Nqkv, D, m->a, D, B, e);
    CK(pj.rc);
    pend(pf, wq + B * (D + m->Nqkv) * es, 2.0 * B * m->Nqkv * D);
    if (e.qk_raw) {
      pbeg(pf, "decode_qk_norm");
      CK(launch_qk_norm_rope(lc, m->fp32, e, B));
      pend(pf, static_cast<double>(B) * (m->H + m->G) * m->d * (4 + es), 0);
    }

    AttnArgs at = base_attn(m, l, bt);
    at.ctx = ctx;
    at.S = 1;
    at.splits = splits;
    at.part = attn_part ? attn_part : m->attn_part;
    at.counter = attn_cnt ? attn_cnt : m->attn_cnt;
    at.o_lo = m->o_lo;
    at.q_lo = m->q_lo;
    pbeg(pf, "decode_attention");
    CK(launch_attn_decode(lc, m->fp32, at, B));
    pend(pf, kv_tokens * 2.0 * m->G * m->d * es + 2.0 * B * Hd * es, 4.0 * kv_tokens * m->H * m->d);

    EpiArgs r = base_epi(m);
    r.S = 1;
    r.ctx = ctx;
    r.x = m->x;
    r.a_out = m->a;
    r.gain = w.g2;
    r.a_lo_out = m->a_lo;
    r.ss_out = m->ss;
    r.ss_out_stride = m->Pmax;
    pbeg(pf, "decode_o");
    ns = pj.run(EPI_RESID, w.wo, &w.m_o, D, Hd, m->o, Hd, B, r);
    CK(pj.rc);
    pend(pf, wo + B * (Hd * es + D * (8 + es)), 2.0 * B * D * Hd);

    EpiArgs row = base_epi(m);
    row.S = 1;
    row.ctx = ctx;
    CK_RC(enqueue_mlp(m, l, pj, lc, pf, row, B, true, ns));
  }
  EpiArgs h = base_epi(m);
  h.S = 1;
  h.ctx = ctx;
  set_norm(m, ns, h);
  h.keys = m->keys;
  h.logits = logits;
  h.logits_stride = m->V;
  pbeg(pf, "decode_lm_head");
  pj.run(EPI_LOGITS, m->head, &m->m_head, m->V, D, m->a, D, B, h);
  CK(pj.rc);
  pend(pf, whd + B * (D * es + (logits ? 4.0 * m->V : 0.0)), 2.0 * B * m->V * D);
  pbeg(pf, "finalize");
  CK(launch_finalize(lc, m->keys, B, 1, 0, B, next, ctx));
  pend(pf, 16.0 * B, 0);
  return AXON_OK;
}

}  // namespace

// Direct-launch decode step with caller-supplied attention merge scratch
// (used by the allocation-free entry point in noalloc.cu). Not exported.
int axon_internal_decode_direct(axon_model* m, const int32_t* tokens, int B, int32_t* ctx, const int32_t* bt,
                                float* logits, int32_t* next, cudaStream_t st, float* attn_part, int* attn_cnt,
                                int attn_rows_cap, int* head_dim, int* kv_heads) {
  if (head_dim) *head_dim = m->d;
  if (kv_heads) *kv_heads = m->G;
  if (!tokens) return AXON_OK;  // query only
  return enqueue_decode(m, tokens, B, ctx, bt, logits, next, st, nullptr, 0, attn_part, attn_cnt, attn_rows_cap);
}

// Validation shared with axon_decode_step. Not exported.
int axon_internal_decode_args_ok(const axon_model* m, const int32_t* d_tokens, int32_t B, const int32_t* d_ctx,
                                 const int32_t* d_block_table, const int32_t* d_next) {
  if (!m || !d_tokens || !d_ctx || !d_next) return AXON_ERR_INVALID_ARG;
  if (B < 1 || B > m->cfg.max_batch || B > 64) return AXON_ERR_INVALID_ARG;
  const bool paged = m->cfg.kv_layout == AXON_KV_PAGED;
  if (paged != (d_block_table != nullptr)) return AXON_ERR_INVALID_ARG;
  if (m->fp32) return AXON_ERR_UNSUPPORTED;
  return AXON_OK;
}

namespace {

void free_model(axon_model* m) {
  if (!m) return;
  for (auto& kv : m->graphs) cudaGraphExecDestroy(kv.second);
  m->graphs.clear();
  if (m->cap_stream) cudaStreamDestroy(m->cap_stream);
  for (void* p : m->allocs) cudaFree(p);
  delete m;
}

}  // namespace

extern "C" {

const char* axon_status_string(int status) {
  switch (status) {
    case AXON_OK: return "ok";
    case AXON_ERR_INVALID_ARG: return "invalid argument";
    case AXON_ERR_SHAPE_MISMATCH: return "weight shape does not match the config";
    case AXON_ERR_MISSING_WEIGHT: return "required weight missing";
    case AXON_ERR_UNSUPPORTED: return "configuration not supported by the kernels";
    case AXON_ERR_OOM: return "device out of memory";
    case AXON_ERR_CUDA: return "CUDA runtime error";
    case AXON_ERR_TIMEOUT: return "bounded device wait expired";
    case AXON_ERR_DEVICE_CHECK: return "device-side range check failed";
    default: return "unknown status";
  }
}

int axon_model_create(const axon_config* cfg, const axon_tensor* weights, int32_t n_weights, void* stream,
                      axon_model** out) {
  if (!out) return AXON_ERR_INVALID_ARG;
  *out = nullptr;
  if (!cfg || (!weights && n_weights > 0) || n_weights < 0) return AXON_ERR_INVALID_ARG;
  int rc = validate_config(cfg);
  if (rc) return rc;
  axon_model* m = new axon_model();
  m->cfg = *cfg;
  if (m->cfg.max_prefill_tokens <= 0) m->cfg.max_prefill_tokens = cfg->max_batch * cfg->max_context;
  m->L = cfg->num_hidden_layers;
  m->D = cfg->hidden_size;
  m->H = cfg->num_attention_heads;
  m->G = cfg->num_key_value_heads;
  m->d = cfg->head_dim;
  m->F = cfg->intermediate_size;
  m->V = cfg->vocab_size;
  m->Nqkv = (m->H + 2 * m->G) * m->d;
  m->fp32 = cfg->precision == AXON_FP32_DEBUG;
  m->f16 = cfg->precision == AXON_FP16;
  m->esz = m->fp32 ? 4 : 2;
  m->use_graphs = !env_flag("AXON_NO_GRAPH");
  m->use_pdl = !env_flag("AXON_NO_PDL");
  if (const char* v = getenv("AXON_PERSIST_SPLIT_BLOCKS")) {
    const int t = atoi(v);
    if (t >= 8 && t <= 4096) m->persist_split_blocks = t;
  }
  if (const char* v = getenv("AXON_DECODE_GEMV_MAX")) {
    const int t = atoi(v);
    if (t >= 0 && t <= 64) m->decode_gemv_max = t;
  }
  if (const char* v = getenv("AXON_QKV_SPLITK")) m->qkv_split = atoi(v) != 0;
  g_trace = env_flag("AXON_TRACE");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  auto fail = [&](int code) {
    cudaStreamSynchronize(st);
    free_model(m);
    return code;
  };
  if (cudaGetDevice(&m->device) != cudaSuccess) return fail(AXON_ERR_CUDA);
  cudaDeviceGetAttribute(&m->num_sms, cudaDevAttrMultiProcessorCount, m->device);
  m->attn_target_ctas = 0;
  if (const char* v = getenv("AXON_ATTN_TARGET_CTAS")) {
    const int t = atoi(v);
    if (t >= 1 && t <= 1 << 20) m->attn_target_ctas = t;
  }
  int major = 0;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, m->device);
  if (major < 10) return fail(AXON_ERR_UNSUPPORTED);
  if (prepare_attn_kernels() != cudaSuccess || prepare_gemm_kernels() != cudaSuccess ||
      prepare_gemv_kernels() != cudaSuccess)
    return fail(AXON_ERR_CUDA);

  Builder bl{m, weights, n_weights, st};
  const int D = m->D, Hd = m->H * m->d, Gd = m->G * m->d, F = m->F, V = m->V;
  // ---- validate every name and shape before allocating
  if ((rc = bl.check(bl.find("model.embed_tokens.weight"), V, D))) return fail(rc);
  if ((rc = bl.check(bl.find("model.norm.weight"), D, -1))) return fail(rc);
  if (!cfg->tie_word_embeddings && (rc = bl.check(bl.find("lm_head.weight"), V, D))) return fail(rc);
  for (int l = 0; l < m->L; ++l) {
    const std::string p = "model.layers." + std::to_string(l) + ".";
    if ((rc = bl.check(bl.find(p + "input_layernorm.weight"), D, -1))) return fail(rc);
    if ((rc = bl.check(bl.find(p + "post_attention_layernorm.weight"), D, -1))) return fail(rc);
    if ((rc = bl.check(bl.find(p + "self_attn.q_proj.weight"), Hd, D))) return fail(rc);
    if ((rc = bl.check(bl.find(p + "self_attn.k_proj.weight"), Gd, D))) return fail(rc);
    if ((rc = bl.check(bl.find(p + "self_attn.v_proj.weight"), Gd, D))) return fail(rc);
    if ((rc = bl.check(bl.find(p + "self_attn.o_proj.weight"), D, Hd))) return fail(rc);
    if (cfg->n_routed_experts > 0 && l >= cfg->first_k_dense_replace) {
      const int E = cfg->n_routed_experts, Fe = cfg->moe_intermediate_size, Fs = cfg->n_shared_experts * Fe;
      if ((rc = bl.check(bl.find(p + "mlp.gate.weight"), E, D))) return fail(rc);
      for (int e = 0; e < E; ++e) {
        const std::string q = p + "mlp.experts." + std::to_string(e) + ".";
        if ((rc = bl.check(bl.find(q + "gate_proj.weight"), Fe, D))) return fail(rc);
        if ((rc = bl.check(bl.find(q + "up_proj.weight"), Fe, D))) return fail(rc);
        if ((rc = bl.check(bl.find(q + "down_proj.weight"), D, Fe))) return fail(rc);
      }
      if (Fs) {
        const std::string q = p + "mlp.shared_experts.";
        if ((rc = bl.check(bl.find(q + "gate_proj.weight"), Fs, D))) return fail(rc);
        if ((rc = bl.check(bl.find(q + "up_proj.weight"), Fs, D))) return fail(rc);
        if ((rc = bl.check(bl.find(q + "down_proj.weight"), D, Fs))) return fail(rc);
      }
    } else {
      if ((rc = bl.check(bl.find(p + "mlp.gate_proj.weight"), F, D))) return fail(rc);
      if ((rc = bl.check(bl.find(p + "mlp.up_proj.weight"), F, D))) return fail(rc);
      if ((rc = bl.check(bl.find(p + "mlp.down_proj.weight"), D, F))) return fail(rc);
    }
    if (cfg->qk_norm) {
      if ((rc = bl.check(bl.find(p + "self_attn.q_norm.weight"), m->d, -1))) return fail(rc);
      if ((rc = bl.check(bl.find(p + "self_attn.k_norm.weight"), m->d, -1))) return fail(rc);
    }
    if (cfg->attention_bias) {
      if ((rc = bl.check(bl.find(p + "self_attn.q_proj.bias"), Hd, -1))) return fail(rc);
      if ((rc = bl.check(bl.find(p + "self_attn.k_proj.bias"), Gd, -1))) return fail(rc);
      if ((rc = bl.check(bl.find(p + "self_attn.v_proj.bias"), Gd, -1))) return fail(rc);
    }
  }

  // ---- weights
  const bool f32 = m->fp32;
  const size_t es = m->esz;
  if ((rc = dev_alloc(m, &m->embed, static_cast<size_t>(V) * D * es))) return fail(rc);
  if ((rc = bl.gather(m->embed, f32, bl.find("model.embed_tokens.weight"), nullptr, V, D))) return fail(rc);
  if (cfg->tie_word_embeddings) {
    m->head = m->embed;
  } else {
    if ((rc = dev_alloc(m, &m->head, static_cast<size_t>(V) * D * es))) return fail(rc);
    if ((rc = bl.gather(m->head, f32, bl.find("lm_head.weight"), nullptr, V, D))) return fail(rc);
  }
  void* gfp = nullptr;
  if ((rc = dev_alloc(m, &gfp, D * 4))) return fail(rc);
  m->gf = static_cast<float*>(gfp);
  if ((rc = bl.gather(m->gf, true, bl.find("model.norm.weight"), nullptr, 1, D))) return fail(rc);

  std::vector<int> qmap(Hd), kmap(Gd), gmap(F), umap(F);
  for (int h = 0; h < m->H; ++h)
    for (int p = 0; p < m->d; ++p) qmap[h * m->d + p] = h * m->d + qkv_natural(p, m->d);
  for (int h = 0; h < m->G; ++h)
    for (int p = 0; p < m->d; ++p) kmap[h * m->d + p] = h * m->d + qkv_natural(p, m->d);
  m->layers.resize(m->L);
  for (int l = 0; l < m->L; ++l) {
    LayerW& w = m->layers[l];
    const std::string p = "model.layers." + std::to_string(l) + ".";
    if ((rc = dev_alloc(m, &w.wqkv, static_cast<size_t>(m->Nqkv) * D * es))) return fail(rc);
    char* q0 = static_cast<char*>(w.wqkv);
    if ((rc = bl.gather(q0, f32, bl.find(p + "self_attn.q_proj.weight"), &qmap, Hd, D))) return fail(rc);
    if ((rc = bl.gather(q0 + static_cast<size_t>(Hd) * D * es, f32, bl.find(p + "self_attn.k_proj.weight"), &kmap,
                        Gd, D)))
      return fail(rc);
    if ((rc = bl.gather(q0 + static_cast<size_t>(Hd + Gd) * D * es, f32, bl.find(p + "self_attn.v_proj.weight"),
                        &kmap, Gd, D)))
      return fail(rc);
    if (cfg->attention_bias) {
      void* bp = nullptr;
      if ((rc = dev_alloc(m, &bp, static_cast<size_t>(m->Nqkv) * 4))) return fail(rc);
      w.bqkv = static_cast<float*>(bp);
      // A bias vector is a [n, 1] matrix for the gather.
      axon_tensor tq = *bl.find(p + "self_attn.q_proj.bias"), tk = *bl.find(p + "self_attn.k_proj.bias"),
                  tv = *bl.find(p + "self_attn.v_proj.bias");
      tq.ndim = tk.ndim = tv.ndim = 2;
      tq.shape[1] = tk.shape[1] = tv.shape[1] = 1;
      if ((rc = bl.gather(w.bqkv, true, &tq, &qmap, Hd, 1))) return fail(rc);
      if ((rc = bl.gather(w.bqkv + Hd, true, &tk, &kmap, Gd, 1))) return fail(rc);
      if ((rc = bl.gather(w.bqkv + Hd + Gd, true, &tv, &kmap, Gd, 1))) return fail(rc);
    }
    if ((rc = dev_alloc(m, &w.wo, static_cast<size_t>(D) * Hd * es))) return fail(rc);
    if ((rc = bl.gather(w.wo, f32, bl.find(p + "self_attn.o_proj.weight"), nullptr, D, Hd))) return fail(rc);
    // gate/up interleave: packed row r: chunk r/16, slots 0..7 gate, 8..15 up.
    // gate row j -> packed row (j/8)*16 + j%8, up row j -> (j/8)*16 + 8 + j%8
    auto pack_mlp = [&](const std::string& q, int width, void* gu, void* dn) {
      std::vector<int> to_gate(width), to_up(width);
      for (int j = 0; j < width; ++j) {
        to_gate[j] = (j >> 3) * 16 + (j & 7);
        to_up[j] = (j >> 3) * 16 + 8 + (j & 7);
      }
      int r = bl.gather(gu, f32, bl.find(q + "gate_proj.weight"), nullptr, width, D, &to_gate);
      if (!r) r = bl.gather(gu, f32, bl.find(q + "up_proj.weight"), nullptr, width, D, &to_up);
      if (!r) r = bl.gather(dn, f32, bl.find(q + "down_proj.weight"), nullptr, D, width);
      return r;
    };
    const bool moe_layer = cfg->n_routed_experts > 0 && l >= cfg->first_k_dense_replace;
    w.Fl = moe_layer ? cfg->n_shared_experts * cfg->moe_intermediate_size : F;
    if (w.Fl) {
      if ((rc = dev_alloc(m, &w.wgu, static_cast<size_t>(2 * w.Fl) * D * es))) return fail(rc);
      if ((rc = dev_alloc(m, &w.wd, static_cast<size_t>(D) * w.Fl * es))) return fail(rc);
      if ((rc = pack_mlp(moe_layer ? p + "mlp.shared_experts." : p + "mlp.", w.Fl, w.wgu, w.wd))) return fail(rc);
    }
    if (moe_layer) {
      // the stacked-experts formulation: expert e's gate/up rows at
      // e * 2Fe, its down rows at e * D, of one tensor each
      const int E = cfg->n_routed_experts, Fe = cfg->moe_intermediate_size;
      w.moe = true;
      if ((rc = dev_alloc(m, &w.router, static_cast<size_t>(E) * D * es))) return fail(rc);
      if ((rc = bl.gather(w.router, f32, bl.find(p + "mlp.gate.weight"), nullptr, E, D))) return fail(rc);
      if ((rc = dev_alloc(m, &w.wgu_e, static_cast<size_t>(E) * 2 * Fe * D * es))) return fail(rc);
      if ((rc = dev_alloc(m, &w.wd_e, static_cast<size_t>(E) * D * Fe * es))) return fail(rc);
      for (int e = 0; e < E && !rc; ++e)
        rc = pack_mlp(p + "mlp.experts." + std::to_string(e) + ".", Fe,
                      static_cast<char*>(w.wgu_e) + static_cast<size_t>(e) * 2 * Fe * D * es,
                      static_cast<char*>(w.wd_e) + static_cast<size_t>(e) * D * Fe * es);
      if (rc) return fail(rc);
    }
    void* g1 = nullptr;
    void* g2 = nullptr;
    if ((rc = dev_alloc(m, &g1, D * 4))) return fail(rc);
    if ((rc = dev_alloc(m, &g2, D * 4))) return fail(rc);
    w.g1 = static_cast<float*>(g1);
    w.g2 = static_cast<float*>(g2);
    if ((rc = bl.gather(w.g1, true, bl.find(p + "input_layernorm.weight"), nullptr, 1, D))) return fail(rc);
    if ((rc = bl.gather(w.g2, true, bl.find(p + "post_attention_layernorm.weight"), nullptr, 1, D)))
      return fail(rc);
    if (cfg->qk_norm) {
      void* qn = nullptr;
      void* kn = nullptr;
      if ((rc = dev_alloc(m, &qn, m->d * 4))) return fail(rc);
      if ((rc = dev_alloc(m, &kn, m->d * 4))) return fail(rc);
      w.qn = static_cast<float*>(qn);
      w.kn = static_cast<float*>(kn);
      if ((rc = bl.gather(w.qn, true, bl.find(p + "self_attn.q_norm.weight"), nullptr, 1, m->d))) return fail(rc);
      if ((rc = bl.gather(w.kn, true, bl.find(p + "self_attn.k_norm.weight"), nullptr, 1, m->d))) return fail(rc);
    }
  }

  // ---- KV cache: pools [L][num_blocks][G][16][d]
  m->blocks_per_seq = cfg->max_context / 16;
  m->num_blocks = cfg->kv_layout == AXON_KV_PAGED ? cfg->kv_num_blocks
                                                  : static_cast<long long>(cfg->max_batch) * m->blocks_per_seq;
  m->layer_kv_elems = static_cast<size_t>(m->num_blocks) * m->G * 16 * m->d;
  const size_t kv_bytes = m->layer_kv_elems * m->L * es;
  if ((rc = dev_alloc(m, &m->kpool, kv_bytes))) return fail(rc);
  if ((rc = dev_alloc(m, &m->vpool, kv_bytes))) return fail(rc);
  if (cudaMemsetAsync(m->kpool, 0, kv_bytes, st) != cudaSuccess ||
      cudaMemsetAsync(m->vpool, 0, kv_bytes, st) != cudaSuccess)
    return fail(AXON_ERR_CUDA);

  // ---- RoPE table in double precision: (cos, sin)(p * f_j), f_j =
  // theta^(-2j/d), stretched per band when frequency scaling is configured
  {
    const int half = m->d / 2;
    std::vector<double> freq(half);
    for (int j = 0; j < half; ++j) {
      double f = std::pow(static_cast<double>(cfg->rope_theta), -2.0 * j / m->d);
      if (cfg->rope_scaling_factor > 0.f) {
        const double factor = cfg->rope_scaling_factor, lo = cfg->rope_low_freq_factor,
                     hi = cfg->rope_high_freq_factor, C = cfg->rope_original_max_position;
        const double w = 2.0 * 3.14159265358979323846 / f;
        if (w > C / lo) {
          f = f / factor;
        } else if (w >= C / hi) {
          const double t = (C / w - lo) / (hi - lo);
          f = (1.0 - t) * f / factor + t * f;
        }
      }
      freq[j] = f;
    }
    std::vector<float2> tab(static_cast<size_t>(cfg->max_context) * half);
    for (int pos = 0; pos < cfg->max_context; ++pos)
      for (int j = 0; j < half; ++j) {
        const double ang = pos * freq[j];
        tab[static_cast<size_t>(pos) * half + j] = make_float2(static_cast<float>(std::cos(ang)),
                                                               static_cast<float>(std::sin(ang)));
      }
    void* rp = nullptr;
    if ((rc = dev_alloc(m, &rp, tab.size() * sizeof(float2)))) return fail(rc);
    m->rope = static_cast<float2*>(rp);
    if (cudaMemcpy(m->rope, tab.data(), tab.size() * sizeof(float2), cudaMemcpyHostToDevice) != cudaSuccess)
      return fail(AXON_ERR_CUDA);
  }

  // ---- workspace
  int Mcap = m->cfg.max_prefill_tokens;
  if (Mcap < cfg->max_batch) Mcap = cfg->max_batch;
  Mcap = (Mcap + 127) / 128 * 128;
  m->Mcap = Mcap;
  m->Pmax = D / 16;
  void* p = nullptr;
  if ((rc = dev_alloc(m, &p, static_cast<size_t>(Mcap) * D * 4))) return fail(rc);
  m->x = static_cast<float*>(p);
  if ((rc = dev_alloc(m, &m->a, static_cast<size_t>(Mcap) * D * es))) return fail(rc);
  if (m->f16) {
    if ((rc = dev_alloc(m, &m->a_lo, static_cast<size_t>(Mcap) * D * es))) return fail(rc);
    if (cudaMemsetAsync(m->a_lo, 0, static_cast<size_t>(Mcap) * D * es, st) != cudaSuccess) return fail(AXON_ERR_CUDA);
  }
  if ((rc = dev_alloc(m, &p, static_cast<size_t>(Mcap) * m->Pmax * 4))) return fail(rc);
  m->ss = static_cast<float*>(p);
  if ((rc = dev_alloc(m, &m->q, static_cast<size_t>(Mcap) * Hd * es))) return fail(rc);
  if ((rc = dev_alloc(m, &m->o, static_cast<size_t>(Mcap) * Hd * es))) return fail(rc);
  int Fmax = 0;  // widest dense MLP of any layer (shared experts included)
  for (const LayerW& w : m->layers) Fmax = w.Fl > Fmax ? w.Fl : Fmax;
  if (Fmax == 0) Fmax = 64;
  if ((rc = dev_alloc(m, &m->u, static_cast<size_t>(Mcap) * Fmax * es))) return fail(rc);
  if (!f32) {
    const size_t rows = static_cast<size_t>(cfg->max_batch < 64 ? cfg->max_batch : 64);
    if ((rc = dev_alloc(m, &m->q_lo, rows * Hd * es))) return fail(rc);
  }
  if (m->f16) {
    if ((rc = dev_alloc(m, &m->o_lo, static_cast<size_t>(m->cfg.max_batch) * Hd * es))) return fail(rc);
    if ((rc = dev_alloc(m, &m->u_lo, static_cast<size_t>(m->cfg.max_batch) * Fmax * es))) return fail(rc);
  }
  if ((rc = dev_alloc(m, &p, static_cast<size_t>(Mcap) * 8))) return fail(rc);
  m->keys = static_cast<unsigned long long*>(p);
  if ((rc = dev_alloc(m, &p, static_cast<size_t>(Mcap) * 4))) return fail(rc);
  m->rinv = static_cast<float*>(p);
  if ((rc = dev_alloc(m, &p, static_cast<size_t>(Mcap) * sizeof(int2)))) return fail(rc);
  m->rowmap = static_cast<int2*>(p);
  if (cfg->qk_norm) {
    if ((rc = dev_alloc(m, &p, static_cast<size_t>(Mcap) * (m->H + m->G) * m->d * 4))) return fail(rc);
    m->qk_raw = static_cast<float*>(p);
  }
  if (cfg->n_routed_experts > 0 && cfg->first_k_dense_replace < m->L) {
    // sorted rows: every (token, expert) slot plus, per expert in use, up to
    // 127 rows of padding to a whole 128-row block
    m->moe = true;
    m->E = cfg->n_routed_experts;
    m->topk = cfg->num_experts_per_tok;
    m->Fe = cfg->moe_intermediate_size;
    const long long slots = static_cast<long long>(Mcap) * m->topk;
    m->R_cap = (slots + std::min<long long>(m->E, slots) * 127 + 127) / 128 * 128;
    const size_t R = static_cast<size_t>(m->R_cap);
    if ((rc = dev_alloc(m, &p, slots * 4))) return fail(rc);
    m->moe_topk_idx = static_cast<int*>(p);
    if ((rc = dev_alloc(m, &p, slots * 4))) return fail(rc);
    m->moe_topk_w = static_cast<float*>(p);
    if ((rc = dev_alloc(m, &p, slots * 4))) return fail(rc);
    m->moe_slot_row = static_cast<int*>(p);
    if ((rc = dev_alloc(m, &p, R * 4))) return fail(rc);
    m->moe_row_tok = static_cast<int*>(p);
    if ((rc = dev_alloc(m, &p, R * 4))) return fail(rc);
    m->moe_row_w = static_cast<float*>(p);
    if ((rc = dev_alloc(m, &p, (R / 128) * 4 + 16))) return fail(rc);
    m->moe_mb_expert = static_cast<int*>(p);
    if ((rc = dev_alloc(m, &p, 16))) return fail(rc);
    m->moe_nmb = static_cast<int*>(p);
    if ((rc = dev_alloc(m, &p, static_cast<size_t>(Mcap) * m->E * 4))) return fail(rc);
    m->moe_logits = static_cast<float*>(p);
    if ((rc = dev_alloc(m, &p, static_cast<size_t>(Mcap) * 8))) return fail(rc);
    m->moe_keys = static_cast<unsigned long long*>(p);
    if ((rc = dev_alloc(m, &p, 16))) return fail(rc);
    m->moe_ones = static_cast<float*>(p);
    const float one = 1.0f;
    if (cudaMemcpy(m->moe_ones, &one, 4, cudaMemcpyHostToDevice) != cudaSuccess) return fail(AXON_ERR_CUDA);
    if ((rc = dev_alloc(m, &m->moe_a_sorted, R * D * es))) return fail(rc);
    if ((rc = dev_alloc(m, &m->moe_u_sorted, R * m->Fe * es))) return fail(rc);
    if ((rc = dev_alloc(m, &p, R * D * 4))) return fail(rc);
    m->moe_y_sorted = static_cast<float*>(p);
    if (cudaMemsetAsync(m->moe_row_tok, 0xff, R * 4, st) != cudaSuccess ||
        cudaMemsetAsync(m->moe_nmb, 0, 16, st) != cudaSuccess)
      return fail(AXON_ERR_CUDA);
    if (prepare_moe_kernels(D, m->E) != cudaSuccess) return fail(AXON_ERR_CUDA);
  }
  if ((rc = dev_alloc(m, &m->a_last, static_cast<size_t>(cfg->max_batch) * D * es))) return fail(rc);
  if (m->f16 && (rc = dev_alloc(m, &m->a_lo_last, static_cast<size_t>(cfg->max_batch) * D * es))) return fail(rc);
  if ((rc = dev_alloc(m, &p, static_cast<size_t>(cfg->max_batch) * 4))) return fail(rc);
  m->rinv_last = static_cast<float*>(p);
  if ((rc = dev_alloc(m, &p, 16))) return fail(rc);
  m->ticket = static_cast<int*>(p);
  m->splitk.max_tiles = 1024;
  m->splitk.max_ctas = 2048;
  if ((rc = dev_alloc(m, &p, static_cast<size_t>(m->splitk.max_ctas) * 16 * 64 * 4))) return fail(rc);
  m->splitk.part = static_cast<float*>(p);
  if ((rc = dev_alloc(m, &p, static_cast<size_t>(m->splitk.max_tiles) * 4))) return fail(rc);
  m->splitk.ticket = static_cast<int*>(p);
  if (cudaMemsetAsync(m->splitk.ticket, 0, static_cast<size_t>(m->splitk.max_tiles) * 4, st) != cudaSuccess)
    return fail(AXON_ERR_CUDA);
  if (!f32) {
    // decode-sized tensor-core GEMMs with too few tiles split K (<= 128 rows)
    const int nmax = std::max(std::max(m->Nqkv, 2 * F), std::max(D, V));
    m->gemm_sk.max_tiles = (nmax + 255) / 256;
    if ((rc = dev_alloc(m, &p, static_cast<size_t>(GEMM_MAX_UNITS) * 128 * 256 * 4))) return fail(rc);
    m->gemm_sk.ws = static_cast<float*>(p);
    if ((rc = dev_alloc(m, &p, static_cast<size_t>(m->gemm_sk.max_tiles) * 4))) return fail(rc);
    m->gemm_sk.tickets = static_cast<int*>(p);
    if (cudaMemsetAsync(m->gemm_sk.tickets, 0, static_cast<size_t>(m->gemm_sk.max_tiles) * 4, st) != cudaSuccess)
      return fail(AXON_ERR_CUDA);
  }
  m->max_splits = 64;
  const int dec_b = cfg->max_batch < 64 ? cfg->max_batch : 64;
  if ((rc = dev_alloc(m, &p, static_cast<size_t>(dec_b) * m->G * m->max_splits * 16 * (m->d + 2) * 4))) return fail(rc);
  m->attn_part = static_cast<float*>(p);
  if ((rc = dev_alloc(m, &p, static_cast<size_t>(dec_b) * m->G * 4))) return fail(rc);
  m->attn_cnt = static_cast<int*>(p);
  if ((rc = dev_alloc(m, &p, 16))) return fail(rc);
  m->err = static_cast<int*>(p);
  if (cudaMemsetAsync(m->keys, 0, static_cast<size_t>(Mcap) * 8, st) != cudaSuccess ||
      cudaMemsetAsync(m->attn_cnt, 0, static_cast<size_t>(dec_b) * m->G * 4, st) != cudaSuccess ||
      cudaMemsetAsync(m->err, 0, 16, st) != cudaSuccess || cudaMemsetAsync(m->ticket, 0, 16, st) != cudaSuccess ||
      cudaMemsetAsync(m->x, 0, static_cast<size_t>(Mcap) * D * 4, st) != cudaSuccess ||
      cudaMemsetAsync(m->a, 0, static_cast<size_t>(Mcap) * D * es, st) != cudaSuccess ||
      cudaMemsetAsync(m->o, 0, static_cast<size_t>(Mcap) * Hd * es, st) != cudaSuccess ||
      cudaMemsetAsync(m->u, 0, static_cast<size_t>(Mcap) * Fmax * es, st) != cudaSuccess)
    return fail(AXON_ERR_CUDA);

  // ---- TMA descriptors (bf16 tensor-core path)
  if (!f32) {
    bool ok = make_tma_2d_16(&m->t_a, m->a, Mcap, D, 128, m->f16) && make_tma_2d_16(&m->t_o, m->o, Mcap, Hd, 128, m->f16);
    if (ok && m->moe)
      ok = make_tma_2d_16(&m->t_asorted, m->moe_a_sorted, m->R_cap, D, 128, m->f16) &&
           make_tma_2d_16(&m->t_usorted, m->moe_u_sorted, m->R_cap, m->Fe, 128, m->f16);
    if (ok && m->a_lo) ok = make_tma_2d_16(&m->t_alo, m->a_lo, Mcap, D, 128, m->f16);
    ok = ok && make_tma_2d_16(&m->t_a16, m->a, Mcap, D, 16, m->f16) &&
         make_tma_2d_16(&m->t_o16, m->o, Mcap, Hd, 16, m->f16) &&
         make_tma_2d_16(&m->t_a64, m->a, Mcap, D, 64, m->f16) && make_tma_2d_16(&m->t_o64, m->o, Mcap, Hd, 64, m->f16);
    if (ok && m->a_lo)
      ok = make_tma_2d_16(&m->t_alo16, m->a_lo, Mcap, D, 16, m->f16) &&
           make_tma_2d_16(&m->t_alo64, m->a_lo, Mcap, D, 64, m->f16);
    auto small_a = [&](GemmMaps& g, const CUtensorMap& a16, const CUtensorMap& a64) {
      g.a16 = a16;
      g.a64 = a64;
      if (g.split) {
        g.a_lo16 = m->t_alo16;
        g.a_lo64 = m->t_alo64;
      }
      g.has16 = g.has64 = true;
    };
    for (int l = 0; l < m->L && ok; ++l) {
      LayerW& w = m->layers[l];
      w.m_qkv.a = m->t_a;
      ok = ok && make_tma_2d_16(&w.m_qkv.w, w.wqkv, m->Nqkv, D, 256, m->f16);
      if (m->a_lo) {
        w.m_qkv.a_lo = m->t_alo;
        w.m_qkv.split = true;
      }
      w.m_o.a = m->t_o;
      ok = ok && make_tma_2d_16(&w.m_o.w, w.wo, D, Hd, 256, m->f16);
      small_a(w.m_qkv, m->t_a16, m->t_a64);
      small_a(w.m_o, m->t_o16, m->t_o64);
      if (w.Fl) {
        w.m_gu.a = m->t_a;
        ok = ok && make_tma_2d_16(&w.m_gu.w, w.wgu, 2 * w.Fl, D, 256, m->f16);
        // the down projection reads u with this layer's row stride
        ok = ok && make_tma_2d_16(&w.m_d.a, m->u, Mcap, w.Fl, 128, m->f16);
        ok = ok && make_tma_2d_16(&w.m_d.w, w.wd, D, w.Fl, 256, m->f16);
        small_a(w.m_gu, m->t_a16, m->t_a64);
        CUtensorMap u16, u64;
        ok = ok && make_tma_2d_16(&u16, m->u, Mcap, w.Fl, 16, m->f16) &&
             make_tma_2d_16(&u64, m->u, Mcap, w.Fl, 64, m->f16);
        small_a(w.m_d, u16, u64);
      }
      if (w.moe) {
        const int E = m->E, Fe = m->Fe;
        w.m_router.a = m->t_a;
        if (m->a_lo) {
          w.m_router.a_lo = m->t_alo;
          w.m_router.split = true;
        }
        ok = ok && make_tma_2d_16(&w.m_router.w, w.router, E, D, 256, m->f16);
        w.m_router128 = w.m_router;
        ok = ok && make_tma_2d_16(&w.m_router128.w, w.router, E, D, 128, m->f16);
        w.m_router.n128 = &w.m_router128;
        w.m_gu_e.a = m->t_asorted;
        ok = ok && make_tma_2d_16(&w.m_gu_e.w, w.wgu_e, static_cast<uint64_t>(E) * 2 * Fe, D, 256, m->f16);
        w.m_d_e.a = m->t_usorted;
        ok = ok && make_tma_2d_16(&w.m_d_e.w, w.wd_e, static_cast<uint64_t>(E) * D, Fe, 256, m->f16);
        w.m_gu_e128 = w.m_gu_e;
        ok = ok && make_tma_2d_16(&w.m_gu_e128.w, w.wgu_e, static_cast<uint64_t>(E) * 2 * Fe, D, 128, m->f16);
        w.m_gu_e.n128 = &w.m_gu_e128;
        w.m_d_e128 = w.m_d_e;
        ok = ok && make_tma_2d_16(&w.m_d_e128.w, w.wd_e, static_cast<uint64_t>(E) * D, Fe, 128, m->f16);
        w.m_d_e.n128 = &w.m_d_e128;
      }
    }
    m->m_head.a = m->t_a;
    ok = ok && make_tma_2d_16(&m->m_head.w, m->head, V, D, 256, m->f16);
    small_a(m->m_head, m->t_a16, m->t_a64);
    // decode projections: weight boxes of 128 rows, activation boxes of 8..64 token rows
    for (int l = 0; l < m->L && ok; ++l) {
      LayerW& w = m->layers[l];
      ok = make_tma_2d_16(&w.v_qkv, w.wqkv, m->Nqkv, D, 128, m->f16) && make_tma_2d_16(&w.v_o, w.wo, D, Hd, 128, m->f16);
      if (ok && w.Fl)
        ok = make_tma_2d_16(&w.v_gu, w.wgu, 2 * w.Fl, D, 128, m->f16) &&
             make_tma_2d_16(&w.v_d, w.wd, D, w.Fl, 128, m->f16);
    }
    ok = ok && make_tma_2d_16(&m->v_head, m->head, V, D, 128, m->f16);
    // 128-wide output tiles reuse the 128-row weight boxes of the decode maps
    for (int l = 0; l < m->L && ok; ++l) {
      LayerW& w = m->layers[l];
      w.m_qkv128 = w.m_qkv;
      w.m_qkv128.w = w.v_qkv;
      w.m_qkv.n128 = &w.m_qkv128;
      w.m_o128 = w.m_o;
      w.m_o128.w = w.v_o;
      w.m_o.n128 = &w.m_o128;
      w.m_gu128 = w.m_gu;
      w.m_gu128.w = w.v_gu;
      w.m_gu.n128 = &w.m_gu128;
      w.m_d128 = w.m_d;
      w.m_d128.w = w.v_d;
      w.m_d.n128 = &w.m_d128;
    }
    m->m_head128 = m->m_head;
    m->m_head128.w = m->v_head;
    m->m_head.n128 = &m->m_head128;
    if (!ok) return fail(AXON_ERR_CUDA);
  }
  // ---- persistent decode step: layer table and grid barrier state
  // default for B <= PERSIST_MAX_B; AXON_NO_PERSIST=1 keeps the launch chain
  if (!f32 && !m->moe && !env_flag("AXON_NO_PERSIST") && (m->d == 64 || m->d == 128)) {
    const int per_sm = persist_ctas_per_sm(m->d, m->f16);
    if (per_sm >= 1) {
      std::vector<PersistLayer> pl(m->L);
      for (int l = 0; l < m->L; ++l) {
        const LayerW& w = m->layers[l];
        PersistLayer& t = pl[l];
        t.wqkv = w.wqkv;
        t.bqkv = w.bqkv;
        t.wo = w.wo;
        t.wgu = w.wgu;
        t.wd = w.wd;
        t.g1 = w.g1;
        t.g2 = w.g2;
        t.gnext = l + 1 < m->L ? m->layers[l + 1].g1 : m->gf;
        t.kc = static_cast<char*>(m->kpool) + static_cast<size_t>(l) * m->layer_kv_elems * m->esz;
        t.vc = static_cast<char*>(m->vpool) + static_cast<size_t>(l) * m->layer_kv_elems * m->esz;
      }
      if ((rc = dev_alloc(m, &p, sizeof(PersistLayer) * (m->L > 0 ? m->L : 1)))) return fail(rc);
      m->players = static_cast<PersistLayer*>(p);
      if (m->L > 0 && cudaMemcpy(m->players, pl.data(), sizeof(PersistLayer) * m->L, cudaMemcpyHostToDevice) !=
                          cudaSuccess)
        return fail(AXON_ERR_CUDA);
      std::vector<CUtensorMap> maps(4 * m->L + 1);
      bool ok = true;
      for (int l = 0; l < m->L && ok; ++l) {
        const LayerW& w = m->layers[l];
        ok = make_tma_2d_plain(&maps[4 * l + 0], w.wqkv, m->Nqkv, D, PERSIST_BOX_COLS, 16, m->f16) &&
             make_tma_2d_plain(&maps[4 * l + 1], w.wo, D, Hd, PERSIST_BOX_COLS, 16, m->f16) &&
             make_tma_2d_plain(&maps[4 * l + 2], w.wgu, 2 * F, D, PERSIST_BOX_COLS, 16, m->f16) &&
             make_tma_2d_plain(&maps[4 * l + 3], w.wd, D, F, PERSIST_BOX_COLS, 16, m->f16);
      }
      ok = ok && make_tma_2d_plain(&maps[4 * m->L], m->head, V, D, PERSIST_BOX_COLS, 16, m->f16);
      if (!ok) return fail(AXON_ERR_CUDA);
      if ((rc = dev_alloc(m, &p, sizeof(CUtensorMap) * maps.size()))) return fail(rc);
      m->pmaps = static_cast<CUtensorMap*>(p);
      if (cudaMemcpy(m->pmaps, maps.data(), sizeof(CUtensorMap) * maps.size(), cudaMemcpyHostToDevice) != cudaSuccess)
        return fail(AXON_ERR_CUDA);
      if ((rc = dev_alloc(m, &p, sizeof(PersistGrid)))) return fail(rc);
      m->pgrid = static_cast<PersistGrid*>(p);
      if (cudaMemsetAsync(m->pgrid, 0, sizeof(PersistGrid), st) != cudaSuccess) return fail(AXON_ERR_CUDA);
      m->persist_ctas = m->num_sms;  // one CTA per SM
    }
  }
  if (cudaStreamCreateWithFlags(&m->cap_stream, cudaStreamNonBlocking) != cudaSuccess) return fail(AXON_ERR_CUDA);
  if (cudaStreamSynchronize(st) != cudaSuccess) return fail(AXON_ERR_CUDA);
  *out = m;
  return AXON_OK;
}

int axon_prefill(axon_model* m, const int32_t* d_ids, int32_t B, int32_t S, const int32_t* d_block_table,
                 int32_t logits_mode, float* d_logits, int32_t* d_next, void* stream) {
  if (!m || !d_ids) return AXON_ERR_INVALID_ARG;
  if (B < 1 || B > m->cfg.max_batch || S < 1 || S > m->cfg.max_context) return AXON_ERR_INVALID_ARG;
  if (static_cast<long long>(B) * S > m->cfg.max_prefill_tokens) return AXON_ERR_INVALID_ARG;
  if (logits_mode != AXON_LOGITS_LAST && logits_mode != AXON_LOGITS_ALL) return AXON_ERR_INVALID_ARG;
  if (B > 64 && logits_mode == AXON_LOGITS_LAST) return AXON_ERR_UNSUPPORTED;
  const bool paged = m->cfg.kv_layout == AXON_KV_PAGED;
  if (paged != (d_block_table != nullptr)) return AXON_ERR_INVALID_ARG;
  return enqueue_prefill(m, d_ids, B, S, d_block_table, logits_mode, d_logits, d_next,
                         static_cast<cudaStream_t>(stream));
}

int axon_prefill_varlen(axon_model* m, const int32_t* d_ids, int32_t B, int32_t T, const int32_t* d_cu_seqlens,
                        int32_t* d_context_lens, int32_t max_chunk, const int32_t* d_block_table, int32_t logits_mode,
                        float* d_logits, int32_t* d_next, void* stream) {
  if (!m || !d_ids || !d_cu_seqlens || !d_context_lens) return AXON_ERR_INVALID_ARG;
  if (B < 1 || B > m->cfg.max_batch || T < B || T > m->cfg.max_prefill_tokens) return AXON_ERR_INVALID_ARG;
  if (max_chunk < 1 || max_chunk > m->cfg.max_context || max_chunk > T) return AXON_ERR_INVALID_ARG;
  if (logits_mode != AXON_LOGITS_LAST && logits_mode != AXON_LOGITS_ALL) return AXON_ERR_INVALID_ARG;
  const bool paged = m->cfg.kv_layout == AXON_KV_PAGED;
  if (paged != (d_block_table != nullptr)) return AXON_ERR_INVALID_ARG;
  const VarlenBatch vl{d_cu_seqlens, d_context_lens, T, max_chunk};
  return enqueue_prefill(m, d_ids, B, max_chunk, d_block_table, logits_mode, d_logits, d_next,
                         static_cast<cudaStream_t>(stream), nullptr, &vl);
}

int axon_decode_step(axon_model* m, const int32_t* d_tokens, int32_t B, int32_t* d_context_lens,
                     const int32_t* d_block_table, float* d_logits, int32_t* d_next, void* stream) {
  if (!m || !d_tokens || !d_context_lens || !d_next) return AXON_ERR_INVALID_ARG;
  if (B < 1 || B > m->cfg.max_batch || B > 64) return AXON_ERR_INVALID_ARG;
  const bool paged = m->cfg.kv_layout == AXON_KV_PAGED;
  if (paged != (d_block_table != nullptr)) return AXON_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // The persistent step is a single launch: nothing for a graph to save.
  if (!m->use_graphs || persist_eligible(m, B))
    return enqueue_decode(m, d_tokens, B, d_context_lens, d_block_table, d_logits, d_next, st);
  const GraphKey key{B, d_tokens, d_context_lens, d_block_table, d_logits, d_next};
  auto it = m->graphs.find(key);
  if (it == m->graphs.end()) {
    if (m->graphs.size() >= 64) {
      for (auto& kv : m->graphs) cudaGraphExecDestroy(kv.second);
      m->graphs.clear();
    }
    cudaGraph_t g = nullptr;
    CK(cudaStreamBeginCapture(m->cap_stream, cudaStreamCaptureModeThreadLocal));
    const int rc = enqueue_decode(m, d_tokens, B, d_context_lens, d_block_table, d_logits, d_next, m->cap_stream);
    const cudaError_t ec = cudaStreamEndCapture(m->cap_stream, &g);
    if (rc != AXON_OK || ec != cudaSuccess) {
      if (g) cudaGraphDestroy(g);
      cudaGetLastError();
      return rc != AXON_OK ? rc : AXON_ERR_CUDA;
    }
    cudaGraphExec_t ex = nullptr;
    const cudaError_t ei = cudaGraphInstantiate(&ex, g, 0);
    cudaGraphDestroy(g);
    if (ei != cudaSuccess) {
      cudaGetLastError();
      return AXON_ERR_CUDA;
    }
    it = m->graphs.emplace(key, ex).first;
  }
  CK(cudaGraphLaunch(it->second, st));
  return AXON_OK;
}

namespace {
int collect_profile(Prof& pf, axon_kernel_time* out, int32_t max_out, int32_t* n_out) {
  CK(cudaStreamSynchronize(pf.st));
  std::vector<axon_kernel_time> agg;
  for (auto& e : pf.entries) {
    float ms = 0.f;
    CK(cudaEventElapsedTime(&ms, e.a, e.b));
    axon_kernel_time* slot = nullptr;
    for (auto& a : agg)
      if (e.name == a.name) slot = &a;
    if (!slot) {
      axon_kernel_time t;
      memset(&t, 0, sizeof(t));
      snprintf(t.name, sizeof(t.name), "%s", e.name.c_str());
      agg.push_back(t);
      slot = &agg.back();
    }
    slot->launches += 1;
    slot->total_ms += ms;
    slot->bytes += e.bytes;
    slot->flops += e.flops;
  }
  const int n = static_cast<int>(agg.size()) < max_out ? static_cast<int>(agg.size()) : max_out;
  for (int i = 0; i < n; ++i) out[i] = agg[i];
  if (n_out) *n_out = n;
  return AXON_OK;
}
}  // namespace

int axon_profile_decode_step(axon_model* m, const int32_t* d_tokens, int32_t B, int32_t* d_context_lens,
                             const int32_t* d_block_table, int32_t* d_next, void* stream, axon_kernel_time* out,
                             int32_t max_out, int32_t* n_out) {
  if (!m || !d_tokens || !d_context_lens || !d_next || !out || max_out < 1) return AXON_ERR_INVALID_ARG;
  if (B < 1 || B > m->cfg.max_batch || B > 64) return AXON_ERR_INVALID_ARG;
  const bool paged = m->cfg.kv_layout == AXON_KV_PAGED;
  if (paged != (d_block_table != nullptr)) return AXON_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  std::vector<int32_t> h(B);
  CK(cudaMemcpyAsync(h.data(), d_context_lens, B * sizeof(int32_t), cudaMemcpyDeviceToHost, st));
  CK(cudaStreamSynchronize(st));
  double kv_tokens = 0;
  for (int b = 0; b < B; ++b) kv_tokens += h[b] + 1;
  Prof pf;
  pf.st = st;
  const int rc = enqueue_decode(m, d_tokens, B, d_context_lens, d_block_table, nullptr, d_next, st, &pf, kv_tokens);
  if (rc) return rc;
  return collect_profile(pf, out, max_out, n_out);
}

int axon_profile_prefill(axon_model* m, const int32_t* d_ids, int32_t B, int32_t S, const int32_t* d_block_table,
                         int32_t* d_next, void* stream, axon_kernel_time* out, int32_t max_out, int32_t* n_out) {
  if (!m || !d_ids || !out || max_out < 1) return AXON_ERR_INVALID_ARG;
  if (B < 1 || B > m->cfg.max_batch || S < 1 || S > m->cfg.max_context) return AXON_ERR_INVALID_ARG;
  if (static_cast<long long>(B) * S > m->cfg.max_prefill_tokens || B > 64) return AXON_ERR_INVALID_ARG;
  const bool paged = m->cfg.kv_layout == AXON_KV_PAGED;
  if (paged != (d_block_table != nullptr)) return AXON_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  Prof pf;
  pf.st = st;
  const int rc = enqueue_prefill(m, d_ids, B, S, d_block_table, AXON_LOGITS_LAST, nullptr, d_next, st, &pf);
  if (rc) return rc;
  return collect_profile(pf, out, max_out, n_out);
}

int axon_moe_routing_record(axon_model* m, int32_t* d_experts, int32_t rows) {
  if (!m) return AXON_ERR_INVALID_ARG;
  if (!m->moe) return AXON_ERR_UNSUPPORTED;
  if (d_experts && rows < 1) return AXON_ERR_INVALID_ARG;
  m->moe_record = d_experts;
  m->moe_record_rows = d_experts ? rows : 0;
  // recorded launches must not replay from graphs built without the record
  for (auto& kv : m->graphs) cudaGraphExecDestroy(kv.second);
  m->graphs.clear();
  return AXON_OK;
}

int axon_reset(axon_model* m) {
  if (!m) return AXON_ERR_INVALID_ARG;
  CK(cudaDeviceSynchronize());
  const size_t kv_bytes = m->layer_kv_elems * m->L * m->esz;
  CK(cudaMemset(m->kpool, 0, kv_bytes));
  CK(cudaMemset(m->vpool, 0, kv_bytes));
  CK(cudaMemset(m->err, 0, 16));
  CK(cudaDeviceSynchronize());
  return AXON_OK;
}

int axon_check_device(axon_model* m, void* stream, int32_t* bits) {
  if (!m) return AXON_ERR_INVALID_ARG;
  CK(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
  int word = 0;
  CK(cudaMemcpy(&word, m->err, sizeof(int), cudaMemcpyDeviceToHost));
  CK(cudaMemset(m->err, 0, sizeof(int)));
  if (bits) *bits = word;
  if (word & DEVERR_TIMEOUT) return AXON_ERR_TIMEOUT;
  if (word) return AXON_ERR_DEVICE_CHECK;
  return AXON_OK;
}

int axon_kv_view_get(const axon_model* m, axon_kv_view* out) {
  if (!m || !out) return AXON_ERR_INVALID_ARG;
  out->k_pool = m->kpool;
  out->v_pool = m->vpool;
  out->num_blocks = m->num_blocks;
  out->blocks_per_seq = m->blocks_per_seq;
  out->block_size = 16;
  out->elem_bytes = static_cast<int32_t>(m->esz);
  return AXON_OK;
}

void axon_free(axon_model* m) {
  if (!m) return;
  cudaDeviceSynchronize();
  free_model(m);
}

}  // extern "C"
