// Allocation-free decode step.
//
// axon_decode_step records each (batch size, pointer set) into a CUDA graph
// the first time it sees it, and instantiating a graph allocates device and
// host memory. axon_decode_step_noalloc runs the same kernels launched one
// after another instead, and the one kernel of the step that needs scratch
// beyond the model's own buffers -- the split-KV attention, which merges the
// partial softmax states of its key splits -- takes that scratch from the
// fixed file-scope array below rather than from anything allocated per call.
//
// The array lives in every device that loads this library, for the life of
// the process: NOALLOC_ROWS merge slots of (16 head rows x (head_dim + 2))
// floats plus one ticket per (sequence, kv head), about 2.1 MB.
#include <cuda.h>
#include <cuda_runtime.h>

#include <mutex>

#include "../../include/axon.h"
#include "kernels.h"

int axon_internal_decode_direct(axon_model* m, const int32_t* tokens, int B, int32_t* ctx, const int32_t* bt,
                                float* logits, int32_t* next, cudaStream_t st, float* attn_part, int* attn_cnt,
                                int attn_rows_cap, int* head_dim, int* kv_heads);
int axon_internal_decode_args_ok(const axon_model* m, const int32_t* d_tokens, int32_t B, const int32_t* d_ctx,
                                 const int32_t* d_block_table, const int32_t* d_next);

namespace {

constexpr int NOALLOC_ROWS = 256;  // (sequence, kv head, key split) merge slots
constexpr int NOALLOC_MAX_HEAD_DIM = 128;
constexpr int NOALLOC_PART_FLOATS = NOALLOC_ROWS * 16 * (NOALLOC_MAX_HEAD_DIM + 2);

// Partial (O, running max, running sum) states of the attention key splits,
// followed by the per-(sequence, kv head) tickets that pick the merging CTA.
static __device__ __align__(256) float g_noalloc_scratch[NOALLOC_PART_FLOATS + NOALLOC_ROWS];

// Device address of g_noalloc_scratch per device, resolved with that device
// current (in host code the symbol's name is only a host-side stand-in, never
// a device address). The address belongs to the context the module was
// loaded into: after cudaDeviceReset (or any teardown of the primary
// context) the module is loaded again, possibly elsewhere, so each entry
// remembers its context and is resolved again when the current one differs.
typedef CUresult (*CtxGetCurrentFn)(CUcontext*);

CtxGetCurrentFn ctx_get_current() {
  static CtxGetCurrentFn fn = nullptr;
  static bool tried = false;
  if (!tried) {
    tried = true;
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<CtxGetCurrentFn>(p);
  }
  return fn;
}

struct Resolved {
  CUcontext ctx = nullptr;
  float* addr = nullptr;
};
std::mutex g_mu;
Resolved g_addr[64];

float* scratch_on_current_device(int* status) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    *status = AXON_ERR_CUDA;
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(g_mu);
  CtxGetCurrentFn get = ctx_get_current();
  CUcontext ctx = nullptr;
  if (!get || get(&ctx) != CUDA_SUCCESS) {
    *status = AXON_ERR_CUDA;
    return nullptr;
  }
  Resolved& r = g_addr[dev];
  if (!r.addr || !ctx || r.ctx != ctx) {
    // cudaGetSymbolAddress also binds the device's primary context to this
    // thread when nothing is bound yet; the context is read again after it
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p || get(&ctx) != CUDA_SUCCESS || !ctx) {
      cudaGetLastError();
      *status = AXON_ERR_CUDA;
      return nullptr;
    }
    r.addr = static_cast<float*>(p);
    r.ctx = ctx;
  }
  *status = AXON_OK;
  return r.addr;
}

}  // namespace

extern "C" int axon_decode_step_noalloc(axon_model* m, const int32_t* d_tokens, int32_t B, int32_t* d_context_lens,
                                        const int32_t* d_block_table, float* d_logits, int32_t* d_next,
                                        void* stream) {
  int rc = axon_internal_decode_args_ok(m, d_tokens, B, d_context_lens, d_block_table, d_next);
  if (rc != AXON_OK) return rc;
  int head_dim = 0, kv_heads = 0;
  axon_internal_decode_direct(m, nullptr, 0, nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, 0,
                              &head_dim, &kv_heads);
  if (head_dim > NOALLOC_MAX_HEAD_DIM || B * kv_heads > NOALLOC_ROWS) return AXON_ERR_UNSUPPORTED;
  float* part = scratch_on_current_device(&rc);
  if (!part) return rc;
  int* tickets = reinterpret_cast<int*>(part + NOALLOC_PART_FLOATS);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // Tickets must start at zero; the partial states are always written before
  // they are read, so they need no clearing.
  if (cudaMemsetAsync(tickets, 0, static_cast<size_t>(B) * kv_heads * sizeof(int), st) != cudaSuccess) {
    cudaGetLastError();
    return AXON_ERR_CUDA;
  }
  return axon_internal_decode_direct(m, d_tokens, B, d_context_lens, d_block_table, d_logits, d_next, st, part,
                                     tickets, NOALLOC_ROWS, nullptr, nullptr);
}
