// Variable-length batches: several sequences each append one chunk of new
// tokens after the tokens they already hold in the cache (a whole prompt, a
// further piece of one, or a single decode token), packed row after row into
// one batch (Positions.position_ids with a past length per sequence and
// Cache.update, Sec. Built-In Libraries; vLLM's continuous batching over
// PagedAttention, Sec. Related Work).
//
// Sequence b's chunk is rows cu[b] .. cu[b+1]-1 and row cu[b] + i sits at
// position past[b] + i. The projections see only rows; these kernels give
// each row its (sequence, position), gather the last row of every chunk for
// the LM head, and turn the head's argmax keys into next tokens.
#include "kernels.h"

namespace {

// One thread per row: the sequence is the last b with cu[b] <= m (binary
// search over the B+1 offsets). Thread 0 of block 0 also checks the offsets.
__global__ void __launch_bounds__(256) varlen_rows_kernel(const int* cu, const int* past, int B, int T, int max_chunk,
                                                         int max_pos, int2* rowmap, int* err) {
  grid_dep_launch();
  grid_dep_wait();
  if (blockIdx.x == 0) {
    for (int b = threadIdx.x; b < B; b += blockDim.x) {
      const int n = cu[b + 1] - cu[b];
      if (n < 1 || n > max_chunk || (b == 0 && cu[0] != 0) || (b == B - 1 && cu[B] != T)) set_err(err, DEVERR_SEQ);
      if (past[b] < 0 || past[b] + n > max_pos) set_err(err, DEVERR_POS);
    }
  }
  const int m = blockIdx.x * blockDim.x + threadIdx.x;
  if (m >= T) return;
  int lo = 0, hi = B - 1;  // invariant: the answer lies in [lo, hi]
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (cu[mid] <= m) lo = mid;
    else hi = mid - 1;
  }
  const int i = m - cu[lo];
  const int pos = past[lo] + i;
  const bool ok = i >= 0 && m < cu[lo + 1] && past[lo] >= 0 && pos < max_pos;
  rowmap[m] = ok ? make_int2(lo, pos) : make_int2(0, -1);
}

// One CTA per sequence: copy the chunk's last row of a (and a_lo) with
// 16-byte accesses, and reduce its inverse RMS.
__global__ void __launch_bounds__(128) gather_last_kernel(const int* cu, int T, const uint4* a, const uint4* a_lo,
                                                         int row_vecs, const float* rinv, const float* ss,
                                                         int ss_stride, int parts, float inv_D, float eps, uint4* a_out,
                                                         uint4* a_lo_out, float* rinv_out) {
  grid_dep_launch();
  grid_dep_wait();
  const int b = blockIdx.x;
  int row = cu[b + 1] - 1;
  row = row < 0 ? 0 : (row >= T ? T - 1 : row);  // inconsistent offsets were reported
  const long long src = static_cast<long long>(row) * row_vecs, dst = static_cast<long long>(b) * row_vecs;
  for (int i = threadIdx.x; i < row_vecs; i += blockDim.x) {
    a_out[dst + i] = a[src + i];
    if (a_lo) a_lo_out[dst + i] = a_lo[src + i];
  }
  if (threadIdx.x == 0) {
    float r;
    if (rinv) {
      r = rinv[row];
    } else {
      const float* p = ss + static_cast<long long>(row) * ss_stride;
      float s = 0.f;
      for (int i = 0; i < parts; ++i) s += p[i];  // the producers' partials, in order
      r = 1.0f / sqrtf(s * inv_D + eps);
    }
    rinv_out[b] = r;
  }
}

__global__ void __launch_bounds__(1024) finalize_varlen_kernel(unsigned long long* keys, int n_keys, const int* cu,
                                                              int last_rows, int B, int* next, int* ctx) {
  grid_dep_launch();
  grid_dep_wait();
  for (int b = threadIdx.x; b < B; b += blockDim.x) {
    int k = b;
    if (last_rows) {
      k = cu[b + 1] - 1;
      k = k < 0 ? 0 : (k >= n_keys ? n_keys - 1 : k);
    }
    if (next) next[b] = static_cast<int>(0xffffffffu - static_cast<uint32_t>(keys[k] & 0xffffffffull));
    if (ctx) ctx[b] += cu[b + 1] - cu[b];
  }
  __syncthreads();
  for (int j = threadIdx.x; j < n_keys; j += blockDim.x) keys[j] = 0ull;
}

// qk-norm of Qwen3-family layers (the RMSNorm built-in applied to each
// head's d values of q and k before RoPE): one warp per (row, head); heads
// 0 .. H-1 are q, H .. H+G-1 are k. Reads the QKV epilogue's fp32 values,
// sums their squares in a fixed order, scales by 1 / sqrt(mean + eps) and
// the gains, rotates the (j, j + d/2) pairs, and stores q (with its second
// 16-bit term when q_lo_out is set) or k into the row's cache slot: one
// rounding, as without the norm.
template <typename T>
__global__ void __launch_bounds__(32) qk_norm_rope_kernel(EpiArgs e) {
  grid_dep_launch();
  grid_dep_wait();
  const int m = blockIdx.x, h = blockIdx.y, lane = threadIdx.x;
  const int d = e.d, half = d >> 1;
  const float* x = e.qk_raw + (static_cast<long long>(m) * (e.H + e.G) + h) * d;
  float ss = 0.f;
  for (int i = lane; i < d; i += 32) ss += x[i] * x[i];
  ss = warp_sum(ss);
  const float r = 1.0f / sqrtf(ss / static_cast<float>(d) + e.eps);
  const bool is_q = h < e.H;
  const float* gn = is_q ? e.qn_gain : e.kn_gain;
  int b;
  const int pos = row_seq_pos(e, m, b);
  T* dst;
  T* dlo = nullptr;
  if (is_q) {
    const long long off = (static_cast<long long>(m) * e.H + h) * d;
    dst = static_cast<T*>(e.q_out) + off;
    if (e.q_lo_out) dlo = static_cast<T*>(e.q_lo_out) + off;
  } else {
    const long long off = kv_offset(e, b, pos, h - e.H);
    if (off < 0) return;  // reported where v was stored
    dst = static_cast<T*>(e.k_cache) + off;
  }
  const float2* cs = e.rope + static_cast<long long>(min(max(pos, 0), e.max_pos - 1)) * half;
  for (int j = lane; j < half; j += 32) {
    const float a = x[j] * r * gn[j], bb = x[j + half] * r * gn[j + half];
    const float2 t = cs[j];
    const float o0 = a * t.x - bb * t.y, o1 = bb * t.x + a * t.y;
    const T h0 = from_f<T>(o0), h1 = from_f<T>(o1);
    dst[j] = h0;
    dst[j + half] = h1;
    if (dlo) {
      dlo[j] = from_f<T>(o0 - to_f(h0));
      dlo[j + half] = from_f<T>(o1 - to_f(h1));
    }
  }
}

template <typename K, typename... Args>
cudaError_t launch_k(const LaunchCtx& lc, K kernel, dim3 grid, dim3 block, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.stream = lc.stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = lc.pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

}  // namespace

cudaError_t launch_varlen_rows(const LaunchCtx& lc, const int* cu, const int* past, int B, int T, int max_chunk,
                               int max_pos, int2* rowmap, int* err) {
  if (B < 1 || T < 1) return cudaErrorInvalidValue;
  return launch_k(lc, varlen_rows_kernel, dim3((T + 255) / 256), dim3(256), cu, past, B, T, max_chunk, max_pos,
                  rowmap, err);
}

cudaError_t launch_gather_last(const LaunchCtx& lc, const int* cu, int B, int T, const void* a, const void* a_lo,
                               int row_bytes, const float* rinv, const float* ss, int ss_stride, int parts,
                               float inv_D, float eps, void* a_out, void* a_lo_out, float* rinv_out) {
  if (B < 1 || T < 1 || row_bytes % 16 != 0) return cudaErrorInvalidValue;
  return launch_k(lc, gather_last_kernel, dim3(B), dim3(128), cu, T, static_cast<const uint4*>(a),
                  static_cast<const uint4*>(a_lo), row_bytes / 16, rinv, ss, ss_stride, parts, inv_D, eps,
                  static_cast<uint4*>(a_out), static_cast<uint4*>(a_lo_out), rinv_out);
}

cudaError_t launch_finalize_varlen(const LaunchCtx& lc, unsigned long long* keys, int n_keys, const int* cu,
                                   int last_rows, int B, int* next, int* ctx) {
  return launch_k(lc, finalize_varlen_kernel, dim3(1), dim3(1024), keys, n_keys, cu, last_rows, B, next, ctx);
}

cudaError_t launch_qk_norm_rope(const LaunchCtx& lc, bool fp32, const EpiArgs& e, int rows) {
  if (rows < 1 || !e.qk_raw || !e.qn_gain || !e.kn_gain) return cudaErrorInvalidValue;
  const dim3 grid(rows, e.H + e.G);
  if (fp32) return launch_k(lc, qk_norm_rope_kernel<float>, grid, dim3(32), e);
  if (lc.f16) return launch_k(lc, qk_norm_rope_kernel<f16>, grid, dim3(32), e);
  return launch_k(lc, qk_norm_rope_kernel<bf16>, grid, dim3(32), e);
}
