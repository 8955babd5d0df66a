// Decode-side kernels: the weight-streaming projection (skinny GEMV on
// tensor cores), the embedding gather and the greedy-token finaliser.
//
// Projection layout: one CTA owns 16 consecutive weight rows and all B <= 64
// tokens; its KW warps split K into 64-wide chunks. Each lane streams 2 rows
// x 32 bytes per chunk with 16-byte L1-bypassing loads (4 lanes cover 128
// contiguous bytes of a row), so the whole matrix is read exactly once at
// full 128-byte-line efficiency. Products run on mma.sync m16n8k16 with the
// weights as the 16-row A operand and tokens as the 8-wide N operand: the
// dot product is order-free in k, so each lane feeds its contiguous 16
// elements into the fragment slots in a fixed permutation that the token
// operand mirrors. Partial sums meet in shared memory in a fixed warp order
// (deterministic), then one thread per token runs the fused epilogue.
#include "kernels.h"

namespace {

constexpr int GEMV_KW = 8;  // warps per CTA along K

// Inverse RMS of each token for the consuming epilogue: either read back
// (producer already reduced it) or summed from the producer's partials by
// one warp.
AXON_DEV void load_rinv(const EpiArgs& ep, int B, float* rinv_s, int lane) {
  if (ep.rinv) {
    for (int b = lane; b < B; b += 32) rinv_s[b] = ep.rinv[static_cast<long long>(b) * ep.rinv_stride];
    return;
  }
  for (int b = 0; b < B; ++b) {
    const float* p = ep.ss + static_cast<long long>(b) * ep.ss_stride;
    float s = 0.f;
    for (int i = lane; i < ep.ss_parts; i += 32) s += p[i];
    s = warp_sum(s);
    if (lane == 0) rinv_s[b] = 1.0f / sqrtf(s * ep.inv_D + ep.eps);
  }
}

// Residual producers: the last CTA to finish reduces every token's partial
// sums of squares (fixed order, deterministic) into rinv_out and re-arms the
// ticket. No CTA waits on another.
AXON_DEV void finish_rinv(const EpiArgs& ep, int B, int nparts) {
  __shared__ int is_last;
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) is_last = (atomicAdd(ep.ticket, 1) == static_cast<int>(gridDim.x) - 1);
  __syncthreads();
  if (!is_last) return;
  __threadfence();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  for (int b = warp; b < B; b += nw) {
    const float* p = ep.ss_out + static_cast<long long>(b) * ep.ss_out_stride;
    float s = 0.f;
    for (int i = lane; i < nparts; i += 32) s += __ldcg(p + i);
    s = warp_sum(s);
    if (lane == 0) ep.rinv_out[b] = 1.0f / sqrtf(s * ep.inv_D + ep.eps);
  }
  if (threadIdx.x == 0) *ep.ticket = 0;
}

// LO: the activation operand is the sum of two 16-bit terms, act (the
// rounded value) and act_lo (what that rounding lost, same layout), and
// every k-step runs two MMAs into one accumulator: ~22 significant bits
// per activation instead of 11. The MMAs run in every lane whatever the
// token count (unused token slots feed zeros): mma.sync is warp-collective.
template <int NT, int KIND, typename T16, bool LO>
__global__ void __launch_bounds__(GEMV_KW * 32) gemv_mma_kernel(const T16* __restrict__ W, int N, int K,
                                                               const T16* __restrict__ act, long long act_stride,
                                                               int B, EpiArgs ep, SplitK sk,
                                                               const T16* __restrict__ act_lo) {
  constexpr int TOK = NT * 8;
  __shared__ float red[GEMV_KW][16][TOK + 1];
  __shared__ float rinv_s[TOK];

  // Let the next kernel in the stream start launching now: it only reads our
  // outputs after its own griddepcontrol.wait.
  grid_dep_launch();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = lane >> 2, q = lane & 3;
  const int n0 = blockIdx.x * 16;
  const int row0 = min(n0 + r, N - 1), row1 = min(n0 + r + 8, N - 1);
  // K-split blockIdx.y covers chunks [c_begin, c_end) of 64 columns.
  const int per = (K >> 6) / sk.count;
  const int c_begin = blockIdx.y * per;
  const int nchunks = (blockIdx.y == sk.count - 1) ? (K >> 6) - c_begin : per;
  const T16* w0 = W + static_cast<long long>(row0) * K + 16 * q + c_begin * 64;
  const T16* w1 = W + static_cast<long long>(row1) * K + 16 * q + c_begin * 64;

  float acc[NT][4];
#pragma unroll
  for (int t = 0; t < NT; ++t) acc[t][0] = acc[t][1] = acc[t][2] = acc[t][3] = 0.f;

  const T16* arow[NT];
  const T16* lrow[NT];
  bool aval[NT];
#pragma unroll
  for (int t = 0; t < NT; ++t) {
    const int tok = t * 8 + r;
    aval[t] = tok < B;
    const long long off = static_cast<long long>(aval[t] ? tok : 0) * act_stride + 16 * q + c_begin * 64;
    arow[t] = act + off;
    lrow[t] = LO ? act_lo + off : nullptr;
  }

  auto chunk = [&](int c, const uint4& wa0, const uint4& wa1, const uint4& wb0, const uint4& wb1) {
    const uint32_t A0[8] = {wa0.x, wa0.y, wa0.z, wa0.w, wa1.x, wa1.y, wa1.z, wa1.w};
    const uint32_t A1[8] = {wb0.x, wb0.y, wb0.z, wb0.w, wb1.x, wb1.y, wb1.z, wb1.w};
#pragma unroll
    for (int t = 0; t < NT; ++t) {
      uint4 x0 = make_uint4(0, 0, 0, 0), x1 = make_uint4(0, 0, 0, 0);
      if (aval[t]) {
        x0 = ld16(arow[t] + c * 64);
        x1 = ld16(arow[t] + c * 64 + 8);
      }
      const uint32_t Bv[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint32_t a[4] = {A0[2 * j], A1[2 * j], A0[2 * j + 1], A1[2 * j + 1]};
        const uint32_t bb[2] = {Bv[2 * j], Bv[2 * j + 1]};
        mma16816<T16>(acc[t], a, bb);
      }
      if (LO) {
        uint4 y0 = make_uint4(0, 0, 0, 0), y1 = make_uint4(0, 0, 0, 0);
        if (aval[t]) {
          y0 = ld16(lrow[t] + c * 64);
          y1 = ld16(lrow[t] + c * 64 + 8);
        }
        const uint32_t Bl[8] = {y0.x, y0.y, y0.z, y0.w, y1.x, y1.y, y1.z, y1.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint32_t a[4] = {A0[2 * j], A1[2 * j], A0[2 * j + 1], A1[2 * j + 1]};
          const uint32_t bb[2] = {Bl[2 * j], Bl[2 * j + 1]};
          mma16816<T16>(acc[t], a, bb);
        }
      }
    }
  };

  // Weights do not depend on earlier kernels: the first iteration's weight
  // loads are in flight before waiting for the activations.
  int c = warp;
  const uint4 z = make_uint4(0, 0, 0, 0);
  uint4 a0 = z, a1 = z, b0 = z, b1 = z, a2 = z, a3 = z, b2 = z, b3 = z;
  if (c < nchunks) {
    a0 = ld_stream16(w0 + c * 64);
    a1 = ld_stream16(w0 + c * 64 + 8);
    b0 = ld_stream16(w1 + c * 64);
    b1 = ld_stream16(w1 + c * 64 + 8);
  }
  if (c + GEMV_KW < nchunks) {
    const int c2 = c + GEMV_KW;
    a2 = ld_stream16(w0 + c2 * 64);
    a3 = ld_stream16(w0 + c2 * 64 + 8);
    b2 = ld_stream16(w1 + c2 * 64);
    b3 = ld_stream16(w1 + c2 * 64 + 8);
  }
  grid_dep_wait();
  if (c < nchunks) chunk(c, a0, a1, b0, b1);
  if (c + GEMV_KW < nchunks) chunk(c + GEMV_KW, a2, a3, b2, b3);
  for (c += 2 * GEMV_KW; c + GEMV_KW < nchunks; c += 2 * GEMV_KW) {
    const int c2 = c + GEMV_KW;
    a0 = ld_stream16(w0 + c * 64);
    a1 = ld_stream16(w0 + c * 64 + 8);
    b0 = ld_stream16(w1 + c * 64);
    b1 = ld_stream16(w1 + c * 64 + 8);
    a2 = ld_stream16(w0 + c2 * 64);
    a3 = ld_stream16(w0 + c2 * 64 + 8);
    b2 = ld_stream16(w1 + c2 * 64);
    b3 = ld_stream16(w1 + c2 * 64 + 8);
    chunk(c, a0, a1, b0, b1);
    chunk(c2, a2, a3, b2, b3);
  }
  if (c < nchunks) {
    a0 = ld_stream16(w0 + c * 64);
    a1 = ld_stream16(w0 + c * 64 + 8);
    b0 = ld_stream16(w1 + c * 64);
    b1 = ld_stream16(w1 + c * 64 + 8);
    chunk(c, a0, a1, b0, b1);
  }

  if (KIND != EPI_RESID && warp == GEMV_KW - 1) load_rinv(ep, B, rinv_s, lane);
#pragma unroll
  for (int t = 0; t < NT; ++t) {
    red[warp][r][t * 8 + 2 * q] = acc[t][0];
    red[warp][r][t * 8 + 2 * q + 1] = acc[t][1];
    red[warp][r + 8][t * 8 + 2 * q] = acc[t][2];
    red[warp][r + 8][t * 8 + 2 * q + 1] = acc[t][3];
  }
  __syncthreads();

  const int b = threadIdx.x;
  float v[16];
  if (b < B) {
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      float s = 0.f;
#pragma unroll
      for (int w = 0; w < GEMV_KW; ++w) s += red[w][i][b];
      v[i] = s;
    }
  }
  if (sk.count > 1) {
    // Cross-CTA split-K: publish this split's partial tile; the last split to
    // arrive sums all of them in split order (deterministic) and runs the
    // epilogue. No CTA waits on another.
    __shared__ int last_split;
    float* pt = sk.part + (static_cast<long long>(blockIdx.x) * sk.count) * 16 * 64;
    if (b < B) {
#pragma unroll
      for (int i = 0; i < 16; ++i) pt[(blockIdx.y * 16 + i) * 64 + b] = v[i];
    }
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) last_split = (atomicAdd(sk.ticket + blockIdx.x, 1) == sk.count - 1);
    __syncthreads();
    if (!last_split) return;
    __threadfence();
    if (b < B) {
#pragma unroll
      for (int i = 0; i < 16; ++i) v[i] = 0.f;
      for (int y = 0; y < sk.count; ++y) {
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] += __ldcg(pt + (y * 16 + i) * 64 + b);
      }
    }
    if (threadIdx.x == 0) sk.ticket[blockIdx.x] = 0;
  }
  if (b < B) {
    if (KIND == EPI_QKV) {
      epi_qkv16<T16>(ep, b, n0, v, rinv_s[b]);
    } else if (KIND == EPI_RESID) {
      const float s = epi_resid16<T16>(ep, b, n0, v);
      ep.ss_out[static_cast<long long>(b) * ep.ss_out_stride + blockIdx.x] = s;
    } else if (KIND == EPI_SWIGLU) {
      epi_swiglu16<T16>(ep, b, n0, v, rinv_s[b]);
    } else {
      const unsigned long long k = epi_logits16(ep, b, n0, v, rinv_s[b]);
      argmax_commit(ep.keys + b, k);
    }
  }
  if (KIND == EPI_RESID && ep.rinv_out) finish_rinv(ep, B, gridDim.x);
}

// fp32 debug projection: same CTA shape, CUDA-core FMAs on fp32 weights.
template <int KIND>
__global__ void __launch_bounds__(GEMV_KW * 32) gemv_f32_kernel(const float* __restrict__ W, int N, int K,
                                                               const float* __restrict__ act, long long act_stride,
                                                               int B, EpiArgs ep) {
  __shared__ float red[GEMV_KW][16][65];
  __shared__ float rinv_s[64];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n0 = blockIdx.x * 16;
  grid_dep_launch();
  grid_dep_wait();
  if (KIND != EPI_RESID && warp == GEMV_KW - 1) load_rinv(ep, B, rinv_s, lane);
  // Warp w: rows n0 + 2w, n0 + 2w + 1; lanes stride over K.
  for (int rr = 0; rr < 2; ++rr) {
    const int i = warp * 2 + rr;
    const int row = min(n0 + i, N - 1);
    const float* w = W + static_cast<long long>(row) * K;
    for (int b = 0; b < B; ++b) {
      const float* a = act + static_cast<long long>(b) * act_stride;
      float s = 0.f;
      for (int k = lane; k < K; k += 32) s = fmaf(w[k], a[k], s);
      s = warp_sum(s);
      if (lane == 0) red[0][i][b] = s;
    }
  }
  __syncthreads();
  const int b = threadIdx.x;
  if (b < B) {
    float v[16];
    for (int i = 0; i < 16; ++i) v[i] = red[0][i][b];
    if (KIND == EPI_QKV) {
      epi_qkv16<float>(ep, b, n0, v, rinv_s[b]);
    } else if (KIND == EPI_RESID) {
      const float s = epi_resid16<float>(ep, b, n0, v);
      ep.ss_out[static_cast<long long>(b) * ep.ss_out_stride + blockIdx.x] = s;
    } else if (KIND == EPI_SWIGLU) {
      epi_swiglu16<float>(ep, b, n0, v, rinv_s[b]);
    } else {
      const unsigned long long k = epi_logits16(ep, b, n0, v, rinv_s[b]);
      argmax_commit(ep.keys + b, k);
    }
  }
  if (KIND == EPI_RESID && ep.rinv_out) finish_rinv(ep, B, gridDim.x);
}

template <typename T>
__global__ void __launch_bounds__(256) embed_kernel(const T* __restrict__ E, int V, int D, const int* __restrict__ ids,
                                                    float* __restrict__ x, T* __restrict__ a,
                                                    const float* __restrict__ g, float* __restrict__ ss, int ss_stride,
                                                    float* __restrict__ rinv, float eps, int* err, T* __restrict__ a_lo) {
  __shared__ float red[8];
  grid_dep_launch();
  grid_dep_wait();
  const int m = blockIdx.x;
  int id = ids[m];
  if (id < 0 || id >= V) {
    if (threadIdx.x == 0) set_err(err, DEVERR_TOKEN);
    id = 0;
  }
  const T* e = E + static_cast<long long>(id) * D;
  float* xr = x + static_cast<long long>(m) * D;
  T* ar = a + static_cast<long long>(m) * D;
  float s = 0.f;
  // 8 consecutive elements per thread and step (D is a multiple of 64).
  for (int k = threadIdx.x * 8; k < D; k += blockDim.x * 8) {
    float v[8], ag[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = to_f(e[k + i]);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      ag[i] = v[i] * g[k + i];
      s += v[i] * v[i];
    }
    reinterpret_cast<float4*>(xr + k)[0] = make_float4(v[0], v[1], v[2], v[3]);
    reinterpret_cast<float4*>(xr + k)[1] = make_float4(v[4], v[5], v[6], v[7]);
    store8<T>(ar + k, ag);
    if (a_lo) {
      float lo[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) lo[i] = ag[i] - to_f(from_f<T>(ag[i]));
      store8<T>(a_lo + static_cast<long long>(m) * D + k, lo);
    }
  }
  s = warp_sum(s);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    float tot = 0.f;
    for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) tot += red[w];
    ss[static_cast<long long>(m) * ss_stride] = tot;
    if (rinv) rinv[m] = 1.0f / sqrtf(tot / static_cast<float>(D) + eps);
  }
}

// One CTA: read the B greedy tokens, then clear every key row used.
__global__ void __launch_bounds__(1024) finalize_kernel(unsigned long long* keys, int n_keys, int key_stride,
                                                        int key_offset, int B, int* next, int* ctx) {
  grid_dep_launch();
  grid_dep_wait();
  const int i = threadIdx.x;
  if (i < B) {
    const unsigned long long k = keys[static_cast<long long>(i) * key_stride + key_offset];
    if (next) next[i] = static_cast<int>(0xffffffffu - static_cast<uint32_t>(k & 0xffffffffull));
    if (ctx) ctx[i] += 1;
  }
  __syncthreads();
  for (int j = i; j < n_keys; j += blockDim.x) keys[j] = 0ull;
}

template <typename K, typename... Args>
cudaError_t launch_k(const LaunchCtx& lc, K kernel, dim3 grid, dim3 block, size_t smem, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = lc.stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = lc.pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

template <int NT, typename T16, bool LO>
cudaError_t gemv_nt_lo(const LaunchCtx& lc, int kind, const T16* w, int N, int K, const T16* a, long long st, int B,
                       const EpiArgs& ep, SplitK sk, const T16* al) {
  const dim3 grid((N + 15) / 16, sk.count), block(GEMV_KW * 32);
  switch (kind) {
    case EPI_QKV:
      return launch_k(lc, gemv_mma_kernel<NT, EPI_QKV, T16, LO>, grid, block, 0, w, N, K, a, st, B, ep, sk, al);
    case EPI_RESID:
      return launch_k(lc, gemv_mma_kernel<NT, EPI_RESID, T16, LO>, grid, block, 0, w, N, K, a, st, B, ep, sk, al);
    case EPI_SWIGLU:
      return launch_k(lc, gemv_mma_kernel<NT, EPI_SWIGLU, T16, LO>, grid, block, 0, w, N, K, a, st, B, ep, sk, al);
    default:
      return launch_k(lc, gemv_mma_kernel<NT, EPI_LOGITS, T16, LO>, grid, block, 0, w, N, K, a, st, B, ep, sk, al);
  }
}
template <int NT>
cudaError_t gemv_nt(const LaunchCtx& lc, int kind, const void* W, int N, int K, const void* act, long long st, int B,
                    const EpiArgs& ep, SplitK sk, const void* act_lo) {
  if (lc.f16) {
    const f16* w = static_cast<const f16*>(W);
    const f16* a = static_cast<const f16*>(act);
    if (act_lo)
      return gemv_nt_lo<NT, f16, true>(lc, kind, w, N, K, a, st, B, ep, sk, static_cast<const f16*>(act_lo));
    return gemv_nt_lo<NT, f16, false>(lc, kind, w, N, K, a, st, B, ep, sk, nullptr);
  }
  return gemv_nt_lo<NT, bf16, false>(lc, kind, static_cast<const bf16*>(W), N, K, static_cast<const bf16*>(act), st, B,
                                     ep, sk, nullptr);
}

// Resident CTAs per SM of each projection instantiation (occupancy API),
// filled by prepare_gemv_kernels().
int g_resident[4][4] = {};  // [NT index][kind]

// K-split count minimising the modelled time of the launch:
// waves(tiles * ks) * (chunks per CTA + per-CTA overhead), with waves
// counted against the resident-CTA capacity of the whole GPU. Each warp
// keeps >= 2 chunks; the partial-tile workspace bounds tiles * ks.
SplitK choose_split(const LaunchCtx& lc, int nt_idx, int kind, int N, int K, const SplitKWork& wk) {
  SplitK sk{1, wk.part, wk.ticket};
  if (!wk.part || !wk.ticket) return sk;
  const int tiles = (N + 15) / 16;
  if (tiles > wk.max_tiles) return sk;
  const int per_sm = g_resident[nt_idx][kind] > 0 ? g_resident[nt_idx][kind] : 2;
  const long long cap = static_cast<long long>(per_sm) * lc.num_sms;
  const int nch = K >> 6;
  const int max_ks = nch / (2 * GEMV_KW);
  constexpr double OVERHEAD_CHUNKS = 8.0;  // launch + first-load latency + merge, in chunk-times
  double best = 1e30;
  for (int ks = 1; ks <= (max_ks < 1 ? 1 : max_ks); ++ks) {
    const long long total = static_cast<long long>(tiles) * ks;
    if (ks > 1 && total > wk.max_ctas) break;
    const long long waves = (total + cap - 1) / cap;
    const double t = static_cast<double>(waves) * (static_cast<double>(nch) / ks / GEMV_KW + OVERHEAD_CHUNKS);
    if (t < best - 1e-9) {
      best = t;
      sk.count = ks;
    }
  }
  return sk;
}

}  // namespace

cudaError_t launch_gemv(const LaunchCtx& lc, int kind, bool fp32, const void* W, int N, int K, const void* act,
                        long long act_stride, int B, const EpiArgs& ep, const SplitKWork& wk,
                        const void* act_lo) {
  if (B < 1 || B > 64 || (K & 63) || N < 1) return cudaErrorInvalidValue;
  if (fp32) {
    const dim3 grid((N + 15) / 16), block(GEMV_KW * 32);
    const float* w = static_cast<const float*>(W);
    const float* a = static_cast<const float*>(act);
    switch (kind) {
      case EPI_QKV: return launch_k(lc, gemv_f32_kernel<EPI_QKV>, grid, block, 0, w, N, K, a, act_stride, B, ep);
      case EPI_RESID: return launch_k(lc, gemv_f32_kernel<EPI_RESID>, grid, block, 0, w, N, K, a, act_stride, B, ep);
      case EPI_SWIGLU: return launch_k(lc, gemv_f32_kernel<EPI_SWIGLU>, grid, block, 0, w, N, K, a, act_stride, B, ep);
      default: return launch_k(lc, gemv_f32_kernel<EPI_LOGITS>, grid, block, 0, w, N, K, a, act_stride, B, ep);
    }
  }
  const int nt_idx = B <= 8 ? 0 : (B <= 16 ? 1 : (B <= 32 ? 2 : 3));
  const SplitK sk = choose_split(lc, nt_idx, kind, N, K, wk);
  if (B <= 8) return gemv_nt<1>(lc, kind, W, N, K, act, act_stride, B, ep, sk, act_lo);
  if (B <= 16) return gemv_nt<2>(lc, kind, W, N, K, act, act_stride, B, ep, sk, act_lo);
  if (B <= 32) return gemv_nt<4>(lc, kind, W, N, K, act, act_stride, B, ep, sk, act_lo);
  return gemv_nt<8>(lc, kind, W, N, K, act, act_stride, B, ep, sk, act_lo);
}

namespace {
// Resident CTAs per SM of a projection kind: the smaller of the plain bf16
// variant and the fp16 split-operand variant (which holds more registers).
template <int NT, int KIND>
cudaError_t occupancy_kind(int idx) {
  const int threads = GEMV_KW * 32;
  int a = 0, b = 0;
  cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&a, gemv_mma_kernel<NT, KIND, bf16, false>, threads, 0);
  b = a;
  if (e == cudaSuccess)
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, gemv_mma_kernel<NT, KIND, f16, true>, threads, 0);
  g_resident[idx][KIND] = a < b ? a : b;
  return e;
}
template <int NT>
cudaError_t occupancy_nt(int idx) {
  cudaError_t e = occupancy_kind<NT, EPI_QKV>(idx);
  if (e == cudaSuccess) e = occupancy_kind<NT, EPI_RESID>(idx);
  if (e == cudaSuccess) e = occupancy_kind<NT, EPI_SWIGLU>(idx);
  if (e == cudaSuccess) e = occupancy_kind<NT, EPI_LOGITS>(idx);
  return e;
}
}  // namespace

cudaError_t prepare_gemv_kernels() {
  cudaError_t e = occupancy_nt<1>(0);
  if (e == cudaSuccess) e = occupancy_nt<2>(1);
  if (e == cudaSuccess) e = occupancy_nt<4>(2);
  if (e == cudaSuccess) e = occupancy_nt<8>(3);
  return e;
}

cudaError_t launch_embed(const LaunchCtx& lc, bool fp32, const void* E, int V, int D, const int* ids, int M, float* x,
                         void* a, const float* g, float* ss, int ss_stride, float* rinv, float eps, int* err,
                         void* a_lo) {
  if (fp32)
    return launch_k(lc, embed_kernel<float>, dim3(M), dim3(256), 0, static_cast<const float*>(E), V, D, ids, x,
                    static_cast<float*>(a), g, ss, ss_stride, rinv, eps, err, static_cast<float*>(nullptr));
  if (lc.f16)
    return launch_k(lc, embed_kernel<f16>, dim3(M), dim3(256), 0, static_cast<const f16*>(E), V, D, ids, x,
                    static_cast<f16*>(a), g, ss, ss_stride, rinv, eps, err, static_cast<f16*>(a_lo));
  return launch_k(lc, embed_kernel<bf16>, dim3(M), dim3(256), 0, static_cast<const bf16*>(E), V, D, ids, x,
                  static_cast<bf16*>(a), g, ss, ss_stride, rinv, eps, err, static_cast<bf16*>(a_lo));
}

cudaError_t launch_finalize(const LaunchCtx& lc, unsigned long long* keys, int n_keys, int key_stride, int key_offset,
                            int B, int* next, int* ctx) {
  if (B > 1024) return cudaErrorInvalidValue;
  return launch_k(lc, finalize_kernel, dim3(1), dim3(1024), 0, keys, n_keys, key_stride, key_offset, B, next, ctx);
}
