// Mixture-of-experts MLP (the MoE built-ins' softmax top-k router and
// grouped experts; the stacked-experts formulation that the paper's graph
// rewriting puts in place of a loop over experts):
//
//   moe_route_kernel    per token: h = (a [+ a_lo]) * r, the normalised
//                       input (r from the producer's norm partials), router
//                       logits h . Wr[e] in fp32, softmax, top-k (lowest
//                       index on ties), weights (optionally renormalised);
//                       h is also stored as 16-bit operand terms;
//   moe_plan_kernel     one CTA: a stable counting sort of the T x k
//                       (token, expert) slots by expert into segments padded
//                       to 128-row blocks: the sorted row of every slot, the
//                       token and weight of every sorted row (token -1 for
//                       padding), the expert of every 128-row block and the
//                       block count -- the grouped GEMM's tile list;
//   moe_gather_kernel   the sorted operand rows (padding rows zero);
//   [grouped tcgen05 GEMM gate/up + SwiGLU, grouped GEMM down scaled by the
//    row's weight: k_gemm.cu]
//   moe_combine_kernel  per token: x += the sum of its k expert outputs in
//                       slot order; optionally the residual epilogue's
//                       next-norm operand and partial sums of squares.
// Every step is deterministic: no floating-point atomics.
#include "kernels.h"

namespace {

constexpr int ROUTE_THREADS = 256;
constexpr int PLAN_THREADS = 1024;

template <typename T16>
__global__ void __launch_bounds__(ROUTE_THREADS) moe_route_kernel(MoeArgs a, EpiArgs ns) {
  grid_dep_launch();
  grid_dep_wait();
  extern __shared__ float sh[];  // [D] normalised h, then [E] logits
  const int t = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int D = a.D, E = a.E, k = a.k;
  float* lg = sh + D;
  const float r = row_rinv(ns, t);
  const T16* ah = static_cast<const T16*>(a.act) + static_cast<long long>(t) * a.act_stride;
  const T16* al = a.act_lo ? static_cast<const T16*>(a.act_lo) + static_cast<long long>(t) * a.act_stride : nullptr;
  T16* hh = static_cast<T16*>(a.h_hi) + static_cast<long long>(t) * D;
  T16* hl = a.h_lo ? static_cast<T16*>(a.h_lo) + static_cast<long long>(t) * D : nullptr;
  for (int i = tid; i < D; i += ROUTE_THREADS) {
    const float v = (to_f(ah[i]) + (al ? to_f(al[i]) : 0.f)) * r;
    sh[i] = v;
    const T16 h16 = from_f<T16>(v);
    hh[i] = h16;
    if (hl) hl[i] = from_f<T16>(v - to_f(h16));
  }
  __syncthreads();
  for (int e = warp; e < E; e += ROUTE_THREADS / 32) {
    const float* w = a.router + static_cast<long long>(e) * D;
    float s = 0.f;
    for (int i = lane; i < D; i += 32) s = fmaf(sh[i], w[i], s);
    s = warp_sum(s);
    if (lane == 0) lg[e] = s;
  }
  __syncthreads();
  if (warp != 0) return;
  float mx = -INFINITY;
  for (int e = lane; e < E; e += 32) mx = fmaxf(mx, lg[e]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  float den = 0.f;
  for (int e = lane; e < E; e += 32) {
    const float p = expf(lg[e] - mx);
    lg[e] = p;
    den += p;
  }
  den = warp_sum(den);
  __syncwarp();
  // top-k by repeated arg-max over (probability, lowest index)
  float wsum = 0.f, wk[8];
  int ik[8];
  for (int j = 0; j < k; ++j) {
    float bv = -1.f;
    int bi = 0x7fffffff;
    for (int e = lane; e < E; e += 32) {
      const float p = lg[e];
      if (p > bv || (p == bv && e < bi)) {
        bv = p;
        bi = e;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
      if (ov > bv || (ov == bv && oi < bi)) {
        bv = ov;
        bi = oi;
      }
    }
    ik[j] = bi;
    wk[j] = bv / den;
    wsum += wk[j];
    __syncwarp();
    if (lane == 0) lg[bi] = -2.f;  // taken
    __syncwarp();
  }
  if (lane < k) {
    float w = 0.f;
    int e = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (j == lane) {
        w = wk[j];
        e = ik[j];
      }
    a.topk_idx[static_cast<long long>(t) * k + lane] = e;
    a.topk_w[static_cast<long long>(t) * k + lane] = a.norm_topk ? w / wsum : w;
    if (a.record && t < a.record_rows) a.record[static_cast<long long>(t) * k + lane] = e;
  }
}

// Stable counting sort of the n = T * k slots by expert, in rounds of
// PLAN_THREADS slots: within a warp, slots of one expert are ranked by
// lane (match_any), warps are ranked in order by a per-expert prefix over
// the round's warp counts, rounds in order by the running counts.
__global__ void __launch_bounds__(PLAN_THREADS) moe_plan_kernel(MoeArgs a, int T) {
  grid_dep_launch();
  grid_dep_wait();
  __shared__ int cnt[MOE_MAX_EXPERTS];
  __shared__ int seg[MOE_MAX_EXPERTS];
  __shared__ int wcnt[PLAN_THREADS / 32][MOE_MAX_EXPERTS];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int E = a.E, n = T * a.k;
  for (int e = tid; e < E; e += PLAN_THREADS) cnt[e] = 0;
  for (int base = 0; base < n; base += PLAN_THREADS) {
    for (int c = tid; c < (PLAN_THREADS / 32) * E; c += PLAN_THREADS) wcnt[c / E][c % E] = 0;
    __syncthreads();
    const int i = base + tid;
    int e = i < n ? a.topk_idx[i] : -1;
    if (e >= E || e < -1) {
      set_err(a.err, DEVERR_SEQ);
      e = -1;
    }
    const unsigned peers = __match_any_sync(0xffffffffu, e);
    const int rank_w = __popc(peers & ((1u << lane) - 1u));
    if (e >= 0 && rank_w == 0) wcnt[warp][e] = __popc(peers);
    __syncthreads();
    for (int x = tid; x < E; x += PLAN_THREADS) {
      int s = cnt[x];
      for (int w = 0; w < PLAN_THREADS / 32; ++w) {
        const int c = wcnt[w][x];
        wcnt[w][x] = s;
        s += c;
      }
      cnt[x] = s;
    }
    __syncthreads();
    if (e >= 0) a.slot_row[i] = wcnt[warp][e] + rank_w;  // rank within the expert, for now
    else if (i < n) a.slot_row[i] = -1;
    __syncthreads();
  }
  if (tid == 0) {
    int acc = 0;
    for (int e = 0; e < E; ++e) {
      seg[e] = acc;
      const int blocks = (cnt[e] + 127) >> 7;
      for (int b = 0; b < blocks; ++b) a.mb_expert[(acc >> 7) + b] = e;
      acc += blocks << 7;
    }
    *a.n_mblocks = acc >> 7;
  }
  __syncthreads();
  for (int i = tid; i < n; i += PLAN_THREADS) {
    const int e = a.topk_idx[i];
    const int rk = a.slot_row[i];
    if (rk < 0 || e < 0 || e >= E) continue;
    const int row = seg[e] + rk;
    a.slot_row[i] = row;
    a.row_tok[row] = i / a.k;
    a.row_w[row] = a.topk_w[i];
  }
  // padding rows of each segment
  for (int e = 0; e < E; ++e) {
    const int pad0 = seg[e] + cnt[e], pad1 = seg[e] + (((cnt[e] + 127) >> 7) << 7);
    for (int row = pad0 + tid; row < pad1; row += PLAN_THREADS) {
      a.row_tok[row] = -1;
      a.row_w[row] = 0.f;
    }
  }
}

// Sorted operand rows: row r is token row_tok[r]'s normalised h (both
// terms), or zeros for padding. One warp per row, 16-byte copies.
template <typename T16>
__global__ void __launch_bounds__(256) moe_gather_kernel(MoeArgs a) {
  grid_dep_launch();
  grid_dep_wait();
  const int rows = __ldcg(a.n_mblocks) * 128;
  const int per_row = a.D / 8;  // 16-byte pieces
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  const int nwarps = (gridDim.x * blockDim.x) >> 5;
  for (int r = warp; r < rows; r += nwarps) {
    const int tok = __ldcg(a.row_tok + r);
    const uint4* sh = reinterpret_cast<const uint4*>(static_cast<const T16*>(a.h_hi) + static_cast<long long>(tok) * a.D);
    uint4* dh = reinterpret_cast<uint4*>(static_cast<T16*>(a.a_sorted) + static_cast<long long>(r) * a.D);
    const uint4* sl = a.h_lo ? reinterpret_cast<const uint4*>(static_cast<const T16*>(a.h_lo) + static_cast<long long>(tok) * a.D) : nullptr;
    uint4* dl = a.a_sorted_lo ? reinterpret_cast<uint4*>(static_cast<T16*>(a.a_sorted_lo) + static_cast<long long>(r) * a.D) : nullptr;
    const uint4 z = make_uint4(0, 0, 0, 0);
    for (int c = lane; c < per_row; c += 32) {
      dh[c] = tok >= 0 ? __ldcg(sh + c) : z;
      if (dl) dl[c] = (tok >= 0 && sl) ? __ldcg(sl + c) : z;
    }
  }
}

// x[t] += sum over j of y[slot_row[t * k + j]] (j in order); with the
// residual epilogue (ep.a_out set): the next norm's operand and partial sums
// of squares per 16 columns as well. One thread per 16 columns.
template <typename T16>
__global__ void __launch_bounds__(1024) moe_combine_kernel(MoeArgs a, EpiArgs ep) {
  grid_dep_launch();
  grid_dep_wait();
  const int t = blockIdx.x, c = threadIdx.x;
  const int n0 = c * 16;
  if (n0 >= a.D) return;
  float v[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = 0.f;
  for (int j = 0; j < a.k; ++j) {
    const int row = a.slot_row[static_cast<long long>(t) * a.k + j];
    if (row < 0) continue;
    const float4* y = reinterpret_cast<const float4*>(a.y_sorted + static_cast<long long>(row) * a.D + n0);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float4 f = __ldcg(y + q);
      v[4 * q] += f.x;
      v[4 * q + 1] += f.y;
      v[4 * q + 2] += f.z;
      v[4 * q + 3] += f.w;
    }
  }
  float4 xin[4];
  load_resid16(ep, t, n0, xin);
  if (ep.a_out) {
    const float s = epi_resid16x<T16>(ep, t, n0, v, xin);
    ep.ss_out[static_cast<long long>(t) * ep.ss_out_stride + c] = s;
  } else {
    float4* xp = reinterpret_cast<float4*>(ep.x + static_cast<long long>(t) * ep.N + n0);
#pragma unroll
    for (int q = 0; q < 4; ++q)
      xp[q] = make_float4(xin[q].x + v[4 * q], xin[q].y + v[4 * q + 1], xin[q].z + v[4 * q + 2],
                          xin[q].w + v[4 * q + 3]);
  }
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

}  // namespace

cudaError_t prepare_moe_kernels(int D, int E) {
  const int smem = (D + E) * 4;
  cudaError_t e = cudaFuncSetAttribute(moe_route_kernel<bf16>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(moe_route_kernel<f16>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  return e;
}

cudaError_t launch_moe_route(const LaunchCtx& lc, const MoeArgs& a, int T, const EpiArgs& ns) {
  if (T < 1 || a.k < 1 || a.k > 8 || a.k > a.E || a.E > MOE_MAX_EXPERTS) return cudaErrorInvalidValue;
  const size_t smem = static_cast<size_t>(a.D + a.E) * 4;
  if (lc.f16) return launch_k(lc, moe_route_kernel<f16>, dim3(T), dim3(ROUTE_THREADS), smem, a, ns);
  return launch_k(lc, moe_route_kernel<bf16>, dim3(T), dim3(ROUTE_THREADS), smem, a, ns);
}

cudaError_t launch_moe_plan(const LaunchCtx& lc, const MoeArgs& a, int T) {
  return launch_k(lc, moe_plan_kernel, dim3(1), dim3(PLAN_THREADS), 0, a, T);
}

cudaError_t launch_moe_gather(const LaunchCtx& lc, const MoeArgs& a) {
  if (a.D % 8) return cudaErrorInvalidValue;
  if (lc.f16) return launch_k(lc, moe_gather_kernel<f16>, dim3(2 * lc.num_sms), dim3(256), 0, a);
  return launch_k(lc, moe_gather_kernel<bf16>, dim3(2 * lc.num_sms), dim3(256), 0, a);
}

cudaError_t launch_moe_combine(const LaunchCtx& lc, const MoeArgs& a, int T, const EpiArgs& ep) {
  if (a.D % 16 || a.D / 16 > 1024) return cudaErrorInvalidValue;
  const dim3 block((a.D / 16 + 31) / 32 * 32);
  if (lc.f16) return launch_k(lc, moe_combine_kernel<f16>, dim3(T), block, 0, a, ep);
  return launch_k(lc, moe_combine_kernel<bf16>, dim3(T), block, 0, a, ep);
}
