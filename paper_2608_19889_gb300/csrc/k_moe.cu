// Mixture-of-experts MLP (the MoE built-ins' softmax top-k router and
// grouped experts; the stacked-experts formulation that the paper's graph
// rewriting puts in place of a loop over experts):
//
//   [router logits: the decode GEMV or the tcgen05 GEMM with the LOGITS
//    epilogue (norm scale applied), fp32 [T][E]]
//   moe_route_kernel    per token: softmax of the router logits, top-k
//                       (lowest index on ties), weights (optionally
//                       renormalised); for few tokens the plan kernel's
//                       CTA does this itself;
//   moe_plan_kernel     one CTA: a stable counting sort of the T x k
//                       (token, expert) slots by expert into segments padded
//                       to 128-row blocks: the sorted row of every slot, the
//                       token and weight of every sorted row (token -1 for
//                       padding), the expert of every 128-row block and the
//                       block count -- the grouped GEMM's tile list;
//   moe_gather_kernel   the sorted operand rows: the normalised input
//                       h = (a [+ a_lo]) * r, rounded once to 16 bits;
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
// Token counts up to which one CTA both routes and sorts (the decode path).
constexpr int FUSED_ROUTE_MAX_T = 256;

// Token t: softmax of its router logits, top-k by repeated arg-max over
// (probability, lowest index), the weights (renormalised over the k chosen
// when norm_topk). One warp; lg is the warp's [E] scratch.
AXON_DEV void route_token(const MoeArgs& a, int t, float* lg, int lane) {
  const int E = a.E, k = a.k;
  __syncwarp();
  for (int e = lane; e < E; e += 32) lg[e] = a.logits[static_cast<long long>(t) * E + e];
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

// One warp per token (many tokens: prefill).
__global__ void __launch_bounds__(ROUTE_THREADS) moe_route_kernel(MoeArgs a, int T) {
  grid_dep_launch();
  grid_dep_wait();
  extern __shared__ float sh[];  // [warps][E]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t = blockIdx.x * (ROUTE_THREADS / 32) + warp;
  if (t < T) route_token(a, t, sh + warp * a.E, lane);
}

// Stable counting sort of the n = T * k slots by expert, in rounds of
// PLAN_THREADS slots: within a warp, slots of one expert are ranked by
// lane (match_any), warps are ranked in order by a per-expert prefix over
// the round's warp counts, rounds in order by the running counts.
// With ROUTE, the CTA's warps first route the T tokens themselves (the
// per-warp scratch is the count table, unused until then).
template <bool ROUTE>
__global__ void __launch_bounds__(PLAN_THREADS) moe_plan_kernel(MoeArgs a, int T) {
  grid_dep_launch();
  grid_dep_wait();
  __shared__ int cnt[MOE_MAX_EXPERTS];
  __shared__ int seg[MOE_MAX_EXPERTS];
  __shared__ int wcnt[PLAN_THREADS / 32][MOE_MAX_EXPERTS];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int E = a.E, n = T * a.k;
  if (ROUTE) {
    for (int t = warp; t < T; t += PLAN_THREADS / 32) route_token(a, t, reinterpret_cast<float*>(wcnt[warp]), lane);
    __syncthreads();
  }
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

// Sorted operand rows: slot i = (token t, j) goes to row slot_row[i] as the
// normalised input h = (a [+ a_lo]) * r of token t, rounded once to 16 bits.
// Padding rows are left as they are: a row of the grouped GEMMs' operand
// only reaches its own output row, which the epilogues skip. One warp per
// slot, 8 elements per lane step.
template <typename T16>
__global__ void __launch_bounds__(256) moe_gather_kernel(MoeArgs a, int T, EpiArgs ns) {
  grid_dep_launch();
  grid_dep_wait();
  const int n = T * a.k, per_row = a.D / 8;
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  const int nwarps = (gridDim.x * blockDim.x) >> 5;
  for (int i = warp; i < n; i += nwarps) {
    const int row = a.slot_row[i];
    if (row < 0) continue;
    const int t = i / a.k;
    const float r = row_rinv(ns, t);
    const uint4* sh = reinterpret_cast<const uint4*>(static_cast<const T16*>(a.act) + t * a.act_stride);
    const uint4* sl = a.act_lo ? reinterpret_cast<const uint4*>(static_cast<const T16*>(a.act_lo) + t * a.act_stride)
                               : nullptr;
    uint4* dh = reinterpret_cast<uint4*>(static_cast<T16*>(a.a_sorted) + static_cast<long long>(row) * a.D);
    for (int c = lane; c < per_row; c += 32) {
      const uint4 hv = sh[c];
      const T16* h8 = reinterpret_cast<const T16*>(&hv);
      float v[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) v[q] = to_f(h8[q]);
      if (sl) {
        const uint4 lv = sl[c];
        const T16* l8 = reinterpret_cast<const T16*>(&lv);
#pragma unroll
        for (int q = 0; q < 8; ++q) v[q] += to_f(l8[q]);
      }
      uint4 o;
      T16* o8 = reinterpret_cast<T16*>(&o);
#pragma unroll
      for (int q = 0; q < 8; ++q) o8[q] = from_f<T16>(v[q] * r);
      dh[c] = o;
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
  (void)D;
  (void)E;
  return cudaSuccess;
}

cudaError_t launch_moe_route_plan(const LaunchCtx& lc, const MoeArgs& a, int T) {
  if (T < 1 || a.k < 1 || a.k > 8 || a.k > a.E || a.E > MOE_MAX_EXPERTS) return cudaErrorInvalidValue;
  if (T <= FUSED_ROUTE_MAX_T) return launch_k(lc, moe_plan_kernel<true>, dim3(1), dim3(PLAN_THREADS), 0, a, T);
  const int warps = ROUTE_THREADS / 32;
  const size_t smem = static_cast<size_t>(warps) * a.E * 4;
  cudaError_t e = launch_k(lc, moe_route_kernel, dim3((T + warps - 1) / warps), dim3(ROUTE_THREADS), smem, a, T);
  if (e != cudaSuccess) return e;
  return launch_k(lc, moe_plan_kernel<false>, dim3(1), dim3(PLAN_THREADS), 0, a, T);
}

cudaError_t launch_moe_gather(const LaunchCtx& lc, const MoeArgs& a, int T, const EpiArgs& ns) {
  if (a.D % 8) return cudaErrorInvalidValue;
  const long long warps = static_cast<long long>(T) * a.k;
  const int grid = static_cast<int>(std::min<long long>((warps + 7) / 8, 4LL * lc.num_sms));
  if (lc.f16) return launch_k(lc, moe_gather_kernel<f16>, dim3(grid), dim3(256), 0, a, T, ns);
  return launch_k(lc, moe_gather_kernel<bf16>, dim3(grid), dim3(256), 0, a, T, ns);
}

cudaError_t launch_moe_combine(const LaunchCtx& lc, const MoeArgs& a, int T, const EpiArgs& ep) {
  if (a.D % 16 || a.D / 16 > 1024) return cudaErrorInvalidValue;
  const dim3 block((a.D / 16 + 31) / 32 * 32);
  if (lc.f16) return launch_k(lc, moe_combine_kernel<f16>, dim3(T), block, 0, a, ep);
  return launch_k(lc, moe_combine_kernel<bf16>, dim3(T), block, 0, a, ep);
}
