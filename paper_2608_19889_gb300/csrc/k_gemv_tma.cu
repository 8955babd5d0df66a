// Decode projections, TMA-fed: out[b][n] = act[b] . W[n] for B <= 64 tokens,
// a persistent stream-K kernel with one CTA per SM.
//
//   * Work = (row block of 128 weight rows) x (64-wide k stage); the
//     RB * KB iterations are cut into equal contiguous ranges, one per CTA,
//     so every SM streams the same number of bytes whatever N and K are.
//   * Warp 8 is the producer: one lane issues, per iteration, a TMA load of
//     the 128x64 weight tile and of the 64-wide activation tile (TOK token
//     rows) into an NSTAGE-deep shared-memory ring (128-byte swizzle),
//     completion tracked by mbarrier transaction bytes. Weight tiles for the
//     first stages are requested before griddepcontrol.wait: they do not
//     depend on the previous kernel.
//   * Warps 0..7 consume: warp w owns rows 16w..16w+15 of the row block,
//     reads A (weights) and B (tokens) fragments with ldmatrix and
//     accumulates with mma.sync m16n8k16 (bf16 in, fp32 out).
//   * A row block split between CTAs leaves partial tiles; per 16-row warp
//     slice, the last contributor to arrive (atomic ticket, no waiting) sums
//     the partials in CTA order -- deterministic -- and runs the fused
//     epilogue. Residual producers also reduce each token's sum of squares
//     into the inverse RMS of the next norm (last slice to finish).
// Every mbarrier wait is bounded (DEVERR_TIMEOUT instead of a hang).
#include "kernels.h"

namespace {

constexpr int CW = 8;              // consumer warps
constexpr int ROWS = 16 * CW;      // weight rows per row block
constexpr int KST = 64;            // k per stage
constexpr int W_BYTES = ROWS * KST * 2;
constexpr int NTHREADS = (CW + 1) * 32;

template <int NT>
struct Cfg {
  static constexpr int TOK = 8 * NT;
  static constexpr int A_BYTES = TOK * KST * 2;
  static constexpr int NSTAGE = NT <= 2 ? 8 : (NT == 4 ? 7 : 6);
  static constexpr int STAGE = W_BYTES + A_BYTES;
  static constexpr int EPI_FLOATS = CW * 16 * (TOK + 1);
  static constexpr int SMEM = NSTAGE * STAGE + EPI_FLOATS * 4 + 16 * NSTAGE + 1024;
};

struct StreamK {
  float* part;        // [grid][2][ROWS][64]
  int* slice_ticket;  // [row blocks][CW], zero between launches
  int* rinv_ticket;   // [1]
};

// CTA range of iteration t for `grid` CTAs over T iterations (ranges
// [floor(i*T/grid), floor((i+1)*T/grid))).
AXON_DEV int cta_of(long long t, long long T, int grid) {
  return static_cast<int>(((t + 1) * grid - 1) / T);
}
AXON_DEV long long range_begin(int i, long long T, int grid) { return (static_cast<long long>(i) * T) / grid; }

AXON_DEV uint32_t swz128(uint32_t base, int row, int chunk) {
  return base + row * 128 + ((chunk ^ (row & 7)) << 4);
}

template <int NT, int KIND>
__global__ void __launch_bounds__(NTHREADS, 1)
    gemv_tma_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmA, int N, int K,
                    int B, EpiArgs ep, StreamK sk) {
  using C = Cfg<NT>;
  constexpr int TOK = C::TOK;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* base_ptr = smem_raw + (base - raw);
  float* epi = reinterpret_cast<float*>(base_ptr + C::NSTAGE * C::STAGE);
  const uint32_t bars = base + C::NSTAGE * C::STAGE + C::EPI_FLOATS * 4;
  auto full_bar = [&](int s) { return bars + 8 * s; };
  auto empty_bar = [&](int s) { return bars + 8 * (C::NSTAGE + s); };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NSTAGE; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), CW);
    }
    fence_mbar_init();
    fence_proxy_async();
  }
  __syncthreads();
  grid_dep_launch();

  const int RB = (N + ROWS - 1) / ROWS;
  const int KB = K / KST;
  const long long T = static_cast<long long>(RB) * KB;
  const int grid = gridDim.x;
  const long long beg = range_begin(blockIdx.x, T, grid), end = range_begin(blockIdx.x + 1, T, grid);

  if (warp == CW) {
    // ---------------- producer
    if (lane == 0) {
      tma_prefetch_desc(&tmW);
      tma_prefetch_desc(&tmA);
      const long long pre_end = (end - beg < C::NSTAGE) ? end : beg + C::NSTAGE;
      for (long long t = beg; t < pre_end; ++t) {
        const int s = static_cast<int>((t - beg) % C::NSTAGE);
        const int u = static_cast<int>(t / KB), kb = static_cast<int>(t % KB);
        mbar_arrive_expect_tx(full_bar(s), C::STAGE);
        tma_load_2d(base + s * C::STAGE, &tmW, full_bar(s), kb * KST, u * ROWS);
      }
      grid_dep_wait();
      for (long long t = beg; t < pre_end; ++t) {
        const int s = static_cast<int>((t - beg) % C::NSTAGE);
        const int kb = static_cast<int>(t % KB);
        tma_load_2d(base + s * C::STAGE + W_BYTES, &tmA, full_bar(s), kb * KST, 0);
      }
      for (long long t = pre_end; t < end; ++t) {
        const long long it = t - beg;
        const int s = static_cast<int>(it % C::NSTAGE);
        const uint32_t ph = static_cast<uint32_t>((it / C::NSTAGE) & 1);
        if (!mbar_wait(empty_bar(s), ph ^ 1, ep.err)) break;
        const int u = static_cast<int>(t / KB), kb = static_cast<int>(t % KB);
        mbar_arrive_expect_tx(full_bar(s), C::STAGE);
        tma_load_2d(base + s * C::STAGE, &tmW, full_bar(s), kb * KST, u * ROWS);
        tma_load_2d(base + s * C::STAGE + W_BYTES, &tmA, full_bar(s), kb * KST, 0);
      }
    }
    __syncwarp();
    return;
  }

  // ---------------- consumers
  grid_dep_wait();
  const int r = lane >> 2, q = lane & 3;
  float* my_epi = epi + warp * 16 * (TOK + 1);
  float acc[NT][4];
  long long seg_start = beg;
  bool first_seg = true;
  for (long long t = beg; t < end; ++t) {
    const long long it = t - beg;
    const int s = static_cast<int>(it % C::NSTAGE);
    const uint32_t ph = static_cast<uint32_t>((it / C::NSTAGE) & 1);
    const int u = static_cast<int>(t / KB), kb = static_cast<int>(t % KB);
    if (t == seg_start) {
#pragma unroll
      for (int n = 0; n < NT; ++n) acc[n][0] = acc[n][1] = acc[n][2] = acc[n][3] = 0.f;
    }
    if (!mbar_wait(full_bar(s), ph, ep.err)) break;
    const uint32_t ws = base + s * C::STAGE, as = ws + W_BYTES;
#pragma unroll
    for (int kk = 0; kk < KST / 16; ++kk) {
      uint32_t a[4];
      ldsm_x4(a, swz128(ws, warp * 16 + (lane & 15), 2 * kk + (lane >> 4)));
#pragma unroll
      for (int n2 = 0; n2 < (NT + 1) / 2; ++n2) {
        // x4: (tokens n2*16+0..7, k lo), (same, k hi), (tokens +8..15, k lo), (+8..15, k hi)
        uint32_t bfr[4];
        const int mi = lane >> 3, li = lane & 7;
        const int tok = n2 * 16 + (mi >> 1) * 8 + li;
        ldsm_x4(bfr, swz128(as, tok < TOK ? tok : 0, 2 * kk + (mi & 1)));
        {
          const uint32_t b0[2] = {bfr[0], bfr[1]};
          mma_bf16_16816(acc[2 * n2], a, b0);
        }
        if (2 * n2 + 1 < NT) {
          const uint32_t b1[2] = {bfr[2], bfr[3]};
          mma_bf16_16816(acc[2 * n2 + 1], a, b1);
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(empty_bar(s));

    const bool seg_end = (kb == KB - 1) || (t == end - 1);
    if (!seg_end) continue;
    // ---- a segment of row block u ends here
    const bool complete = (seg_start == static_cast<long long>(u) * KB) && (kb == KB - 1);
    const int slice_row0 = u * ROWS + warp * 16;
    bool do_epi = true;
    if (complete) {
#pragma unroll
      for (int n = 0; n < NT; ++n) {
        my_epi[r * (TOK + 1) + n * 8 + 2 * q] = acc[n][0];
        my_epi[r * (TOK + 1) + n * 8 + 2 * q + 1] = acc[n][1];
        my_epi[(r + 8) * (TOK + 1) + n * 8 + 2 * q] = acc[n][2];
        my_epi[(r + 8) * (TOK + 1) + n * 8 + 2 * q + 1] = acc[n][3];
      }
    } else {
      // publish this warp's partial slice, then see whether it completes the slice
      const int slot = first_seg ? 0 : 1;
      float* mine = sk.part + ((static_cast<long long>(blockIdx.x) * 2 + slot) * ROWS + warp * 16) * 64;
#pragma unroll
      for (int n = 0; n < NT; ++n) {
        mine[r * 64 + n * 8 + 2 * q] = acc[n][0];
        mine[r * 64 + n * 8 + 2 * q + 1] = acc[n][1];
        mine[(r + 8) * 64 + n * 8 + 2 * q] = acc[n][2];
        mine[(r + 8) * 64 + n * 8 + 2 * q + 1] = acc[n][3];
      }
      __threadfence();
      __syncwarp();
      const int i_first = cta_of(static_cast<long long>(u) * KB, T, grid);
      const int i_last = cta_of(static_cast<long long>(u) * KB + KB - 1, T, grid);
      const int count = i_last - i_first + 1;
      int last = 0;
      if (lane == 0) last = (atomicAdd(sk.slice_ticket + u * CW + warp, 1) == count - 1);
      last = __shfl_sync(0xffffffffu, last, 0);
      do_epi = last != 0;
      if (do_epi) {
        __threadfence();
        // Sum the contributors' slices in CTA order (fixed order: deterministic);
        // eight contributors' loads are in flight at a time.
        const long long u0 = static_cast<long long>(u) * KB;
        auto slice_src = [&](int i) {
          const int slot_i = (i == i_first && range_begin(i, T, grid) < u0) ? 1 : 0;
          return sk.part + ((static_cast<long long>(i) * 2 + slot_i) * ROWS + warp * 16) * 64;
        };
        for (int e = lane; e < 16 * TOK; e += 32) {
          const int off = (e / TOK) * 64 + (e % TOK);
          float sum = 0.f;
          int i = i_first;
          for (; i + 8 <= i_last + 1; i += 8) {
            float v[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) v[j] = __ldcg(slice_src(i + j) + off);
#pragma unroll
            for (int j = 0; j < 8; ++j) sum += v[j];
          }
          for (; i <= i_last; ++i) sum += __ldcg(slice_src(i) + off);
          my_epi[(e / TOK) * (TOK + 1) + (e % TOK)] = sum;
        }
        if (lane == 0) sk.slice_ticket[u * CW + warp] = 0;
      }
    }
    first_seg = false;
    seg_start = t + 1;
    if (!do_epi) continue;
    __syncwarp();
    for (int b = lane; b < B; b += 32) {
      if (slice_row0 >= N) break;
      float v[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) v[i] = my_epi[i * (TOK + 1) + b];
      if (KIND == EPI_QKV) {
        epi_qkv16<bf16>(ep, b, slice_row0, v, row_rinv(ep, b));
      } else if (KIND == EPI_RESID) {
        const float ssum = epi_resid16<bf16>(ep, b, slice_row0, v);
        ep.ss_out[static_cast<long long>(b) * ep.ss_out_stride + slice_row0 / 16] = ssum;
      } else if (KIND == EPI_SWIGLU) {
        epi_swiglu16<bf16>(ep, b, slice_row0, v, row_rinv(ep, b));
      } else {
        argmax_commit(ep.keys + b, epi_logits16(ep, b, slice_row0, v, row_rinv(ep, b)));
      }
    }
    __syncwarp();
    if (KIND == EPI_RESID && ep.rinv_out && slice_row0 < N) {
      // The warp finishing the last 16-row slice reduces every token's
      // partial sums of squares into the next norm's inverse RMS.
      const int nslices = (N + 15) / 16;
      __threadfence();
      int last = 0;
      if (lane == 0) last = (atomicAdd(sk.rinv_ticket, 1) == nslices - 1);
      last = __shfl_sync(0xffffffffu, last, 0);
      if (last) {
        __threadfence();
        for (int b = 0; b < B; ++b) {
          const float* p = ep.ss_out + static_cast<long long>(b) * ep.ss_out_stride;
          float sum = 0.f;
          for (int i = lane; i < nslices; i += 32) sum += __ldcg(p + i);
          sum = warp_sum(sum);
          if (lane == 0) ep.rinv_out[b] = 1.0f / sqrtf(sum * ep.inv_D + ep.eps);
        }
        if (lane == 0) *sk.rinv_ticket = 0;
      }
    }
  }
}

template <int NT, int KIND>
cudaError_t launch_one(const LaunchCtx& lc, const CUtensorMap& w, const CUtensorMap& a, int N, int K, int B,
                       const EpiArgs& ep, const StreamK& sk) {
  // At least MIN_ITERS k-stages per CTA, so that no 16-row slice collects
  // partial sums from more than a handful of CTAs.
  constexpr long long MIN_ITERS = 4;
  const long long T = static_cast<long long>((N + ROWS - 1) / ROWS) * (K / KST);
  long long want = (T + MIN_ITERS - 1) / MIN_ITERS;
  if (want > lc.num_sms) want = lc.num_sms;
  const int grid = static_cast<int>(want < 1 ? 1 : want);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(NTHREADS);
  cfg.dynamicSmemBytes = Cfg<NT>::SMEM;
  cfg.stream = lc.stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = lc.pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, gemv_tma_kernel<NT, KIND>, w, a, N, K, B, ep, sk);
}

template <int NT>
cudaError_t launch_nt(const LaunchCtx& lc, int kind, const CUtensorMap& w, const CUtensorMap& a, int N, int K, int B,
                      const EpiArgs& ep, const StreamK& sk) {
  switch (kind) {
    case EPI_QKV: return launch_one<NT, EPI_QKV>(lc, w, a, N, K, B, ep, sk);
    case EPI_RESID: return launch_one<NT, EPI_RESID>(lc, w, a, N, K, B, ep, sk);
    case EPI_SWIGLU: return launch_one<NT, EPI_SWIGLU>(lc, w, a, N, K, B, ep, sk);
    default: return launch_one<NT, EPI_LOGITS>(lc, w, a, N, K, B, ep, sk);
  }
}

template <int NT>
cudaError_t prepare_nt() {
  cudaError_t e = cudaSuccess;
  const int smem = Cfg<NT>::SMEM;
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(gemv_tma_kernel<NT, EPI_QKV>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(gemv_tma_kernel<NT, EPI_RESID>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(gemv_tma_kernel<NT, EPI_SWIGLU>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(gemv_tma_kernel<NT, EPI_LOGITS>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  return e;
}

}  // namespace

int gemv_tma_tokens(int B) { return B <= 8 ? 8 : (B <= 16 ? 16 : (B <= 32 ? 32 : 64)); }

cudaError_t prepare_gemv_tma_kernels() {
  cudaError_t e = prepare_nt<1>();
  if (e == cudaSuccess) e = prepare_nt<2>();
  if (e == cudaSuccess) e = prepare_nt<4>();
  if (e == cudaSuccess) e = prepare_nt<8>();
  return e;
}

cudaError_t launch_gemv_tma(const LaunchCtx& lc, int kind, const CUtensorMap& w, const CUtensorMap& a, int N, int K,
                            int B, const EpiArgs& ep, const GemvTmaWork& wk) {
  if (B < 1 || B > 64 || (K % KST) || N < 1) return cudaErrorInvalidValue;
  if ((N + ROWS - 1) / ROWS > wk.max_row_blocks || lc.num_sms > wk.max_grid) return cudaErrorInvalidValue;
  const StreamK sk{wk.part, wk.slice_ticket, wk.rinv_ticket};
  if (B <= 8) return launch_nt<1>(lc, kind, w, a, N, K, B, ep, sk);
  if (B <= 16) return launch_nt<2>(lc, kind, w, a, N, K, B, ep, sk);
  if (B <= 32) return launch_nt<4>(lc, kind, w, a, N, K, B, ep, sk);
  return launch_nt<8>(lc, kind, w, a, N, K, B, ep, sk);
}
