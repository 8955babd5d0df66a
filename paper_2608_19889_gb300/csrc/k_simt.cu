// fp32 debug projections: a plain shared-memory-tiled CUDA-core GEMM
// (64x64 tile, 4x4 outputs per thread) followed by the same fused
// epilogues as the tensor-core paths, on fp32 activations, weights and
// cache. Used only in AXON_FP32_DEBUG mode, where exactness matters and
// speed does not.
#include "kernels.h"

namespace {

constexpr int TM = 64, TN = 64, TK = 16;

template <int KIND>
__global__ void __launch_bounds__(256) gemm_simt_kernel(const float* __restrict__ A, long long a_stride,
                                                        const float* __restrict__ W, int M, int N, int K, EpiArgs ep) {
  __shared__ float As[TK][TM + 1];
  __shared__ float Ws[TK][TN + 1];
  __shared__ float C[TM][TN + 1];
  grid_dep_wait();
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const int m0 = blockIdx.y * TM, n0 = blockIdx.x * TN;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += TK) {
    for (int i = threadIdx.x; i < TM * TK; i += 256) {
      const int mm = i / TK, kk = i % TK;
      const int gm = m0 + mm, gk = k0 + kk;
      As[kk][mm] = (gm < M && gk < K) ? A[static_cast<long long>(gm) * a_stride + gk] : 0.f;
      const int gn = n0 + mm;
      Ws[kk][mm] = (gn < N && gk < K) ? W[static_cast<long long>(gn) * K + gk] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < TK; ++kk) {
      float a[4], w[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        a[i] = As[kk][ty * 4 + i];
        w[i] = Ws[kk][tx * 4 + i];
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], w[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) C[ty * 4 + i][tx * 4 + j] = acc[i][j];
  __syncthreads();
  grid_dep_launch();
  // Epilogue: thread -> (row, 16-column chunk).
  const int row = threadIdx.x >> 2, chunk = threadIdx.x & 3;
  const int m = m0 + row, nc = n0 + chunk * 16;
  if (m >= M || nc >= N) return;
  float v[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = C[row][chunk * 16 + i];
  if (KIND == EPI_QKV) {
    epi_qkv16<float>(ep, m, nc, v, row_rinv(ep, m));
  } else if (KIND == EPI_RESID) {
    const float s = epi_resid16<float>(ep, m, nc, v);
    ep.ss_out[static_cast<long long>(m) * ep.ss_out_stride + nc / 16] = s;
  } else if (KIND == EPI_SWIGLU) {
    epi_swiglu16<float>(ep, m, nc, v, row_rinv(ep, m));
  } else {
    argmax_commit(ep.keys + m, epi_logits16(ep, m, nc, v, row_rinv(ep, m)));
  }
}

template <int KIND>
cudaError_t launch_kind(const LaunchCtx& lc, const float* A, long long a_stride, const float* W, int M, int N, int K,
                        const EpiArgs& ep) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((N + TN - 1) / TN, (M + TM - 1) / TM);
  cfg.blockDim = dim3(256);
  cfg.stream = lc.stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = lc.pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, gemm_simt_kernel<KIND>, A, a_stride, W, M, N, K, ep);
}

}  // namespace

cudaError_t launch_gemm_simt(const LaunchCtx& lc, int kind, const float* A, long long a_stride, const float* W, int M,
                             int N, int K, const EpiArgs& ep) {
  if (M < 1 || N < 1 || K < 1) return cudaErrorInvalidValue;
  switch (kind) {
    case EPI_QKV: return launch_kind<EPI_QKV>(lc, A, a_stride, W, M, N, K, ep);
    case EPI_RESID: return launch_kind<EPI_RESID>(lc, A, a_stride, W, M, N, K, ep);
    case EPI_SWIGLU: return launch_kind<EPI_SWIGLU>(lc, A, a_stride, W, M, N, K, ep);
    default: return launch_kind<EPI_LOGITS>(lc, A, a_stride, W, M, N, K, ep);
  }
}
