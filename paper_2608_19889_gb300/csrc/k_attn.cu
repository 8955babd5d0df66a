// Causal grouped-query attention over the block-structured KV cache
// (Attention.attention + Masking.causal_mask; the scale 1/sqrt(d) of the
// scale_heads listing; Sec. Built-In Libraries).
//
// Cache layout (both contiguous and paged): per layer a pool of 16-token
// blocks [num_blocks][G][16][d], so one (block, kv head) tile is 16*d
// contiguous elements. A sequence's logical block j is block_table[b][j]
// (paged) or b*blocks_per_seq + j (contiguous).
//
// One warp works on 16 "rows" that share a KV head: for decode the H/G query
// heads of one token (padded to 16), for prefill PW positions x H/G heads.
// Q stays in registers as mma.sync A fragments; each 16-key tile is staged in
// shared memory (16-byte chunks XOR-swizzled by row so ldmatrix is
// conflict-free), S = Q K^T and O += P V run on m16n8k16 bf16 tensor-core
// MMAs with fp32 accumulation, and the softmax is the online (running max,
// running sum) form with warp-shuffle row reductions.
//
// Decode splits each sequence's keys over `splits` CTAs (x 4 warps); the
// last CTA of a (sequence, kv head) to finish -- found with an atomic ticket,
// no waiting -- merges the partial (max, sum, O) triples.
#include "attn_tile.cuh"

namespace {

// --------------------------------------------------------------- decode
template <int HD, typename T16>
__global__ void __launch_bounds__(DEC_WARPS * 32) attn_decode_kernel(AttnArgs p) {
  extern __shared__ __align__(128) uint8_t sm[];
  grid_dep_launch();
  grid_dep_wait();
  attn_decode_item<HD, T16, false>(p, blockIdx.x, blockIdx.y, blockIdx.z, sm, threadIdx.x);
}

// -------------------------------------------------------------- prefill
// CTA: 4 warps x PW positions x (H/G) heads of one kv head g of sequence b;
// key tiles staged 4 blocks (64 keys) at a time, double-buffered, shared by
// the 4 warps.
template <int HD, typename T16>
__global__ void __launch_bounds__(128) attn_prefill_kernel(AttnArgs p, int PW, AttnVarlen vl) {
  extern __shared__ __align__(128) uint8_t sm[];
  constexpr int TILE = 16 * HD * 2;
  constexpr int STAGE = 4 * 2 * TILE;  // 4 blocks x (K, V)
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, r = lane >> 2, q = lane & 3;
  const int HPG = p.H / p.G;
  const int PC = 4 * PW;
  // grid (kv head, position block, sequence), position blocks counted down
  // from the end: under the causal mask the last blocks carry the most keys,
  // and dispatching them first keeps the tail of the launch short.
  const int b = blockIdx.z, g = blockIdx.x, p0 = (gridDim.y - 1 - blockIdx.y) * PC;
  grid_dep_launch();
  grid_dep_wait();
  // The sequence's chunk: rows row0 .. row0+S-1 of q / o, at positions
  // past .. past+S-1 (a prompt from an empty cache: past = 0, row0 = b*S).
  int S = p.S, row0 = b * p.S, past = 0;
  if (vl.cu) {
    row0 = vl.cu[b];
    const int row1 = vl.cu[b + 1];
    past = vl.past[b];
    S = row1 - row0;
    // inconsistent offsets (reported by the row-map kernel): no work
    if (row0 < 0 || row1 > vl.rows || S < 0 || S > p.S || past < 0 || past + S > p.blocks_per_seq * 16) S = 0;
  }
  if (p0 >= S) return;

  // local index i of the chunk -> absolute position past + i (or -1: padding)
  auto row_info = [&](int i, int& pos, int& h) {
    const int pl = i / HPG;
    h = i - pl * HPG;
    pos = p0 + warp * PW + pl;
    if (i >= PW * HPG || pos >= S) pos = -1;
  };
  int i0, h0, i1, h1;
  row_info(r, i0, h0);
  row_info(r + 8, i1, h1);
  const int pos0 = i0 >= 0 ? past + i0 : -1, pos1 = i1 >= 0 ? past + i1 : -1;
  const uint16_t* qbase = static_cast<const uint16_t*>(p.q);
  const long long Hd = static_cast<long long>(p.H) * HD;
  const uint16_t* qr0 =
      i0 >= 0 ? qbase + (static_cast<long long>(row0) + i0) * Hd + (g * HPG + h0) * HD : nullptr;
  const uint16_t* qr1 =
      i1 >= 0 ? qbase + (static_cast<long long>(row0) + i1) * Hd + (g * HPG + h1) * HD : nullptr;
  uint32_t qa[HD / 16][4];
  load_q<HD>(qa, qr0, qr1, q);

  WarpState<HD> st;
  st.init();
  // Keys klo .. pend-1 are visible to some row of the CTA (klo > 0 only
  // under a sliding window); staging starts at klo's block.
  const int W = p.window;
  const int pend = past + min(p0 + PC, S);
  const int klo = (W > 0 && past + p0 >= W) ? past + p0 - W + 1 : 0;
  const int jlo = klo >> 4;
  const int nblk = ((pend + 15) >> 4) - jlo;
  const int nst = (nblk + 3) >> 2;
  const int wfirst = p0 + warp * PW;
  const int wmax = past + min(wfirst + PW - 1, S - 1);
  // row lower limits (key index) and the warp's lowest one
  const int lo0 = (W > 0 && pos0 >= W) ? pos0 - W + 1 : 0, lo1 = (W > 0 && pos1 >= W) ? pos1 - W + 1 : 0;
  const int wlo = (W > 0 && past + wfirst >= W) ? past + wfirst - W + 1 : 0;
  const uint32_t base = smem_u32(sm);
  const uint16_t* kp = static_cast<const uint16_t*>(p.k);
  const uint16_t* vp = static_cast<const uint16_t*>(p.v);
  auto issue = [&](int stage_idx, int buf) {
    for (int jj = 0; jj < 4; ++jj) {
      const int j = jlo + stage_idx * 4 + jj;
      if (j >= jlo + nblk) break;
      bool ok;
      const int blk = block_of(p, b, j, ok);
      const long long off = (static_cast<long long>(blk) * p.G + g) * 16 * HD;
      const uint32_t dst = base + buf * STAGE + jj * 2 * TILE;
      stage_tile<HD>(dst, kp + off, ok, threadIdx.x, 128);
      stage_tile<HD>(dst + TILE, vp + off, ok, threadIdx.x, 128);
    }
    cp_async_commit();
  };
  issue(0, 0);
  int buf = 0;
  for (int sidx = 0; sidx < nst; ++sidx) {
    if (sidx + 1 < nst) {
      issue(sidx + 1, buf ^ 1);
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    if (wfirst < S) {
      // blocks in pairs where both are needed (32-key tiles), else singly
      for (int jj = 0; jj < 4;) {
        const int j = jlo + sidx * 4 + jj;
        if (j >= jlo + nblk || j * 16 > wmax) break;
        if (j * 16 + 15 < wlo) {  // slid out of every row of this warp
          ++jj;
          continue;
        }
        const uint32_t t = base + buf * STAGE + jj * 2 * TILE;
        if (jj + 1 < 4 && j + 1 < jlo + nblk && (j + 1) * 16 <= wmax) {
          attn_tile32<HD, T16>(t, t + TILE, t + 2 * TILE, t + 3 * TILE, qa, st, j * 16, lo0, pos0, lo1, pos1,
                               p.scale_log2, lane);
          jj += 2;
        } else {
          attn_tile16<HD, T16>(t, t + TILE, qa, st, j * 16, lo0, pos0, lo1, pos1, p.scale_log2, lane);
          ++jj;
        }
      }
    }
    __syncthreads();
    buf ^= 1;
  }
  st.l0 += __shfl_xor_sync(0xffffffffu, st.l0, 1);
  st.l0 += __shfl_xor_sync(0xffffffffu, st.l0, 2);
  st.l1 += __shfl_xor_sync(0xffffffffu, st.l1, 1);
  st.l1 += __shfl_xor_sync(0xffffffffu, st.l1, 2);
  T16* ob = static_cast<T16*>(p.o);
  const float inv0 = st.l0 > 0.f ? 1.f / st.l0 : 0.f, inv1 = st.l1 > 0.f ? 1.f / st.l1 : 0.f;
#pragma unroll
  for (int nd = 0; nd < HD / 8; ++nd) {
    if (i0 >= 0) {
      T16* d0 = ob + (static_cast<long long>(row0) + i0) * Hd + (g * HPG + h0) * HD + nd * 8 + 2 * q;
      *reinterpret_cast<uint32_t*>(d0) = pack2<T16>(st.o[nd][0] * inv0, st.o[nd][1] * inv0);
    }
    if (i1 >= 0) {
      T16* d1 = ob + (static_cast<long long>(row0) + i1) * Hd + (g * HPG + h1) * HD + nd * 8 + 2 * q;
      *reinterpret_cast<uint32_t*>(d1) = pack2<T16>(st.o[nd][2] * inv1, st.o[nd][3] * inv1);
    }
  }
}

// ------------------------------------------------------- fp32 debug path
// One warp per (row, query head): plain online softmax over visible keys.
__global__ void __launch_bounds__(32) attn_f32_kernel(AttnArgs p, int decode, AttnVarlen vl) {
  grid_dep_launch();
  grid_dep_wait();
  const int m = blockIdx.x, h = blockIdx.y, lane = threadIdx.x;
  const int d = p.d, HPG = p.H / p.G, g = h / HPG;
  int b, pos;
  if (decode) {
    b = m;
    pos = p.ctx[m];
  } else if (vl.rowmap) {
    const int2 rm = vl.rowmap[m];
    b = rm.x;
    pos = rm.y < 0 ? 0 : rm.y;  // unplaced row (already reported): any finite output
  } else {
    b = m / p.S;
    pos = m - b * p.S;
  }
  const int tmax = p.blocks_per_seq * 16;
  if (pos >= tmax) {
    if (lane == 0) set_err(p.err, DEVERR_POS);
    pos = tmax - 1;
  }
  const float* qr = static_cast<const float*>(p.q) + (static_cast<long long>(m) * p.H + h) * d;
  float qv[4], ov[4] = {0.f, 0.f, 0.f, 0.f};
  for (int i = 0; i < 4; ++i) qv[i] = (lane + 32 * i < d) ? qr[lane + 32 * i] : 0.f;
  float mx = NEG_INF, l = 0.f;
  const float* kp = static_cast<const float*>(p.k);
  const float* vp = static_cast<const float*>(p.v);
  const int t0 = (p.window > 0 && pos >= p.window) ? pos - p.window + 1 : 0;
  for (int t = t0; t <= pos; ++t) {
    bool ok;
    const int blk = block_of(p, b, t >> 4, ok);
    if (!ok) continue;
    const long long off = ((static_cast<long long>(blk) * p.G + g) * 16 + (t & 15)) * d;
    float s = 0.f;
    for (int i = 0; i < 4; ++i)
      if (lane + 32 * i < d) s += qv[i] * kp[off + lane + 32 * i];
    s = warp_sum(s) * p.scale_log2;
    const float nm = fmaxf(mx, s);
    const float a = exp2f(mx - nm), e = exp2f(s - nm);
    l = l * a + e;
    for (int i = 0; i < 4; ++i)
      if (lane + 32 * i < d) ov[i] = ov[i] * a + e * vp[off + lane + 32 * i];
    mx = nm;
  }
  float* orow = static_cast<float*>(p.o) + (static_cast<long long>(m) * p.H + h) * d;
  for (int i = 0; i < 4; ++i)
    if (lane + 32 * i < d) orow[lane + 32 * i] = ov[i] / l;
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

template <int HD>
constexpr size_t prefill_smem() { return 2 * 4 * 2 * 16 * HD * 2; }  // 2 stages x 4 blocks x (K, V)

template <int HD>
cudaError_t decode_hd(const LaunchCtx& lc, const AttnArgs& a, int B) {
  const size_t smem = decode_smem<HD>();
  if (lc.f16) return launch_k(lc, attn_decode_kernel<HD, f16>, dim3(a.splits, a.G, B), dim3(DEC_WARPS * 32), smem, a);
  return launch_k(lc, attn_decode_kernel<HD, bf16>, dim3(a.splits, a.G, B), dim3(DEC_WARPS * 32), smem, a);
}

template <int HD>
cudaError_t prefill_hd(const LaunchCtx& lc, const AttnArgs& a, int B, const AttnVarlen& vl) {
  const size_t smem = prefill_smem<HD>();
  const int HPG = a.H / a.G;
  const int PW = 16 / HPG;
  const int PC = 4 * PW;
  const dim3 grid(a.G, (a.S + PC - 1) / PC, B);
  if (lc.f16) return launch_k(lc, attn_prefill_kernel<HD, f16>, grid, dim3(128), smem, a, PW, vl);
  return launch_k(lc, attn_prefill_kernel<HD, bf16>, grid, dim3(128), smem, a, PW, vl);
}

}  // namespace

namespace {
template <typename T16>
cudaError_t prepare_attn_t() {
  cudaError_t e = cudaSuccess;
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attn_decode_kernel<64, T16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)decode_smem<64>());
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attn_decode_kernel<128, T16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)decode_smem<128>());
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attn_prefill_kernel<64, T16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)prefill_smem<64>());
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attn_prefill_kernel<128, T16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)prefill_smem<128>());
  return e;
}
}  // namespace

cudaError_t prepare_attn_kernels() {
  cudaError_t e = prepare_attn_t<bf16>();
  if (e == cudaSuccess) e = prepare_attn_t<f16>();
  return e;
}

int attn_decode_splits(int B, int G, int max_blocks, int num_sms, int target_ctas) {
  const int bg = B * G;
  const int smax = max_blocks < 64 ? max_blocks : 64;
  if (target_ctas > 0) {  // explicit grid budget
    const int want = target_ctas / bg;
    return want < 1 ? 1 : (want > smax ? smax : want);
  }
  // B x G CTAs already cover every SM: no split (with ragged contexts,
  // measured on 64 sequences of 512-4096 tokens, one split beats two).
  if (bg >= num_sms) return 1;
  // One resident CTA per SM (128 KB of staging): choose the split count with
  // the smallest makespan, waves x (key blocks per split + a per-CTA cost of
  // about 4 blocks), where a split holds at least one block per warp.
  int best = 1;
  long long best_cost = -1;
  for (int s = 1; s <= smax; ++s) {
    const int per = max((max_blocks + s - 1) / s, DEC_WARPS);
    const int used = (max_blocks + per - 1) / per;
    if (used < s) break;  // further splits would exit at once
    const long long waves = (static_cast<long long>(bg) * used + num_sms - 1) / num_sms;
    const long long cost = waves * (per + 4);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best = s;
    }
  }
  return best;
}

cudaError_t launch_attn_decode(const LaunchCtx& lc, bool fp32, const AttnArgs& a, int B) {
  if (fp32) return launch_k(lc, attn_f32_kernel, dim3(B, a.H), dim3(32), 0, a, 1, AttnVarlen{});
  if (a.H / a.G > 16) return cudaErrorInvalidValue;
  if (a.d == 64) return decode_hd<64>(lc, a, B);
  if (a.d == 128) return decode_hd<128>(lc, a, B);
  return cudaErrorInvalidValue;
}

cudaError_t launch_attn_prefill(const LaunchCtx& lc, bool fp32, const AttnArgs& a, int B, const AttnVarlen* vl) {
  const AttnVarlen v = vl ? *vl : AttnVarlen{};
  if (fp32) return launch_k(lc, attn_f32_kernel, dim3(vl ? v.rows : B * a.S, a.H), dim3(32), 0, a, 0, v);
  if (a.H / a.G > 16) return cudaErrorInvalidValue;
  if (a.d == 64) return prefill_hd<64>(lc, a, B, v);
  if (a.d == 128) return prefill_hd<128>(lc, a, B, v);
  return cudaErrorInvalidValue;
}
