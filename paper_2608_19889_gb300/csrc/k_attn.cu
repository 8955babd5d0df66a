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
#include "kernels.h"

#include <math.h>

namespace {

constexpr float NEG_INF = -INFINITY;
constexpr int DEC_WARPS = 8;  // warps per decode CTA (one key block each per round)

template <int HD>
AXON_DEV uint32_t swz(uint32_t base, int tok, int ch) {
  return base + tok * (HD * 2) + ((ch ^ (tok & 7)) << 4);
}

// Copy one (block, kv head) tile of 16 x HD bf16 into swizzled shared memory
// with `nthreads` cooperating threads starting at `tid`.
template <int HD>
AXON_DEV void stage_tile(uint32_t dst, const uint16_t* src, bool valid, int tid, int nthreads) {
  constexpr int CH = HD / 8;
  for (int c = tid; c < 16 * CH; c += nthreads) {
    const int tok = c / CH, ch = c % CH;
    cp_async16_zfill(swz<HD>(dst, tok, ch), valid ? src + tok * HD + ch * 8 : src, valid);
  }
}

template <int HD>
AXON_DEV void load_q(uint32_t (&qa)[HD / 16][4], const uint16_t* row0, const uint16_t* row1, int q) {
#pragma unroll
  for (int kk = 0; kk < HD / 16; ++kk) {
    const int k = kk * 16 + 2 * q;
    qa[kk][0] = row0 ? *reinterpret_cast<const uint32_t*>(row0 + k) : 0u;
    qa[kk][1] = row1 ? *reinterpret_cast<const uint32_t*>(row1 + k) : 0u;
    qa[kk][2] = row0 ? *reinterpret_cast<const uint32_t*>(row0 + k + 8) : 0u;
    qa[kk][3] = row1 ? *reinterpret_cast<const uint32_t*>(row1 + k + 8) : 0u;
  }
}

template <int HD>
struct WarpState {
  float m0, m1, l0, l1;
  float o[HD / 8][4];
  AXON_DEV void init() {
    m0 = m1 = NEG_INF;
    l0 = l1 = 0.f;
#pragma unroll
    for (int i = 0; i < HD / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  }
};

// One 16-key tile: keys tok0 .. tok0+15; key t is visible to row r (r+8)
// iff t <= lim0 (lim1).
template <int HD, typename T16>
AXON_DEV void attn_tile16(uint32_t ks, uint32_t vs, const uint32_t (&qa)[HD / 16][4], WarpState<HD>& st, int tok0,
                          int lim0, int lim1, float sl2, int lane) {
  const int q = lane & 3;
  const int mi = lane >> 3, li = lane & 7;
  float s[2][4];
#pragma unroll
  for (int i = 0; i < 2; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
#pragma unroll
  for (int kk = 0; kk < HD / 16; ++kk) {
    uint32_t kb[4];
    const int tok = (mi >> 1) * 8 + li, ch = 2 * kk + (mi & 1);
    ldsm_x4(kb, swz<HD>(ks, tok, ch));
    const uint32_t b0[2] = {kb[0], kb[1]}, b1[2] = {kb[2], kb[3]};
    mma16816<T16>(s[0], qa[kk], b0);
    mma16816<T16>(s[1], qa[kk], b1);
  }
  float mx0 = NEG_INF, mx1 = NEG_INF;
#pragma unroll
  for (int nt = 0; nt < 2; ++nt) {
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const int t = tok0 + nt * 8 + 2 * q + e;
      s[nt][e] = (t <= lim0) ? s[nt][e] * sl2 : NEG_INF;
      s[nt][2 + e] = (t <= lim1) ? s[nt][2 + e] * sl2 : NEG_INF;
      mx0 = fmaxf(mx0, s[nt][e]);
      mx1 = fmaxf(mx1, s[nt][2 + e]);
    }
  }
  mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
  mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
  mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
  mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
  const float nm0 = fmaxf(st.m0, mx0), nm1 = fmaxf(st.m1, mx1);
  const float base0 = (nm0 == NEG_INF) ? 0.f : nm0, base1 = (nm1 == NEG_INF) ? 0.f : nm1;
  const float a0 = exp2f(st.m0 - base0), a1 = exp2f(st.m1 - base1);
  float ps0 = 0.f, ps1 = 0.f;
#pragma unroll
  for (int nt = 0; nt < 2; ++nt) {
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      s[nt][e] = exp2f(s[nt][e] - base0);
      s[nt][2 + e] = exp2f(s[nt][2 + e] - base1);
      ps0 += s[nt][e];
      ps1 += s[nt][2 + e];
    }
  }
  st.l0 = st.l0 * a0 + ps0;
  st.l1 = st.l1 * a1 + ps1;
  st.m0 = nm0;
  st.m1 = nm1;
#pragma unroll
  for (int nd = 0; nd < HD / 8; ++nd) {
    st.o[nd][0] *= a0;
    st.o[nd][1] *= a0;
    st.o[nd][2] *= a1;
    st.o[nd][3] *= a1;
  }
  const uint32_t pa[4] = {pack2<T16>(s[0][0], s[0][1]), pack2<T16>(s[0][2], s[0][3]),
                          pack2<T16>(s[1][0], s[1][1]), pack2<T16>(s[1][2], s[1][3])};
#pragma unroll
  for (int nd2 = 0; nd2 < HD / 16; ++nd2) {
    uint32_t vb[4];
    const int tok = (mi & 1) * 8 + li, ch = 2 * nd2 + (mi >> 1);
    ldsm_x4_t(vb, swz<HD>(vs, tok, ch));
    const uint32_t b0[2] = {vb[0], vb[1]}, b1[2] = {vb[2], vb[3]};
    mma16816<T16>(st.o[2 * nd2], pa, b0);
    mma16816<T16>(st.o[2 * nd2 + 1], pa, b1);
  }
}

AXON_DEV int block_of(const AttnArgs& p, int b, int j, bool& ok) {
  const int blk = p.block_table ? p.block_table[static_cast<long long>(b) * p.bt_stride + j] : b * p.blocks_per_seq + j;
  ok = blk >= 0 && blk < p.num_blocks;
  if (!ok) set_err(p.err, DEVERR_BLOCK);
  return ok ? blk : 0;
}

// --------------------------------------------------------------- decode
template <int HD, typename T16>
__global__ void __launch_bounds__(DEC_WARPS * 32) attn_decode_kernel(AttnArgs p) {
  extern __shared__ __align__(128) uint8_t sm[];
  constexpr int TILE = 16 * HD * 2;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, r = lane >> 2, q = lane & 3;
  const int s = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int HPG = p.H / p.G;
  grid_dep_launch();
  grid_dep_wait();

  int T = p.ctx[b] + 1;
  const int tmax = p.blocks_per_seq * 16;
  if (T > tmax) {
    if (threadIdx.x == 0) set_err(p.err, DEVERR_POS);
    T = tmax;
  }
  if (T < 1) T = 1;
  const int nblk = (T + 15) >> 4;
  // At least one block per warp; splits beyond the ones needed exit at once.
  const int per = max((nblk + p.splits - 1) / p.splits, DEC_WARPS);
  const int n_used = (nblk + per - 1) / per;
  if (s >= n_used) return;
  const int jb = s * per, je = min(jb + per, nblk);

  const uint16_t* qg = static_cast<const uint16_t*>(p.q) + (static_cast<long long>(b) * p.H + g * HPG) * HD;
  uint32_t qa[HD / 16][4];
  load_q<HD>(qa, r < HPG ? qg + r * HD : nullptr, r + 8 < HPG ? qg + (r + 8) * HD : nullptr, q);

  WarpState<HD> st;
  st.init();
  const uint32_t wbase = smem_u32(sm) + warp * 4 * TILE;  // per warp: [stage][K | V]
  const uint16_t* kp = static_cast<const uint16_t*>(p.k);
  const uint16_t* vp = static_cast<const uint16_t*>(p.v);
  auto issue = [&](int j, int stg) {
    bool ok;
    const int blk = block_of(p, b, j, ok);
    const long long off = (static_cast<long long>(blk) * p.G + g) * 16 * HD;
    stage_tile<HD>(wbase + stg * 2 * TILE, kp + off, ok, lane, 32);
    stage_tile<HD>(wbase + stg * 2 * TILE + TILE, vp + off, ok, lane, 32);
    cp_async_commit();
  };
  int j = jb + warp, stg = 0;
  if (j < je) issue(j, 0);
  for (; j < je; j += DEC_WARPS) {
    const int jn = j + DEC_WARPS;
    if (jn < je) {
      issue(jn, stg ^ 1);
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncwarp();
    attn_tile16<HD, T16>(wbase + stg * 2 * TILE, wbase + stg * 2 * TILE + TILE, qa, st, j * 16, T - 1, T - 1,
                         p.scale_log2, lane);
    __syncwarp();
    stg ^= 1;
  }
  st.l0 += __shfl_xor_sync(0xffffffffu, st.l0, 1);
  st.l0 += __shfl_xor_sync(0xffffffffu, st.l0, 2);
  st.l1 += __shfl_xor_sync(0xffffffffu, st.l1, 1);
  st.l1 += __shfl_xor_sync(0xffffffffu, st.l1, 2);
  __syncthreads();

  // Merge the warps' states in shared memory.
  float* wm = reinterpret_cast<float*>(sm);  // [DEC_WARPS][16]
  float* wl = wm + DEC_WARPS * 16;           // [DEC_WARPS][16]
  float* wo = wl + DEC_WARPS * 16;           // [DEC_WARPS][16][HD]
  if (q == 0) {
    wm[warp * 16 + r] = st.m0;
    wm[warp * 16 + r + 8] = st.m1;
    wl[warp * 16 + r] = st.l0;
    wl[warp * 16 + r + 8] = st.l1;
  }
#pragma unroll
  for (int nd = 0; nd < HD / 8; ++nd) {
    float* o0 = wo + (warp * 16 + r) * HD + nd * 8 + 2 * q;
    float* o1 = wo + (warp * 16 + r + 8) * HD + nd * 8 + 2 * q;
    o0[0] = st.o[nd][0];
    o0[1] = st.o[nd][1];
    o1[0] = st.o[nd][2];
    o1[1] = st.o[nd][3];
  }
  __syncthreads();

  const int rowlen = HD + 2;
  float* part = p.part + ((static_cast<long long>(b) * p.G + g) * p.splits) * 16 * rowlen;
  for (int idx = threadIdx.x; idx < HPG * HD; idx += blockDim.x) {
    const int i = idx / HD, dd = idx - i * HD;
    float M = NEG_INF;
#pragma unroll
    for (int w = 0; w < DEC_WARPS; ++w) M = fmaxf(M, wm[w * 16 + i]);
    float O = 0.f, L = 0.f;
    if (M != NEG_INF) {
#pragma unroll
      for (int w = 0; w < DEC_WARPS; ++w) {
        const float f = exp2f(wm[w * 16 + i] - M);
        O += wo[(w * 16 + i) * HD + dd] * f;
        L += wl[w * 16 + i] * f;
      }
    }
    if (n_used == 1) {
      T16* og = static_cast<T16*>(p.o) + (static_cast<long long>(b) * p.H + g * HPG + i) * HD + dd;
      *og = from_f<T16>(L > 0.f ? O / L : 0.f);
    } else {
      float* pr = part + (static_cast<long long>(s) * 16 + i) * rowlen;
      pr[dd] = O;
      if (dd == 0) {
        pr[HD] = M;
        pr[HD + 1] = L;
      }
    }
  }
  if (n_used == 1) return;

  // Last CTA of this (sequence, kv head) merges the n_used partial states.
  __shared__ int is_last;
  __shared__ float cw[16][64];
  __shared__ float cinv[16];
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) is_last = (atomicAdd(p.counter + b * p.G + g, 1) == n_used - 1);
  __syncthreads();
  if (!is_last) return;
  __threadfence();
  float* cl = wo;  // reuse: [16][64] running sums
  for (int idx = threadIdx.x; idx < HPG * n_used; idx += blockDim.x) {
    const int i = idx / n_used, t = idx - i * n_used;
    const float* pr = part + (static_cast<long long>(t) * 16 + i) * rowlen;
    cw[i][t] = __ldcg(pr + HD);
    cl[i * 64 + t] = __ldcg(pr + HD + 1);
  }
  __syncthreads();
  if (threadIdx.x < HPG) {
    const int i = threadIdx.x;
    float M = NEG_INF;
    for (int t = 0; t < n_used; ++t) M = fmaxf(M, cw[i][t]);
    float L = 0.f;
    for (int t = 0; t < n_used; ++t) {
      const float f = (cw[i][t] == NEG_INF) ? 0.f : exp2f(cw[i][t] - M);
      cw[i][t] = f;
      L += cl[i * 64 + t] * f;
    }
    cinv[i] = L > 0.f ? 1.f / L : 0.f;
  }
  __syncthreads();
  for (int idx = threadIdx.x; idx < HPG * HD; idx += blockDim.x) {
    const int i = idx / HD, dd = idx - i * HD;
    const float* pc = part + static_cast<long long>(i) * rowlen + dd;
    float O0 = 0.f, O1 = 0.f, O2 = 0.f, O3 = 0.f;
    int t = 0;
    for (; t + 4 <= n_used; t += 4) {
      const float v0 = __ldcg(pc + (t + 0) * 16 * rowlen), v1 = __ldcg(pc + (t + 1) * 16 * rowlen);
      const float v2 = __ldcg(pc + (t + 2) * 16 * rowlen), v3 = __ldcg(pc + (t + 3) * 16 * rowlen);
      O0 += cw[i][t] * v0;
      O1 += cw[i][t + 1] * v1;
      O2 += cw[i][t + 2] * v2;
      O3 += cw[i][t + 3] * v3;
    }
    for (; t < n_used; ++t) O0 += cw[i][t] * __ldcg(pc + t * 16 * rowlen);
    T16* og = static_cast<T16*>(p.o) + (static_cast<long long>(b) * p.H + g * HPG + i) * HD + dd;
    *og = from_f<T16>(((O0 + O1) + (O2 + O3)) * cinv[i]);
  }
  if (threadIdx.x == 0) p.counter[b * p.G + g] = 0;
}

// -------------------------------------------------------------- prefill
// CTA: 4 warps x PW positions x (H/G) heads of one kv head g of sequence b;
// key tiles staged 4 blocks (64 keys) at a time, double-buffered, shared by
// the 4 warps.
template <int HD, typename T16>
__global__ void __launch_bounds__(128) attn_prefill_kernel(AttnArgs p, int PW) {
  extern __shared__ __align__(128) uint8_t sm[];
  constexpr int TILE = 16 * HD * 2;
  constexpr int STAGE = 4 * 2 * TILE;  // 4 blocks x (K, V)
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, r = lane >> 2, q = lane & 3;
  const int HPG = p.H / p.G, S = p.S;
  const int PC = 4 * PW;
  const int b = blockIdx.z, g = blockIdx.y, p0 = blockIdx.x * PC;
  grid_dep_launch();
  grid_dep_wait();

  auto row_info = [&](int i, int& pos, int& h) {
    const int pl = i / HPG;
    h = i - pl * HPG;
    pos = p0 + warp * PW + pl;
    if (i >= PW * HPG || pos >= S) pos = -1;
  };
  int pos0, h0, pos1, h1;
  row_info(r, pos0, h0);
  row_info(r + 8, pos1, h1);
  const uint16_t* qbase = static_cast<const uint16_t*>(p.q);
  const long long Hd = static_cast<long long>(p.H) * HD;
  const uint16_t* qr0 =
      pos0 >= 0 ? qbase + (static_cast<long long>(b) * S + pos0) * Hd + (g * HPG + h0) * HD : nullptr;
  const uint16_t* qr1 =
      pos1 >= 0 ? qbase + (static_cast<long long>(b) * S + pos1) * Hd + (g * HPG + h1) * HD : nullptr;
  uint32_t qa[HD / 16][4];
  load_q<HD>(qa, qr0, qr1, q);

  WarpState<HD> st;
  st.init();
  const int pend = min(p0 + PC, S);
  const int nblk = (pend + 15) >> 4;
  const int nst = (nblk + 3) >> 2;
  const int wfirst = p0 + warp * PW;
  const int wmax = min(wfirst + PW - 1, S - 1);
  const uint32_t base = smem_u32(sm);
  const uint16_t* kp = static_cast<const uint16_t*>(p.k);
  const uint16_t* vp = static_cast<const uint16_t*>(p.v);
  auto issue = [&](int stage_idx, int buf) {
    for (int jj = 0; jj < 4; ++jj) {
      const int j = stage_idx * 4 + jj;
      if (j >= nblk) break;
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
      for (int jj = 0; jj < 4; ++jj) {
        const int j = sidx * 4 + jj;
        if (j >= nblk || j * 16 > wmax) break;
        const uint32_t t = base + buf * STAGE + jj * 2 * TILE;
        attn_tile16<HD, T16>(t, t + TILE, qa, st, j * 16, pos0, pos1, p.scale_log2, lane);
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
    if (pos0 >= 0) {
      T16* d0 = ob + (static_cast<long long>(b) * S + pos0) * Hd + (g * HPG + h0) * HD + nd * 8 + 2 * q;
      *reinterpret_cast<uint32_t*>(d0) = pack2<T16>(st.o[nd][0] * inv0, st.o[nd][1] * inv0);
    }
    if (pos1 >= 0) {
      T16* d1 = ob + (static_cast<long long>(b) * S + pos1) * Hd + (g * HPG + h1) * HD + nd * 8 + 2 * q;
      *reinterpret_cast<uint32_t*>(d1) = pack2<T16>(st.o[nd][2] * inv1, st.o[nd][3] * inv1);
    }
  }
}

// ------------------------------------------------------- fp32 debug path
// One warp per (row, query head): plain online softmax over visible keys.
__global__ void __launch_bounds__(32) attn_f32_kernel(AttnArgs p, int decode) {
  grid_dep_launch();
  grid_dep_wait();
  const int m = blockIdx.x, h = blockIdx.y, lane = threadIdx.x;
  const int d = p.d, HPG = p.H / p.G, g = h / HPG;
  int b, pos;
  if (decode) {
    b = m;
    pos = p.ctx[m];
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
  for (int t = 0; t <= pos; ++t) {
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
constexpr size_t decode_smem() { return DEC_WARPS * 4 * 16 * HD * 2; }  // warps x 2 stages x (K, V)
template <int HD>
constexpr size_t prefill_smem() { return 2 * 4 * 2 * 16 * HD * 2; }  // 2 stages x 4 blocks x (K, V)

template <int HD>
cudaError_t decode_hd(const LaunchCtx& lc, const AttnArgs& a, int B) {
  const size_t smem = decode_smem<HD>();
  if (lc.f16) return launch_k(lc, attn_decode_kernel<HD, f16>, dim3(a.splits, a.G, B), dim3(DEC_WARPS * 32), smem, a);
  return launch_k(lc, attn_decode_kernel<HD, bf16>, dim3(a.splits, a.G, B), dim3(DEC_WARPS * 32), smem, a);
}

template <int HD>
cudaError_t prefill_hd(const LaunchCtx& lc, const AttnArgs& a, int B) {
  const size_t smem = prefill_smem<HD>();
  const int HPG = a.H / a.G;
  const int PW = 16 / HPG;
  const int PC = 4 * PW;
  const dim3 grid((a.S + PC - 1) / PC, a.G, B);
  if (lc.f16) return launch_k(lc, attn_prefill_kernel<HD, f16>, grid, dim3(128), smem, a, PW);
  return launch_k(lc, attn_prefill_kernel<HD, bf16>, grid, dim3(128), smem, a, PW);
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

int attn_decode_splits(int B, int G, int max_blocks, int num_sms) {
  int want = (2 * num_sms + B * G - 1) / (B * G);
  if (want > max_blocks) want = max_blocks;
  if (want > 64) want = 64;
  return want < 1 ? 1 : want;
}

cudaError_t launch_attn_decode(const LaunchCtx& lc, bool fp32, const AttnArgs& a, int B) {
  if (fp32) return launch_k(lc, attn_f32_kernel, dim3(B, a.H), dim3(32), 0, a, 1);
  if (a.H / a.G > 16) return cudaErrorInvalidValue;
  if (a.d == 64) return decode_hd<64>(lc, a, B);
  if (a.d == 128) return decode_hd<128>(lc, a, B);
  return cudaErrorInvalidValue;
}

cudaError_t launch_attn_prefill(const LaunchCtx& lc, bool fp32, const AttnArgs& a, int B) {
  if (fp32) return launch_k(lc, attn_f32_kernel, dim3(B * a.S, a.H), dim3(32), 0, a, 0);
  if (a.H / a.G > 16) return cudaErrorInvalidValue;
  if (a.d == 64) return prefill_hd<64>(lc, a, B);
  if (a.d == 128) return prefill_hd<128>(lc, a, B);
  return cudaErrorInvalidValue;
}
