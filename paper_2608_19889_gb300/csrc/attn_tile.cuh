// Decode-attention building blocks shared by the decode attention kernel
// (k_attn.cu) and the persistent decode step (k_persist.cu): the swizzled
// key/value tile staging, the per-warp online-softmax tile update and one
// split-KV work item with its last-arriver merge. The file's comment in
// k_attn.cu describes the scheme.
#pragma once

#include <math.h>

#include <type_traits>

#include "kernels.h"

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
    qa[kk][0] = row0 ? __ldcg(reinterpret_cast<const unsigned int*>(row0 + k)) : 0u;
    qa[kk][1] = row1 ? __ldcg(reinterpret_cast<const unsigned int*>(row1 + k)) : 0u;
    qa[kk][2] = row0 ? __ldcg(reinterpret_cast<const unsigned int*>(row0 + k + 8)) : 0u;
    qa[kk][3] = row1 ? __ldcg(reinterpret_cast<const unsigned int*>(row1 + k + 8)) : 0u;
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
// iff lo0 <= t <= lim0 (lo1 <= t <= lim1); lo is 0 without a sliding
// window, else position - window + 1.
//
// PAIRED (decode with at most 8 query heads per kv head, whose rows 8..15
// would be padding): row r + 8 carries the second 16-bit term of row r's
// query instead of another head. The score of row r is the sum of the two
// rows' products, and the probabilities enter the P.V product the same way
// -- their 16-bit rounding in row r, what it lost in row r + 8 -- so both
// accumulator rows add up to head r's output (folded by the caller). The
// second terms cost no extra MMA. Only row r's softmax state is used.
template <int HD, typename T16, bool PAIRED = false>
AXON_DEV void attn_tile16(uint32_t ks, uint32_t vs, const uint32_t (&qa)[HD / 16][4], WarpState<HD>& st, int tok0,
                          int lo0, int lim0, int lo1, int lim1, float sl2, int lane) {
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
  if (PAIRED) {
#pragma unroll
    for (int nt = 0; nt < 2; ++nt) {
      s[nt][0] += s[nt][2];
      s[nt][1] += s[nt][3];
    }
  }
  float mx0 = NEG_INF, mx1 = NEG_INF;
#pragma unroll
  for (int nt = 0; nt < 2; ++nt) {
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const int t = tok0 + nt * 8 + 2 * q + e;
      s[nt][e] = (t <= lim0 && t >= lo0) ? s[nt][e] * sl2 : NEG_INF;
      mx0 = fmaxf(mx0, s[nt][e]);
      if (!PAIRED) {
        s[nt][2 + e] = (t <= lim1 && t >= lo1) ? s[nt][2 + e] * sl2 : NEG_INF;
        mx1 = fmaxf(mx1, s[nt][2 + e]);
      }
    }
  }
  mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
  mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
  if (!PAIRED) {
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
  }
  const float nm0 = fmaxf(st.m0, mx0), nm1 = PAIRED ? NEG_INF : fmaxf(st.m1, mx1);
  const float base0 = (nm0 == NEG_INF) ? 0.f : nm0, base1 = (nm1 == NEG_INF) ? 0.f : nm1;
  const float a0 = exp2f(st.m0 - base0), a1 = PAIRED ? a0 : exp2f(st.m1 - base1);
  float ps0 = 0.f, ps1 = 0.f;
#pragma unroll
  for (int nt = 0; nt < 2; ++nt) {
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      s[nt][e] = exp2f(s[nt][e] - base0);
      ps0 += s[nt][e];
      if (!PAIRED) {
        s[nt][2 + e] = exp2f(s[nt][2 + e] - base1);
        ps1 += s[nt][2 + e];
      }
    }
  }
  st.l0 = st.l0 * a0 + ps0;
  st.m0 = nm0;
  if (!PAIRED) {
    st.l1 = st.l1 * a1 + ps1;
    st.m1 = nm1;
  }
#pragma unroll
  for (int nd = 0; nd < HD / 8; ++nd) {
    st.o[nd][0] *= a0;
    st.o[nd][1] *= a0;
    st.o[nd][2] *= a1;
    st.o[nd][3] *= a1;
  }
  if (PAIRED) {
    // row r + 8: what the 16-bit rounding of row r's probabilities lost
#pragma unroll
    for (int nt = 0; nt < 2; ++nt) {
      s[nt][2] = s[nt][0] - to_f(from_f<T16>(s[nt][0]));
      s[nt][3] = s[nt][1] - to_f(from_f<T16>(s[nt][1]));
    }
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

// Two consecutive 16-key blocks (keys tok0 .. tok0+31; block A's K and V at
// ksa / vsa, block B's at ksb / vsb) as one tile: four independent score
// accumulators in the QK^T loop instead of two, one online-softmax rescale
// of the output for 32 keys instead of two. Rows as in attn_tile16 (not
// paired).
template <int HD, typename T16>
AXON_DEV void attn_tile32(uint32_t ksa, uint32_t vsa, uint32_t ksb, uint32_t vsb, const uint32_t (&qa)[HD / 16][4],
                          WarpState<HD>& st, int tok0, int lo0, int lim0, int lo1, int lim1, float sl2, int lane) {
  const int q = lane & 3;
  const int mi = lane >> 3, li = lane & 7;
  float s[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
#pragma unroll
  for (int kk = 0; kk < HD / 16; ++kk) {
    uint32_t ka[4], kb[4];
    const int tok = (mi >> 1) * 8 + li, ch = 2 * kk + (mi & 1);
    ldsm_x4(ka, swz<HD>(ksa, tok, ch));
    ldsm_x4(kb, swz<HD>(ksb, tok, ch));
    const uint32_t b0[2] = {ka[0], ka[1]}, b1[2] = {ka[2], ka[3]}, b2[2] = {kb[0], kb[1]}, b3[2] = {kb[2], kb[3]};
    mma16816<T16>(s[0], qa[kk], b0);
    mma16816<T16>(s[1], qa[kk], b1);
    mma16816<T16>(s[2], qa[kk], b2);
    mma16816<T16>(s[3], qa[kk], b3);
  }
  float mx0 = NEG_INF, mx1 = NEG_INF;
#pragma unroll
  for (int nt = 0; nt < 4; ++nt) {
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const int t = tok0 + nt * 8 + 2 * q + e;
      s[nt][e] = (t <= lim0 && t >= lo0) ? s[nt][e] * sl2 : NEG_INF;
      s[nt][2 + e] = (t <= lim1 && t >= lo1) ? s[nt][2 + e] * sl2 : NEG_INF;
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
  for (int nt = 0; nt < 4; ++nt) {
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
  const uint32_t pa[4] = {pack2<T16>(s[0][0], s[0][1]), pack2<T16>(s[0][2], s[0][3]), pack2<T16>(s[1][0], s[1][1]),
                          pack2<T16>(s[1][2], s[1][3])};
  const uint32_t pb[4] = {pack2<T16>(s[2][0], s[2][1]), pack2<T16>(s[2][2], s[2][3]), pack2<T16>(s[3][0], s[3][1]),
                          pack2<T16>(s[3][2], s[3][3])};
#pragma unroll
  for (int nd2 = 0; nd2 < HD / 16; ++nd2) {
    uint32_t va[4], vb[4];
    const int tok = (mi & 1) * 8 + li, ch = 2 * nd2 + (mi >> 1);
    ldsm_x4_t(va, swz<HD>(vsa, tok, ch));
    ldsm_x4_t(vb, swz<HD>(vsb, tok, ch));
    const uint32_t a0v[2] = {va[0], va[1]}, a1v[2] = {va[2], va[3]}, b0v[2] = {vb[0], vb[1]}, b1v[2] = {vb[2], vb[3]};
    mma16816<T16>(st.o[2 * nd2], pa, a0v);
    mma16816<T16>(st.o[2 * nd2 + 1], pa, a1v);
    mma16816<T16>(st.o[2 * nd2], pb, b0v);
    mma16816<T16>(st.o[2 * nd2 + 1], pb, b1v);
  }
}

// After the last PAIRED tile: add row r + 8's partial output into row r and
// leave row r + 8 empty.
template <int HD>
AXON_DEV void fold_paired(WarpState<HD>& st) {
#pragma unroll
  for (int nd = 0; nd < HD / 8; ++nd) {
    st.o[nd][0] += st.o[nd][2];
    st.o[nd][1] += st.o[nd][3];
    st.o[nd][2] = st.o[nd][3] = 0.f;
  }
  st.m1 = NEG_INF;
  st.l1 = 0.f;
}

AXON_DEV int block_of(const AttnArgs& p, int b, int j, bool& ok) {
  const int blk = p.block_table ? p.block_table[static_cast<long long>(b) * p.bt_stride + j] : b * p.blocks_per_seq + j;
  ok = blk >= 0 && blk < p.num_blocks;
  if (!ok) set_err(p.err, DEVERR_BLOCK);
  return ok ? blk : 0;
}

// Barrier over the DEC_WARPS * 32 threads that run a decode item: the whole
// CTA, or (NAMED) named barrier 1 when the CTA holds other warps too.
template <bool NAMED>
AXON_DEV void dec_sync() {
  if (NAMED)
    asm volatile("bar.sync 1, %0;" ::"n"(DEC_WARPS * 32) : "memory");
  else
    __syncthreads();
}

// One decode work item: split s of the keys of (kv head g, sequence b), run
// by DEC_WARPS warps (thread `tid` of them) with `sm` as staging memory
// (decode_smem<HD>() bytes). Reads of q and of the merge partials bypass L1:
// they may have been written by another SM earlier in the same kernel.
// PAIR = 1: the caller guarantees a second term of q and at most 8 query
// heads per kv head, so only the paired tile loop is compiled; PAIR = 0:
// chosen at run time.
template <int HD, typename T16, bool NAMED, int PAIR = 0, int STAGES = 2>
AXON_DEV void attn_decode_item(const AttnArgs& p, int s, int g, int b, uint8_t* sm, int tid) {
  constexpr int TILE = 16 * HD * 2;
  const int warp = tid >> 5, lane = tid & 31, r = lane >> 2, q = lane & 3;
  const int HPG = p.H / p.G;

  int T = p.ctx[b] + 1;
  const int tmax = p.blocks_per_seq * 16;
  if (T > tmax) {
    if (tid == 0) set_err(p.err, DEVERR_POS);
    T = tmax;
  }
  if (T < 1) T = 1;
  // keys klo .. T-1: all of them, or the last `window`
  const int klo = (p.window > 0 && T > p.window) ? T - p.window : 0;
  const int jlo = klo >> 4, nblk = ((T + 15) >> 4) - jlo;
  // At least one block per warp; splits beyond the ones needed exit at once.
  const int per = max((nblk + p.splits - 1) / p.splits, DEC_WARPS);
  const int n_used = (nblk + per - 1) / per;
  if (s >= n_used) return;
  const int jb = jlo + s * per, je = min(jb + per, jlo + nblk);

  const uint32_t wbase = smem_u32(sm) + warp * STAGES * 2 * TILE;  // per warp: [stage][K | V]
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
  // The first key/value tile is requested before q is read: the two round
  // trips overlap.
  int j = jb + warp, stg = 0;
  if (j < je) issue(j, 0);

  // With a second term of q and at most 8 query heads per kv head, rows
  // r + 8 of the MMA tiles carry the second terms (attn_tile16, PAIRED).
  const long long qoff = (static_cast<long long>(b) * p.H + g * HPG) * HD;
  const uint16_t* qg = static_cast<const uint16_t*>(p.q) + qoff;
  const bool paired = PAIR == 1 || (p.q_lo != nullptr && HPG <= 8);
  const uint16_t* qg1 = paired ? static_cast<const uint16_t*>(p.q_lo) + qoff + r * HD : qg + (r + 8) * HD;
  uint32_t qa[HD / 16][4];
  load_q<HD>(qa, r < HPG ? qg + r * HD : nullptr, (paired ? r : r + 8) < HPG ? qg1 : nullptr, q);

  WarpState<HD> st;
  st.init();
  auto run_tiles = [&](auto paired_tag) {
    constexpr bool PAIRED = decltype(paired_tag)::value;
    for (; j < je; j += DEC_WARPS) {
      const int jn = j + DEC_WARPS;
      if (STAGES == 2 && jn < je) {
        issue(jn, stg ^ 1);
        cp_async_wait<1>();
      } else {
        cp_async_wait<0>();
      }
      __syncwarp();
      attn_tile16<HD, T16, PAIRED>(wbase + stg * 2 * TILE, wbase + stg * 2 * TILE + TILE, qa, st, j * 16, klo, T - 1,
                                   klo, T - 1, p.scale_log2, lane);
      __syncwarp();
      if (STAGES == 2)
        stg ^= 1;
      else if (jn < je)
        issue(jn, 0);  // one stage: the next block loads once this one is consumed
    }
    if (PAIRED) fold_paired<HD>(st);
  };
  if constexpr (PAIR == 1) {
    run_tiles(std::true_type{});
  } else {
    if (paired)
      run_tiles(std::true_type{});
    else
      run_tiles(std::false_type{});
  }
  st.l0 += __shfl_xor_sync(0xffffffffu, st.l0, 1);
  st.l0 += __shfl_xor_sync(0xffffffffu, st.l0, 2);
  st.l1 += __shfl_xor_sync(0xffffffffu, st.l1, 1);
  st.l1 += __shfl_xor_sync(0xffffffffu, st.l1, 2);
  dec_sync<NAMED>();

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
  dec_sync<NAMED>();

  const int rowlen = HD + 2;
  float* part = p.part + ((static_cast<long long>(b) * p.G + g) * p.splits) * 16 * rowlen;
  for (int idx = tid; idx < HPG * HD; idx += DEC_WARPS * 32) {
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
      const float ov = L > 0.f ? O / L : 0.f;
      *og = from_f<T16>(ov);
      if (p.o_lo) static_cast<T16*>(p.o_lo)[og - static_cast<T16*>(p.o)] = from_f<T16>(ov - to_f(from_f<T16>(ov)));
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
  // The ticket is taken after the CTA barrier by one thread with an
  // acquire-release atomic: its release covers the CTA's partial stores, its
  // acquire (passed on by the second barrier) the other CTAs'.
  __shared__ int is_last;
  dec_sync<NAMED>();
  if (tid == 0) is_last = (atom_add_acq_rel_gpu(p.counter + b * p.G + g, 1) == n_used - 1);
  dec_sync<NAMED>();
  if (!is_last) return;
  // Each thread folds the n_used (m, l, O) partial states of its outputs in
  // split order with the online-softmax update; the loads of sixteen splits
  // are issued together, so up to sixteen splits cost one L2 round trip.
  for (int idx = tid; idx < HPG * HD; idx += DEC_WARPS * 32) {
    const int i = idx / HD, dd = idx - i * HD;
    const float* pc = part + static_cast<long long>(i) * rowlen;
    float M = NEG_INF, L = 0.f, O = 0.f;
    for (int t0 = 0; t0 < n_used; t0 += 16) {
      float mv[16], lv[16], ov[16];
#pragma unroll
      for (int u = 0; u < 16; ++u) {
        const bool in = t0 + u < n_used;
        const float* pr = pc + static_cast<long long>(in ? t0 + u : 0) * 16 * rowlen;
        mv[u] = in ? __ldcg(pr + HD) : NEG_INF;
        lv[u] = in ? __ldcg(pr + HD + 1) : 0.f;
        ov[u] = in ? __ldcg(pr + dd) : 0.f;
      }
#pragma unroll
      for (int u = 0; u < 16; ++u) {
        if (mv[u] == NEG_INF) continue;  // a split with no visible key
        const float nm = fmaxf(M, mv[u]);
        const float a = exp2f(M - nm), f = exp2f(mv[u] - nm);  // a = 0 while M = -inf
        L = L * a + lv[u] * f;
        O = O * a + ov[u] * f;
        M = nm;
      }
    }
    T16* og = static_cast<T16*>(p.o) + (static_cast<long long>(b) * p.H + g * HPG + i) * HD + dd;
    const float res = L > 0.f ? O / L : 0.f;
    *og = from_f<T16>(res);
    if (p.o_lo) static_cast<T16*>(p.o_lo)[og - static_cast<T16*>(p.o)] = from_f<T16>(res - to_f(from_f<T16>(res)));
  }
  if (tid == 0) p.counter[b * p.G + g] = 0;
}


template <int HD>
constexpr size_t decode_smem() { return DEC_WARPS * 4 * 16 * HD * 2; }  // warps x 2 stages x (K, V)
// One stage per warp (STAGES = 1), or the merge buffers of attn_decode_item
// ([warps][16] maxima and sums, [warps][16][HD] outputs), whichever is larger.
template <int HD>
constexpr size_t decode_smem1() {
  return DEC_WARPS * 2 * 16 * HD * 2 > (2 * DEC_WARPS * 16 + DEC_WARPS * 16 * HD) * 4
             ? DEC_WARPS * 2 * 16 * HD * 2
             : (2 * DEC_WARPS * 16 + DEC_WARPS * 16 * HD) * 4;
}

}  // namespace
