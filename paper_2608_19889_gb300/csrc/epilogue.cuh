// Fused epilogues of the projection kernels (decode GEMV and prefill GEMM).
//
// Every projection's output tile reaches an epilogue as a row chunk: row m
// (a token), 16 consecutive packed output columns n0 .. n0+15 (n0 % 16 == 0)
// holding pairs (v[i], v[8+i]), i < 8. The weight repack arranges rows so the
// pair a step needs lands in one chunk:
//   * QKV: within each head, chunk c holds dims c*8+i (v[i]) and
//     c*8+i+d/2 (v[8+i]) -- the rotate-half RoPE partners;
//   * gate/up: chunk c holds gate row c*8+i (v[i]) and up row c*8+i (v[8+i]);
//   * o_proj, down_proj and the LM head keep natural order.
//
// RMSNorm is split across producer and consumer so that no separate
// normalisation kernel runs: a residual-producing epilogue writes the fp32
// residual x, the bf16 operand a = x * g (gain of the NEXT norm) and a
// partial sum of x^2 per (row, chunk of columns); the consuming projection
// scales its accumulator by r = 1 / sqrt(sum / D + eps), since
// rms(x) * g . W^T = r * ((x * g) . W^T).
#pragma once

#include "common.cuh"

enum EpiKind : int { EPI_QKV = 0, EPI_RESID = 1, EPI_SWIGLU = 2, EPI_LOGITS = 3, EPI_ROWSCALE = 4 };
// Gate activation of the gated MLP (axon_config.hidden_act).
enum ActKind : int { ACT_SILU = 0, ACT_GELU_TANH = 1 };

struct EpiArgs {
  int M;  // rows (tokens)
  int N;  // packed output columns
  // row m -> (sequence b, position): variable-length batch (rowmap !=
  // null): (b, pos) = rowmap[m]; decode (ctx != null): b = m,
  // pos = ctx[m]; prefill: b = m / S, pos = m % S.
  int S;
  const int* ctx;
  const int2* rowmap;
  int max_pos;
  // A-operand normalisation (QKV, SWIGLU, LOGITS): partial sums of squares
  // of the producer, ss_parts per row, rows ss_stride floats apart.
  const float* ss;
  int ss_stride;
  int ss_parts;
  float inv_D;
  float eps;
  // ... or, when the producer already reduced them, r itself: rinv[m * rinv_stride].
  const float* rinv;
  int rinv_stride;
  // QKV
  const float* bias;   // packed [N] or null
  const float2* rope;  // [max_pos][d/2] (cos, sin)
  int H, G, d;
  void* q_out;  // [M][H*d]
  void* q_lo_out;  // optional [M][H*d] (decode): q - q_out, the second 16-bit term of q
  // qk-norm (null when off): q and k leave the epilogue unrotated and
  // unrounded, [M][H + G][d] fp32 (natural dimension order), for the
  // kernel that normalises each head, applies the gains and RoPE and stores
  // them (launch_qk_norm_rope); v is stored as usual.
  float* qk_raw;
  const float* qn_gain;  // [d]
  const float* kn_gain;  // [d]
  void* k_cache;  // this layer's pool [num_blocks][G][16][d]
  void* v_cache;
  const int* block_table;  // paged: [B][bt_stride]; null = contiguous
  int bt_stride;
  int blocks_per_seq;
  int num_blocks;
  // RESID
  float* x;            // [M][N] residual (in/out)
  void* a_out;         // [M][N] x * gain
  void* a_lo_out;      // optional [M][N]: x * gain - a_out (residual of the rounding), same type
  const float* gain;   // [N]
  float* ss_out;       // [M][ss_out_stride]
  int ss_out_stride;
  // Decode projections: the last CTA to finish reduces the partials into
  // rinv_out[m] (ticket: a zeroed counter it resets).
  float* rinv_out;
  int* ticket;
  // SWIGLU
  void* u_out;     // [M][N/2]
  void* u_lo_out;  // optional [M][N/2]: u - u_out (second term of the down projection's operand)
  int act;         // gate activation: ACT_SILU or ACT_GELU_TANH
  // LOGITS
  float* logits;  // [M][logits_stride] or null
  long long logits_stride;
  unsigned long long* keys;  // [M] argmax keys
  // ROWSCALE (mixture-of-experts down projection): y_out[m][n] = v * row_w[m], fp32, row stride N
  float* y_out;
  const float* row_w;
  int* err;
};

AXON_DEV float row_rinv(const EpiArgs& e, int m) {
  if (e.rinv) return e.rinv[static_cast<long long>(m) * e.rinv_stride];
  const float* p = e.ss + static_cast<long long>(m) * e.ss_stride;
  float s = 0.f;
  for (int i = 0; i < e.ss_parts; ++i) s += p[i];
  return 1.0f / sqrtf(s * e.inv_D + e.eps);
}

AXON_DEV int row_seq_pos(const EpiArgs& e, int m, int& b) {
  if (e.rowmap) {
    const int2 r = e.rowmap[m];
    b = r.x;
    return r.y;
  }
  if (e.ctx) {
    b = m;
    return e.ctx[m];
  }
  b = m / e.S;
  return m - b * e.S;
}

// Element offset of (sequence b, position pos, kv head g, dim 0) in a pool,
// or -1 (error recorded) when the block table or position is out of range.
AXON_DEV long long kv_offset(const EpiArgs& e, int b, int pos, int g) {
  if (pos < 0 || pos >= e.max_pos) {
    set_err(e.err, DEVERR_POS);
    return -1;
  }
  const int j = pos >> 4;
  const int blk = e.block_table ? e.block_table[static_cast<long long>(b) * e.bt_stride + j] : b * e.blocks_per_seq + j;
  if (blk < 0 || blk >= e.num_blocks) {
    set_err(e.err, DEVERR_BLOCK);
    return -1;
  }
  return ((static_cast<long long>(blk) * e.G + g) * 16 + (pos & 15)) * e.d;
}

template <typename T>
AXON_DEV void store8(T* dst, const float* v);
template <>
AXON_DEV void store8<bf16>(bf16* dst, const float* v) {
  uint4 u;
  u.x = pack_bf2(v[0], v[1]);
  u.y = pack_bf2(v[2], v[3]);
  u.z = pack_bf2(v[4], v[5]);
  u.w = pack_bf2(v[6], v[7]);
  *reinterpret_cast<uint4*>(dst) = u;
}
template <>
AXON_DEV void store8<f16>(f16* dst, const float* v) {
  uint4 u;
  u.x = pack_h2(v[0], v[1]);
  u.y = pack_h2(v[2], v[3]);
  u.z = pack_h2(v[4], v[5]);
  u.w = pack_h2(v[6], v[7]);
  *reinterpret_cast<uint4*>(dst) = u;
}
template <>
AXON_DEV void store8<float>(float* dst, const float* v) {
  reinterpret_cast<float4*>(dst)[0] = make_float4(v[0], v[1], v[2], v[3]);
  reinterpret_cast<float4*>(dst)[1] = make_float4(v[4], v[5], v[6], v[7]);
}

// Global inputs of one QKV chunk: the RoPE (cos, sin) pairs of its 8
// rotation frequencies at the row's position, and its 16 biases.
struct QkvIn {
  float2 cs[8];
  float b[16];
};

AXON_DEV void load_qkv16(const EpiArgs& e, int m, int n0, QkvIn& in) {
  const int Hd = e.H * e.d, Gd = e.G * e.d;
  const int c = n0 < Hd ? n0 % e.d : (n0 < Hd + Gd ? (n0 - Hd) % e.d : (n0 - Hd - Gd) % e.d);
  int b;
  const int pos = row_seq_pos(e, m, b);
  if (n0 < Hd + Gd) {
    const int pc = min(max(pos, 0), e.max_pos - 1);
    const float2* cs = e.rope + static_cast<long long>(pc) * (e.d >> 1) + (c >> 4) * 8;
#pragma unroll
    for (int i = 0; i < 8; ++i) in.cs[i] = cs[i];
  }
#pragma unroll
  for (int i = 0; i < 16; ++i) in.b[i] = e.bias ? e.bias[n0 + i] : 0.f;
}

// q/k/v: scale by r, add bias, rotate q and k, store q to the q buffer and
// k, v into the cache slot of (b, pos). `in`: the chunk's loaded inputs.
template <typename T>
AXON_DEV void epi_qkv16x(const EpiArgs& e, int m, int n0, const float* v, float r, const QkvIn& in) {
  const int Hd = e.H * e.d, Gd = e.G * e.d;
  int region, head, c;
  if (n0 < Hd) {
    region = 0; head = n0 / e.d; c = n0 - head * e.d;
  } else if (n0 < Hd + Gd) {
    region = 1; head = (n0 - Hd) / e.d; c = n0 - Hd - head * e.d;
  } else {
    region = 2; head = (n0 - Hd - Gd) / e.d; c = n0 - Hd - Gd - head * e.d;
  }
  const int j0 = (c >> 4) * 8, half = e.d >> 1;
  int b;
  const int pos = row_seq_pos(e, m, b);
  float lo[8], hi[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    lo[i] = v[i] * r + in.b[i];
    hi[i] = v[8 + i] * r + in.b[8 + i];
  }
  if (region < 2 && e.qk_raw) {
    float* raw = e.qk_raw + (static_cast<long long>(m) * (e.H + e.G) + (region == 0 ? head : e.H + head)) * e.d + j0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      raw[i] = lo[i];
      raw[half + i] = hi[i];
    }
    return;
  }
  if (region < 2) {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float2 t = in.cs[i];
      const float a = lo[i], bb = hi[i];
      lo[i] = a * t.x - bb * t.y;
      hi[i] = bb * t.x + a * t.y;
    }
  }
  if (region == 0) {
    const long long qo = static_cast<long long>(m) * Hd + head * e.d + j0;
    T* dst = reinterpret_cast<T*>(e.q_out) + qo;
    store8<T>(dst, lo);
    store8<T>(dst + half, hi);
    if (e.q_lo_out) {
      // what the 16-bit rounding of q lost: the decode attention multiplies
      // both terms with the keys
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        lo[i] -= to_f(from_f<T>(lo[i]));
        hi[i] -= to_f(from_f<T>(hi[i]));
      }
      T* ld = reinterpret_cast<T*>(e.q_lo_out) + qo;
      store8<T>(ld, lo);
      store8<T>(ld + half, hi);
    }
  } else {
    const long long off = kv_offset(e, b, pos, head);
    if (off < 0) return;
    T* dst = reinterpret_cast<T*>(region == 1 ? e.k_cache : e.v_cache) + off + j0;
    store8<T>(dst, lo);
    store8<T>(dst + half, hi);
  }
}

template <typename T>
AXON_DEV void epi_qkv16(const EpiArgs& e, int m, int n0, const float* v, float r) {
  QkvIn in;
  load_qkv16(e, m, n0, in);
  epi_qkv16x<T>(e, m, n0, v, r, in);
}

// x += v; a = x * gain; returns sum of x^2 over the 16 columns. `xin`:
// the 16 current residual values, already loaded by the caller.
template <typename T>
AXON_DEV float epi_resid16x(const EpiArgs& e, int m, int n0, const float* v, const float4* xin) {
  float* xp = e.x + static_cast<long long>(m) * e.N + n0;
  float xn[16];
#pragma unroll
  for (int i = 0; i < 16; i += 4) {
    const float4 t = xin[i >> 2];
    xn[i] = t.x + v[i];
    xn[i + 1] = t.y + v[i + 1];
    xn[i + 2] = t.z + v[i + 2];
    xn[i + 3] = t.w + v[i + 3];
    *reinterpret_cast<float4*>(xp + i) = make_float4(xn[i], xn[i + 1], xn[i + 2], xn[i + 3]);
  }
  float ag[16], s = 0.f;
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    ag[i] = xn[i] * e.gain[n0 + i];
    s += xn[i] * xn[i];
  }
  T* ap = reinterpret_cast<T*>(e.a_out) + static_cast<long long>(m) * e.N + n0;
  store8<T>(ap, ag);
  store8<T>(ap + 8, ag + 8);
  if (e.a_lo_out) {
    // second 16-bit term: what rounding a_out lost (split operand for the
    // next QKV projection)
    float lo[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) lo[i] = ag[i] - to_f(from_f<T>(ag[i]));
    T* lp = reinterpret_cast<T*>(e.a_lo_out) + static_cast<long long>(m) * e.N + n0;
    store8<T>(lp, lo);
    store8<T>(lp + 8, lo + 8);
  }
  return s;
}

// Loads the 16 residual values of (m, n0..n0+15) from L2: the previous
// writer of this slice may be another SM of the same (persistent) kernel,
// whose writes L1 does not see.
AXON_DEV void load_resid16(const EpiArgs& e, int m, int n0, float4* xin) {
  const float* xp = e.x + static_cast<long long>(m) * e.N + n0;
#pragma unroll
  for (int i = 0; i < 4; ++i) xin[i] = __ldcg(reinterpret_cast<const float4*>(xp + 4 * i));
}

template <typename T>
AXON_DEV float epi_resid16(const EpiArgs& e, int m, int n0, const float* v) {
  float4 xin[4];
  load_resid16(e, m, n0, xin);
  return epi_resid16x<T>(e, m, n0, v, xin);
}

// Both gate activations are z * sigmoid(k(z)): silu with k(z) = z, and
// gelu_new, 0.5 z (1 + tanh(sqrt(2/pi) (z + 0.044715 z^3))), with
// k(z) = 2 sqrt(2/pi) (z + 0.044715 z^3), since (1 + tanh(a)) / 2 =
// sigmoid(2a).
AXON_DEV float gate_act(float z, bool gelu) {
  const float k = gelu ? 1.5957691216057308f * fmaf(0.044715f * z, z * z, z) : z;
  return z / (1.0f + expf(-k));
}

template <typename T>
AXON_DEV void epi_swiglu16(const EpiArgs& e, int m, int n0, const float* v, float r) {
  float u[8];
  const bool gelu = e.act == ACT_GELU_TANH;
#pragma unroll
  for (int i = 0; i < 8; ++i) u[i] = gate_act(v[i] * r, gelu) * (v[8 + i] * r);
  T* up = reinterpret_cast<T*>(e.u_out) + static_cast<long long>(m) * (e.N >> 1) + (n0 >> 1);
  store8<T>(up, u);
  if (e.u_lo_out) {
    float lo[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) lo[i] = u[i] - to_f(from_f<T>(u[i]));
    store8<T>(reinterpret_cast<T*>(e.u_lo_out) + static_cast<long long>(m) * (e.N >> 1) + (n0 >> 1), lo);
  }
}

// Mixture-of-experts down projection: the 16 outputs of sorted row m times
// the row's routing weight, stored fp32 for the combine kernel.
AXON_DEV void epi_rowscale16(const EpiArgs& e, int m, int n0, const float* v) {
  const float w = e.row_w[m];
  float4* y = reinterpret_cast<float4*>(e.y_out + static_cast<long long>(m) * e.N + n0);
#pragma unroll
  for (int i = 0; i < 4; ++i) y[i] = make_float4(v[4 * i] * w, v[4 * i + 1] * w, v[4 * i + 2] * w, v[4 * i + 3] * w);
}

// logits = r * v (columns >= N dropped); returns this chunk's argmax key.
AXON_DEV unsigned long long epi_logits16(const EpiArgs& e, int m, int n0, const float* v, float r) {
  unsigned long long best = 0ull;
  float* lp = e.logits ? e.logits + static_cast<long long>(m) * e.logits_stride + n0 : nullptr;
  if (n0 + 16 <= e.N) {
    float l[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      l[i] = v[i] * r;
      const unsigned long long k = argmax_key(l[i], n0 + i);
      best = k > best ? k : best;
    }
    if (lp) {
      // Rows of a vocabulary that is not a multiple of 4 are not 16-byte
      // aligned: vector stores only where the address allows them.
      if ((reinterpret_cast<uintptr_t>(lp) & 15) == 0) {
#pragma unroll
        for (int i = 0; i < 16; i += 4)
          *reinterpret_cast<float4*>(lp + i) = make_float4(l[i], l[i + 1], l[i + 2], l[i + 3]);
      } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) lp[i] = l[i];
      }
    }
  } else {
    for (int i = 0; i < 16 && n0 + i < e.N; ++i) {
      const float l = v[i] * r;
      const unsigned long long k = argmax_key(l, n0 + i);
      best = k > best ? k : best;
      if (lp) lp[i] = l;
    }
  }
  return best;
}

// Fold a candidate into the row's argmax key: read first, so that most
// chunks (whose best loses) issue no atomic.
AXON_DEV void argmax_commit(unsigned long long* key, unsigned long long cand) {
  if (cand > *reinterpret_cast<volatile unsigned long long*>(key)) atomicMax(key, cand);
}
