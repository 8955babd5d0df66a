// Persistent decode step: one cooperative launch runs a whole decode step
// (embedding, L x [QKV, attention, O, gate/up, down], LM head, greedy token)
// for B <= 8 sequences, with one CTA per SM.
//
// Why: at decode, every projection of a small model moves a few MB, which the
// GPU streams in a microsecond or two, while a chain of ~5L+3 dependent
// kernel launches pays the kernel boundary (grid drain, launch, first loads)
// at every link. Here the links are grid-wide barriers inside one kernel, and
// the weights -- which do not depend on the activations -- never wait for
// them: in every CTA a producer warp streams that CTA's share of every
// weight matrix of the step, in consumption order, through a shared-memory
// ring (2D TMA tensor copies completing on mbarriers), running ahead across
// layer and phase boundaries as far as the ring allows. The eight consumer
// warps wait at the barriers, take weight tiles from the ring and activation
// fragments from L2, and run the same mma.sync products, reductions and fused
// epilogues as the decode GEMV kernels.
//
// Work split: a projection phase is cut into items of 16 weight rows x all
// of K; item i of a phase goes to CTA (i + rot) mod grid, rot advancing by
// the phase's item count so that consecutive phases continue the round
// robin and every CTA streams about the same number of bytes per step. The
// producer and the consumers of a CTA walk the same item sequence. Attention
// items are the (split, kv head, sequence) triples of the split-KV decode
// attention, run by the consumer warps with the shared decode-attention code
// (last-arriver merge across splits).
//
// Coherence: every read of data written earlier in the same launch by
// another SM (residual stream, activations, q, norm partials, merge
// partials, argmax keys) goes to L2 (ld.global.cg / cp.async.cg); L1 is not
// coherent across SMs.
//
// Waits: every wait (ring mbarriers, grid barrier) gives up after 2 s, sets
// DEVERR_TIMEOUT and a grid-wide abort flag; after that no wait blocks, the
// producer issues no further copies, the kernel runs to its end on garbage
// (same barrier sequence, so named barriers stay matched) and the host sees
// the error bit. Before it exits, the producer waits (bounded) for its copies
// in flight.
#include <type_traits>

#include "attn_tile.cuh"

namespace {

constexpr int PCW = 8;                     // consumer warps (= DEC_WARPS)
constexpr int PTHREADS = (PCW + 1) * 32;   // + 1 producer warp
constexpr int KC = 512;                    // weight columns per ring stage (one 64-column chunk per warp)
constexpr int BOXC = PERSIST_BOX_COLS;     // columns per TMA box: a stage is 2 boxes of 16 rows x 256
constexpr int BOX_BYTES = 16 * BOXC * 2;   // 8 KB, rows dense (512 bytes)
constexpr int STAGE_BYTES = 2 * BOX_BYTES;
constexpr int RED_FLOATS = PCW * 16 * 9;   // cross-warp partials of one item: [warp][row][token + pad]
constexpr uint64_t PWAIT_NS = 2000000000ull;
constexpr int SMEM_LIMIT = 232448;         // 227 KB opt-in per CTA

static_assert(PCW == DEC_WARPS, "attention items run on the consumer warps");

// How the 16-bit operand terms of the projections enter the MMAs (proj_phase).
constexpr int TERMS_ONE = 0, TERMS_PAIRED = 1, TERMS_TWO = 2;

// Shared-memory layout. SM ("small", head_dim 128): the attention items stage
// one key block per warp (decode_smem1), so the weight ring gets the space a
// second stage would take: 9 ring stages instead of 5.
template <int HD, bool SM>
struct PLayout {
  static constexpr int ATTN = SM ? static_cast<int>(decode_smem1<HD>()) : static_cast<int>(decode_smem<HD>());
  static constexpr int RED = 2 * RED_FLOATS * 4;
  static constexpr int MISC = 256;  // rinv[8], abort flag
  static constexpr int STATIC_EST = 1024;  // static shared (the merge flag), with margin
  static constexpr int NS = (SMEM_LIMIT - ATTN - RED - MISC - STATIC_EST - 1024) / (STAGE_BYTES + 16);
  static constexpr int BARS = 2 * NS * 8;
  static constexpr int RING_OFF = 0;
  static constexpr int ATTN_OFF = RING_OFF + NS * STAGE_BYTES;
  static constexpr int RED_OFF = ATTN_OFF + ATTN;
  static constexpr int BAR_OFF = RED_OFF + RED;
  static constexpr int MISC_OFF = BAR_OFF + BARS;
  static constexpr int BYTES = MISC_OFF + MISC + 1024;  // + alignment slack
  static_assert(NS >= 3, "ring too small");
};

AXON_DEV void consumer_sync() { asm volatile("bar.sync 1, %0;" ::"n"(PCW * 32) : "memory"); }

AXON_DEV unsigned ld_acquire(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
AXON_DEV unsigned ld_volatile(const unsigned* p) { return *reinterpret_cast<const volatile unsigned*>(p); }

AXON_DEV uint4 lds16(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
  return v;
}

// Wait for phase `parity` of a ring mbarrier: bounded, and a no-op once the
// launch is aborting. The poll loop touches nothing but the barrier; the
// clock is read every 1024 polls and the grid-wide abort flag only after a
// millisecond of waiting, so that a completed phase is seen at once.
AXON_DEV bool ring_wait(uint32_t bar, uint32_t parity, PersistGrid* g, volatile int* s_abort, int* err) {
  if (mbar_try_wait(bar, parity)) return true;
  if (*s_abort) return false;
  uint64_t t0 = 0;
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 1023u) == 0) {
      const uint64_t now = global_ns();
      if (t0 == 0) {
        t0 = now;
      } else if (now - t0 > 1000000ull) {
        if (*s_abort || ld_volatile(&g->abort)) {
          *s_abort = 1;
          return false;
        }
        if (now - t0 > PWAIT_NS) {
          set_err(err, DEVERR_TIMEOUT);
          atomicExch(&g->abort, 1u);
          *s_abort = 1;
          return false;
        }
      }
    }
  }
}

AXON_DEV void red_release_add(unsigned* p, unsigned v) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Grid-wide barrier of the consumer warps (the producer never takes part):
// the CTA's writes are ordered before its arrival by the CTA barrier and the
// release of the arrival (cumulative); the acquiring poll orders every later
// read after all arrivals, and the closing CTA barrier passes that on.
AXON_DEV void grid_sync(PersistGrid* g, unsigned& epoch, int tid, volatile int* s_abort, int* err) {
  consumer_sync();
  if (tid == 0) {
    ++epoch;
    red_release_add(&g->count, 1u);
    const unsigned target = epoch * gridDim.x;
    if (!*s_abort) {
      const uint64_t t0 = global_ns();
      int spins = 0;
      while (ld_acquire(&g->count) < target) {
        if ((++spins & 255) == 0) {
          if (ld_volatile(&g->abort)) {
            *s_abort = 1;
            break;
          }
          if (global_ns() - t0 > PWAIT_NS) {
            set_err(err, DEVERR_TIMEOUT);
            atomicExch(&g->abort, 1u);
            *s_abort = 1;
            break;
          }
        }
      }
    }
  }
  consumer_sync();
}

AXON_DEV int first_item(int rot) {
  const int n = static_cast<int>(gridDim.x);
  return ((static_cast<int>(blockIdx.x) - rot) % n + n) % n;
}

template <int HD, bool SM>
struct Ring {
  uint32_t base;  // shared address of stage 0
  uint32_t bars;  // full[NS] then empty[NS]
  AXON_DEV uint32_t full(int s) const { return bars + 8 * s; }
  AXON_DEV uint32_t empty(int s) const { return bars + 8 * (PLayout<HD, SM>::NS + s); }
};

// ----------------------------------------------------------------- producer
// Streams this CTA's items of one matrix (in the item order the consumers
// walk): per ring stage one or two TMA boxes of 16 rows x 256 columns, one
// instruction each; rows >= N and columns >= K arrive as zeros.
template <int HD, bool SM>
AXON_DEV void stream_matrix(const Ring<HD, SM>& R, const CUtensorMap* map, int N, int K, int& rot, uint32_t& stage,
                            bool& stop, PersistGrid* g, volatile int* s_abort, int* err, int lane) {
  constexpr int NS = PLayout<HD, SM>::NS;
  const int n = (N + 15) >> 4;
  const int i0 = first_item(rot);
  rot = (rot + n) % static_cast<int>(gridDim.x);
  // Weights are read once per step: they should not evict the key/value
  // cache or the activations from L2.
  const uint64_t policy = createpolicy_evict_first();
  for (int i = i0; i < n && !stop; i += gridDim.x) {
    for (int k0 = 0; k0 < K && !stop; k0 += KC) {
      const int slot = static_cast<int>(stage % NS);
      int ok = 1;
      if (lane == 0) {
        if (stage >= static_cast<uint32_t>(NS))  // the consumers released this slot's previous use?
          ok = ring_wait(R.empty(slot), ((stage / NS) - 1) & 1u, g, s_abort, err) ? 1 : 0;
        if (ok) {
          const bool two = k0 + BOXC < K;
          mbar_arrive_expect_tx(R.full(slot), two ? STAGE_BYTES : BOX_BYTES);
          const uint32_t dst = R.base + slot * STAGE_BYTES;
          tma_load_2d_hint(dst, map, R.full(slot), k0, i * 16, policy);
          if (two) tma_load_2d_hint(dst + BOX_BYTES, map, R.full(slot), k0 + BOXC, i * 16, policy);
        }
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) {
        stop = true;
        break;
      }
      ++stage;
    }
  }
}

// ----------------------------------------------------------------- consumers
struct CState {
  int rot = 0;
  uint32_t stage = 0;
  int buf = 0;
};

// Stage t of a phase's stage sequence (spi stages per item): wait for the
// ring slot, copy this warp's weight fragments (rows r, r+8 x 16 columns)
// and the token-r activation fragments to registers, release the slot.
template <int HD, bool SM, typename T16, bool WANT_Y>
AXON_DEV void load_stage(const Ring<HD, SM>& R, CState& cs, const PersistArgs& A, PersistGrid* g, volatile int* s_abort,
                         int t, int spi, int K, int warp, int lane, int r, int q, bool tok_ok, bool staged,
                         const uint8_t* act_sm, int pitch, const T16* xsrc, const T16* ysrc, int xrow_s, int yrow_s,
                         uint4& w0, uint4& w1, uint4& w2, uint4& w3, uint4& x0, uint4& x1, uint4& y0,
                         uint4& y1, bool& on) {
  constexpr int NS = PLayout<HD, SM>::NS;
  const int k0 = (t % spi) * KC;
  const int kc = min(KC, K - k0);
  const int sl = static_cast<int>(cs.stage % NS);
  ring_wait(R.full(sl), (cs.stage / NS) & 1u, g, s_abort, A.err);
  on = warp * 64 < kc;
  x0 = x1 = y0 = y1 = make_uint4(0, 0, 0, 0);
  if (on) {
    // chunk `warp` = box warp/4, columns (warp%4)*64 of its dense 512-byte rows
    const uint32_t rs = R.base + sl * STAGE_BYTES + (warp >> 2) * BOX_BYTES + (warp & 3) * 128 + q * 32;
    w0 = lds16(rs + r * (BOXC * 2));
    w1 = lds16(rs + r * (BOXC * 2) + 16);
    w2 = lds16(rs + (r + 8) * (BOXC * 2));
    w3 = lds16(rs + (r + 8) * (BOXC * 2) + 16);
    const int k = k0 + warp * 64;
    if (tok_ok) {
      if (staged) {
        const uint32_t sa = smem_u32(act_sm) + xrow_s * pitch + (k + 16 * q) * 2;
        x0 = lds16(sa);
        x1 = lds16(sa + 16);
        if (WANT_Y) {
          const uint32_t sb = smem_u32(act_sm) + yrow_s * pitch + (k + 16 * q) * 2;
          y0 = lds16(sb);
          y1 = lds16(sb + 16);
        }
      } else {
        x0 = __ldcg(reinterpret_cast<const uint4*>(xsrc + k));
        x1 = __ldcg(reinterpret_cast<const uint4*>(xsrc + k + 8));
        if (WANT_Y) {
          y0 = __ldcg(reinterpret_cast<const uint4*>(ysrc + k));
          y1 = __ldcg(reinterpret_cast<const uint4*>(ysrc + k + 8));
        }
      }
    }
  } else {
    w0 = w1 = w2 = w3 = make_uint4(0, 0, 0, 0);
  }
  __syncwarp();
  if (lane == 0) mbar_arrive(R.empty(sl));  // fragments are in registers: slot free
  ++cs.stage;
}

// One projection phase: items of 16 rows x K, products on mma.sync with the
// weight tile from the ring and the B <= 8 token rows of `act` (and of its
// second term `act_lo` in the two-term modes); epilogue `KIND`.
//
// MODE (compile time, so that each kernel carries only its own inner loop):
//   TERMS_ONE    one 16-bit term per token (bf16 mode);
//   TERMS_PAIRED two terms, B <= 4: token slot 2b of the MMA's N dimension
//                holds token b's first term and slot 2b+1 its second, and
//                the reduction adds the two accumulator columns (no extra
//                MMA, no extra load);
//   TERMS_TWO    two terms, B = 5..8: a second MMA set takes the second
//                terms.
//
// Per item the consumer warps only run the products and the cross-warp sum;
// the item's 16 x B sums go to a shared buffer and the epilogues run in
// batches of up to 64 items, spread over all consumer threads, so that their
// global reads (residual, rope table, bias, gains) overlap instead of
// stalling the weight stream item after item. The LM head's argmax keeps a
// per-CTA best key per token in shared memory and commits it once per phase.
template <int HD, bool SM, int KIND, typename T16, int MODE>
AXON_DEV void proj_phase(const Ring<HD, SM>& R, CState& cs, const PersistArgs& A, const T16* W, int N, int K,
                         const T16* act, const T16* act_lo, int act_stride, const EpiArgs& ep, float* red_base,
                         float* rinv_s, unsigned long long* best_s, uint8_t* act_sm, PersistGrid* g,
                         volatile int* s_abort, int tid) {
  constexpr int ATTN = PLayout<HD, SM>::ATTN;
  constexpr bool LO = MODE != TERMS_ONE;
  constexpr bool paired = MODE == TERMS_PAIRED;
  const int warp = tid >> 5, lane = tid & 31, r = lane >> 2, q = lane & 3;
  const int B = A.B;
  const int n = (N + 15) >> 4;
  const int i_first = first_item(cs.rot);
  cs.rot = (cs.rot + n) % static_cast<int>(gridDim.x);
  if (i_first >= n) return;
  // Every item of the phase reads the same B x K activations: copy them
  // (and their second term) to shared memory once, rows padded by 16 bytes
  // so that the 8 token rows of a fragment load hit distinct banks. The
  // ring stages then cost no L2 round trip. Falls back to L2 reads when
  // they do not fit next to the epilogue buffer (the attention staging
  // region is free during a projection phase).
  // Residual phases also keep, per buffered item, the 16 x B residual
  // values that its epilogue updates (prefetched, see below).
  constexpr int PER_ITEM = (KIND == EPI_RESID ? 2 : 1) * 16 * 4;  // bytes per item and token
  const int pitch = K * 2 + 16;
  const int act_bytes = B * pitch * (LO ? 2 : 1);
  const bool staged = act_bytes <= ATTN - 8 * B * PER_ITEM;
  const int act_off = staged ? ((act_bytes + 15) & ~15) : 0;
  int cap = (ATTN - act_off) / (B * PER_ITEM);
  cap = cap > 64 ? 64 : cap;
  float* vbuf = reinterpret_cast<float*>(act_sm + act_off);
  float* xpre = vbuf + cap * B * 16;  // residual phases: [slot][token][16]
  const int my_items = (n - i_first + static_cast<int>(gridDim.x) - 1) / static_cast<int>(gridDim.x);
  // Residual phases: the residual slices of the next `cap` items go to
  // shared memory (L2-only copies: they were written by other SMs before the
  // phase barrier), in flight while the products run.
  auto prefetch_x = [&](int first, int count) {
    if (KIND != EPI_RESID) return;
    const uint32_t dst = smem_u32(xpre);
    for (int t = tid; t < count * B * 4; t += PCW * 32) {
      const int slot = t / (B * 4), rem = t - slot * (B * 4), b = rem >> 2, piece = rem & 3;
      const int item = first + slot * static_cast<int>(gridDim.x);
      cp_async16(dst + ((slot * B + b) * 16 + piece * 4) * 4,
                 A.x + static_cast<long long>(b) * A.D + item * 16 + piece * 4);
    }
    cp_async_commit();
  };
  if (KIND == EPI_LOGITS && tid < B) best_s[tid] = 0ull;
  if (staged) {
    const int per_row = K >> 3;  // 16-byte pieces per row
    const int total = B * per_row * (LO ? 2 : 1);
    const uint32_t base = smem_u32(act_sm);
    for (int c = tid; c < total; c += PCW * 32) {
      const int t = c / per_row, piece = c - t * per_row;
      const int term = LO ? t / B : 0, b = LO ? t - term * B : t;
      const T16* src = (term ? act_lo : act) + static_cast<long long>(b) * act_stride + piece * 8;
      cp_async16(base + (term * B + b) * pitch + piece * 16, src);
    }
    cp_async_commit();
    cp_async_wait<0>();
  }
  consumer_sync();
  prefetch_x(i_first, my_items < cap ? my_items : cap);
  // The norm scale of this phase's input: sum of the producer's partials,
  // loads issued now and reduced before the first epilogue batch.
  float rp = 0.f;
  bool rinv_pending = KIND != EPI_RESID;
  if (KIND != EPI_RESID && warp < B)
    for (int j = lane; j < A.Pmax; j += 32) rp += __ldcg(A.ss + warp * A.Pmax + j);
  // Token slot r of the MMA's N dimension holds token r, or (paired) the
  // first or second term of token r / 2.
  const int tb = paired ? (r >> 1) : r;
  const bool term_lo = paired && (r & 1);
  const bool tok_ok = tb < B;
  const int tsafe = tok_ok ? tb : 0;
  const T16* xsrc = (term_lo ? act_lo : act) + static_cast<long long>(tsafe) * act_stride + 16 * q;
  const T16* ysrc = LO ? act_lo + static_cast<long long>(tsafe) * act_stride + 16 * q : nullptr;
  const int xrow_s = term_lo ? B + tsafe : tsafe, yrow_s = B + tsafe;
  constexpr bool want_y = LO && !paired;

  // Epilogues of the buffered items slot 0 .. nslots-1 (items i0 + slot * grid).
  auto flush = [&](int i0, int nslots) {
    if (rinv_pending) {
      rp = warp_sum(rp);
      if (lane == 0 && warp < B) rinv_s[warp] = 1.0f / sqrtf(rp * A.inv_D + A.eps);
      rinv_pending = false;
    }
    cp_async_wait<0>();  // this thread's residual prefetch
    consumer_sync();     // sums of the last item, the prefetch and the norm scale visible
    unsigned long long best = 0ull;
    for (int t = tid; t < nslots * B; t += PCW * 32) {
      const int slot = t / B, b = t - slot * B;
      const int item = i0 + slot * static_cast<int>(gridDim.x);
      const int n0 = item * 16;
      float v[16];
#pragma unroll
      for (int rr = 0; rr < 16; ++rr) v[rr] = vbuf[(slot * B + b) * 16 + rr];
      if (KIND == EPI_QKV) {
        epi_qkv16<T16>(ep, b, n0, v, rinv_s[b]);
      } else if (KIND == EPI_RESID) {
        const float4* xp = reinterpret_cast<const float4*>(xpre + (slot * B + b) * 16);
        const float4 xin[4] = {xp[0], xp[1], xp[2], xp[3]};
        A.ss[b * A.Pmax + item] = epi_resid16x<T16>(ep, b, n0, v, xin);
      } else if (KIND == EPI_SWIGLU) {
        epi_swiglu16<T16>(ep, b, n0, v, rinv_s[b]);
      } else {
        best = epi_logits16(ep, b, n0, v, rinv_s[b]);
        atomicMax(best_s + b, best);
      }
    }
    consumer_sync();  // buffer free again
  };

  const int spi = (K + KC - 1) / KC;
  int slot = 0, i0 = i_first;
  for (int i = i_first; i < n; i += gridDim.x) {
    float acc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
    for (int t = 0; t < spi; ++t) {
      uint4 w0, w1, w2, w3, x0, x1, y0, y1;
      bool on;
      load_stage<HD, SM, T16, want_y>(R, cs, A, g, s_abort, t, spi, K, warp, lane, r, q, tok_ok, staged, act_sm,
                                      pitch, xsrc, ysrc, xrow_s, yrow_s, w0, w1, w2, w3, x0, x1, y0, y1, on);
      if (on) {
        const uint32_t A0[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
        const uint32_t A1[8] = {w2.x, w2.y, w2.z, w2.w, w3.x, w3.y, w3.z, w3.w};
        const uint32_t Bv[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
        // Every lane issues every MMA (mma.sync is warp-collective); token
        // slots >= B feed zeros. Two accumulators halve the dependent chain.
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint32_t a[4] = {A0[2 * j], A1[2 * j], A0[2 * j + 1], A1[2 * j + 1]};
          const uint32_t bb[2] = {Bv[2 * j], Bv[2 * j + 1]};
          mma16816<T16>(acc[j & 1], a, bb);
        }
        if (want_y) {
          const uint32_t Bl[8] = {y0.x, y0.y, y0.z, y0.w, y1.x, y1.y, y1.z, y1.w};
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const uint32_t a[4] = {A0[2 * j], A1[2 * j], A0[2 * j + 1], A1[2 * j + 1]};
            const uint32_t bb[2] = {Bl[2 * j], Bl[2 * j + 1]};
            mma16816<T16>(acc[j & 1], a, bb);
          }
        }
      }
    }
    // Accumulator of lane (r, q): rows r, r+8 x token slots 2q, 2q+1.
    float* red = red_base + cs.buf * RED_FLOATS;
    if (paired) {  // slots 2q, 2q+1 = the two terms of token q
      red[(warp * 16 + r) * 9 + q] = (acc[0][0] + acc[1][0]) + (acc[0][1] + acc[1][1]);
      red[(warp * 16 + r + 8) * 9 + q] = (acc[0][2] + acc[1][2]) + (acc[0][3] + acc[1][3]);
    } else {
      red[(warp * 16 + r) * 9 + 2 * q] = acc[0][0] + acc[1][0];
      red[(warp * 16 + r) * 9 + 2 * q + 1] = acc[0][1] + acc[1][1];
      red[(warp * 16 + r + 8) * 9 + 2 * q] = acc[0][2] + acc[1][2];
      red[(warp * 16 + r + 8) * 9 + 2 * q + 1] = acc[0][3] + acc[1][3];
    }
    consumer_sync();
    if (tid < B * 16) {
      const int b = tid >> 4, rr = tid & 15;
      float sum = 0.f;
#pragma unroll
      for (int w = 0; w < PCW; ++w) sum += red[(w * 16 + rr) * 9 + b];
      vbuf[(slot * B + b) * 16 + rr] = sum;
    }
    cs.buf ^= 1;
    if (++slot == cap) {
      flush(i0, slot);
      i0 = i + static_cast<int>(gridDim.x);
      slot = 0;
      const int left = (n - i0 + static_cast<int>(gridDim.x) - 1) / static_cast<int>(gridDim.x);
      if (left > 0) prefetch_x(i0, left < cap ? left : cap);
    }
  }
  if (slot > 0) flush(i0, slot);
  if (KIND == EPI_LOGITS && tid < B) argmax_commit(A.keys + tid, best_s[tid]);
}

AXON_DEV EpiArgs base_ep(const PersistArgs& A) {
  EpiArgs e;
  memset(&e, 0, sizeof(e));
  e.M = A.B;
  e.S = 1;
  e.ctx = A.ctx;
  e.max_pos = A.max_pos;
  e.inv_D = A.inv_D;
  e.eps = A.eps;
  e.act = A.act;
  e.H = A.H;
  e.G = A.G;
  e.d = A.d;
  e.rope = A.rope;
  e.err = A.err;
  return e;
}

template <int HD, bool SM, typename T16, int MODE>
__global__ void __launch_bounds__(PTHREADS, 1) persist_decode_kernel(PersistArgs A) {
  constexpr bool LO = MODE != TERMS_ONE;  // fp16 mode carries the split operand
  constexpr int NS = PLayout<HD, SM>::NS;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  Ring<HD, SM> R;
  R.base = smem_u32(sm + PLayout<HD, SM>::RING_OFF);
  R.bars = smem_u32(sm + PLayout<HD, SM>::BAR_OFF);
  uint8_t* attn_sm = sm + PLayout<HD, SM>::ATTN_OFF;
  float* red_base = reinterpret_cast<float*>(sm + PLayout<HD, SM>::RED_OFF);
  float* rinv_s = reinterpret_cast<float*>(sm + PLayout<HD, SM>::MISC_OFF);
  volatile int* s_abort = reinterpret_cast<volatile int*>(sm + PLayout<HD, SM>::MISC_OFF + 64);
  unsigned long long* best_s = reinterpret_cast<unsigned long long*>(sm + PLayout<HD, SM>::MISC_OFF + 128);
  PersistGrid* g = A.grid;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(R.full(s), 1);
      mbar_init(R.empty(s), PCW);
    }
    *s_abort = 0;
    fence_mbar_init();
  }
  __syncthreads();

  const int Hd = A.H * A.d;
  if (warp == PCW) {
    // ------------------------------------------------------------ producer
    int rot = 0;
    uint32_t stage = 0;
    bool stop = false;
    for (int l = 0; l < A.L && !stop; ++l) {
      stream_matrix<HD, SM>(R, A.wmaps + 4 * l + 0, A.Nqkv, A.D, rot, stage, stop, g, s_abort, A.err, lane);
      stream_matrix<HD, SM>(R, A.wmaps + 4 * l + 1, A.D, Hd, rot, stage, stop, g, s_abort, A.err, lane);
      stream_matrix<HD, SM>(R, A.wmaps + 4 * l + 2, 2 * A.F, A.D, rot, stage, stop, g, s_abort, A.err, lane);
      stream_matrix<HD, SM>(R, A.wmaps + 4 * l + 3, A.D, A.F, rot, stage, stop, g, s_abort, A.err, lane);
    }
    if (!stop)
      stream_matrix<HD, SM>(R, A.wmaps + 4 * A.L, A.V, A.D, rot, stage, stop, g, s_abort, A.err, lane);
    // Copies still in flight must land before the CTA's shared memory goes
    // away: wait for the last use of every slot.
    if (lane == 0) {
      for (uint32_t j = stage > static_cast<uint32_t>(NS) ? stage - NS : 0u; j < stage; ++j) {
        if (!mbar_try_wait(R.full(static_cast<int>(j % NS)), (j / NS) & 1u)) {
          const uint64_t t0 = global_ns();
          while (!mbar_try_wait(R.full(static_cast<int>(j % NS)), (j / NS) & 1u))
            if (global_ns() - t0 > PWAIT_NS) {
              set_err(A.err, DEVERR_TIMEOUT);
              break;
            }
        }
      }
    }
    return;
  }

  // -------------------------------------------------------------- consumers
  const int tid = threadIdx.x;
  unsigned epoch = 0;
  CState cs;
  const int B = A.B;

  // Embedding: x = E[token], a = x * g (+ its second term), sum of squares per
  // 16-column chunk (the norm partials the first projection reads).
  {
    const int chunks = A.D >> 4;
    const float* g0 = A.L > 0 ? A.layers[0].g1 : A.gf;
    const T16* E = static_cast<const T16*>(A.embed);
    for (int it = blockIdx.x * (PCW * 32) + tid; it < B * chunks; it += gridDim.x * (PCW * 32)) {
      const int b = it / chunks, c = it - b * chunks;
      int id = A.tokens[b];
      if (id < 0 || id >= A.V) {
        set_err(A.err, DEVERR_TOKEN);
        id = 0;
      }
      const T16* e = E + static_cast<long long>(id) * A.D + c * 16;
      float v[16], ag[16], s = 0.f;
#pragma unroll
      for (int k = 0; k < 16; ++k) {
        v[k] = to_f(e[k]);
        ag[k] = v[k] * g0[c * 16 + k];
        s += v[k] * v[k];
      }
      float* xr = A.x + static_cast<long long>(b) * A.D + c * 16;
#pragma unroll
      for (int k = 0; k < 16; k += 4) *reinterpret_cast<float4*>(xr + k) = make_float4(v[k], v[k + 1], v[k + 2], v[k + 3]);
      T16* ar = static_cast<T16*>(A.a) + static_cast<long long>(b) * A.D + c * 16;
      store8<T16>(ar, ag);
      store8<T16>(ar + 8, ag + 8);
      if (LO) {
        float lo[16];
#pragma unroll
        for (int k = 0; k < 16; ++k) lo[k] = ag[k] - to_f(from_f<T16>(ag[k]));
        T16* lr = static_cast<T16*>(A.a_lo) + static_cast<long long>(b) * A.D + c * 16;
        store8<T16>(lr, lo);
        store8<T16>(lr + 8, lo + 8);
      }
      A.ss[b * A.Pmax + c] = s;
    }
  }
  grid_sync(g, epoch, tid, s_abort, A.err);

  const T16* a16 = static_cast<const T16*>(A.a);
  const T16* alo16 = LO ? static_cast<const T16*>(A.a_lo) : nullptr;
  for (int l = 0; l < A.L; ++l) {
    const PersistLayer& w = A.layers[l];
    // QKV + bias + RoPE + KV store
    {
      EpiArgs e = base_ep(A);
      e.N = A.Nqkv;
      e.bias = w.bqkv;
      e.q_out = A.q;
      e.q_lo_out = A.q_lo;
      e.k_cache = w.kc;
      e.v_cache = w.vc;
      e.block_table = A.block_table;
      e.bt_stride = A.blocks_per_seq;
      e.blocks_per_seq = A.blocks_per_seq;
      e.num_blocks = A.num_blocks;
      proj_phase<HD, SM, EPI_QKV, T16, MODE>(R, cs, A, static_cast<const T16*>(w.wqkv), A.Nqkv, A.D, a16, alo16, A.D, e,
                                       red_base, rinv_s, best_s, attn_sm, g, s_abort, tid);
    }
    grid_sync(g, epoch, tid, s_abort, A.err);
    // split-KV attention
    {
      AttnArgs p;
      memset(&p, 0, sizeof(p));
      p.q = A.q;
      p.k = w.kc;
      p.v = w.vc;
      p.o = A.o;
      p.ctx = A.ctx;
      p.block_table = A.block_table;
      p.bt_stride = A.blocks_per_seq;
      p.blocks_per_seq = A.blocks_per_seq;
      p.num_blocks = A.num_blocks;
      p.H = A.H;
      p.G = A.G;
      p.d = A.d;
      p.S = 1;
      p.splits = A.splits;
      p.window = A.window;
      p.scale_log2 = A.scale_log2;
      p.part = A.attn_part;
      p.counter = A.attn_cnt;
      p.o_lo = A.o_lo;
      p.q_lo = A.q_lo;
      p.err = A.err;
      const int items = A.splits * A.G * B;
      for (int it = blockIdx.x; it < items; it += gridDim.x) {
        const int s = it % A.splits, gg = (it / A.splits) % A.G, b = it / (A.splits * A.G);
        attn_decode_item<HD, T16, true, 1, SM ? 1 : 2>(p, s, gg, b, attn_sm, tid);
      }
    }
    grid_sync(g, epoch, tid, s_abort, A.err);
    // O projection + residual; next operand a = x * g2
    {
      EpiArgs e = base_ep(A);
      e.N = A.D;
      e.x = A.x;
      e.a_out = A.a;
      e.a_lo_out = A.a_lo;
      e.gain = w.g2;
      proj_phase<HD, SM, EPI_RESID, T16, MODE>(R, cs, A, static_cast<const T16*>(w.wo), A.D, Hd,
                                         static_cast<const T16*>(A.o), static_cast<const T16*>(A.o_lo), Hd, e,
                                         red_base, rinv_s, best_s, attn_sm, g, s_abort, tid);
    }
    grid_sync(g, epoch, tid, s_abort, A.err);
    // gate/up + SwiGLU
    {
      EpiArgs e = base_ep(A);
      e.N = 2 * A.F;
      e.u_out = A.u;
      e.u_lo_out = A.u_lo;
      proj_phase<HD, SM, EPI_SWIGLU, T16, MODE>(R, cs, A, static_cast<const T16*>(w.wgu), 2 * A.F, A.D, a16, alo16, A.D, e,
                                          red_base, rinv_s, best_s, attn_sm, g, s_abort, tid);
    }
    grid_sync(g, epoch, tid, s_abort, A.err);
    // down projection + residual; next operand a = x * (next norm's gain)
    {
      EpiArgs e = base_ep(A);
      e.N = A.D;
      e.x = A.x;
      e.a_out = A.a;
      e.a_lo_out = A.a_lo;
      e.gain = w.gnext;
      proj_phase<HD, SM, EPI_RESID, T16, MODE>(R, cs, A, static_cast<const T16*>(w.wd), A.D, A.F,
                                         static_cast<const T16*>(A.u), static_cast<const T16*>(A.u_lo), A.F, e,
                                         red_base, rinv_s, best_s, attn_sm, g, s_abort, tid);
    }
    grid_sync(g, epoch, tid, s_abort, A.err);
  }
  // final norm + LM head + argmax
  {
    EpiArgs e = base_ep(A);
    e.N = A.V;
    e.logits = A.logits;
    e.logits_stride = A.V;
    e.keys = A.keys;
    proj_phase<HD, SM, EPI_LOGITS, T16, MODE>(R, cs, A, static_cast<const T16*>(A.head), A.V, A.D, a16, alo16, A.D, e,
                                        red_base, rinv_s, best_s, attn_sm, g, s_abort, tid);
  }
  grid_sync(g, epoch, tid, s_abort, A.err);
  // greedy token, context advance, keys cleared for the next step
  if (blockIdx.x == 0 && tid < B) {
    const unsigned long long k = __ldcg(A.keys + tid);
    if (A.next) A.next[tid] = static_cast<int>(0xffffffffu - static_cast<uint32_t>(k & 0xffffffffull));
    A.ctx[tid] += 1;
    A.keys[tid] = 0ull;
  }
  // Last CTA out resets the grid barrier for the next launch (every CTA has
  // passed its final barrier once it counts itself out).
  if (tid == 0) {
    __threadfence();
    if (atomicAdd(&g->exit, 1u) == gridDim.x - 1) {
      g->count = 0u;
      g->abort = 0u;
      __threadfence();
      g->exit = 0u;
    }
  }
}

template <int HD, bool SM, typename T16, int MODE>
cudaError_t launch_t(const PersistArgs& a, int nctas, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(nctas);
  cfg.blockDim = dim3(PTHREADS);
  cfg.dynamicSmemBytes = PLayout<HD, SM>::BYTES;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, persist_decode_kernel<HD, SM, T16, MODE>, a);
}

template <int HD, bool SM, typename T16, int MODE>
cudaError_t prepare_one(int* per_sm) {
  cudaError_t e = cudaFuncSetAttribute(persist_decode_kernel<HD, SM, T16, MODE>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, PLayout<HD, SM>::BYTES);
  if (e != cudaSuccess) return e;
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(per_sm, persist_decode_kernel<HD, SM, T16, MODE>, PTHREADS,
                                                       PLayout<HD, SM>::BYTES);
}

// The kernels a (head_dim, type) launches: bf16 one term; fp16 paired
// (B <= 4) and two sets (B > 4). Head_dim 64 takes the layout whose
// attention region stages two key blocks per warp, head_dim 128 the small
// one (measured at head_dim 128: the two-stage layout's 5-stage ring lost to
// the launch chain at 8B width, B = 8, bf16, 4.19 against 3.59 ms per step,
// and tied it at 32B width, B = 1, fp16). Resident CTAs per SM = the smaller
// count.
template <int HD, typename T16>
cudaError_t prepare_t(int* per_sm) {
  constexpr bool SMALL = HD == 128;
  if constexpr (!std::is_same<T16, f16>::value) {
    return prepare_one<HD, SMALL, T16, TERMS_ONE>(per_sm);
  } else {
    int a = 0, b = 0;
    cudaError_t e = prepare_one<HD, SMALL, T16, TERMS_PAIRED>(&a);
    if (e == cudaSuccess) e = prepare_one<HD, SMALL, T16, TERMS_TWO>(&b);
    *per_sm = a < b ? a : b;
    return e;
  }
}

template <int HD, typename T16>
cudaError_t launch_mode(const PersistArgs& a, int nctas, cudaStream_t st) {
  constexpr bool SMALL = HD == 128;
  if constexpr (!std::is_same<T16, f16>::value)
    return launch_t<HD, SMALL, T16, TERMS_ONE>(a, nctas, st);
  else
    return a.B <= 4 ? launch_t<HD, SMALL, T16, TERMS_PAIRED>(a, nctas, st)
                    : launch_t<HD, SMALL, T16, TERMS_TWO>(a, nctas, st);
}

// Whether B activation rows (two terms each in fp16 mode) of K columns stage
// in an attention region of `attn` bytes next to the epilogue buffer.
bool stages_in(int attn, bool use_f16, int B, int K) {
  const int rows = use_f16 ? 2 * B : B;
  return static_cast<long long>(rows) * (K * 2 + 16) <= attn - 8 * B * 16 * 4;
}

}  // namespace

int persist_ctas_per_sm(int head_dim, bool use_f16) {
  int n = 0;
  cudaError_t e;
  if (head_dim == 64)
    e = use_f16 ? prepare_t<64, f16>(&n) : prepare_t<64, bf16>(&n);
  else if (head_dim == 128)
    e = use_f16 ? prepare_t<128, f16>(&n) : prepare_t<128, bf16>(&n);
  else
    return 0;
  if (e != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

bool persist_fits(int head_dim, bool use_f16, int B, int D, int kmax) {
  if (B < 1 || B > PERSIST_MAX_B) return false;
  // Head_dim 64: the normed operand of QKV, gate/up and the LM head (K = D)
  // must stage in shared memory next to the epilogue buffer; streaming it
  // from L2 stage by stage is slower than the launch chain. Head_dim 128
  // (small layout): every projection's operand (K up to kmax) must.
  if (head_dim == 64) return stages_in(PLayout<64, false>::ATTN, use_f16, B, D);
  if (head_dim == 128) return stages_in(PLayout<128, true>::ATTN, use_f16, B, kmax);
  return false;
}

cudaError_t launch_persist_decode(const PersistArgs& a, int head_dim, bool use_f16, int nctas, cudaStream_t st) {
  if (a.B < 1 || a.B > PERSIST_MAX_B || (a.D & 63) || (a.F & 63) || ((a.H * a.d) & 63)) return cudaErrorInvalidValue;
  if (head_dim == 64) return use_f16 ? launch_mode<64, f16>(a, nctas, st) : launch_mode<64, bf16>(a, nctas, st);
  if (head_dim == 128) return use_f16 ? launch_mode<128, f16>(a, nctas, st) : launch_mode<128, bf16>(a, nctas, st);
  return cudaErrorInvalidValue;
}
