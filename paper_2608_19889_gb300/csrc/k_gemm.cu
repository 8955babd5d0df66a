// Prefill projections on the 5th-generation tensor cores: a persistent,
// warp-specialised tcgen05 GEMM, out[m][n] = A[m] . W[n] (A = bf16
// activations [M][K], W = bf16 weights [N][K], fp32 accumulation in TMEM),
// followed by the fused epilogues of epilogue.cuh.
//
//   warp 0      : TMA producer -- one lane streams 128x64 A and 256x64 W
//                 tiles (128-byte swizzle) into a 4-stage shared-memory ring,
//                 completion tracked by mbarrier transaction bytes;
//   warp 1      : MMA issuer -- allocates 512 TMEM columns (two 128x256 fp32
//                 accumulators), one lane issues tcgen05.mma kind::f16
//                 (M=128, N=256, K=16) and frees ring slots / publishes
//                 finished accumulators with tcgen05.commit;
//   warps 2..5  : epilogue -- each reads its 32 TMEM lanes (rows) 16 columns
//                 at a time with tcgen05.ld and applies the fused epilogue,
//                 overlapping the next tile's main loop (double-buffered
//                 accumulators).
// Tiles are visited in groups of 8 M-blocks per N sweep so the A and W
// working sets of the concurrently running CTAs stay L2-resident.
// Every mbarrier wait is bounded (DEVERR_TIMEOUT instead of a hang).
#include "kernels.h"

#include <cudaTypedefs.h>

namespace {

constexpr int BM = 128, BK = 64, GROUP_M = 8;
constexpr int A_BYTES = BM * BK * 2;  // 16 KB
constexpr int NUM_THREADS = 192;

// BN_: columns of the output tile (256, or 128 where 256-wide tiles leave
// the last wave mostly empty). SPLIT: the A operand is the sum of two
// 16-bit terms (hi + lo) and every k-step issues two MMAs into the same
// accumulator. The ring takes as many stages as fit in 200 KB, at most 6
// (BN 256: 4, split 3; BN 128: 6, split 4).
//
// AROWS < 128 (at most AROWS activation rows, decode: 16 or 64): each stage
// holds [A (AROWS rows) | A_lo (AROWS rows, SPLIT) | B]; the MMA still reads
// 128 A rows from the tile, rows AROWS..127 falling in the same stage's
// following bytes (landed, so stable; their accumulator rows are never
// stored). Without the padding rows a stage is smaller, so more of them --
// more weight bytes in flight per SM -- fit (up to 12).
//
// RING: the ring's byte budget. The residual kind at BN 256 keeps 8 KB of
// static shared memory for its row sums, so its ring gets 196 KB.
template <bool SPLIT, int BN_, int AROWS = 128, int RING = 200 * 1024>
struct GCfg {
  static constexpr int BN = BN_;
  static constexpr int B_BYTES = BN * BK * 2;
  static constexpr uint32_t TMEM_COLS = 2 * BN;
  static constexpr int A_TERMS = SPLIT ? 2 : 1;
  static constexpr bool SMALL = AROWS < BM;
  static constexpr int A_TILE = AROWS * BK * 2;  // bytes of one A term in a stage
  static constexpr int STAGE_BYTES = A_TERMS * A_TILE + B_BYTES;
  static constexpr int MAX_STAGES = SMALL ? 12 : 6;
  static constexpr int STAGES = RING / STAGE_BYTES > MAX_STAGES ? MAX_STAGES : RING / STAGE_BYTES;
  static_assert(!SMALL || STAGE_BYTES - (A_TERMS - 1) * A_TILE >= A_BYTES, "the MMA's 128-row read stays in its stage");
  static constexpr int BAR_BYTES = 8 * (2 * STAGES + 4) + 16;
  static constexpr int SMEM = STAGES * STAGE_BYTES + BAR_BYTES + 1024;
};

template <int KIND, int BN>
constexpr int ring_budget() { return KIND == EPI_RESID && BN == 256 ? 196 * 1024 : 200 * 1024; }
template <int KIND, bool SPLIT, int BN, int AROWS>
using GCfgK = GCfg<SPLIT, BN, AROWS, ring_budget<KIND, BN>()>;

// Residual epilogue staging: each epilogue warp's 32 rows x 32 accumulator
// columns, rows padded to 36 floats (float4 stores of 8 consecutive rows
// hit distinct banks).
constexpr int EPI_TP = 36;
template <int KIND>
constexpr int epi_smem() { return KIND == EPI_RESID ? 4 * 32 * EPI_TP * 4 : 0; }

AXON_DEV void tile_coords(int t, int num_m, int num_n, int& mb, int& nb) {
  const int per_group = GROUP_M * num_n;
  const int g = t / per_group;
  const int first_m = g * GROUP_M;
  const int gm = min(GROUP_M, num_m - first_m);
  const int local = t - g * per_group;
  nb = local / gm;
  mb = first_m + (local - nb * gm);
}

template <int KIND, typename T16, bool SPLIT, int BN_, int AROWS>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmAlo, int M, int N, int K, EpiArgs ep, int ks, float* ws,
                   int* tickets, GemmGroup grp) {
  using C = GCfgK<KIND, SPLIT, BN_, AROWS>;
  constexpr bool SMALL = C::SMALL;
  constexpr int BN = C::BN;
  constexpr int B_BYTES = C::B_BYTES;
  constexpr uint32_t TMEM_COLS = C::TMEM_COLS;
  constexpr int STAGES = C::STAGES;
  constexpr int STAGE_BYTES = C::STAGE_BYTES;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  // ring: [STAGES] A tiles, [STAGES] A_lo tiles (SPLIT), [STAGES] B tiles;
  // AROWS < 128: per stage [A | A_lo | B]
  const uint32_t sA = base, sAlo = base + STAGES * A_BYTES, sB = base + STAGES * A_BYTES * C::A_TERMS;
  auto a_at = [&](int s) { return SMALL ? base + s * STAGE_BYTES : sA + s * A_BYTES; };
  auto alo_at = [&](int s) { return SMALL ? base + s * STAGE_BYTES + C::A_TILE : sAlo + s * A_BYTES; };
  auto b_at = [&](int s) { return SMALL ? base + s * STAGE_BYTES + C::A_TERMS * C::A_TILE : sB + s * B_BYTES; };
  const uint32_t bars = base + STAGES * STAGE_BYTES;
  const uint32_t tmem_slot = bars + 8 * (2 * STAGES + 4);
  float* const epi_tile = reinterpret_cast<float*>(smem_raw + (bars + C::BAR_BYTES - raw));  // epi_smem<KIND>()
  const uint32_t* tmem_slot_ptr =
      reinterpret_cast<const uint32_t*>(smem_raw + (tmem_slot - raw));
  auto full_bar = [&](int s) { return bars + 8 * s; };
  auto empty_bar = [&](int s) { return bars + 8 * (STAGES + s); };
  auto accf_bar = [&](int i) { return bars + 8 * (2 * STAGES + i); };
  auto acce_bar = [&](int i) { return bars + 8 * (2 * STAGES + 2 + i); };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(accf_bar(i), 1);
      mbar_init(acce_bar(i), 128);
    }
    fence_mbar_init();
    fence_proxy_async();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    if (SPLIT) tma_prefetch_desc(&tmAlo);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot_ptr;

  grid_dep_wait();
  // grouped: the m-blocks the routing plan laid out (read after the wait,
  // when the plan kernel's writes are visible)
  const bool grouped = grp.mb_expert != nullptr;
  const int num_m = grouped ? __ldcg(grp.n_mblocks) : (M + BM - 1) / BM, num_n = (N + BN - 1) / BN;
  const int tiles = num_m * num_n, KB = K / BK;
  // Work units: (tile, K split) pairs, the ks splits of a tile adjacent.
  // ks > 1 only with one M tile (M <= BM): each unit leaves its partial tile
  // in `ws` and the last of a tile's units to finish sums them.
  const int units = tiles * ks;

  if (warp == 0) {
    if (lane == 0) {
      int it = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
        const int t = u / ks, sp = u - t * ks;
        int mb, nb;
        tile_coords(t, num_m, num_n, mb, nb);
        if (grouped) {
          mb = t / num_n;
          nb = t - mb * num_n;
        }
        const int wrow = grouped ? __ldcg(grp.mb_expert + mb) * N + nb * BN : nb * BN;
        const int kb1 = (sp + 1) * KB / ks;
        for (int kb = sp * KB / ks; kb < kb1; ++kb, ++it) {
          const int s = it % STAGES;
          const uint32_t ph = (it / STAGES) & 1;
          if (!mbar_wait(empty_bar(s), ph ^ 1, ep.err)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(full_bar(s), STAGE_BYTES);
          tma_load_2d(a_at(s), &tmA, full_bar(s), kb * BK, mb * BM);
          if (SPLIT) tma_load_2d(alo_at(s), &tmAlo, full_bar(s), kb * BK, mb * BM);
          tma_load_2d(b_at(s), &tmB, full_bar(s), kb * BK, wrow);
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_f32acc(BM, BN, MmaFmt<T16>::v);
      int it = 0, lt = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x, ++lt) {
        const int sp = u % ks;
        const int kb0 = sp * KB / ks, kb1 = (sp + 1) * KB / ks;
        const int buf = lt & 1;
        const uint32_t aph = (lt >> 1) & 1;
        if (!mbar_wait(acce_bar(buf), aph ^ 1, ep.err)) break;
        tc_fence_after();
        const uint32_t d = tmem + buf * BN;
        for (int kb = kb0; kb < kb1; ++kb, ++it) {
          const int s = it % STAGES;
          const uint32_t ph = (it / STAGES) & 1;
          if (!mbar_wait(full_bar(s), ph, ep.err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t ad = smem_desc_sw128(a_at(s));
          const uint64_t bd = smem_desc_sw128(b_at(s));
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)  // +32 bytes along K inside the swizzle atom
            tc_mma_f16(d, ad + 2 * k, bd + 2 * k, idesc, (kb != kb0 || k != 0) ? 1u : 0u);
          if (SPLIT) {
            const uint64_t ald = smem_desc_sw128(alo_at(s));
#pragma unroll
            for (int k = 0; k < BK / 16; ++k) tc_mma_f16(d, ald + 2 * k, bd + 2 * k, idesc, 1u);
          }
          tc_commit(empty_bar(s));
        }
        if (ok) tc_commit(accf_bar(buf));
      }
    }
    __syncwarp();
  } else {
    const int q4 = warp & 3;  // TMEM lane quarter this warp may read
    const int row = q4 * 32 + lane;
    const int etid = threadIdx.x - 64;  // 0..127 over the 4 epilogue warps
    __shared__ int s_last;
    __shared__ float s_rinv[BM];
    __shared__ float s_ssp[KIND == EPI_RESID ? BM : 1][KIND == EPI_RESID ? BN / 16 : 1];
    int lt = 0;
    for (int u = blockIdx.x; u < units; u += gridDim.x, ++lt) {
      const int t = u / ks;
      int mb, nb;
      tile_coords(t, num_m, num_n, mb, nb);
      if (grouped) {
        mb = t / num_n;
        nb = t - mb * num_n;
      }
      const int buf = lt & 1;
      const uint32_t aph = (lt >> 1) & 1;
      const bool got = mbar_wait(accf_bar(buf), aph, ep.err);
      __syncwarp();
      if (!got) break;
      tc_fence_after();
      if (ks > 1) {
        // 1. this unit's partial tile -> workspace (rows < M; mb == 0)
        const uint32_t taddr = tmem + (static_cast<uint32_t>(q4 * 32) << 16) + buf * BN;
        float* wp = ws + (static_cast<long long>(u) * BM + row) * BN;
#pragma unroll 1
        for (int c = 0; c < BN; c += 16) {
          uint32_t v[16];
          tmem_ld16(taddr + c, v);
          tmem_wait_ld();
          if (row < M) {
#pragma unroll
            for (int i = 0; i < 16; i += 4)
              *reinterpret_cast<float4*>(wp + c + i) =
                  make_float4(__uint_as_float(v[i]), __uint_as_float(v[i + 1]), __uint_as_float(v[i + 2]),
                              __uint_as_float(v[i + 3]));
          }
        }
        tc_fence_before();
        mbar_arrive(acce_bar(buf));
        // ticket after the epilogue warps' barrier: one acquire-release atomic
        // publishes the four warps' partial stores and, for the last unit,
        // orders its loads of the other units' partials after theirs
        asm volatile("bar.sync 1, 128;" ::: "memory");
        if (etid == 0) s_last = (atom_add_acq_rel_gpu(tickets + t, 1) == ks - 1);
        asm volatile("bar.sync 1, 128;" ::: "memory");
        if (s_last) {
          // 2. last unit of the tile: sum the ks partials in split order
          // (deterministic) and run the epilogue, as (row, 16 columns) tasks
          if (KIND != EPI_RESID && etid < M) s_rinv[etid] = row_rinv(ep, etid);
          asm volatile("bar.sync 1, 128;" ::: "memory");
          constexpr int CH = BN / 16;
          for (int task = etid; task < M * CH; task += 128) {
            const int m = task / CH, c = (task - m * CH) * 16;
            const int n0 = nb * BN + c;
            if (n0 >= N) continue;
            float f[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) f[i] = 0.f;
            // four splits' loads in flight per round trip, added in split order
            for (int sp0 = 0; sp0 < ks; sp0 += 4) {
              float4 a4[4][4];
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                const bool in = sp0 + u < ks;
                const float* pp = ws + ((static_cast<long long>(t) * ks + (in ? sp0 + u : 0)) * BM + m) * BN + c;
#pragma unroll
                for (int i = 0; i < 4; ++i)
                  a4[u][i] = in ? __ldcg(reinterpret_cast<const float4*>(pp + 4 * i)) : make_float4(0.f, 0.f, 0.f, 0.f);
              }
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                if (sp0 + u >= ks) break;
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                  f[4 * i] += a4[u][i].x;
                  f[4 * i + 1] += a4[u][i].y;
                  f[4 * i + 2] += a4[u][i].z;
                  f[4 * i + 3] += a4[u][i].w;
                }
              }
            }
            if (KIND == EPI_QKV) {
              epi_qkv16<T16>(ep, m, n0, f, s_rinv[m]);
            } else if (KIND == EPI_RESID) {
              s_ssp[m][c >> 4] = epi_resid16<T16>(ep, m, n0, f);
            } else if (KIND == EPI_SWIGLU) {
              epi_swiglu16<T16>(ep, m, n0, f, s_rinv[m]);
            } else {
              argmax_commit(ep.keys + m, epi_logits16(ep, m, n0, f, s_rinv[m]));
            }
          }
          asm volatile("bar.sync 1, 128;" ::: "memory");
          if (KIND == EPI_RESID && etid < M) {
            // the row's norm partial for this 256-wide tile, chunks summed in order
            // (as the unsplit tile would); chunks past N count zero
            float ssum = 0.f;
            for (int c = 0; c < BN / 16; ++c)
              if (nb * BN + c * 16 < N) ssum += s_ssp[etid][c];
            ep.ss_out[static_cast<long long>(etid) * ep.ss_out_stride + nb] = ssum;
          }
          if (etid == 0) tickets[t] = 0;
        }
        continue;
      }
      const int m = mb * BM + row;
      const bool mval = m < M && (!grp.row_valid || grp.row_valid[m] >= 0);
      float rinv = 1.f;
      if (KIND != EPI_RESID && KIND != EPI_ROWSCALE && mval) rinv = row_rinv(ep, m);
      unsigned long long best = 0ull;
      const uint32_t taddr = tmem + (static_cast<uint32_t>(q4 * 32) << 16) + buf * BN;
      if (KIND == EPI_RESID) {
        // Through shared memory, 32 columns at a time: the warp stages its 32
        // rows x 32 accumulator columns, then every global access (residual
        // read, x, a and a_lo writes) covers 4 rows x 128 bytes per
        // instruction, lane (r, c) taking row 4i + r, columns 4c .. 4c+3.
        float* tw = epi_tile + q4 * 32 * EPI_TP;
        const int lr = lane >> 3, lc = (lane & 7) * 4;
        const int mrow = mb * BM + q4 * 32 + lr;  // + 4i: the lane's rows
        bool rv[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int mm = mrow + 4 * i;
          rv[i] = mm < M && (!grp.row_valid || grp.row_valid[mm] >= 0);
        }
        // residual slices of group c0 (8 rows x 4 columns per lane), loaded
        // one group ahead so that their round trip overlaps the previous
        // group's stores
        auto load_x = [&](int c0, float4 (&xr)[8]) {
          const int n = nb * BN + c0 + lc;
#pragma unroll
          for (int i = 0; i < 8; ++i)
            xr[i] = (rv[i] && n < N) ? __ldcg(reinterpret_cast<const float4*>(
                                           ep.x + static_cast<long long>(mrow + 4 * i) * ep.N + n))
                                     : make_float4(0.f, 0.f, 0.f, 0.f);
        };
        float rs[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) rs[i] = 0.f;
        float4 xcur[8], xnext[8];
        load_x(0, xcur);
#pragma unroll 1
        for (int c0 = 0; c0 < BN; c0 += 32) {
          if (c0 + 32 < BN) load_x(c0 + 32, xnext);
          uint32_t v[2][16];
          tmem_ld16(taddr + c0, v[0]);
          tmem_ld16(taddr + c0 + 16, v[1]);
          tmem_wait_ld();
#pragma unroll
          for (int j = 0; j < 8; ++j)
            *reinterpret_cast<float4*>(tw + lane * EPI_TP + 4 * j) =
                make_float4(__uint_as_float(v[j >> 2][(j & 3) * 4]), __uint_as_float(v[j >> 2][(j & 3) * 4 + 1]),
                            __uint_as_float(v[j >> 2][(j & 3) * 4 + 2]), __uint_as_float(v[j >> 2][(j & 3) * 4 + 3]));
          __syncwarp();
          const int n = nb * BN + c0 + lc;
          const float4 g4 = n < N ? *reinterpret_cast<const float4*>(ep.gain + n) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const int rl = 4 * i + lr;
            float part = 0.f;
            if (rv[i] && n < N) {
              const float4 acc = *reinterpret_cast<const float4*>(tw + rl * EPI_TP + lc);
              const float4 xo = xcur[i];
              const float xn[4] = {xo.x + acc.x, xo.y + acc.y, xo.z + acc.z, xo.w + acc.w};
              const long long off = static_cast<long long>(mrow + 4 * i) * ep.N + n;
              *reinterpret_cast<float4*>(ep.x + off) = make_float4(xn[0], xn[1], xn[2], xn[3]);
              const float ag[4] = {xn[0] * g4.x, xn[1] * g4.y, xn[2] * g4.z, xn[3] * g4.w};
              *reinterpret_cast<uint2*>(static_cast<T16*>(ep.a_out) + off) =
                  make_uint2(pack2<T16>(ag[0], ag[1]), pack2<T16>(ag[2], ag[3]));
              if (ep.a_lo_out) {
                float lo[4];
#pragma unroll
                for (int k = 0; k < 4; ++k) lo[k] = ag[k] - to_f(from_f<T16>(ag[k]));
                *reinterpret_cast<uint2*>(static_cast<T16*>(ep.a_lo_out) + off) =
                    make_uint2(pack2<T16>(lo[0], lo[1]), pack2<T16>(lo[2], lo[3]));
              }
              part = ((xn[0] * xn[0] + xn[1] * xn[1]) + xn[2] * xn[2]) + xn[3] * xn[3];
            }
            // the row's 32 columns: the 8 lanes of the row, fixed tree order
            part += __shfl_xor_sync(0xffffffffu, part, 1);
            part += __shfl_xor_sync(0xffffffffu, part, 2);
            part += __shfl_xor_sync(0xffffffffu, part, 4);
            rs[i] += part;
          }
          __syncwarp();
#pragma unroll
          for (int i = 0; i < 8; ++i) xcur[i] = xnext[i];
        }
        if ((lane & 7) == 0) {
#pragma unroll
          for (int i = 0; i < 8; ++i)
            if (rv[i]) ep.ss_out[static_cast<long long>(mrow + 4 * i) * ep.ss_out_stride + nb] = rs[i];
        }
      }
#pragma unroll 1
      for (int c = 0; c < BN && KIND != EPI_RESID; c += 16) {
        uint32_t v[16];
        tmem_ld16(taddr + c, v);
        tmem_wait_ld();
        const int n0 = nb * BN + c;
        if (mval && n0 < N) {
          float f[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) f[i] = __uint_as_float(v[i]);
          if (KIND == EPI_QKV) {
            epi_qkv16<T16>(ep, m, n0, f, rinv);
          } else if (KIND == EPI_SWIGLU) {
            epi_swiglu16<T16>(ep, m, n0, f, rinv);
          } else if (KIND == EPI_ROWSCALE) {
            epi_rowscale16(ep, m, n0, f);
          } else {
            const unsigned long long k = epi_logits16(ep, m, n0, f, rinv);
            best = k > best ? k : best;
          }
        }
      }
      tc_fence_before();
      mbar_arrive(acce_bar(buf));

      if (KIND == EPI_LOGITS && mval) argmax_commit(ep.keys + m, best);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

template <int KIND, typename T16, bool SPLIT, int BN, int AROWS>
cudaError_t launch_kind(const LaunchCtx& lc, const GemmMaps& maps, int M, int N, int K, const EpiArgs& ep,
                        const GemmSplitK& sk, const GemmGroup& grp) {
  const int tiles = ((M + BM - 1) / BM) * ((N + BN - 1) / BN) * sk.ks;
  // grouped: the tile count is known only on the device; one CTA per SM
  const int grid = grp.mb_expert ? lc.num_sms : (tiles < lc.num_sms ? tiles : lc.num_sms);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(NUM_THREADS);
  cfg.dynamicSmemBytes = GCfgK<KIND, SPLIT, BN, AROWS>::SMEM + epi_smem<KIND>();
  cfg.stream = lc.stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = lc.pdl ? 1 : 0;
  const GemmMaps& g = BN == 256 ? maps : *maps.n128;
  const CUtensorMap& ta = AROWS == 16 ? g.a16 : (AROWS == 64 ? g.a64 : g.a);
  const CUtensorMap& tlo = SPLIT ? (AROWS == 16 ? g.a_lo16 : (AROWS == 64 ? g.a_lo64 : g.a_lo)) : ta;
  return cudaLaunchKernelEx(&cfg, gemm_tc_kernel<KIND, T16, SPLIT, BN, AROWS>, ta, g.w, tlo, M, N, K, ep, sk.ks,
                            sk.ws, sk.tickets, grp);
}

}  // namespace

bool make_tma_2d_16(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows, bool f16) {
  PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
  if (!fn || (reinterpret_cast<uintptr_t>(base) & 15) || ((cols * 2) & 15)) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(BK), box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, f16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool make_tma_2d_plain(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_cols,
                       uint32_t box_rows, bool f16) {
  PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
  if (!fn || (reinterpret_cast<uintptr_t>(base) & 15) || ((cols * 2) & 15) || ((box_cols * 2) & 15)) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {box_cols, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, f16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base),
            dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

namespace {
template <int KIND, typename T16, bool SPLIT, int BN, int AROWS>
cudaError_t set_smem1() {
  return cudaFuncSetAttribute(gemm_tc_kernel<KIND, T16, SPLIT, BN, AROWS>,
                              cudaFuncAttributeMaxDynamicSharedMemorySize,
                              GCfgK<KIND, SPLIT, BN, AROWS>::SMEM + epi_smem<KIND>());
}
template <int KIND, typename T16, bool SPLIT>
cudaError_t set_smem() {
  cudaError_t e = set_smem1<KIND, T16, SPLIT, 256, 128>();
  if (e == cudaSuccess) e = set_smem1<KIND, T16, SPLIT, 128, 128>();
  if constexpr (KIND != EPI_ROWSCALE) {  // the small-M layouts (decode kinds)
    if (e == cudaSuccess) e = set_smem1<KIND, T16, SPLIT, 256, 16>();
    if (e == cudaSuccess) e = set_smem1<KIND, T16, SPLIT, 128, 16>();
    if (e == cudaSuccess) e = set_smem1<KIND, T16, SPLIT, 256, 64>();
    if (e == cudaSuccess) e = set_smem1<KIND, T16, SPLIT, 128, 64>();
  }
  return e;
}
template <typename T16>
cudaError_t prepare_gemm_t() {
  cudaError_t e = set_smem<EPI_QKV, T16, false>();
  if (e == cudaSuccess) e = set_smem<EPI_QKV, T16, true>();
  if (e == cudaSuccess) e = set_smem<EPI_RESID, T16, false>();
  if (e == cudaSuccess) e = set_smem<EPI_SWIGLU, T16, false>();
  if (e == cudaSuccess) e = set_smem<EPI_LOGITS, T16, false>();
  if (e == cudaSuccess) e = set_smem<EPI_ROWSCALE, T16, false>();
  return e;
}
template <typename T16, int BN, int AROWS>
cudaError_t launch_t(const LaunchCtx& lc, int kind, const GemmMaps& maps, int M, int N, int K, const EpiArgs& ep,
                     const GemmSplitK& sk, const GemmGroup& grp) {
  switch (kind) {
    case EPI_QKV:
      return maps.split ? launch_kind<EPI_QKV, T16, true, BN, AROWS>(lc, maps, M, N, K, ep, sk, grp)
                        : launch_kind<EPI_QKV, T16, false, BN, AROWS>(lc, maps, M, N, K, ep, sk, grp);
    case EPI_RESID: return launch_kind<EPI_RESID, T16, false, BN, AROWS>(lc, maps, M, N, K, ep, sk, grp);
    case EPI_SWIGLU: return launch_kind<EPI_SWIGLU, T16, false, BN, AROWS>(lc, maps, M, N, K, ep, sk, grp);
    case EPI_ROWSCALE: return launch_kind<EPI_ROWSCALE, T16, false, BN, 128>(lc, maps, M, N, K, ep, sk, grp);
    default: return launch_kind<EPI_LOGITS, T16, false, BN, AROWS>(lc, maps, M, N, K, ep, sk, grp);
  }
}
template <int BN, int AROWS>
cudaError_t launch_ar(const LaunchCtx& lc, int kind, const GemmMaps& maps, int M, int N, int K, const EpiArgs& ep,
                      const GemmSplitK& sk, const GemmGroup& grp) {
  return lc.f16 ? launch_t<f16, BN, AROWS>(lc, kind, maps, M, N, K, ep, sk, grp)
                : launch_t<bf16, BN, AROWS>(lc, kind, maps, M, N, K, ep, sk, grp);
}
template <int BN>
cudaError_t launch_bn(const LaunchCtx& lc, int kind, const GemmMaps& maps, int M, int N, int K, const EpiArgs& ep,
                      const GemmSplitK& sk, const GemmGroup& grp, int arows) {
  if (arows == 16) return launch_ar<BN, 16>(lc, kind, maps, M, N, K, ep, sk, grp);
  if (arows == 64) return launch_ar<BN, 64>(lc, kind, maps, M, N, K, ep, sk, grp);
  return launch_ar<BN, 128>(lc, kind, maps, M, N, K, ep, sk, grp);
}
}  // namespace

// Output-tile width for an M x N product: 128 where 256-wide tiles leave
// the last wave mostly idle (cost in column-waves: waves x width, plus a
// per-tile overhead worth 16 columns), 256 otherwise.
int gemm_tile_n(const LaunchCtx& lc, const GemmMaps& maps, int M, int N) {
  if (!maps.n128) return 256;
  const long long mt = (M + BM - 1) / BM;
  const long long t256 = mt * ((N + 255) / 256), t128 = mt * ((N + 127) / 128);
  const long long w256 = (t256 + lc.num_sms - 1) / lc.num_sms, w128 = (t128 + lc.num_sms - 1) / lc.num_sms;
  const long long c256 = w256 * (256 + 16), c128 = w128 * (128 + 16);
  return c128 * 100 < c256 * 85 ? 128 : 256;
}

cudaError_t prepare_gemm_kernels() {
  cudaError_t e = prepare_gemm_t<bf16>();
  if (e == cudaSuccess) e = prepare_gemm_t<f16>();
  return e;
}

cudaError_t launch_gemm_tc(const LaunchCtx& lc, int kind, const GemmMaps& maps, int M, int N, int K,
                           const EpiArgs& ep, int tile_n, const GemmSplitK* split, const GemmGroup* group) {
  if (M < 1 || N < 1 || K < BK || (K % BK)) return cudaErrorInvalidValue;
  const GemmGroup grp = group ? *group : GemmGroup{};
  if (grp.mb_expert && (!grp.n_mblocks || (split && split->ks > 1) || (M % BM))) return cudaErrorInvalidValue;
  if (kind == EPI_ROWSCALE && !grp.mb_expert) return cudaErrorInvalidValue;
  GemmSplitK sk;
  if (split && split->ks > 1) {
    // one M tile, 256-wide tiles, at most GEMM_MAX_UNITS units, at least one K block per unit
    const int tiles = (N + 255) / 256;
    if (M > BM || tile_n != 256 || !split->ws || !split->tickets || tiles * split->ks > GEMM_MAX_UNITS ||
        split->ks > K / BK || tiles > split->max_tiles)
      return cudaErrorInvalidValue;
    sk = *split;
  }
  // at most 16 (64) rows -- one M block -- and activation boxes of 16 (64)
  // rows: the small-M stage layouts
  const bool dec = !grp.mb_expert && kind != EPI_ROWSCALE;
  const int arows = (dec && M <= 16 && maps.has16) ? 16 : ((dec && M <= 64 && maps.has64) ? 64 : 128);
  if (tile_n == 128) {
    if (!maps.n128) return cudaErrorInvalidValue;
    return launch_bn<128>(lc, kind, maps, M, N, K, ep, sk, grp, arows);
  }
  return launch_bn<256>(lc, kind, maps, M, N, K, ep, sk, grp, arows);
}

int gemm_split_k(const LaunchCtx& lc, int M, int N, int K) {
  if (M > BM) return 1;
  const int tiles = (N + 255) / 256;
  if (2 * tiles >= lc.num_sms) return 1;
  int ks = lc.num_sms / tiles;
  const int kmax = K / BK / 4;  // keep >= 4 K blocks per unit
  if (ks > kmax) ks = kmax;
  if (ks > 16) ks = 16;
  if (tiles * ks > GEMM_MAX_UNITS) ks = GEMM_MAX_UNITS / tiles;
  return ks < 2 ? 1 : ks;
}
