// Device utilities shared by the kernels: bf16 packing, warp reductions,
// and inline-PTX wrappers for the sm_103a features the kernels use
// (mma.sync for skinny decode products, ldmatrix/cp.async for attention
// tiles, mbarrier + TMA + tcgen05/TMEM for the prefill GEMM).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda.h>
#include <stdint.h>

#define AXON_DEV __device__ __forceinline__

typedef __nv_bfloat16 bf16;
typedef __half f16;

// Device error word bits (read by axon_check_device).
enum : int {
  DEVERR_TOKEN = 1,    // token id outside [0, V)
  DEVERR_BLOCK = 2,    // block-table entry outside [0, num_blocks)
  DEVERR_POS = 4,      // position outside [0, max_context)
  DEVERR_TIMEOUT = 8,  // a bounded mbarrier wait expired
  DEVERR_SEQ = 16,     // variable-length batch: row offsets or cached lengths inconsistent
};

AXON_DEV void set_err(int* err, int bit) {
  if (err) atomicOr(err, bit);
}

// ------------------------------------------------------------------ bf16
AXON_DEV float bf_lo(uint32_t v) { return __uint_as_float(v << 16); }
AXON_DEV float bf_hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }
AXON_DEV uint32_t pack_bf2(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}
// fp16 operands saturate at the largest finite half (NaN passes through).
AXON_DEV float sat_half(float v) { return fabsf(v) > 65504.f ? copysignf(65504.f, v) : v; }
AXON_DEV uint32_t pack_h2(float lo, float hi) {
  __half2 h = __floats2half2_rn(sat_half(lo), sat_half(hi));
  return *reinterpret_cast<uint32_t*>(&h);
}
template <typename T> AXON_DEV uint32_t pack2(float lo, float hi);
template <> AXON_DEV uint32_t pack2<bf16>(float lo, float hi) { return pack_bf2(lo, hi); }
template <> AXON_DEV uint32_t pack2<f16>(float lo, float hi) { return pack_h2(lo, hi); }
AXON_DEV float to_f(bf16 v) { return __bfloat162float(v); }
AXON_DEV float to_f(f16 v) { return __half2float(v); }
AXON_DEV float to_f(float v) { return v; }
template <typename T> AXON_DEV T from_f(float v);
template <> AXON_DEV float from_f<float>(float v) { return v; }
template <> AXON_DEV bf16 from_f<bf16>(float v) { return __float2bfloat16_rn(v); }
template <> AXON_DEV f16 from_f<f16>(float v) { return __float2half_rn(sat_half(v)); }

// --------------------------------------------------------------- reductions
AXON_DEV float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
AXON_DEV float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// Orderable 64-bit argmax key: larger value wins, lower index wins ties.
AXON_DEV unsigned long long argmax_key(float v, int idx) {
  uint32_t b = __float_as_uint(v);
  b = (b & 0x80000000u) ? ~b : (b | 0x80000000u);
  return (static_cast<unsigned long long>(b) << 32) | (0xffffffffu - static_cast<uint32_t>(idx));
}

// ------------------------------------------------------------ global loads
// Streaming 16-byte load that bypasses L1 allocation (weights: read once).
AXON_DEV uint4 ld_stream16(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}
// Cached 16-byte load (activations: reused by every warp of the SM).
AXON_DEV uint4 ld16(const void* p) { return *reinterpret_cast<const uint4*>(p); }

AXON_DEV void prefetch_l2(const void* p) { asm volatile("prefetch.global.L2 [%0];" ::"l"(p)); }

// ------------------------------------------------------- programmatic launch
// Wait until the preceding kernel in the stream has completed and its
// writes are visible (no-op when launched without programmatic dependency).
AXON_DEV void grid_dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
// Allow the next kernel in the stream to begin launching.
AXON_DEV void grid_dep_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// ---------------------------------------------------------------- mma.sync
AXON_DEV void mma_bf16_16816(float* c, const uint32_t* a, const uint32_t* b) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}

AXON_DEV void mma_f16_16816(float* c, const uint32_t* a, const uint32_t* b) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}
// m16n8k16 with fp32 accumulation on 16-bit operands of type T (bf16 or fp16).
template <typename T> AXON_DEV void mma16816(float* c, const uint32_t* a, const uint32_t* b);
template <> AXON_DEV void mma16816<bf16>(float* c, const uint32_t* a, const uint32_t* b) { mma_bf16_16816(c, a, b); }
template <> AXON_DEV void mma16816<f16>(float* c, const uint32_t* a, const uint32_t* b) { mma_f16_16816(c, a, b); }

AXON_DEV uint32_t smem_u32(const void* p) { return static_cast<uint32_t>(__cvta_generic_to_shared(p)); }

AXON_DEV void ldsm_x4(uint32_t* r, uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
AXON_DEV void ldsm_x4_t(uint32_t* r, uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}

AXON_DEV void cp_async16(uint32_t smem, const void* g) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem), "l"(g) : "memory");
}
AXON_DEV void cp_async16_zfill(uint32_t smem, const void* g, bool valid) {
  int n = valid ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem), "l"(g), "r"(n) : "memory");
}
AXON_DEV void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
AXON_DEV void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// ---------------------------------------------------------------- mbarrier
AXON_DEV void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
AXON_DEV void fence_mbar_init() { asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory"); }
AXON_DEV void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }
AXON_DEV void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
AXON_DEV void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
AXON_DEV bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
AXON_DEV uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// Bounded wait on an mbarrier phase: gives up after ~`limit_ns` and
// reports DEVERR_TIMEOUT instead of spinning forever.
AXON_DEV bool mbar_wait(uint32_t bar, uint32_t parity, int* err, uint64_t limit_ns = 2000000000ull) {
  if (mbar_try_wait(bar, parity)) return true;
  uint64_t t0 = global_ns();
  while (true) {
    for (int i = 0; i < 64; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (global_ns() - t0 > limit_ns) {
      set_err(err, DEVERR_TIMEOUT);
      return false;
    }
  }
}

// --------------------------------------------------------------------- TMA
AXON_DEV void tma_load_2d(uint32_t dst, const CUtensorMap* map, uint32_t bar, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}
// The same load with an L2 eviction policy (createpolicy_evict_first): data
// read once per pass should not push reusable lines out of L2.
AXON_DEV void tma_load_2d_hint(uint32_t dst, const CUtensorMap* map, uint32_t bar, int x, int y, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1, {%2, "
      "%3}], [%4], %5;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar), "l"(policy)
      : "memory");
}
AXON_DEV uint64_t createpolicy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
// Atomic add at gpu scope with acquire-release semantics; returns the old
// value. After a CTA barrier, one thread's release covers the CTA's writes.
AXON_DEV int atom_add_acq_rel_gpu(int* p, int v) {
  int old;
  asm volatile("atom.add.acq_rel.gpu.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}
AXON_DEV void tma_prefetch_desc(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

// ------------------------------------------------------------ tcgen05/TMEM
AXON_DEV void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
               : "memory");
}
AXON_DEV void tmem_relinquish() { asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory"); }
AXON_DEV void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
AXON_DEV void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
AXON_DEV void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
// D[tmem] (+)= A[smem desc] * B[smem desc]^T, kind::f16 (bf16 in, fp32 acc).
AXON_DEV void tc_mma_f16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(
          d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive on an mbarrier once every previously issued tcgen05.mma completed.
AXON_DEV void tc_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}
// 32 lanes x 16 consecutive 32-bit TMEM columns; thread i gets lane (base+i).
AXON_DEV void tmem_ld16(uint32_t taddr, uint32_t* r) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr)
      : "memory");
}
AXON_DEV void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// Shared-memory matrix descriptor for tcgen05 (K-major operand, 128-byte
// swizzle, 8-row core groups 1024 bytes apart).
AXON_DEV uint64_t smem_desc_sw128(uint32_t addr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((addr >> 4) & 0x3FFFu);          // start address
  d |= static_cast<uint64_t>(1u) << 16;                      // leading byte offset (unused for SW128 K-major)
  d |= static_cast<uint64_t>(1024u >> 4) << 32;              // stride byte offset: 8 rows x 128 B
  d |= static_cast<uint64_t>(1u) << 46;                      // descriptor version (tcgen05)
  d |= static_cast<uint64_t>(2u) << 61;                      // swizzle: 128B
  return d;
}
// Instruction descriptor: kind::f16, A=B=bf16 (ab_fmt 1) or fp16 (ab_fmt 0),
// D=fp32, both K-major.
__host__ __device__ constexpr uint32_t idesc_f32acc(int M, int N, uint32_t ab_fmt) {
  return (1u << 4)                                 // D format fp32
         | (ab_fmt << 7)                           // A format
         | (ab_fmt << 10)                          // B format
         | (static_cast<uint32_t>(N >> 3) << 17)   // N / 8
         | (static_cast<uint32_t>(M >> 4) << 24);  // M / 16
}
template <typename T> struct MmaFmt;
template <> struct MmaFmt<bf16> { static constexpr uint32_t v = 1; };
template <> struct MmaFmt<f16> { static constexpr uint32_t v = 0; };
