// Inline-PTX wrappers for the 5th-generation tensor cores (tcgen05 / TMEM) and mbarriers on sm_103a.
//
// Conventions used by the kernels that include this file:
//  * Operand tiles in shared memory are K-major with the 128-byte swizzle: rows of 64 16-bit elements
//    (128 B); 8 rows form a 1024-byte atom; the 16-byte chunk j of row r sits at chunk position j ^ (r % 8).
//    Tiles start on 1024-byte boundaries. One MMA consumes K = 16 elements (32 B) of every row; the k-th
//    16-element slice of a 64-wide tile is addressed by advancing the descriptor's start address by 32 B.
//  * The accumulator D (M = 128 rows) lives in tensor memory, row i in lane i, one fp32 column per N index.
//  * Every wait is bounded: after kWaitNs of spinning a wait gives up, records kErrTimeout in the kernel's
//    error word and returns false, so a broken pipeline ends the kernel instead of hanging the GPU.
#pragma once

#include <cuda_fp16.h>
#include <stdint.h>

namespace externd {

constexpr unsigned kErrTimeout = 1u;
constexpr unsigned long long kWaitNs = 2000000000ull;   // 2 s

__device__ __forceinline__ uint32_t smem_addr(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("{\n\t.reg .b64 st;\n\tmbarrier.arrive.shared::cta.b64 st, [%0];\n\t}" ::"r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\tselp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Waits for the phase with the given parity to complete; false (and the error word set) after kWaitNs.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, unsigned* err) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 255u) == 0 && global_ns() - t0 > kWaitNs) {
      atomicOr(err, kErrTimeout);
      return false;
    }
  }
}

// Arrives once on the mbarrier and adds `bytes` to the transaction count its current phase waits for.
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

// Orders this thread's generic-proxy shared-memory accesses before later async-proxy ones: its writes become
// visible to the tensor core, and its reads of a buffer complete before a bulk copy refills the buffer.
__device__ __forceinline__ void fence_async_shared() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// ---- tensor memory
__device__ __forceinline__ void tmem_alloc(uint32_t result_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(result_smem), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// 32 lanes x 16 consecutive 32-bit columns starting at taddr (lane field = the warp's quadrant).
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&v)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
        "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// ---- MMA
// Shared-memory matrix descriptor of a K-major, 128-byte-swizzled tile starting at saddr (1024-aligned atom
// base plus a multiple of 32 B for the K slice): stride between 8-row atoms 1024 B, descriptor version 1.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
         ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

// Instruction descriptor of kind::f16 with fp16 A and B, fp32 D, both operands K-major, M x N.
__host__ __device__ constexpr uint32_t f16_idesc(uint32_t M, uint32_t N) {
  return (1u << 4) | (0u << 7) | (0u << 10) | ((N >> 3) << 17) | ((M >> 4) << 24);
}

// D[tmem] (+)= A[smem] * B[smem]^T, issued by one thread.
__device__ __forceinline__ void mma_f16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                        uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// The same with A in tensor memory (M rows in lanes, two 16-bit K elements per 32-bit column from a_tmem on).
__device__ __forceinline__ void mma_f16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc,
                                           uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// 32 lanes x 4 consecutive 32-bit columns from taddr (lane field = the warp's quadrant): each thread its lane.
__device__ __forceinline__ void tmem_st4(uint32_t taddr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x4.b32 [%0], {%1, %2, %3, %4};" ::"r"(taddr), "r"(a), "r"(b), "r"(c),
               "r"(d)
               : "memory");
}
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// Arrives (once) on the mbarrier when every MMA issued so far by this thread has completed.
__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}

// ---- operand packing
__device__ __forceinline__ uint32_t pack_half2(float lo_elem, float hi_elem) {
  const __half a = __float2half_rn(lo_elem), b = __float2half_rn(hi_elem);
  return (uint32_t)__half_as_ushort(a) | ((uint32_t)__half_as_ushort(b) << 16);
}

// Splits x (already scaled into fp16 range) into hi + lo fp16 parts: hi = RN16(x), lo = RN16(x - hi); the
// residual x - hi is exact in float32, so hi + lo carries ~22 significant bits of x.
__device__ __forceinline__ void split_f16(float x, __half& hi, __half& lo) {
  hi = __float2half_rn(x);
  lo = __float2half_rn(x - __half2float(hi));
}

// Byte offset of the 16-byte chunk j (0..7) of row r in a 128-byte-swizzled K-major tile.
__device__ __forceinline__ uint32_t sw128_offset(uint32_t r, uint32_t j) {
  return (r >> 3) * 1024u + (r & 7u) * 128u + ((j ^ (r & 7u)) << 4);
}

// Byte offset of element (r, k) in a K-major fp16 operand of `rows` rows stored as 64-wide, 128-byte-swizzled
// K atoms of rows x 128 B each (atom k / 64, 16-byte chunk (k % 64) / 8 of row r, element k % 8).
__host__ __device__ __forceinline__ uint32_t k_major_offset(uint32_t rows, uint32_t r, uint32_t k) {
  return (k >> 6) * rows * 128u + (r >> 3) * 1024u + (r & 7u) * 128u + ((((k & 63u) >> 3) ^ (r & 7u)) << 4) +
         2u * (k & 7u);
}

// Power-of-two exponent s for which mx * 2^s lies in [2^13, 2^14): fp16 hi / lo splits of values up to mx then
// keep their full precision with room for the sums of an MMA. Clamped to [-100, 100]; 14 for mx = 0.
__device__ __forceinline__ int fp16_scale_exp(float mx) {
  int ex = 0;
  if (mx > 0.f && mx <= 3.0e38f) frexpf(mx, &ex);
  return max(-100, min(100, 14 - ex));
}

}  // namespace externd
