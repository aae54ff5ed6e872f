// Device-scope grid barriers and the per-vector Eq. 2 threshold finalize that cooperative launches run after
// one (a barrier counter is one zero word per use; a timed-out wait sets the error word and returns false).
#pragma once
#include "kernels.h"

namespace externd {
namespace {
constexpr unsigned long long kGridWaitNs = 2000000000ull;   // 2 s

__device__ __forceinline__ unsigned long long grid_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Grid barrier on ctr: every CTA adds one (release) and polls until the count reaches target (acquire);
// false after a timeout (then err holds 1). The CTA barrier before the release and after the acquire carries the
// ordering to the other threads of the CTA (release and acquire are cumulative), so no separate fences.
__device__ __forceinline__ bool grid_barrier(unsigned* ctr, unsigned target, unsigned* err) {
  __shared__ int s_ok;
  __syncthreads();
  if (threadIdx.x == 0) {
    asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(ctr) : "memory");
    int ok = 1;
    const unsigned long long t0 = grid_ns();
    for (unsigned it = 0;; ++it) {
      unsigned v;
      asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(ctr) : "memory");
      if (v >= target) break;
      if ((it & 63u) == 63u && grid_ns() - t0 > kGridWaitNs) {
        atomicOr(err, 1u);
        ok = 0;
        break;
      }
    }
    s_ok = ok;
  }
  __syncthreads();
  return s_ok != 0;
}

// Eq. 2 thresholds of vectors c0, c0 + step, ... < nv from all chunks of the statistics, one CTA per vector at a
// time: the threads take chunks tid, tid + 256, ... and the CTA combines them in a fixed order.
__device__ void finalize_range(const Stats& st, int nv, int c0, int step) {
  __shared__ F2 rs[8];
  __shared__ u64 rk[8];
  const int tid = threadIdx.x;
  for (int a = c0; a < nv; a += step) {
    F2 sv;
    u64 key = 0;
    const uint4* pp = reinterpret_cast<const uint4*>(st.part + (long long)a * st.nchunk);
    for (int c = tid; c < st.nchunk; c += 256) {
      const uint4 r = __ldcg(pp + c);
      F2 t;
      t.hi = __uint_as_float(r.x);
      t.lo = __uint_as_float(r.y);
      sv = f2_add(sv, t);
      const u64 kk = ((u64)r.w << 32) | r.z;
      key = kk > key ? kk : key;
    }
    for (int o = 16; o > 0; o >>= 1) {
      sv = f2_add(sv, f2_shfl_xor(sv, o));
      const u64 t = __shfl_xor_sync(0xffffffffu, key, o);
      key = t > key ? t : key;
    }
    if ((tid & 31) == 0) {
      rs[tid >> 5] = sv;
      rk[tid >> 5] = key;
    }
    __syncthreads();
    if (tid == 0) {
      F2 tot = rs[0];
      u64 kmax = rk[0];
      for (int q = 1; q < 8; ++q) {
        tot = f2_add(tot, rs[q]);
        kmax = rk[q] > kmax ? rk[q] : kmax;
      }
      const float th = __double2float_rd(st.th.tau * (f2_value(tot) / (double)st.th.L));
      st.th.theta[a] = th;
      st.th.fallback[a] = !(key_mag(kmax) > th);
      st.th.arg[a] = key_index(kmax);
    }
    __syncthreads();
  }
}

}  // namespace
}  // namespace externd
