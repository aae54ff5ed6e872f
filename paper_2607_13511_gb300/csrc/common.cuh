// Device helpers shared by the ExTernD kernels: reductions, the Eq. 2 threshold test, vector loads.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace externd {

// Ridge of Eq. 3 (and of Eq. 4 for blocks wider than one component), relative to the mean Gram diagonal.
// The paper writes "+ eps I" without a value.
constexpr double kEpsRel = 1e-4;

// Output positions handled by one CTA of every statistics producer: the per-vector partial sums of |x| and
// the argmax key come in chunks of this many positions, and the Eq. 2 threshold sums the chunks in order.
constexpr int kStatChunk = 128;

// Largest block width the library supports (the paper's default block is 256).
constexpr int kMaxBlock = 256;

typedef unsigned long long u64;

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ u64 warp_max(u64 v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    u64 t = __shfl_xor_sync(0xffffffffu, v, o);
    v = t > v ? t : v;
  }
  return v;
}

// Double-float value hi + lo held in two floats (|lo| <= ulp(hi) / 2), added with Knuth's error-free TwoSum. It
// carries ~44 significant bits with float32 arithmetic only: double-precision arithmetic runs at a small fraction
// of the float32 rate on this GPU and is kept out of every per-element and per-thread reduction.
struct F2 {
  float hi = 0.f, lo = 0.f;
};

__device__ __forceinline__ F2 f2_add(F2 a, F2 b) {
  const float s = a.hi + b.hi;
  const float bb = s - a.hi;
  const float err = (a.hi - (s - bb)) + (b.hi - bb);
  const float lo = a.lo + b.lo + err;
  F2 r;
  r.hi = s + lo;
  r.lo = lo - (r.hi - s);
  return r;
}

__device__ __forceinline__ F2 f2_add(F2 a, float x) {
  F2 b;
  b.hi = x;
  return f2_add(a, b);
}

__device__ __forceinline__ F2 f2_shfl_xor(F2 v, int o) {
  F2 r;
  r.hi = __shfl_xor_sync(0xffffffffu, v.hi, o);
  r.lo = __shfl_xor_sync(0xffffffffu, v.lo, o);
  return r;
}

__device__ __forceinline__ F2 warp_sum(F2 v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = f2_add(v, f2_shfl_xor(v, o));
  return v;
}

__device__ __forceinline__ double f2_value(F2 v) { return (double)v.hi + (double)v.lo; }

// Per-thread sum of magnitudes for the Eq. 2 mean.
struct AbsSum {
  F2 acc;
  __device__ __forceinline__ void add(float x) { acc = f2_add(acc, fabsf(x)); }
};

// Key whose maximum picks the largest |x| and, among equal magnitudes, the lowest index.
__device__ __forceinline__ u64 mag_key(float x, uint32_t idx) {
  return ((u64)__float_as_uint(fabsf(x)) << 32) | (u64)(0xffffffffu - idx);
}
__device__ __forceinline__ uint32_t key_index(u64 key) { return 0xffffffffu - (uint32_t)(key & 0xffffffffu); }
__device__ __forceinline__ float key_mag(u64 key) { return __uint_as_float((uint32_t)(key >> 32)); }

// Eq. 2 decision for a float32 entry: |x| > theta with theta = tau * (S / L) held in double. For a float a,
// a > theta  <=>  a > RD_float(theta), so the comparison runs in float against the rounded-down threshold.
__device__ __forceinline__ int8_t ternary_of(float x, float theta_dn) {
  return fabsf(x) > theta_dn ? (x < 0.f ? (int8_t)-1 : (int8_t)1) : (int8_t)0;
}

// Loads 4 consecutive floats p[i..i+3] with i < len masking; vectorised when aligned.
__device__ __forceinline__ float4 load4(const float* __restrict__ p, long long i, long long len, bool vec_ok) {
  if (vec_ok && i + 3 < len) return __ldg(reinterpret_cast<const float4*>(p + i));
  float4 v;
  v.x = (i + 0 < len) ? __ldg(p + i + 0) : 0.f;
  v.y = (i + 1 < len) ? __ldg(p + i + 1) : 0.f;
  v.z = (i + 2 < len) ? __ldg(p + i + 2) : 0.f;
  v.w = (i + 3 < len) ? __ldg(p + i + 3) : 0.f;
  return v;
}

__host__ __device__ __forceinline__ long long round_up(long long x, long long a) { return (x + a - 1) / a * a; }
__host__ __device__ __forceinline__ long long cdiv(long long x, long long a) { return (x + a - 1) / a; }

}  // namespace externd
