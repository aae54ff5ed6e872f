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

// Compensated (Neumaier) float sum of magnitudes: a thread adds a few hundred |x| with ~2^-44 relative error,
// the cross-thread combine runs in double. Keeps the Eq. 2 mean accurate without per-element double math.
struct AbsSum {
  float s = 0.f, c = 0.f;
  __device__ __forceinline__ void add(float x) {
    const float a = fabsf(x);
    const float t = s + a;
    c += (s >= a) ? ((s - t) + a) : ((a - t) + s);
    s = t;
  }
  __device__ __forceinline__ double value() const { return (double)s + (double)c; }
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
