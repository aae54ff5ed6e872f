// Kernels of the two extensions of the block loop: the convergence safeguard of Prop. 2 and the refinement sweeps
// of §2.4. Both compare what a fitted block removes from the residual with an alternative and act on the result
// on the device, so the block loop keeps running as one captured graph.
//
// A block (U, d, V) with r_a = u_a^T R H v_a and K = (U^T U) .* (V^T H V) removes
//   ||R||_H^2 - ||R - U diag(d) V^T||_H^2 = 2 r^T d - d^T K d
// from the weighted squared residual (expand the square; it holds for any d, with or without Eq. 4's ridge).
//
// Safeguard: the best single-entry pair (u = e_i, v = sgn(R_ij) e_j, d = |R_ij|) removes h_j R_ij^2; when that is
// more than the block removes, the block becomes the pair followed by w - 1 zero components.
// Refinement: a revisited block was added back to the residual; its refit replaces it only if it removes at least
// as much as the old block (what the add-back restored: ||R_add||^2 - ||R||^2).
#include <algorithm>

#include "kernels.h"

namespace externd {

namespace {

constexpr int kArgThreads = 256;

__device__ __forceinline__ bool better(float s1, unsigned long long i1, float s2, unsigned long long i2) {
  return s1 > s2 || (s1 == s2 && i1 < i2);
}

// Per-CTA best entry of R by score h_j R_ij^2 (|R_ij| when unweighted: the same order, without rounding); ties go
// to the lower row-major index. CTA c scans rows c, c + grid, ...
__global__ void __launch_bounds__(kArgThreads) entry_argmax_kernel(const float* __restrict__ R, int m, int n,
                                                                   const float* __restrict__ h,
                                                                   EntryBest* __restrict__ part) {
  float bs = -1.f, br = 0.f;
  unsigned long long bi = ~0ull;
  for (long long i = blockIdx.x; i < m; i += gridDim.x) {
    const float* row = R + i * n;
    for (int j = threadIdx.x; j < n; j += kArgThreads) {
      const float x = row[j];
      const float sc = h != nullptr ? h[j] * x * x : fabsf(x);
      const unsigned long long idx = (unsigned long long)i * n + j;
      if (better(sc, idx, bs, bi)) {
        bs = sc;
        br = x;
        bi = idx;
      }
    }
  }
  for (int o = 16; o > 0; o >>= 1) {
    const float s2 = __shfl_xor_sync(0xffffffffu, bs, o), r2 = __shfl_xor_sync(0xffffffffu, br, o);
    const unsigned long long i2 = __shfl_xor_sync(0xffffffffu, bi, o);
    if (better(s2, i2, bs, bi)) {
      bs = s2;
      br = r2;
      bi = i2;
    }
  }
  __shared__ EntryBest wb[kArgThreads / 32];
  const int warp = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) wb[warp] = EntryBest{bs, br, bi};
  __syncthreads();
  if (threadIdx.x == 0) {
    EntryBest b = wb[0];
    for (int k = 1; k < kArgThreads / 32; ++k)
      if (better(wb[k].score, wb[k].idx, b.score, b.idx)) b = wb[k];
    part[blockIdx.x] = b;
  }
}

// 2 r^T d - d^T K d in double by one CTA (w <= 256); result to thread 0.
__device__ double block_decrease(const float* __restrict__ r, const float* __restrict__ d,
                                 const float* __restrict__ K, int w) {
  __shared__ double red[8];
  double acc = 0.0;
  for (int idx = threadIdx.x; idx < w * w; idx += blockDim.x) {
    const int a = idx / w, b = idx - a * w;
    acc -= (double)d[a] * (double)K[idx] * (double)d[b];
    if (a == b) acc += 2.0 * (double)r[a] * (double)d[a];
  }
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
  __syncthreads();
  double t = 0.0;
  if (threadIdx.x == 0)
    for (int k = 0; k < (int)(blockDim.x >> 5); ++k) t += red[k];
  return t;
}

__global__ void __launch_bounds__(256) safeguard_decide_kernel(const EntryBest* __restrict__ part, int nparts, int n,
                                                               const float* __restrict__ h,
                                                               const float* __restrict__ r, float* __restrict__ d,
                                                               const float* __restrict__ K, int w,
                                                               BlockChoice* __restrict__ choice) {
  // the best of the per-CTA entries: strided over the threads, then a warp and a CTA reduction (same order rule)
  EntryBest b{-1.f, 0.f, ~0ull};
  for (int k = threadIdx.x; k < nparts; k += blockDim.x) {
    const EntryBest c = part[k];
    if (better(c.score, c.idx, b.score, b.idx)) b = c;
  }
  for (int o = 16; o > 0; o >>= 1) {
    const float s2 = __shfl_xor_sync(0xffffffffu, b.score, o), r2 = __shfl_xor_sync(0xffffffffu, b.rij, o);
    const unsigned long long i2 = __shfl_xor_sync(0xffffffffu, b.idx, o);
    if (better(s2, i2, b.score, b.idx)) b = EntryBest{s2, r2, i2};
  }
  __shared__ EntryBest wb[8];
  if ((threadIdx.x & 31) == 0) wb[threadIdx.x >> 5] = b;
  const double dec = block_decrease(r, d, K, w);   // contains a CTA barrier, after which wb is complete
  if (threadIdx.x != 0) return;
  b = wb[0];
  for (int k = 1; k < (int)(blockDim.x >> 5); ++k)
    if (better(wb[k].score, wb[k].idx, b.score, b.idx)) b = wb[k];
  const long long i = (long long)(b.idx / (unsigned long long)n), j = (long long)(b.idx % (unsigned long long)n);
  const double single = (h != nullptr ? (double)h[j] : 1.0) * (double)b.rij * (double)b.rij;
  const int take = single > dec ? 1 : 0;
  choice->flag = take;
  choice->row = i;
  choice->col = j;
  choice->sign = b.rij < 0.f ? -1 : 1;
  choice->count += take;
  if (take) {
    d[0] = fabsf(b.rij);
    for (int a = 1; a < w; ++a) d[a] = 0.f;
  }
}

// The single-entry pair in place of the block, in every layout the deflation and the outputs read.
__global__ void safeguard_replace_kernel(const BlockChoice* __restrict__ choice, int w, int m, int n,
                                         int8_t* __restrict__ Ut, long long ldm, int8_t* __restrict__ Vt,
                                         long long ldn, __half* __restrict__ Uk, __half* __restrict__ Vk,
                                         long long ldk) {
  if (choice->flag == 0) return;
  const long long i0 = choice->row, j0 = choice->col;
  const int sg = choice->sign;
  const long long stride = (long long)gridDim.x * blockDim.x;
  const long long t0 = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  for (long long t = t0; t < (long long)w * ldm; t += stride) {
    const long long a = t / ldm, x = t - a * ldm;
    Ut[t] = (a == 0 && x == i0) ? (int8_t)1 : (int8_t)0;
  }
  for (long long t = t0; t < (long long)w * ldn; t += stride) {
    const long long a = t / ldn, x = t - a * ldn;
    Vt[t] = (a == 0 && x == j0) ? (int8_t)sg : (int8_t)0;
  }
  if (Uk != nullptr)
    for (long long t = t0; t < (long long)m * ldk; t += stride) {
      const long long x = t / ldk, a = t - x * ldk;
      Uk[t] = __float2half((a == 0 && x == i0) ? 1.f : 0.f);
    }
  if (Vk != nullptr)
    for (long long t = t0; t < (long long)n * ldk; t += stride) {
      const long long x = t / ldk, a = t - x * ldk;
      Vk[t] = __float2half((a == 0 && x == j0) ? (float)sg : 0.f);
    }
}

__global__ void __launch_bounds__(256) refine_decide_kernel(const double* __restrict__ norm_add,
                                                            const double* __restrict__ norm_prev,
                                                            const float* __restrict__ r, const float* __restrict__ d,
                                                            const float* __restrict__ K, int w,
                                                            BlockChoice* __restrict__ choice) {
  const double gain = block_decrease(r, d, K, w);
  if (threadIdx.x != 0) return;
  const double old = *norm_add - *norm_prev;
  const int take = gain >= old ? 1 : 0;
  choice->flag = take;
  choice->count += take;
}

// With the flag set: B[:, j0 + a] = Ut row a, C[j0 + a, :] = Vt row a, D[j0 + a] = d[a].
__global__ void commit_kernel(const BlockChoice* __restrict__ choice, const int8_t* __restrict__ Ut, long long ldm,
                              const int8_t* __restrict__ Vt, long long ldn, const float* __restrict__ d, int w, int m,
                              int n, int8_t* __restrict__ B, float* __restrict__ D, int8_t* __restrict__ C,
                              long long k, long long j0) {
  if (choice->flag == 0) return;
  const long long stride = (long long)gridDim.x * blockDim.x;
  const long long t0 = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  for (long long t = t0; t < (long long)m * w; t += stride) {
    const long long x = t / w, a = t - x * w;
    B[x * k + j0 + a] = Ut[a * ldm + x];
  }
  for (long long t = t0; t < (long long)w * n; t += stride) {
    const long long a = t / n, x = t - a * n;
    C[(j0 + a) * n + x] = Vt[a * ldn + x];
  }
  if (t0 < w) D[j0 + t0] = d[t0];
}

__global__ void scale_copy_kernel(const float* __restrict__ src, float alpha, int w, float* __restrict__ dst) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t < w) dst[t] = alpha * src[t];
}

__global__ void count_reset_kernel(BlockChoice* __restrict__ choice, long long* __restrict__ out) {
  if (threadIdx.x == 0 && blockIdx.x == 0) {
    if (out != nullptr) *out = choice->count;
    choice->count = 0;
  }
}

int grid_for(long long work) {
  int sms = 152, dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return (int)std::max<long long>(1, std::min<long long>(cdiv(work, 256), 4LL * sms));
}

}  // namespace

int entry_argmax_parts(int m) {
  int sms = 152, dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return std::max(1, std::min(m, 4 * sms));
}

cudaError_t launch_entry_argmax(const float* R, int m, int n, const float* h, EntryBest* part, cudaStream_t s) {
  entry_argmax_kernel<<<(unsigned)entry_argmax_parts(m), kArgThreads, 0, s>>>(R, m, n, h, part);
  return cudaGetLastError();
}

cudaError_t launch_safeguard_decide(const EntryBest* part, int nparts, int n, const float* h, const float* r, float* d,
                                    const float* K, int w, BlockChoice* choice, cudaStream_t s) {
  safeguard_decide_kernel<<<1, 256, 0, s>>>(part, nparts, n, h, r, d, K, w, choice);
  return cudaGetLastError();
}

cudaError_t launch_safeguard_replace(const BlockChoice* choice, int w, int m, int n, int8_t* Ut, long long ldm,
                                     int8_t* Vt, long long ldn, __half* Uk, __half* Vk, long long ldk,
                                     cudaStream_t s) {
  const long long work = std::max({(long long)w * ldm, (long long)w * ldn, Uk ? (long long)m * ldk : 0LL,
                                   Vk ? (long long)n * ldk : 0LL});
  safeguard_replace_kernel<<<grid_for(work), 256, 0, s>>>(choice, w, m, n, Ut, ldm, Vt, ldn, Uk, Vk, ldk);
  return cudaGetLastError();
}

cudaError_t launch_refine_decide(const double* norm_add, const double* norm_prev, const float* r, const float* d,
                                 const float* K, int w, BlockChoice* choice, cudaStream_t s) {
  refine_decide_kernel<<<1, 256, 0, s>>>(norm_add, norm_prev, r, d, K, w, choice);
  return cudaGetLastError();
}

cudaError_t launch_commit(const BlockChoice* choice, const int8_t* Ut, long long ldm, const int8_t* Vt, long long ldn,
                          const float* d, int w, int m, int n, int8_t* B, float* D, int8_t* C, long long k,
                          long long j0, cudaStream_t s) {
  const long long work = std::max((long long)m * w, (long long)w * n);
  commit_kernel<<<grid_for(work), 256, 0, s>>>(choice, Ut, ldm, Vt, ldn, d, w, m, n, B, D, C, k, j0);
  return cudaGetLastError();
}

cudaError_t launch_scale_copy(const float* src, float alpha, int w, float* dst, cudaStream_t s) {
  scale_copy_kernel<<<(unsigned)cdiv(w, 256), 256, 0, s>>>(src, alpha, w, dst);
  return cudaGetLastError();
}

cudaError_t launch_count_reset(BlockChoice* choice, long long* out, cudaStream_t s) {
  count_reset_kernel<<<1, 32, 0, s>>>(choice, out);
  return cudaGetLastError();
}

}  // namespace externd
