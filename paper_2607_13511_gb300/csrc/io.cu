// Caller-buffer indirection for the captured decomposition graph.
//
// A decomposition graph is captured once per (shape, parameters, workspace) and replayed. If the caller's arrays
// (A in, B / D / C out) were baked into its nodes, every new matrix of the same shape -- a model conversion runs
// hundreds of them back to back -- would need a fresh capture and instantiation. Instead the graph's first and
// last touches of caller memory read the addresses from a small device table, which one tiny kernel refreshes on
// the stream before each replay (kernel arguments are copied at launch, so no host buffer can race with it).
#include <cuda_runtime.h>

#include <algorithm>

#include "kernels.h"

namespace externd {
namespace {

__global__ void io_set_kernel(IoTable* t, const float* A, int8_t* B, float* D, int8_t* C) {
  t->A = A;
  t->B = B;
  t->D = D;
  t->C = C;
}

// R = A (count floats), 16-byte accesses when both ends are aligned.
__global__ void __launch_bounds__(256) io_copy_in_kernel(const IoTable* __restrict__ t, float* __restrict__ R,
                                                         long long count) {
  const float* A = t->A;
  const long long tid = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  const long long stride = (long long)gridDim.x * blockDim.x;
  if ((reinterpret_cast<uintptr_t>(A) & 15) == 0 && (reinterpret_cast<uintptr_t>(R) & 15) == 0) {
    const long long n4 = count >> 2;
    const float4* a4 = reinterpret_cast<const float4*>(A);
    float4* r4 = reinterpret_cast<float4*>(R);
    for (long long i = tid; i < n4; i += stride) r4[i] = __ldcs(a4 + i);
    for (long long i = (n4 << 2) + tid; i < count; i += stride) R[i] = A[i];
  } else {
    for (long long i = tid; i < count; i += stride) R[i] = A[i];
  }
}

// C[j0 + a][:] = Vt[a][0 .. n) for a < w (C is k x n row-major int8), 16-byte accesses where the row allows.
__global__ void __launch_bounds__(256) io_write_c_kernel(const int8_t* __restrict__ Vt, long long ldv, int w, int n,
                                                         const IoTable* __restrict__ t, long long j0) {
  const int a = blockIdx.y;
  if (a >= w) return;
  const int8_t* src = Vt + (long long)a * ldv;
  int8_t* dst = t->C + (j0 + a) * (long long)n;
  const int tid = blockIdx.x * blockDim.x + threadIdx.x, stride = gridDim.x * blockDim.x;
  if ((reinterpret_cast<uintptr_t>(dst) & 15) == 0) {   // src rows are 16-byte aligned (ldv % 16 == 0)
    const int n16 = n >> 4;
    for (int i = tid; i < n16; i += stride)
      reinterpret_cast<int4*>(dst)[i] = reinterpret_cast<const int4*>(src)[i];
    for (int i = (n16 << 4) + tid; i < n; i += stride) dst[i] = src[i];
  } else {
    for (int i = tid; i < n; i += stride) dst[i] = src[i];
  }
}

__global__ void io_write_d_kernel(const float* __restrict__ d, int w, const IoTable* __restrict__ t, long long j0) {
  for (int a = threadIdx.x; a < w; a += blockDim.x) t->D[j0 + a] = d[a];
}

}  // namespace

cudaError_t launch_io_set(IoTable* t, const float* A, int8_t* B, float* D, int8_t* C, cudaStream_t s) {
  io_set_kernel<<<1, 1, 0, s>>>(t, A, B, D, C);
  return cudaGetLastError();
}

cudaError_t launch_io_copy_in(const IoTable* t, float* R, long long count, cudaStream_t s) {
  const long long blocks = std::min<long long>(cdiv(cdiv(count, 4), 256), 152LL * 8);
  io_copy_in_kernel<<<(unsigned)std::max<long long>(blocks, 1), 256, 0, s>>>(t, R, count);
  return cudaGetLastError();
}

cudaError_t launch_io_write_c(const int8_t* Vt, long long ldv, int w, int n, const IoTable* t, long long j0,
                              cudaStream_t s) {
  dim3 grid((unsigned)std::min<long long>(cdiv(cdiv(n, 16), 256), 8), (unsigned)w);
  io_write_c_kernel<<<grid, 256, 0, s>>>(Vt, ldv, w, n, t, j0);
  return cudaGetLastError();
}

cudaError_t launch_io_write_d(const float* d, int w, const IoTable* t, long long j0, cudaStream_t s) {
  io_write_d_kernel<<<1, 256, 0, s>>>(d, w, t, j0);
  return cudaGetLastError();
}

}  // namespace externd
