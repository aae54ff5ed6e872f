// externd_energy_noalloc: Eq. 1 from given factors without allocating anything.
//
// Some callers cannot allocate device memory: a process whose framework has taken the whole GPU for its own
// caching allocator and forbids raw cudaMalloc, a latency-critical path that cannot afford the implicit device
// synchronisation of cudaMalloc/cudaFree, or a plugin that is only ever handed buffers. For them this entry
// point keeps its scratch (the per-tile partial sums of the two squared norms and three scalars) in one
// file-scope static __device__ array of EXTERND_ENERGY_NOALLOC_SCRATCH doubles, which every GPU that loads
// the library holds until the process exits. Only inputs and the host result come from the caller.
//
// In host code the array's name is a host-side stand-in, not a device address, so the first call on each
// device (with that device current) looks the address up with cudaGetSymbolAddress and every later call on that
// device reuses it. All calls share the array and overwrite it: nothing in it needs to start at zero (every
// partial is written before it is read), and two calls whose work overlaps on the GPU race on it.
#include <cuda_runtime.h>

#include <mutex>

#include "../../include/externd.h"
#include "kernels.h"

namespace externd {
cudaStream_t library_stream();
std::mutex& library_mutex();
int record_cuda_error(cudaError_t e, const char* where);
}  // namespace externd

namespace {

constexpr int kScratch = EXTERND_ENERGY_NOALLOC_SCRATCH;
__device__ __align__(256) double g_noalloc_scratch[kScratch];

constexpr int kMaxDevices = 64;
double* g_scratch_addr[kMaxDevices] = {};   // device address of g_noalloc_scratch, per device

bool device_reachable(const void* p) {
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged ||
         (at.type == cudaMemoryTypeHost && at.devicePointer != nullptr);
}

}  // namespace

extern "C" int externd_energy_noalloc(const float* A, int64_t m, int64_t n, const int8_t* B, const float* D,
                                      const int8_t* C, int64_t k, const float* weights, double* energy) {
  using namespace externd;
  std::lock_guard<std::mutex> lock(library_mutex());
  if (A == nullptr || B == nullptr || D == nullptr || C == nullptr || energy == nullptr) return EXTERND_EINVAL;
  // the size limits of every other entry point (row tiles of 64 in gridDim.y, m * n <= 2^40) and k below 2^31
  if (m < 1 || n < 1 || k < 1 || m > 65535LL * 64 || n > (1LL << 30) || m * n > (1LL << 40) || k >= (1LL << 31))
    return EXTERND_EINVAL;
  // tiles of 64 rows x 128 columns (the deflation kernel's), counted in 64 bits so no size can wrap
  const long long tiles = cdiv(m, 64) * cdiv(n, 128);
  if (tiles + 3 > kScratch) return EXTERND_EINVAL;   // larger than the fixed scratch: see the header
  if (tiles != (long long)deflate_tiles((int)m, (int)n)) return EXTERND_EINVAL;
  if (!device_reachable(A) || !device_reachable(B) || !device_reachable(D) || !device_reachable(C) ||
      (weights != nullptr && !device_reachable(weights)))
    return EXTERND_EPTR;

  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return record_cuda_error(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) return EXTERND_ENODEV;
  if (g_scratch_addr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return record_cuda_error(e, "cudaGetSymbolAddress(g_noalloc_scratch)");
    g_scratch_addr[dev] = static_cast<double*>(p);
  }
  F2* part = reinterpret_cast<F2*>(g_scratch_addr[dev]);   // [tiles] per-tile partial sums (8 bytes each)
  double* sc = g_scratch_addr[dev] + tiles;                 // ||A||_H^2, ||A - B diag(D) C||_H^2, energy
  cudaStream_t s = library_stream();
  const int mi = (int)m, ni = (int)n;
  if ((e = launch_deflate(A, nullptr, mi, ni, nullptr, 0, false, nullptr, nullptr, 0, 0, weights, nullptr, part,
                          s)) != cudaSuccess)
    return record_cuda_error(e, "energy_noalloc: norm of A");
  if ((e = launch_norm(part, (int)tiles, sc, nullptr, nullptr, s)) != cudaSuccess)
    return record_cuda_error(e, "energy_noalloc: sum");
  if ((e = launch_deflate(A, nullptr, mi, ni, B, k, true, D, C, n, (int)k, weights, nullptr, part, s)) !=
      cudaSuccess)
    return record_cuda_error(e, "energy_noalloc: residual");
  if ((e = launch_norm(part, (int)tiles, sc + 1, sc, sc + 2, s)) != cudaSuccess)
    return record_cuda_error(e, "energy_noalloc: sum");
  if ((e = cudaMemcpyAsync(energy, sc + 2, sizeof(double), cudaMemcpyDeviceToHost, s)) != cudaSuccess)
    return record_cuda_error(e, "energy_noalloc: copy");
  if ((e = cudaStreamSynchronize(s)) != cudaSuccess) return record_cuda_error(e, "energy_noalloc: sync");
  return EXTERND_OK;
}
