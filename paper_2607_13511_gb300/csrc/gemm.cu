// Residual products, decorrelation and deflation on the CUDA cores (float32 FMA, register-tiled).
//
//   V-step product   part[s][a][c] = sum_{r in split s} U[r][a] R[r][c]            (§2.3 step 1, §2.4)
//   U-step product   part[s][a][r] = sum_{c in split s} R[r][c] h[c] V[c][a]        (§2.3 step 1, §2.5)
//   decorrelation    X[a][x] = sum_b Ginv[a][b] sum_s part[s][b][x]               (Eq. 3)
//   deflation        R[r][c] -= sum_a U[r][a] d[a] V[c][a], fused ||R||_H^2 and column energies (§2.3, §2.4)
//
// Every kernel computes a 64 x 128 output tile with 256 threads (4 x 8 outputs per thread) from 16-deep slices
// staged in shared memory. Split-K partials are written, never atomically added, so results are reproducible.
#include <cstdlib>
#include <cstring>

#include "kernels.h"
#include "grid.cuh"

namespace externd {

namespace {

constexpr int TM = 64;   // rows of the output tile (components, or residual rows for the deflation)
constexpr int TN = 128;  // columns of the output tile
constexpr int TK = 16;   // depth of one shared-memory slice

// One 16-deep step of the 64 x 128 tile: acc[i][j] += As[k][ty*4+i] * Bs[k][(j<4 ? 0 : 64) + tx*4 + j%4].
__device__ __forceinline__ void tile_fma(const float (*As)[TM + 4], const float (*Bs)[TN], int tx, int ty,
                                         float acc[4][8]) {
#pragma unroll
  for (int k = 0; k < TK; ++k) {
    const float4 a = *reinterpret_cast<const float4*>(&As[k][ty * 4]);
    const float4 b0 = *reinterpret_cast<const float4*>(&Bs[k][tx * 4]);
    const float4 b1 = *reinterpret_cast<const float4*>(&Bs[k][64 + tx * 4]);
    const float av[4] = {a.x, a.y, a.z, a.w};
    const float bv[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
  }
}

__device__ __forceinline__ int col_of(int tx, int j) { return (j < 4 ? 0 : 64) + tx * 4 + (j & 3); }

// Ternary slice: Ts[ky][a] = T[a0 + a][y0 + ky] for ky < 16, a < 64 (zero outside w / [y0, yend)).
__device__ __forceinline__ void load_ternary_slice(float (*Ts)[TM + 4], const int8_t* __restrict__ T, int ldt, int w,
                                                   int a0, int y0, int yend, int tid) {
  const int a = tid >> 2;
  const int ky = (tid & 3) * 4;
  const int ag = a0 + a;
  int packed = 0;
  if (ag < w) packed = __ldg(reinterpret_cast<const int*>(T + (long long)ag * ldt + y0 + ky));
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int y = y0 + ky + j;
    const int8_t t = (int8_t)((packed >> (8 * j)) & 0xff);
    Ts[ky + j][a] = (y < yend) ? (float)t : 0.f;
  }
}

template <bool USTEP>
__global__ void __launch_bounds__(256) product_kernel(const float* __restrict__ R, int m, int n,
                                                      const int8_t* __restrict__ T, int ldt, int w,
                                                      const float* __restrict__ h, float* __restrict__ part,
                                                      int ychunk) {
  __shared__ __align__(16) float Rs[TK][TN];
  __shared__ __align__(16) float Ts[TK][TM + 4];
  const int Lx = USTEP ? m : n;
  const int Ly = USTEP ? n : m;
  const int x0 = blockIdx.x * TN;
  const int a0 = blockIdx.y * TM;
  const int ybeg = blockIdx.z * ychunk;
  const int yend = min(Ly, ybeg + ychunk);
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const bool vec = (n & 3) == 0;
  float acc[4][8];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;

  for (int y0 = ybeg; y0 < yend; y0 += TK) {
    if (!USTEP) {
      // Rs[ky][kx] = R[y0 + ky][x0 + kx]
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        const int idx = tid + 256 * q;
        const int ky = idx >> 5, kx = (idx & 31) * 4;
        const int y = y0 + ky;
        float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
        if (y < yend) v = load4(R + (long long)y * n, x0 + kx, n, vec);
        *reinterpret_cast<float4*>(&Rs[ky][kx]) = v;
      }
    } else {
      // Rs[ky][kx] = R[x0 + kx][y0 + ky] * h[y0 + ky]
      const int kx = tid & 127, half = tid >> 7;
      const int x = x0 + kx;
      const int yb = y0 + 8 * half;
      float4 v0 = make_float4(0.f, 0.f, 0.f, 0.f), v1 = v0;
      if (x < m) {
        v0 = load4(R + (long long)x * n, yb, yend, vec);
        v1 = load4(R + (long long)x * n, yb + 4, yend, vec);
      }
      float v[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int y = yb + j;
        const float hy = (h != nullptr && y < yend) ? __ldg(h + y) : 1.f;
        Rs[8 * half + j][kx] = v[j] * hy;
      }
    }
    load_ternary_slice(Ts, T, ldt, w, a0, y0, yend, tid);
    __syncthreads();
    tile_fma(Ts, Rs, tx, ty, acc);
    __syncthreads();
  }

  float* out = part + (long long)blockIdx.z * w * Lx;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int a = a0 + ty * 4 + i;
    if (a >= w) continue;
#pragma unroll
    for (int g = 0; g < 2; ++g) {
      const int x = x0 + g * 64 + tx * 4;
      float* o = out + (long long)a * Lx + x;
      if ((Lx & 3) == 0 && x + 3 < Lx) {
        *reinterpret_cast<float4*>(o) = make_float4(acc[i][4 * g], acc[i][4 * g + 1], acc[i][4 * g + 2], acc[i][4 * g + 3]);
      } else {
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (x + j < Lx) o[j] = acc[i][4 * g + j];
      }
    }
  }
}

// X tile of 64 components x DXT positions (DXT = 16 ... 128, chosen per shape so that the grid fills the GPU
// once or twice): thread (ty, tx) owns components ty*4..+3 at positions tx*PX .. +PX-1, PX = DXT / 16. The CTA
// first stages, with every load of a batch in flight before any is used,
//   Ps[b][x]  = sum_s part[s][b][x0 + x]   for all w components b (split order)
//   Gs[b][a]  = Ginv[b][a0 + a]            (Ginv is symmetric: row b holds column b)
// in dynamic shared memory, then runs the w-deep product out of shared memory. One Eq. 2 statistics chunk per
// CTA column: DXT positions.
constexpr int kGsLd = TM + 4;

size_t decorrelate_smem(int w, int dxt) { return (size_t)w * (dxt + kGsLd) * sizeof(float); }

int decorrelate_dx(int L, int w) {
  int sms = 152, dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int dx = 16;
  while (dx < 128 && cdiv(L, dx) * cdiv(w, TM) > 2LL * sms) dx *= 2;
  return dx;
}

// COOP: launched cooperatively; the thresholds are finalized after a grid barrier by every CTA for its share of
// the vectors (bar: 2 zero words, left zero) instead of by the last CTA for all of them.
template <int DXT, bool COOP>
__global__ void __launch_bounds__(256, 2) decorrelate_kernel(const float* __restrict__ Ginv, int w,
                                                          const float* __restrict__ part, int splits, int L,
                                                          float* __restrict__ X, int ldx, Stats st,
                                                          unsigned* __restrict__ bar, unsigned* __restrict__ err) {
  constexpr int PX = DXT / 16;
  extern __shared__ __align__(16) float dsm[];
  float* const Ps = dsm;                 // [w][DXT]
  float* const Gs = dsm + w * DXT;       // [w][kGsLd]
  const int x0 = blockIdx.x * DXT;
  const int a0 = blockIdx.y * TM;
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;

  // Ps: w x DXT/4 float4 slots; a thread owns slots tid + 256 e and walks its (slot, split) pairs in batches of
  // 8 loads, adding each slot's splits in split order through shared memory. The first Ginv rows (w x 16 float4
  // slots) are issued with the first batch. Two CTAs fit on an SM (<= 128 registers).
  {
    constexpr int Q = DXT / 4, NB = 8;
    const bool pvec = (L & 3) == 0, gvec = (w & 3) == 0;
    const long long sstride = (long long)w * L;
    const int nps = w * Q, pper = (nps + 255) / 256, nld = pper * splits;
    const int ngs = w * 16, gper = (ngs + 255) / 256;
    constexpr int GB = 4;
    float4 g[GB];
#pragma unroll
    for (int q = 0; q < GB; ++q) {
      const int i = q * 256 + tid;
      g[q] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (q < gper && i < ngs) g[q] = load4(Ginv + (long long)(i >> 4) * w, a0 + (i & 15) * 4, w, gvec);
    }
    for (int f0 = 0; f0 < nld; f0 += NB) {
      float4 v[NB];
      int e = f0 / splits, sp = f0 - e * splits;
#pragma unroll
      for (int k = 0; k < NB; ++k) {
        const int i = e * 256 + tid;
        v[k] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (f0 + k < nld && i < nps)
          v[k] = load4(part + sp * sstride + (long long)(i / Q) * L, x0 + (i % Q) * 4, L, pvec);
        if (++sp == splits) {
          sp = 0;
          ++e;
        }
      }
      e = f0 / splits;
      sp = f0 - e * splits;
#pragma unroll
      for (int k = 0; k < NB; ++k) {
        const int i = e * 256 + tid;
        if (f0 + k < nld && i < nps) {
          float4* dst = reinterpret_cast<float4*>(&Ps[(i / Q) * DXT + (i % Q) * 4]);
          if (sp == 0) {
            *dst = v[k];
          } else {
            float4 t = *dst;
            t.x += v[k].x;
            t.y += v[k].y;
            t.z += v[k].z;
            t.w += v[k].w;
            *dst = t;
          }
        }
        if (++sp == splits) {
          sp = 0;
          ++e;
        }
      }
    }
#pragma unroll
    for (int q = 0; q < GB; ++q) {
      const int i = q * 256 + tid;
      if (q < gper && i < ngs) *reinterpret_cast<float4*>(&Gs[(i >> 4) * kGsLd + (i & 15) * 4]) = g[q];
    }
    for (int i = GB * 256 + tid; i < ngs; i += 256)   // w > 64 only
      *reinterpret_cast<float4*>(&Gs[(i >> 4) * kGsLd + (i & 15) * 4]) =
          load4(Ginv + (long long)(i >> 4) * w, a0 + (i & 15) * 4, w, gvec);
  }
  __syncthreads();

  float acc[4][PX];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < PX; ++j) acc[i][j] = 0.f;
#pragma unroll 4
  for (int b = 0; b < w; ++b) {
    const float4 g = *reinterpret_cast<const float4*>(&Gs[b * kGsLd + ty * 4]);
    float p[PX];
    if (PX == 1) {
      p[0] = Ps[b * DXT + tx];
    } else if (PX == 2) {
      const float2 t = *reinterpret_cast<const float2*>(&Ps[b * DXT + tx * 2]);
      p[0] = t.x;
      p[PX - 1] = t.y;
    } else {
#pragma unroll
      for (int j = 0; j < PX; j += 4) {
        const float4 t = *reinterpret_cast<const float4*>(&Ps[b * DXT + tx * PX + j]);
        p[j] = t.x;
        p[j + 1] = t.y;
        p[j + 2] = t.z;
        p[j + 3] = t.w;
      }
    }
    const float gv[4] = {g.x, g.y, g.z, g.w};
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < PX; ++j) acc[i][j] = fmaf(gv[i], p[j], acc[i][j]);
  }

#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int a = a0 + ty * 4 + i;
    AbsSum sum;
    u64 key = 0;
    if (a < w) {
#pragma unroll
      for (int j = 0; j < PX; ++j) {
        const int x = x0 + tx * PX + j;
        if (x < L) {
          X[(long long)a * ldx + x] = acc[i][j];
          sum.add(acc[i][j]);
          const u64 kk = mag_key(acc[i][j], (uint32_t)x);
          key = kk > key ? kk : key;
        }
      }
    }
    F2 s = sum.acc;
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) {
      s = f2_add(s, f2_shfl_xor(s, o));
      const u64 t = __shfl_xor_sync(0xffffffffu, key, o);
      key = t > key ? t : key;
    }
    if (tx == 0 && a < w) put_stat(st, a, blockIdx.x, s, key);
  }
  if (!COOP) {
    stats_done(st, w);
    return;
  }
  const unsigned G = gridDim.x * gridDim.y, c = blockIdx.y * gridDim.x + blockIdx.x;
  if (!grid_barrier(bar, G, err)) return;
  finalize_range(st, w, (int)c, (int)G);
  __syncthreads();
  if (threadIdx.x == 0) {   // exit ticket: the last CTA resets both words
    unsigned old;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(old) : "l"(bar + 1) : "memory");
    if (old == G - 1u) {
      bar[0] = 0u;
      bar[1] = 0u;
    }
  }
}

template <int DXT>
cudaError_t launch_decorrelate_dx(const float* Ginv, int w, const float* part, int splits, int L, float* X, int ldx,
                                  Stats st, unsigned* bar, unsigned* err, cudaStream_t s) {
  static int max_coop = -1;
  if (max_coop < 0) {
    cudaError_t e = cudaFuncSetAttribute(decorrelate_kernel<DXT, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)decorrelate_smem(kMaxBlock, DXT));
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(decorrelate_kernel<DXT, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               (int)decorrelate_smem(kMaxBlock, DXT));
    if (e != cudaSuccess) return e;
    int per_sm = 0, sms = 0, dev = 0;
    if (cudaGetDevice(&dev) == cudaSuccess &&
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess &&
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decorrelate_kernel<DXT, true>, 256,
                                                      decorrelate_smem(kMaxBlock, DXT)) == cudaSuccess)
      max_coop = per_sm * sms;
    else
      max_coop = 0;
    cudaGetLastError();
  }
  dim3 grid((unsigned)cdiv(L, DXT), (unsigned)cdiv(w, TM));
  const size_t smem = decorrelate_smem(w, DXT);
  if (bar != nullptr && err != nullptr && (long long)grid.x * grid.y <= max_coop) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(256);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, decorrelate_kernel<DXT, true>, Ginv, w, part, splits, L, X, ldx, st, bar, err);
  }
  decorrelate_kernel<DXT, false><<<grid, 256, smem, s>>>(Ginv, w, part, splits, L, X, ldx, st, nullptr, nullptr);
  return cudaGetLastError();
}

// ---- Decorrelation and ternarization in one cooperative grid (w <= 64 components) ------------------------------
//
// The same X tile as decorrelate_kernel (thread (ty, tx): components 4ty .. 4ty + 3, positions tx * PX ..), kept in
// registers; then
//   barrier 1 -- every CTA has written its Eq. 2 statistics chunk;
//   each CTA finalizes the thresholds of vectors blockIdx.x, blockIdx.x + grid, ... from all chunks;
//   barrier 2 -- every threshold is written;
//   each CTA ternarizes its tile (int8 rows, optional fp16 rows and K-major fp16) and adds its positions' exact
//   Gram entries (bitplanes in shared memory, popcounts, integer atomics into the upper triangle).
// This replaces two launches, the serial tail of the last-CTA finalize and the round trip of X through memory.
// The grid is launched cooperatively (all CTAs resident); each barrier is a device-scope counter that thread 0
// of every CTA increments with release semantics and polls with acquire loads, giving up after kWaitNs (error
// word set, the CTA skips the rest). Counter 0 is reset by CTA 0 after barrier 2 (everyone has left barrier 1),
// counters 1 and 2 by the last CTA to finish (an exit ticket), so the next launch finds them at zero.
template <int DXT>
__global__ void __launch_bounds__(256, 2) decorrelate_apply_kernel(const float* __restrict__ Ginv, int w,
                                                                const float* __restrict__ part, int splits, int L,
                                                                Stats st, int8_t* __restrict__ T, long long ldt,
                                                                int* __restrict__ gram, __half* __restrict__ T16,
                                                                long long ldt16, __half* __restrict__ Tk,
                                                                long long ldk, unsigned* __restrict__ bar,
                                                                unsigned* __restrict__ err) {
  constexpr int PX = DXT / 16, NW = (DXT + 31) / 32;
  extern __shared__ __align__(16) float dsm[];
  float* const Ps = dsm;                 // [w][DXT]
  float* const Gs = dsm + w * DXT;       // [w][kGsLd]
  __shared__ unsigned mz[TM][NW], mp[TM][NW];   // nonzero / positive bitplanes of the tile
  const int x0 = blockIdx.x * DXT;
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const unsigned G = gridDim.x;

  // ---- X tile = Ginv (sum_s part[s])[:, x0 .. x0 + DXT) (as decorrelate_kernel, a0 = 0)
  {
    constexpr int Q = DXT / 4, NB = 8;
    const bool pvec = (L & 3) == 0, gvec = (w & 3) == 0;
    const long long sstride = (long long)w * L;
    const int nps = w * Q, pper = (nps + 255) / 256, nld = pper * splits;
    const int ngs = w * 16, gper = (ngs + 255) / 256;
    constexpr int GB = 4;
    float4 g[GB];
#pragma unroll
    for (int q = 0; q < GB; ++q) {
      const int i = q * 256 + tid;
      g[q] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (q < gper && i < ngs) g[q] = load4(Ginv + (long long)(i >> 4) * w, (i & 15) * 4, w, gvec);
    }
    for (int f0 = 0; f0 < nld; f0 += NB) {
      float4 v[NB];
      int e = f0 / splits, sp = f0 - e * splits;
#pragma unroll
      for (int k = 0; k < NB; ++k) {
        const int i = e * 256 + tid;
        v[k] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (f0 + k < nld && i < nps)
          v[k] = load4(part + sp * sstride + (long long)(i / Q) * L, x0 + (i % Q) * 4, L, pvec);
        if (++sp == splits) {
          sp = 0;
          ++e;
        }
      }
      e = f0 / splits;
      sp = f0 - e * splits;
#pragma unroll
      for (int k = 0; k < NB; ++k) {
        const int i = e * 256 + tid;
        if (f0 + k < nld && i < nps) {
          float4* dst = reinterpret_cast<float4*>(&Ps[(i / Q) * DXT + (i % Q) * 4]);
          if (sp == 0) {
            *dst = v[k];
          } else {
            float4 t = *dst;
            t.x += v[k].x;
            t.y += v[k].y;
            t.z += v[k].z;
            t.w += v[k].w;
            *dst = t;
          }
        }
        if (++sp == splits) {
          sp = 0;
          ++e;
        }
      }
    }
#pragma unroll
    for (int q = 0; q < GB; ++q) {
      const int i = q * 256 + tid;
      if (q < gper && i < ngs) *reinterpret_cast<float4*>(&Gs[(i >> 4) * kGsLd + (i & 15) * 4]) = g[q];
    }
    for (int i = tid; i < TM * NW; i += 256) {
      (&mz[0][0])[i] = 0u;
      (&mp[0][0])[i] = 0u;
    }
  }
  __syncthreads();

  float acc[4][PX];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < PX; ++j) acc[i][j] = 0.f;
#pragma unroll 4
  for (int b = 0; b < w; ++b) {
    const float4 g = *reinterpret_cast<const float4*>(&Gs[b * kGsLd + ty * 4]);
    float p[PX];
#pragma unroll
    for (int j = 0; j < PX; ++j) p[j] = Ps[b * DXT + tx * PX + j];
    const float gv[4] = {g.x, g.y, g.z, g.w};
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < PX; ++j) acc[i][j] = fmaf(gv[i], p[j], acc[i][j]);
  }

  // ---- Eq. 2 statistics of this chunk (one per CTA)
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int a = ty * 4 + i;
    AbsSum sum;
    u64 key = 0;
    if (a < w) {
#pragma unroll
      for (int j = 0; j < PX; ++j) {
        const int x = x0 + tx * PX + j;
        if (x < L) {
          sum.add(acc[i][j]);
          const u64 kk = mag_key(acc[i][j], (uint32_t)x);
          key = kk > key ? kk : key;
        }
      }
    }
    F2 sv = sum.acc;
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) {
      sv = f2_add(sv, f2_shfl_xor(sv, o));
      const u64 t = __shfl_xor_sync(0xffffffffu, key, o);
      key = t > key ? t : key;
    }
    if (tx == 0 && a < w) put_stat(st, a, blockIdx.x, sv, key);
  }
  if (!grid_barrier(bar + 0, G, err)) return;

  // ---- thresholds of vectors blockIdx.x, blockIdx.x + G, ...: all chunks, fixed-order CTA reduction
  finalize_range(st, w, blockIdx.x, G);
  if (!grid_barrier(bar + 1, G, err)) return;
  if (blockIdx.x == 0 && tid == 0) bar[0] = 0u;   // everyone has left barrier 1

  // ---- ternarize the tile, write the factor layouts, bitplanes for the Gram
  {
    float thv[4];
    int fbv[4];
    unsigned argv[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int a = ty * 4 + i;
      thv[i] = a < w ? __ldcg(st.th.theta + a) : 0.f;
      fbv[i] = a < w ? __ldcg(st.th.fallback + a) : 0;
      argv[i] = a < w ? __ldcg(st.th.arg + a) : 0u;
    }
#pragma unroll
    for (int j = 0; j < PX; ++j) {
      const int xl = tx * PX + j, x = x0 + xl;
      if (x >= L) continue;
      short tk[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int a = ty * 4 + i;
        int8_t t = 0;
        if (a < w) {
          t = ternary_of(acc[i][j], thv[i]);
          if (fbv[i] && (uint32_t)x == argv[i]) t = acc[i][j] < 0.f ? (int8_t)-1 : (int8_t)1;
          T[(long long)a * ldt + x] = t;
          if (T16 != nullptr) T16[(long long)a * ldt16 + x] = __short2half_rn((short)t);
          if (gram != nullptr && t != 0) {
            atomicOr(&mz[a][xl >> 5], 1u << (xl & 31));
            if (t > 0) atomicOr(&mp[a][xl >> 5], 1u << (xl & 31));
          }
        }
        tk[i] = t;
      }
      if (Tk != nullptr) {   // components 4ty .. 4ty + 3 of position x: 8 bytes (ldk is a multiple of 8)
        __half* dst = Tk + (long long)x * ldk + ty * 4;
        if (ty * 4 + 3 < w) {
          const __half2 h01 = __halves2half2(__short2half_rn(tk[0]), __short2half_rn(tk[1]));
          const __half2 h23 = __halves2half2(__short2half_rn(tk[2]), __short2half_rn(tk[3]));
          uint2 u;
          u.x = *reinterpret_cast<const unsigned*>(&h01);
          u.y = *reinterpret_cast<const unsigned*>(&h23);
          *reinterpret_cast<uint2*>(dst) = u;
        } else {
          for (int i = 0; i < 4 && ty * 4 + i < w; ++i) dst[i] = __short2half_rn(tk[i]);
        }
      }
    }
  }
  if (gram != nullptr) {
    __syncthreads();
    // G_ab += popc(Z_a & Z_b) - 2 popc(Z_a & Z_b & (P_a ^ P_b)) over this tile's positions, a <= b
    for (int idx = tid; idx < w * w; idx += 256) {
      const int a = idx / w, b = idx - a * w;
      if (b < a) continue;
      int v = 0;
#pragma unroll
      for (int q = 0; q < NW; ++q) {
        const unsigned zz = mz[a][q] & mz[b][q];
        v += __popc(zz) - 2 * __popc(zz & (mp[a][q] ^ mp[b][q]));
      }
      if (v != 0) atomicAdd(&gram[(long long)a * w + b], v);
    }
  }
  // ---- exit ticket: the last CTA resets barrier 2 and the ticket
  __syncthreads();
  if (tid == 0) {
    unsigned old;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(old) : "l"(bar + 2) : "memory");
    if (old == G - 1u) {
      bar[1] = 0u;
      bar[2] = 0u;
    }
  }
}

template <int DXT>
cudaError_t launch_decorrelate_apply_dx(const float* Ginv, int w, const float* part, int splits, int L, Stats st,
                                        int8_t* T, long long ldt, int* gram, __half* T16, long long ldt16, __half* Tk,
                                        long long ldk, unsigned* bar, unsigned* err, cudaStream_t s, bool* used) {
  static int max_grid = -1;
  if (max_grid < 0) {
    cudaError_t e = cudaFuncSetAttribute(decorrelate_apply_kernel<DXT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)decorrelate_smem(TM, DXT));
    if (e != cudaSuccess) return e;
    int per_sm = 0, sms = 0, dev = 0;
    e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e == cudaSuccess)
      e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decorrelate_apply_kernel<DXT>, 256,
                                                        decorrelate_smem(TM, DXT));
    if (e != cudaSuccess) return e;
    max_grid = per_sm * sms;
  }
  const int grid = (int)cdiv(L, DXT);
  *used = grid <= max_grid;
  if (!*used) return cudaSuccess;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(256);
  cfg.dynamicSmemBytes = decorrelate_smem(w, DXT);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, decorrelate_apply_kernel<DXT>, Ginv, w, part, splits, L, st, T, ldt, gram, T16,
                            ldt16, Tk, ldk, bar, err);
}

template <bool UROW>
__global__ void __launch_bounds__(256) deflate_kernel(const float* Rin, float* Rout, int m, int n,
                                                      const int8_t* __restrict__ U, long long ldu,
                                                      const float* __restrict__ d, const int8_t* __restrict__ V,
                                                      long long ldv, int w, const float* __restrict__ h,
                                                      float* __restrict__ colpart, F2* __restrict__ normpart,
                                                      float* __restrict__ maxpart) {
  __shared__ __align__(16) float As[TK][TM + 4];
  __shared__ float wmax[8];
  __shared__ __align__(16) float Bs[TK][TN];
  __shared__ float red[16][TN];
  __shared__ float wred[8];
  const int c0 = blockIdx.x * TN;
  const int r0 = blockIdx.y * TM;
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  float acc[4][8];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;

  for (int a0 = 0; a0 < w; a0 += TK) {
    if (!UROW) {
      const int ka = tid >> 4, r4 = (tid & 15) * 4;
      const int a = a0 + ka;
      const float da = (a < w) ? __ldg(d + a) : 0.f;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int r = r0 + r4 + j;
        const float u = (a < w && r < m) ? (float)__ldg(U + a * ldu + r) : 0.f;
        As[ka][r4 + j] = u * da;
      }
    } else {
      const int r = tid >> 2, a4 = (tid & 3) * 4;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int a = a0 + a4 + j;
        const float u = (a < w && r0 + r < m) ? (float)__ldg(U + (long long)(r0 + r) * ldu + a) : 0.f;
        As[a4 + j][r] = (a < w) ? u * __ldg(d + a) : 0.f;
      }
    }
    {
      const int ka = tid >> 4, c8 = (tid & 15) * 8;
      const int a = a0 + ka;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int c = c0 + c8 + j;
        Bs[ka][c8 + j] = (a < w && c < n) ? (float)__ldg(V + a * ldv + c) : 0.f;
      }
    }
    __syncthreads();
    tile_fma(As, Bs, tx, ty, acc);
    __syncthreads();
  }

  const bool vec = (n & 3) == 0;
  float csum[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) csum[j] = 0.f;
  float nrm = 0.f, vmax = 0.f;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int r = r0 + ty * 4 + i;
    if (r >= m) continue;
#pragma unroll
    for (int g = 0; g < 2; ++g) {
      const int c = c0 + g * 64 + tx * 4;
      const float* src = Rin + (long long)r * n;
      float4 v4;
      if (vec && c + 3 < n) {
        v4 = *reinterpret_cast<const float4*>(src + c);
      } else {
        v4.x = (c + 0 < n) ? src[c + 0] : 0.f;
        v4.y = (c + 1 < n) ? src[c + 1] : 0.f;
        v4.z = (c + 2 < n) ? src[c + 2] : 0.f;
        v4.w = (c + 3 < n) ? src[c + 3] : 0.f;
      }
      float v[4] = {v4.x - acc[i][4 * g], v4.y - acc[i][4 * g + 1], v4.z - acc[i][4 * g + 2], v4.w - acc[i][4 * g + 3]};
      if (Rout != nullptr) {
        float* dst = Rout + (long long)r * n;
        if (vec && c + 3 < n) {
          *reinterpret_cast<float4*>(dst + c) = make_float4(v[0], v[1], v[2], v[3]);
        } else {
#pragma unroll
          for (int j = 0; j < 4; ++j)
            if (c + j < n) dst[c + j] = v[j];
        }
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        if (c + j < n) {
          const float sq = v[j] * v[j];
          csum[4 * g + j] += sq;
          nrm = fmaf(h != nullptr ? __ldg(h + c + j) : 1.f, sq, nrm);
          vmax = fmaxf(vmax, fabsf(v[j]));
        }
      }
    }
  }
  if (colpart != nullptr) {
#pragma unroll
    for (int j = 0; j < 8; ++j) red[ty][col_of(tx, j)] = csum[j];
    __syncthreads();
    if (tid < TN && c0 + tid < n) {
      float s = 0.f;
#pragma unroll
      for (int t = 0; t < 16; ++t) s += red[t][tid];
      colpart[(long long)blockIdx.y * n + c0 + tid] = s;
    }
  }
  const float dn = warp_sum(nrm);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) vmax = fmaxf(vmax, __shfl_xor_sync(0xffffffffu, vmax, o));
  if ((tid & 31) == 0) {
    wred[tid >> 5] = dn;
    wmax[tid >> 5] = vmax;
  }
  __syncthreads();
  if (tid == 0) {
    F2 s;
    float mx = 0.f;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      s = f2_add(s, wred[q]);
      mx = fmaxf(mx, wmax[q]);
    }
    const long long tile = (long long)blockIdx.y * gridDim.x + blockIdx.x;
    normpart[tile] = s;
    if (maxpart != nullptr) maxpart[tile] = mx;
  }
}

// Split-K factor: enough CTAs to cover the GPU twice (the float32 FMA tiles need the warps), each split at
// least 64 deep and a multiple of TK.
void choose_split(int tiles, int Ly, int* splits, int* chunk) {
  int sms = 152;
  int dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int s = (int)cdiv(2 * sms, tiles);
  s = max(1, min(s, (int)cdiv(Ly, 64)));
  int c = (int)round_up(cdiv(Ly, s), TK);
  *chunk = c;
  *splits = (int)cdiv(Ly, c);
}

}  // namespace

int product_splits(int w, int Lx, int Ly) {
  int s, c;
  choose_split((int)(cdiv(Lx, TN) * cdiv(w, TM)), Ly, &s, &c);
  return s;
}

cudaError_t launch_product_v(const float* R, int m, int n, const int8_t* Ut, int ldu, int w, float* part, int splits,
                             cudaStream_t s) {
  // every one of the `splits` partial slices is written (an empty split writes zeros)
  const int chunk = (int)round_up(cdiv(m, splits), TK);
  dim3 grid((unsigned)cdiv(n, TN), (unsigned)cdiv(w, TM), (unsigned)splits);
  product_kernel<false><<<grid, 256, 0, s>>>(R, m, n, Ut, ldu, w, nullptr, part, chunk);
  return cudaGetLastError();
}

cudaError_t launch_product_u(const float* R, int m, int n, const int8_t* Vt, int ldv, int w, const float* h,
                             float* part, int splits, cudaStream_t s) {
  const int chunk = (int)round_up(cdiv(n, splits), TK);
  dim3 grid((unsigned)cdiv(m, TN), (unsigned)cdiv(w, TM), (unsigned)splits);
  product_kernel<true><<<grid, 256, 0, s>>>(R, m, n, Vt, ldv, w, h, part, chunk);
  return cudaGetLastError();
}

namespace {
bool tc_decorrelation(int w) {
  static const bool enabled = [] {
    const char* e = std::getenv("EXTERND_TCDECOR");
    return !(e && std::strcmp(e, "0") == 0);
  }();
  return enabled && decorrelate_tc_eligible(w);
}
}  // namespace

int decorrelate_chunks(int L, int w) {
  return (int)cdiv(L, tc_decorrelation(w) ? decorrelate_tc_positions(L) : decorrelate_dx(L, w));
}

bool decorrelate_needs_operand(int w) { return tc_decorrelation(w); }

cudaError_t launch_decorrelate(const float* Ginv, int w, const float* part, int splits, int L, float* X, int ldx,
                               Stats st, cudaStream_t s, unsigned* bar, unsigned* err, const void* op) {
  if (tc_decorrelation(w)) return launch_decorrelate_tc(op, w, part, splits, L, X, ldx, st, s, bar, err);
  switch (decorrelate_dx(L, w)) {
    case 16: return launch_decorrelate_dx<16>(Ginv, w, part, splits, L, X, ldx, st, bar, err, s);
    case 32: return launch_decorrelate_dx<32>(Ginv, w, part, splits, L, X, ldx, st, bar, err, s);
    case 64: return launch_decorrelate_dx<64>(Ginv, w, part, splits, L, X, ldx, st, bar, err, s);
    default: return launch_decorrelate_dx<128>(Ginv, w, part, splits, L, X, ldx, st, bar, err, s);
  }
}

bool decorrelate_apply_fits(int w, int L) {
  if (w > TM) return false;
  int dx = decorrelate_dx(L, w), per_sm = 0, sms = 0, dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return false;
  cudaError_t e = cudaSuccess;
  switch (dx) {
    case 16: e = cudaFuncSetAttribute(decorrelate_apply_kernel<16>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)decorrelate_smem(TM, 16));
             if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decorrelate_apply_kernel<16>, 256, decorrelate_smem(TM, 16)); break;
    case 32: e = cudaFuncSetAttribute(decorrelate_apply_kernel<32>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)decorrelate_smem(TM, 32));
             if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decorrelate_apply_kernel<32>, 256, decorrelate_smem(TM, 32)); break;
    case 64: e = cudaFuncSetAttribute(decorrelate_apply_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)decorrelate_smem(TM, 64));
             if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decorrelate_apply_kernel<64>, 256, decorrelate_smem(TM, 64)); break;
    default: e = cudaFuncSetAttribute(decorrelate_apply_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)decorrelate_smem(TM, 128));
             if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decorrelate_apply_kernel<128>, 256, decorrelate_smem(TM, 128)); break;
  }
  if (e != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return cdiv(L, dx) <= (long long)per_sm * sms;
}

cudaError_t launch_decorrelate_apply(const float* Ginv, int w, const float* part, int splits, int L, Stats st,
                                     int8_t* T, long long ldt, int* gram, __half* T16, long long ldt16, __half* Tk,
                                     long long ldk, unsigned* bar, unsigned* err, cudaStream_t s, bool* used) {
  *used = false;
  if (w > TM || st.nchunk != decorrelate_chunks(L, w)) return cudaSuccess;
  if (Tk != nullptr && (ldk < round_up(w, 8) || (ldk & 7) != 0)) return cudaErrorInvalidValue;
  switch (decorrelate_dx(L, w)) {
    case 16: return launch_decorrelate_apply_dx<16>(Ginv, w, part, splits, L, st, T, ldt, gram, T16, ldt16, Tk, ldk, bar, err, s, used);
    case 32: return launch_decorrelate_apply_dx<32>(Ginv, w, part, splits, L, st, T, ldt, gram, T16, ldt16, Tk, ldk, bar, err, s, used);
    case 64: return launch_decorrelate_apply_dx<64>(Ginv, w, part, splits, L, st, T, ldt, gram, T16, ldt16, Tk, ldk, bar, err, s, used);
    default: return launch_decorrelate_apply_dx<128>(Ginv, w, part, splits, L, st, T, ldt, gram, T16, ldt16, Tk, ldk, bar, err, s, used);
  }
}

int deflate_row_tiles(int m) { return (int)cdiv(m, TM); }
int deflate_tiles(int m, int n) { return (int)(cdiv(m, TM) * cdiv(n, TN)); }

cudaError_t launch_deflate(const float* Rin, float* Rout, int m, int n, const int8_t* U, long long ldu, bool u_rowmajor,
                           const float* d, const int8_t* Vt, long long ldv, int w, const float* h, float* colpart,
                           F2* normpart, cudaStream_t s, float* maxpart) {
  dim3 grid((unsigned)cdiv(n, TN), (unsigned)cdiv(m, TM));
  if (u_rowmajor)
    deflate_kernel<true><<<grid, 256, 0, s>>>(Rin, Rout, m, n, U, ldu, d, Vt, ldv, w, h, colpart, normpart, maxpart);
  else
    deflate_kernel<false><<<grid, 256, 0, s>>>(Rin, Rout, m, n, U, ldu, d, Vt, ldv, w, h, colpart, normpart, maxpart);
  return cudaGetLastError();
}

}  // namespace externd
