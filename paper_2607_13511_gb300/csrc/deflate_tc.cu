// Deflation on the 5th-generation tensor cores (§2.3, §2.4):
//
//   R[r][c] <- R[r][c] - sum_a U[r][a] d[a] V[c][a]
//
// fused with the statistics the next block needs: per 64-row tile the column sums of R^2 (column energies),
// sum_c h_c R[r][c]^2 (double-float), and max |R|.
//
// A CTA owns a block of 128 columns (the MMA's M: one TMEM lane, and one epilogue thread, per column) and a run
// of row tiles of 128 rows (N), so the epilogue reads and writes R along rows with consecutive lanes on
// consecutive columns. Operands, K-major fp16 in 128-byte-swizzled shared memory: A[c][a] = V[c][a] d[a] 2^s split
// into hi = RN(.) and lo = RN(. - hi) (V is ternary, so both are exact products of d's two fp16 parts), staged
// once per CTA; B[r][a] = U[r][a] (exact), one tile per row tile, double-buffered (cp.async) when w <= 128. The two
// MMAs per K step accumulate D^T[c][r] = sum_a (d_hi + d_lo)[a] V[c][a] U[r][a] in fp32, alternately into two TMEM
// accumulators: the MMA of row tile i + 1 runs while the epilogue of tile i reads and writes R (16 warps, all 32 of
// a thread's values of R in flight at once). The power of two 2^s puts max |d| just under 2^14, and hi + lo keeps
// ~22 significant bits of every d[a].
#include <algorithm>

#include "kernels.h"
#include "umma.cuh"

namespace externd {

namespace {

constexpr int kCols = 128;        // columns per CTA (MMA M)
constexpr int kRows = 128;        // rows per tile (MMA N)
constexpr int kThreads = 512;     // 16 warps: staging, then the epilogue (4 warps per TMEM lane quadrant)
constexpr uint32_t kAtomA = (uint32_t)kCols * 128u;   // one 64-wide K atom of A: 128 rows x 128 B
constexpr uint32_t kAtomB = (uint32_t)kRows * 128u;

struct DeflateArgs {
  float* R;
  int m, n;
  const __half* Uk;   // m x ldk, U[r][a] at Uk[r * ldk + a]
  const __half* Vk;   // n x ldk
  long long ldk;
  const float* d;
  int w, wpad, natoms, nbuf;
  const float* h;
  float* colpart;     // [cdiv(m, 64)][n] or nullptr
  F2* normpart;       // [cdiv(m, 64)][cdiv(n, 128)]
  float* maxpart;     // same shape, or nullptr
  unsigned* err;
};

// U buffers: two (prefetch) up to 128 components, one above (the shared memory holds no second)
int deflate_tc_bufs(int natoms) { return natoms <= 2 ? 2 : 1; }

size_t deflate_tc_smem(int natoms) {
  return 1024 + (size_t)natoms * (2 * kAtomA + (size_t)deflate_tc_bufs(natoms) * kAtomB) +
         2 * kMaxBlock * sizeof(__half) + 64;
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_but_one() { asm volatile("cp.async.wait_group 1;" ::: "memory"); }

__global__ void __launch_bounds__(kThreads, 1) deflate_tc_kernel(const DeflateArgs p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t sbase = (raw + 1023u) & ~1023u;
  uint8_t* const gbase = smem_raw + (sbase - raw);
  const uint32_t natoms = (uint32_t)p.natoms;
  const uint32_t a_hi = sbase, a_lo = sbase + natoms * kAtomA;
  const uint32_t b_base = sbase + 2u * natoms * kAtomA;   // buffer q at b_base + q * natoms * kAtomB
  uint8_t* const g_ahi = gbase;
  uint8_t* const g_alo = gbase + (size_t)natoms * kAtomA;
  __half* const dhi = reinterpret_cast<__half*>(gbase + (size_t)natoms * (2 * kAtomA + p.nbuf * kAtomB));
  __half* const dlo = dhi + kMaxBlock;
  __shared__ uint64_t done_bar[2];
  __shared__ uint32_t tmem_slot;
  __shared__ float red_max[kThreads / 32];
  __shared__ F2 red_sum[kThreads / 32];
  __shared__ float col_sum[4][kCols];   // per 32-row quarter: the column sums of R^2
  __shared__ int s_exp;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int cb = blockIdx.x, c0 = cb * kCols;
  const int RT = (p.m + kRows - 1) / kRows, S = (int)gridDim.y;
  const int t_begin = (int)((long long)blockIdx.y * RT / S), t_end = (int)((long long)(blockIdx.y + 1) * RT / S);
  const int T = t_end - t_begin;
  if (T <= 0) return;   // uniform across the CTA, before any barrier or allocation
  const int kch = p.wpad / 8;   // 16-byte chunks of one operand row
  const int nb = p.nbuf;

  // B = U rows of row tile t into buffer q (async copies; rows beyond m read as zeros), one commit group
  auto stage_u = [&](int t, int q) {
    const int r0 = t * kRows;
    const uint32_t bq = b_base + (uint32_t)q * natoms * kAtomB;
    for (int id = tid; id < kRows * kch; id += kThreads) {
      const int r = id / kch, j = id - r * kch;
      const uint32_t dst = bq + (uint32_t)(j >> 3) * kAtomB + sw128_offset((uint32_t)r, (uint32_t)(j & 7));
      const bool in = r0 + r < p.m;
      cp_async16(dst, p.Uk + (in ? (long long)(r0 + r) * p.ldk + 8 * j : 0), in ? 16u : 0u);
    }
    cp_async_commit();
  };
  stage_u(t_begin, 0);
  if (nb == 2 && T > 1) stage_u(t_begin + 1, 1);
  // scale: 2^s with max |d| * 2^s just under 2^14
  {
    float mx = 0.f;
    for (int a = tid; a < p.w; a += kThreads) mx = fmaxf(mx, fabsf(__ldg(p.d + a)));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    if (lane == 0) red_max[warp] = mx;
    if (tid == 0) {
      mbar_init(smem_addr(&done_bar[0]), 1);
      mbar_init(smem_addr(&done_bar[1]), 1);
      fence_barrier_init();
    }
    __syncthreads();
    if (tid == 0) {
      float t = 0.f;
      for (int q = 0; q < kThreads / 32; ++q) t = fmaxf(t, red_max[q]);
      int ex = 0;
      if (t > 0.f && t <= 3.0e38f) frexpf(t, &ex);
      s_exp = max(-100, min(100, 14 - ex));
    }
    __syncthreads();
    const float scale = ldexpf(1.f, s_exp);
    for (int a = tid; a < p.wpad; a += kThreads) {
      const float x = a < p.w ? __ldg(p.d + a) * scale : 0.f;
      const __half hi = __float2half_rn(x);
      dhi[a] = hi;
      dlo[a] = __float2half_rn(x - __half2float(hi));
    }
  }
  if (warp == 0) {
    tmem_alloc(smem_addr(&tmem_slot), 2u * kRows);   // two accumulators
    tmem_relinquish();
  }
  __syncthreads();
  // A = V rows c0.. times d (hi and lo), once; components >= w and columns >= n are zero
  for (int id = tid; id < kCols * kch; id += kThreads) {
    const int c = id / kch, j = id - c * kch;
    uint4 raw4 = make_uint4(0u, 0u, 0u, 0u);
    if (c0 + c < p.n) raw4 = __ldg(reinterpret_cast<const uint4*>(p.Vk + (long long)(c0 + c) * p.ldk + 8 * j));
    const int valid = p.w - 8 * j;   // components of this chunk below w
    if (valid < 8) {
      uint32_t* wv = reinterpret_cast<uint32_t*>(&raw4);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        if (2 * e >= valid) wv[e] = 0u;
        else if (2 * e + 1 >= valid) wv[e] &= 0xffffu;
      }
    }
    const __half2* v2 = reinterpret_cast<const __half2*>(&raw4);
    const __half2* h2 = reinterpret_cast<const __half2*>(dhi + 8 * j);
    const __half2* l2 = reinterpret_cast<const __half2*>(dlo + 8 * j);
    uint32_t hv[4], lv[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const __half2 ph = __hmul2(v2[e], h2[e]), pl = __hmul2(v2[e], l2[e]);
      hv[e] = *reinterpret_cast<const uint32_t*>(&ph);
      lv[e] = *reinterpret_cast<const uint32_t*>(&pl);
    }
    const uint32_t off = (uint32_t)(j >> 3) * kAtomA + sw128_offset((uint32_t)c, (uint32_t)(j & 7));
    *reinterpret_cast<uint4*>(g_ahi + off) = make_uint4(hv[0], hv[1], hv[2], hv[3]);
    *reinterpret_cast<uint4*>(g_alo + off) = make_uint4(lv[0], lv[1], lv[2], lv[3]);
  }
  if (nb == 2 && T > 1) cp_async_wait_but_one();   // U of the first tile (the second may still be landing)
  else cp_async_wait_all();
  fence_async_shared();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_slot;
  const uint32_t idesc = f16_idesc(kCols, kRows);
  // the MMAs of tile i (B in buffer i % nb) into accumulator i % 2, completion on done_bar[i % 2]
  auto issue = [&](int i) {
    if (tid == 0) {
      const uint32_t bq = b_base + (uint32_t)(i % nb) * natoms * kAtomB;
      const uint32_t d = tmem + (uint32_t)(i & 1) * kRows;
      for (int kk = 0; kk < p.wpad / 16; ++kk) {
        const uint32_t ko = (uint32_t)(kk >> 2), kb = 32u * (uint32_t)(kk & 3);
        const uint64_t bd = sw128_desc(bq + ko * kAtomB + kb);
        mma_f16(d, sw128_desc(a_hi + ko * kAtomA + kb), bd, idesc, kk > 0 ? 1u : 0u);
        mma_f16(d, sw128_desc(a_lo + ko * kAtomA + kb), bd, idesc, 1u);
      }
      mma_commit(smem_addr(&done_bar[i & 1]));
    }
    __syncwarp();
  };
  issue(0);

  // epilogue: warp q reads TMEM lanes 32 (q % 4) .. (columns) for the 32-row quarter q / 4 (2 chunks of 16 rows)
  const int quad = warp & 3, part = warp >> 2, half = part >> 1;
  const int c = c0 + quad * 32 + lane;
  const bool cin = c < p.n;
  const float inv_scale = ldexpf(1.f, -s_exp);
  const float hc = (p.h != nullptr && cin) ? __ldg(p.h + c) : 1.f;
  const int CB = (int)gridDim.x;
  bool ok = true;
  for (int i = 0; i < T; ++i) {
    const int t = t_begin + i, r0 = t * kRows;
    // this thread's 32 values of R for tile t, all in flight before anything waits
    float rv[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const int r = r0 + part * 32 + j;
      rv[j] = (cin && r < p.m) ? p.R[(long long)r * p.n + c] : 0.f;
    }
    if (nb == 2 && i + 1 < T) {   // the next tile's MMAs run during this tile's epilogue
      cp_async_wait_all();
      fence_async_shared();
      tc_fence_before();
      __syncthreads();
      tc_fence_after();
      issue(i + 1);
    }
    const bool got = mbar_wait(smem_addr(&done_bar[i & 1]), (uint32_t)(i >> 1) & 1u, p.err);
    const bool have = ok && __all_sync(0xffffffffu, got) != 0;
    ok = have;
    tc_fence_after();
    if (i + nb < T) stage_u(t_begin + i + nb, i % nb);   // this tile's B buffer is free: the MMAs completed
    float csum = 0.f, vmax = 0.f;
#pragma unroll
    for (int ch = 0; ch < 2; ++ch) {
      const int rb = r0 + part * 32 + ch * 16;
      uint32_t acc[16];
      if (have) {
        tmem_ld16(tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)(i & 1) * kRows + (uint32_t)(part * 32 + ch * 16),
                  acc);
        tmem_wait_ld();
      } else {
#pragma unroll
        for (int j = 0; j < 16; ++j) acc[j] = 0u;
      }
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        if (cin && rb + j < p.m) {
          const float v = rv[16 * ch + j] - __uint_as_float(acc[j]) * inv_scale;
          p.R[(long long)(rb + j) * p.n + c] = v;
          csum = fmaf(v, v, csum);
          vmax = fmaxf(vmax, fabsf(v));
        }
      }
    }
    const int tile_row = 2 * t + half;          // 64-row tile
    const bool row_in = tile_row * 64 < p.m;
    col_sum[part][quad * 32 + lane] = csum;
    F2 s;
    s.hi = hc * csum;
    s = warp_sum(s);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) vmax = fmaxf(vmax, __shfl_xor_sync(0xffffffffu, vmax, o));
    if (lane == 0) {
      red_sum[warp] = s;
      red_max[warp] = vmax;
    }
    tc_fence_before();
    __syncthreads();   // the accumulator is read (free for tile i + 2) and the warp sums are in place
    // column energies of the 64-row tile: its two quarters in order
    if ((part & 1) == 0 && p.colpart != nullptr && cin && row_in)
      p.colpart[(long long)tile_row * p.n + c] = col_sum[part][quad * 32 + lane] + col_sum[part + 1][quad * 32 + lane];
    if ((tid & 255) == 0 && row_in) {   // one thread per 64-row half sums its 8 warps in order
      F2 tsum;
      float mx = 0.f;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        tsum = f2_add(tsum, red_sum[half * 8 + q]);
        mx = fmaxf(mx, red_max[half * 8 + q]);
      }
      const long long tile = (long long)tile_row * CB + cb;
      p.normpart[tile] = tsum;
      if (p.maxpart != nullptr) p.maxpart[tile] = mx;
    }
    if (nb == 1 && i + 1 < T) {   // one buffer: the next tile's operand has landed meanwhile
      cp_async_wait_all();
      fence_async_shared();
      __syncthreads();
      tc_fence_after();
      issue(i + 1);
    } else {
      __syncthreads();   // red_sum / red_max / col_sum are read before the next tile writes them
    }
  }
  cp_async_wait_all();
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, 2u * kRows);
  }
}

// dst[pos * ldk + a] = src[a * lda + pos * ldp] as fp16, for a < w, pos < L.
__global__ void kmajor_kernel(const int8_t* __restrict__ src, long long lda, long long ldp, int w, int L,
                              __half* __restrict__ dst, long long ldk) {
  const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (long long)L * w) return;
  const int pos = (int)(i / w), a = (int)(i - (long long)pos * w);
  dst[(long long)pos * ldk + a] = __short2half_rn((short)src[a * lda + pos * ldp]);
}

}  // namespace

cudaError_t launch_deflate_tc(float* R, int m, int n, const __half* Uk, const __half* Vk, long long ldk,
                              const float* d, int w, const float* h, float* colpart, F2* normpart, float* maxpart,
                              unsigned* err, cudaStream_t s) {
  if (w < 1 || w > kMaxBlock || ldk < round_up(w, 16) || (ldk & 7) != 0 || err == nullptr) return cudaErrorInvalidValue;
  DeflateArgs a;
  a.R = R;
  a.m = m;
  a.n = n;
  a.Uk = Uk;
  a.Vk = Vk;
  a.ldk = ldk;
  a.d = d;
  a.w = w;
  a.wpad = (int)round_up(w, 16);
  a.natoms = (int)cdiv(a.wpad, 64);
  a.nbuf = deflate_tc_bufs(a.natoms);
  a.h = h;
  a.colpart = colpart;
  a.normpart = normpart;
  a.maxpart = maxpart;
  a.err = err;
  static int sms = 0;
  if (sms == 0) {
    int dev = 0, v = 0;
    if (cudaGetDevice(&dev) == cudaSuccess && cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) ==
                                                  cudaSuccess && v > 0)
      sms = v;
    else
      sms = 148;
    cudaGetLastError();
    size_t mx = 0;
    for (int na = 1; na <= (int)cdiv(kMaxBlock, 64); ++na) mx = std::max(mx, deflate_tc_smem(na));
    const cudaError_t e = cudaFuncSetAttribute(deflate_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)mx);
    if (e != cudaSuccess) return e;
  }
  // one CTA per SM: column blocks x row groups, each row group a contiguous run of row tiles
  const int CB = (int)cdiv(n, kCols), RT = (int)cdiv(m, kRows);
  const int S = std::max(1, std::min(RT, (int)cdiv(sms, CB)));
  deflate_tc_kernel<<<dim3((unsigned)CB, (unsigned)S), kThreads, deflate_tc_smem(a.natoms), s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_kmajor(const int8_t* src, long long lda, long long ldp, int w, int L, __half* dst, long long ldk,
                          cudaStream_t s) {
  const long long total = (long long)L * w;
  if (total == 0) return cudaSuccess;
  kmajor_kernel<<<(unsigned)cdiv(total, 256), 256, 0, s>>>(src, lda, ldp, w, L, dst, ldk);
  return cudaGetLastError();
}

}  // namespace externd
