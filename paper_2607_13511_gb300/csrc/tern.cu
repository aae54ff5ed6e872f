// Eq. 2 ternarization (statistics + apply), the start of each block (top-w residual columns), and the small
// data-movement kernels around them.
//
// Eq. 2: T_tau(x)_i = sign(x_i) [|x_i| > tau * (1/L) sum_j |x_j|]; if nothing passes, the single largest |x_i|
// (first index) is kept. The sum is gathered as per-chunk partials (compensated float, combined in double) by
// whichever kernel produces x, then summed in a fixed order by the apply kernel: theta = tau * (S / L) in double,
// compared in float against RD_float(theta), which decides exactly like a double comparison for float x.
#include <algorithm>

#include "kernels.h"

namespace externd {

namespace {

// Per-chunk statistics of vector a over positions [x0, x0 + 128).
__global__ void __launch_bounds__(128) stats_kernel(const float* __restrict__ X, int L, long long ldx, Stats st) {
  __shared__ F2 ssum[4];
  __shared__ u64 skey[4];
  const int a = blockIdx.y;
  const int x = blockIdx.x * kStatChunk + threadIdx.x;
  float v = 0.f;
  bool valid = x < L;
  if (valid) v = __ldg(X + (long long)a * ldx + x);
  F2 s;
  s.hi = valid ? fabsf(v) : 0.f;
  u64 key = valid ? mag_key(v, (uint32_t)x) : 0ull;
  s = warp_sum(s);
  key = warp_max(key);
  const int warp = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) {
    ssum[warp] = s;
    skey[warp] = key;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    F2 t;
    u64 k = 0;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      t = f2_add(t, ssum[q]);
      k = skey[q] > k ? skey[q] : k;
    }
    put_stat(st, a, blockIdx.x, t, k);
  }
  stats_done(st, gridDim.y);
}

// The block start's gather with the per-chunk statistics: Y[a][x] = R[x][J[a]] for one 128-position chunk per
// warp (lanes take positions x0 + lane + 32k, k < 4, the four gathers in flight together), 8 warps per CTA over
// the nv * cdiv(L, 128) (vector, chunk) items, so that few CTAs take the finalize ticket.
__global__ void __launch_bounds__(256) gather_stats_kernel(const float* __restrict__ R, int L, int ncols,
                                                           const int* __restrict__ J, float* __restrict__ Y,
                                                           long long ldy, int nv, Stats st) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nchunk = (L + kStatChunk - 1) / kStatChunk;
  const long long items = (long long)nv * nchunk;
  for (long long it = (long long)blockIdx.x * 8 + warp; it < items; it += (long long)gridDim.x * 8) {
    const int a = (int)(it / nchunk), ch = (int)(it - (long long)a * nchunk);
    const int j = min(max(__ldg(J + a), 0), ncols - 1);   // J comes from select_kernel; never read outside R
    float v[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int x = ch * kStatChunk + lane + 32 * k;
      v[k] = x < L ? __ldg(R + (long long)x * ncols + j) : 0.f;
    }
    F2 s;
    u64 key = 0;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int x = ch * kStatChunk + lane + 32 * k;
      if (x < L) {
        Y[(long long)a * ldy + x] = v[k];
        F2 t;
        t.hi = fabsf(v[k]);
        s = f2_add(s, t);
        const u64 kk = mag_key(v[k], (uint32_t)x);
        key = kk > key ? kk : key;
      }
    }
    s = warp_sum(s);
    key = warp_max(key);
    if (lane == 0) put_stat(st, a, ch, s, key);
  }
  stats_done(st, nv);
}

// T = T_tau(X) for up to 256 vectors per CTA over positions [x0, x0 + P), in 64-position chunks. Each warp
// ternarizes 32 positions of one vector at a time (coalesced reads and byte writes) and records the +1 and -1
// positions as ballot masks; with GRAM the CTA then adds the chunk's exact Gram entries
//   G_ab += popc(P_a & P_b) + popc(N_a & N_b) - popc(P_a & N_b) - popc(N_a & P_b)
// into per-thread integer accumulators (thread: vector a = tid % VB, VB*VB/256 consecutive b), and finally
// atomically adds the upper triangle to gram. Integer sums are exact, so the order of the atomics does not matter.
template <int VB, bool GRAM>
__global__ void __launch_bounds__(256) apply_kernel(const float* __restrict__ X, int nv, int L, long long ldx,
                                                    Thresh th, int8_t* __restrict__ T, long long ldt,
                                                    int* __restrict__ gram, int P, __half* __restrict__ T16,
                                                    long long ldt16, __half* __restrict__ Tk, long long ldk,
                                                    GramScratch gs) {
  // Gram pairs a <= b, folded: row f and row VB-1-f together hold VB+1 pairs; FR = VB/2 folded rows, NPART
  // threads per folded row, PPT pairs per thread (strided along the folded row)
  constexpr int FR = VB / 2, NPART = 256 / FR, PPT = (VB + 1 + NPART - 1) / NPART;
  constexpr int IT = VB / 4;                                      // warp passes per 64-position chunk
  constexpr int KLD = VB + 8;                                     // sK row (halves): 16-byte rows, 4-way stores
  __shared__ unsigned mnz[VB][2], mpos[VB][2];   // per 64-position chunk: nonzero and positive bitplanes
  __shared__ __align__(16) __half sK[64][KLD];                    // the chunk as [position][component]
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int v0 = blockIdx.y * VB;
  const int nvb = min(VB, nv - v0);
  const int xbeg = blockIdx.x * P, xend = min(L, xbeg + P);
  const int gf = tid % FR, gpart = tid / FR;
  int acc[PPT];
#pragma unroll
  for (int k = 0; k < PPT; ++k) acc[k] = 0;
  for (int x0 = xbeg; x0 < xend; x0 += 64) {
    // pass i of warp covers vector a = (warp + 8i) / 2, positions x0 + 32 * ((warp + 8i) % 2) + lane; the
    // loads of a batch of passes (values and thresholds) are all issued before the first is used
    constexpr int IB = IT < 16 ? IT : 16;
#pragma unroll 1
    for (int i0 = 0; i0 < IT; i0 += IB) {
      float xv[IB], thv[IB];
      int fbv[IB];
      unsigned argv[IB];
#pragma unroll
      for (int i = 0; i < IB; ++i) {
        const int u = warp + 8 * (i0 + i), a = u >> 1;
        const int x = x0 + 32 * (u & 1) + lane;
        const bool in = a < nvb && x < xend;
        xv[i] = in ? X[(long long)(v0 + a) * ldx + x] : 0.f;
        thv[i] = a < nvb ? th.theta[v0 + a] : 0.f;
        fbv[i] = a < nvb ? th.fallback[v0 + a] : 0;
        argv[i] = a < nvb ? th.arg[v0 + a] : 0u;
      }
#pragma unroll
      for (int i = 0; i < IB; ++i) {
        const int u = warp + 8 * (i0 + i), a = u >> 1, half = u & 1;
        const int x = x0 + 32 * half + lane;
        int8_t t = 0;
        if (a < nvb && x < xend) {
          const int v = v0 + a;
          t = ternary_of(xv[i], thv[i]);
          if (fbv[i] && (uint32_t)x == argv[i]) t = xv[i] < 0.f ? (int8_t)-1 : (int8_t)1;
          T[(long long)v * ldt + x] = t;
          if (T16 != nullptr) T16[(long long)v * ldt16 + x] = __short2half_rn((short)t);
        }
        if (GRAM) {
          const unsigned zm = __ballot_sync(0xffffffffu, t != 0), pm = __ballot_sync(0xffffffffu, t > 0);
          if (lane == 0) {
            mnz[a][half] = zm;
            mpos[a][half] = pm;
          }
        }
        if (Tk != nullptr) sK[32 * half + lane][a] = __short2half_rn((short)t);
      }
    }
    if (Tk != nullptr) {   // K-major fp16 copy: rows of the chunk's positions, 16-byte chunks of 8 components
      __syncthreads();
      const int kc = (nvb + 7) / 8;
      for (int id = tid; id < 64 * kc; id += 256) {
        const int xl = id / kc, j = id - xl * kc;
        if (x0 + xl < xend)
          *reinterpret_cast<uint4*>(Tk + (long long)(x0 + xl) * ldk + 8 * j) =
              *reinterpret_cast<const uint4*>(&sK[xl][8 * j]);
      }
      __syncthreads();
    }
    if (GRAM) {
      // G_ab += popc(Z_a & Z_b) - 2 popc(Z_a & Z_b & (P_a ^ P_b)): both nonzero, minus twice the opposite signs
      __syncthreads();
      const int a1 = gf, a2 = VB - 1 - gf;
      const unsigned long long z1 = mnz[a1][0] | ((unsigned long long)mnz[a1][1] << 32);
      const unsigned long long p1 = mpos[a1][0] | ((unsigned long long)mpos[a1][1] << 32);
      const unsigned long long z2 = mnz[a2][0] | ((unsigned long long)mnz[a2][1] << 32);
      const unsigned long long p2 = mpos[a2][0] | ((unsigned long long)mpos[a2][1] << 32);
#pragma unroll
      for (int k = 0; k < PPT; ++k) {
        const int e = gpart + NPART * k;          // position along the folded row
        const bool first = e < VB - gf;
        const int b = first ? gf + e : a2 + (e - (VB - gf));
        if (e <= VB) {
          const unsigned long long zb = mnz[b][0] | ((unsigned long long)mnz[b][1] << 32);
          const unsigned long long pb = mpos[b][0] | ((unsigned long long)mpos[b][1] << 32);
          const unsigned long long zz = (first ? z1 : z2) & zb;
          const unsigned long long dd = zz & ((first ? p1 : p2) ^ pb);
          acc[k] += __popcll(zz) - 2 * __popcll(dd);
        }
      }
      __syncthreads();
    }
  }
  if (GRAM) {
    // Few CTAs: every CTA adds its partials atomically. Many CTAs (gs.part given): each CTA stores its partials
    // (slot-major, coalesced) and the last CTA of every group of kGramGroup consecutive CTAs (acquire-release
    // ticket, as for the statistics) sums the group's partials, four slots of loads in flight at a time, and adds
    // them, so one atomic per slot and group reaches L2.
    auto pair_of = [&](int k, int& a, int& b) {
      const int e = gpart + NPART * k;
      const bool first = e < VB - gf;
      a = first ? gf : VB - 1 - gf;
      b = first ? gf + e : VB - 1 - gf + (e - (VB - gf));
      return e <= VB;
    };
    if (gs.part == nullptr) {
#pragma unroll
      for (int k = 0; k < PPT; ++k) {
        int a, b;
        if (pair_of(k, a, b) && a < nvb && b < nvb && acc[k] != 0) atomicAdd(&gram[(long long)a * nv + b], acc[k]);
      }
    } else {
      __shared__ int s_last_g;
      int* mine = gs.part + (long long)blockIdx.x * PPT * 256;
#pragma unroll
      for (int k = 0; k < PPT; ++k) mine[k * 256 + tid] = acc[k];
      __syncthreads();
      const int grp = blockIdx.x / kGramGroup, g0 = grp * kGramGroup;
      const int gn = min(kGramGroup, (int)gridDim.x - g0);
      if (tid == 0) {
        unsigned old;
        asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(old) : "l"(gs.ticket + grp) : "memory");
        s_last_g = (old == (unsigned)gn - 1u);
      }
      __syncthreads();
      if (s_last_g) {
        constexpr int KB = PPT < 4 ? PPT : 4;
        const int* base = gs.part + (long long)g0 * PPT * 256;
#pragma unroll 1
        for (int k0 = 0; k0 < PPT; k0 += KB) {
          int v[KB][kGramGroup];
#pragma unroll
          for (int q = 0; q < KB; ++q)
#pragma unroll
            for (int c = 0; c < kGramGroup; ++c)
              v[q][c] = (k0 + q < PPT && c < gn) ? base[((long long)c * PPT + k0 + q) * 256 + tid] : 0;
#pragma unroll
          for (int q = 0; q < KB; ++q) {
            int sum = 0;
#pragma unroll
            for (int c = 0; c < kGramGroup; ++c) sum += v[q][c];
            int a, b;
            if (k0 + q < PPT && pair_of(k0 + q, a, b) && a < nvb && b < nvb && sum != 0)
              atomicAdd(&gram[(long long)a * nv + b], sum);
          }
        }
        if (tid == 0) gs.ticket[grp] = 0u;
      }
    }
  }
}

// Column energies e_c = h_c * sum_t colpart[t][c].
__global__ void colsum_kernel(const float* __restrict__ colpart, int nrt, int n, const float* __restrict__ h,
                              float* __restrict__ e) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= n) return;
  float s = 0.f;
  for (int t = 0; t < nrt; ++t) s += colpart[(long long)t * n + c];
  e[c] = (h != nullptr) ? s * __ldg(h + c) : s;
}

// Inclusive scan of one int per thread over a 1024-thread block.
__device__ int block_scan_incl(int v, int* sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int t = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += t;
  }
  if (lane == 31) sh[warp] = v;
  __syncthreads();
  if (warp == 0) {
    int t = sh[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int u = __shfl_up_sync(0xffffffffu, t, o);
      if (lane >= o) t += u;
    }
    sh[lane] = t;
  }
  __syncthreads();
  const int r = v + (warp > 0 ? sh[warp - 1] : 0);
  __syncthreads();
  return r;
}

// The w columns with the largest energy (ties to the lower index), in ascending column order. One CTA:
// radix select of the w-th largest key (energies are non-negative floats, so their bits order like the values),
// then an ordered compaction.
__global__ void __launch_bounds__(1024) select_kernel(const float* __restrict__ e, int n, int w, int* __restrict__ J) {
  __shared__ unsigned hist[256];
  __shared__ unsigned s_bin, s_rem;
  __shared__ int scan_sh[32];
  const int tid = threadIdx.x;
  const int per = (int)cdiv(n, 1024);
  const int cb = min(n, tid * per), ce = min(n, cb + per);
  // the thread's keys stay in registers across the passes when they number at most kKeep (n <= 16384)
  constexpr int kKeep = 16;
  const bool keep = per <= kKeep;
  unsigned kr[kKeep];
#pragma unroll
  for (int i = 0; i < kKeep; ++i) kr[i] = (keep && cb + i < ce) ? __float_as_uint(e[cb + i]) : 0u;
  unsigned prefix = 0, mask = 0, remaining = (unsigned)w;
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int i = tid; i < 256; i += 1024) hist[i] = 0;
    __syncthreads();
    if (keep) {
#pragma unroll
      for (int i = 0; i < kKeep; ++i)
        if (cb + i < ce && (kr[i] & mask) == prefix) atomicAdd(&hist[(kr[i] >> shift) & 255u], 1u);
    } else {
      for (int c = cb; c < ce; ++c) {
        const unsigned key = __float_as_uint(e[c]);
        if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
      }
    }
    __syncthreads();
    if (tid < 32) {
      // lane l holds bins 255-8l ... 248-8l (descending)
      unsigned cnt[8], tot = 0;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        cnt[q] = hist[255 - 8 * tid - q];
        tot += cnt[q];
      }
      unsigned incl = tot;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const unsigned t = __shfl_up_sync(0xffffffffu, incl, o);
        if (tid >= o) incl += t;
      }
      const unsigned excl = incl - tot;
      const bool here = excl < remaining && remaining <= incl;
      if (here) {
        unsigned cum = excl;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          if (cum + cnt[q] >= remaining) {
            s_bin = 255 - 8 * tid - q;
            s_rem = remaining - cum;
            break;
          }
          cum += cnt[q];
        }
      }
    }
    __syncthreads();
    prefix |= s_bin << shift;
    mask |= 255u << shift;
    remaining = s_rem;
    __syncthreads();
  }
  // prefix = key of the w-th largest; take every key above it and the first `remaining` keys equal to it.
  // visit(f) calls f(c, key) for the thread's columns in order (keys from registers when kept)
  auto visit = [&](auto&& f) {
    if (keep) {
#pragma unroll
      for (int i = 0; i < kKeep; ++i)
        if (cb + i < ce) f(cb + i, kr[i]);
    } else {
      for (int c = cb; c < ce; ++c) f(c, __float_as_uint(e[c]));
    }
  };
  int eq = 0;
  visit([&](int, unsigned key) { eq += key == prefix; });
  int eq_before = block_scan_incl(eq, scan_sh) - eq;
  int sel = 0;
  {
    int e_seen = eq_before;
    visit([&](int, unsigned key) {
      if (key > prefix) ++sel;
      else if (key == prefix) sel += (unsigned)(e_seen++) < remaining;
    });
  }
  int pos = block_scan_incl(sel, scan_sh) - sel;
  int e_seen = eq_before;
  visit([&](int c, unsigned key) {
    bool take = key > prefix;
    if (key == prefix) take = (unsigned)(e_seen++) < remaining;
    if (take) J[pos++] = c;
  });
}

// One CTA of 1024 threads: thread t adds the partials t, t + 1024, ... (all its loads issued before the first
// addition), then the warps' sums combine by shuffles and the 32 warp sums in warp order: a fixed order, so the
// result is the same on every run.
__global__ void __launch_bounds__(1024) norm_kernel(const F2* __restrict__ part, int count, double* out,
                                                    const double* norm_a, double* trace,
                                                    const float* __restrict__ maxpart, float* maxout) {
  constexpr int kBatch = 8;
  __shared__ F2 red_s[32];
  __shared__ float red_m[32];
  F2 s;
  float mx = 0.f;
  for (int i0 = threadIdx.x; i0 < count; i0 += 1024 * kBatch) {
    F2 v[kBatch];
    float m[kBatch];
#pragma unroll
    for (int b = 0; b < kBatch; ++b) {
      const int i = i0 + 1024 * b;
      v[b] = i < count ? part[i] : F2{};
      m[b] = (maxpart != nullptr && i < count) ? maxpart[i] : 0.f;
    }
#pragma unroll
    for (int b = 0; b < kBatch; ++b) {
      s = f2_add(s, v[b]);
      mx = fmaxf(mx, m[b]);
    }
  }
  s = warp_sum(s);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  if ((threadIdx.x & 31) == 0) {
    red_s[threadIdx.x >> 5] = s;
    red_m[threadIdx.x >> 5] = mx;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    F2 t = red_s[0];
    float tm = red_m[0];
    for (int q = 1; q < 32; ++q) {
      t = f2_add(t, red_s[q]);
      tm = fmaxf(tm, red_m[q]);
    }
    const double v = f2_value(t);
    out[0] = v;
    if (trace != nullptr) trace[0] = 1.0 - v / norm_a[0];
    if (maxout != nullptr) maxout[0] = tm;
  }
}

// out[0] = max |x_i| over n floats (one CTA; the result feeds the fp16 scaling of the tensor-core products).
__global__ void __launch_bounds__(1024) absmax_kernel(const float* __restrict__ x, long long n, float* out) {
  __shared__ float red[32];
  float mx = 0.f;
  for (long long i = threadIdx.x; i < n; i += 1024) mx = fmaxf(mx, fabsf(x[i]));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = mx;
  __syncthreads();
  if (threadIdx.x < 32) {
    mx = red[threadIdx.x];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    if (threadIdx.x == 0) out[0] = mx;
  }
}

// B[r][j0 + a] = Ut[a][r] for a 64-row slab: read Ut rows coalesced, transpose in shared memory, write each
// row's w bytes as 4-byte words when aligned.
__global__ void __launch_bounds__(256) write_b_kernel(const int8_t* __restrict__ Ut, int ldu, int w, int m,
                                                      int8_t* __restrict__ B, long long k, long long j0,
                                                      const IoTable* __restrict__ io) {
  __shared__ int8_t tile[kMaxBlock][68];
  if (io != nullptr) B = io->B;
  const int r0 = blockIdx.x * 64;
  for (int i = threadIdx.x; i < w * 64; i += 256) {
    const int a = i >> 6, r = i & 63;
    tile[a][r] = (r0 + r < m) ? Ut[(long long)a * ldu + r0 + r] : (int8_t)0;
  }
  __syncthreads();
  const bool words = ((k & 3) == 0) && ((j0 & 3) == 0) && ((w & 3) == 0) && ((reinterpret_cast<uintptr_t>(B) & 3) == 0);
  if (words) {
    const int wq = w >> 2;
    for (int i = threadIdx.x; i < 64 * wq; i += 256) {
      const int r = i / wq, q = i % wq;
      if (r0 + r >= m) continue;
      const int v = (int)(uint8_t)tile[4 * q][r] | ((int)(uint8_t)tile[4 * q + 1][r] << 8) |
                    ((int)(uint8_t)tile[4 * q + 2][r] << 16) | ((int)(uint8_t)tile[4 * q + 3][r] << 24);
      *reinterpret_cast<int*>(B + (long long)(r0 + r) * k + j0 + 4 * q) = v;
    }
  } else {
    for (int i = threadIdx.x; i < 64 * w; i += 256) {
      const int r = i / w, a = i % w;
      if (r0 + r < m) B[(long long)(r0 + r) * k + j0 + a] = tile[a][r];
    }
  }
}

template <typename T>
__global__ void transpose_kernel(const T* __restrict__ src, long long lds, int rows, int cols, T* __restrict__ dst,
                                 long long ldd) {
  __shared__ T tile[32][33];
  const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
  for (int i = threadIdx.y; i < 32; i += 8) {
    const int r = r0 + i, c = c0 + threadIdx.x;
    if (r < rows && c < cols) tile[i][threadIdx.x] = src[(long long)r * lds + c];
  }
  __syncthreads();
  for (int i = threadIdx.y; i < 32; i += 8) {
    const int c = c0 + i, r = r0 + threadIdx.x;
    if (r < rows && c < cols) dst[(long long)c * ldd + r] = tile[threadIdx.x][i];
  }
}

__global__ void sum_splits_kernel(const float* __restrict__ part, int splits, int w, int L, float* __restrict__ out,
                                  long long ldo) {
  const int a = blockIdx.y;
  const int x = blockIdx.x * blockDim.x + threadIdx.x;
  if (x >= L) return;
  float s = 0.f;
  for (int q = 0; q < splits; ++q) s += part[((long long)q * w + a) * L + x];
  out[(long long)a * ldo + x] = s;
}

}  // namespace

cudaError_t launch_stats(const float* X, int nv, int L, int ldx, Stats st, cudaStream_t s) {
  dim3 grid((unsigned)cdiv(L, kStatChunk), (unsigned)nv);
  stats_kernel<<<grid, kStatChunk, 0, s>>>(X, L, ldx, st);
  return cudaGetLastError();
}

cudaError_t launch_gather(const float* R, int m, int n, const int* J, int w, float* Y, int ldy, Stats st,
                          cudaStream_t s) {
  static int sms = 0;
  if (sms == 0) {
    int dev = 0, v = 0;
    sms = (cudaGetDevice(&dev) == cudaSuccess &&
           cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && v > 0) ? v : 148;
    cudaGetLastError();
  }
  const long long items = (long long)w * cdiv(m, kStatChunk);
  const long long grid = std::max<long long>(1, std::min<long long>(cdiv(items, 8), 2LL * sms));
  gather_stats_kernel<<<(unsigned)grid, 256, 0, s>>>(R, m, n, J, Y, ldy, w, st);
  return cudaGetLastError();
}

namespace {
// the apply grid: P positions per CTA, gx CTAs
void apply_grid(int L, int* P, int* gx) {
  int sms = 152, dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  *P = 64 * (int)std::max<long long>(1, cdiv(L, 64LL * sms));
  *gx = (int)cdiv(L, *P);
}
}  // namespace

void apply_gram_scratch(int L, size_t* part_ints, size_t* groups) {
  int P, gx;
  apply_grid(L, &P, &gx);
  *part_ints = (size_t)gx * 256 * 33;   // PPT <= 33 (128 vectors)
  *groups = (size_t)cdiv(gx, kGramGroup);
}

cudaError_t launch_apply(const float* X, int nv, int L, int ldx, const Thresh& th, int8_t* T, int ldt, int* gram,
                         cudaStream_t s, __half* T16, long long ldt16, __half* Tk, long long ldk, GramScratch gs) {
  if (Tk != nullptr && (ldk < round_up(nv, 8) || (ldk & 7) != 0)) return cudaErrorInvalidValue;
  // one 64-position chunk per CTA up to one CTA per SM, whole chunks per CTA beyond
  int P, gx;
  apply_grid(L, &P, &gx);
  const bool g = gram != nullptr && nv <= 128;   // 256 vectors would need 256 accumulators per thread
  if (g && (gs.part == nullptr || gs.ticket == nullptr)) return cudaErrorInvalidValue;
  // the grouped reduction pays off once the direct atomics (one per pair and CTA) would number ~400K or more
  if ((long long)gx * nv * (nv + 1) / 2 < 400000) gs = GramScratch{};
#define APPLY_LAUNCH(VB)                                                                                 \
  do {                                                                                                   \
    dim3 grid((unsigned)gx, (unsigned)cdiv(nv, VB));                                                     \
    if (g) apply_kernel<VB, true><<<grid, 256, 0, s>>>(X, nv, L, ldx, th, T, ldt, gram, P, T16, ldt16, Tk, ldk,   \
                                                         gs);                                                \
    else apply_kernel<VB, false><<<grid, 256, 0, s>>>(X, nv, L, ldx, th, T, ldt, nullptr, P, T16, ldt16, Tk, ldk, \
                                                      GramScratch{});                                        \
  } while (0)
  if (nv <= 16) APPLY_LAUNCH(16);
  else if (nv <= 32) APPLY_LAUNCH(32);
  else if (nv <= 64) APPLY_LAUNCH(64);
  else if (nv <= 128) APPLY_LAUNCH(128);
  else {
    dim3 grid((unsigned)gx, (unsigned)cdiv(nv, 256));
    apply_kernel<256, false><<<grid, 256, 0, s>>>(X, nv, L, ldx, th, T, ldt, nullptr, P, T16, ldt16, Tk, ldk,
                                                  GramScratch{});
  }
#undef APPLY_LAUNCH
  return cudaGetLastError();
}

__global__ void i8_to_f16_kernel(const int8_t* __restrict__ src, long long lds, int rows, int cols,
                                 __half* __restrict__ dst, long long ldd) {
  const int r = blockIdx.y;
  for (int c = blockIdx.x * blockDim.x + threadIdx.x; c < cols; c += gridDim.x * blockDim.x)
    dst[(long long)r * ldd + c] = __short2half_rn((short)src[(long long)r * lds + c]);
}

cudaError_t launch_i8_to_f16(const int8_t* src, long long lds, int rows, int cols, __half* dst, long long ldd,
                             cudaStream_t s) {
  if (rows < 1 || cols < 1) return cudaSuccess;
  dim3 grid((unsigned)std::min<long long>(64, cdiv(cols, 256)), (unsigned)rows);
  i8_to_f16_kernel<<<grid, 256, 0, s>>>(src, lds, rows, cols, dst, ldd);
  return cudaGetLastError();
}

// e (n floats) is scratch for the column energies.
cudaError_t launch_select_with(const float* colpart, int nrt, int n, const float* h, int w, int* J, float* e,
                               cudaStream_t s) {
  colsum_kernel<<<(unsigned)cdiv(n, 256), 256, 0, s>>>(colpart, nrt, n, h, e);
  cudaError_t err = cudaGetLastError();
  if (err != cudaSuccess) return err;
  select_kernel<<<1, 1024, 0, s>>>(e, n, w, J);
  return cudaGetLastError();
}

cudaError_t launch_norm(const F2* normpart, int count, double* out, const double* norm_a, double* trace,
                        cudaStream_t s, const float* maxpart, float* maxout) {
  norm_kernel<<<1, 1024, 0, s>>>(normpart, count, out, norm_a, trace, maxpart, maxout);
  return cudaGetLastError();
}

cudaError_t launch_absmax(const float* x, long long n, float* out, cudaStream_t s) {
  absmax_kernel<<<1, 1024, 0, s>>>(x, n, out);
  return cudaGetLastError();
}

cudaError_t launch_write_b(const int8_t* Ut, int ldu, int w, int m, int8_t* B, long long k, long long j0,
                           cudaStream_t s, const IoTable* io) {
  write_b_kernel<<<(unsigned)cdiv(m, 64), 256, 0, s>>>(Ut, ldu, w, m, B, k, j0, io);
  return cudaGetLastError();
}

cudaError_t launch_transpose_i8(const int8_t* src, long long lds, int rows, int cols, int8_t* dst, long long ldd,
                                cudaStream_t s) {
  dim3 grid((unsigned)cdiv(cols, 32), (unsigned)cdiv(rows, 32));
  transpose_kernel<int8_t><<<grid, dim3(32, 8), 0, s>>>(src, lds, rows, cols, dst, ldd);
  return cudaGetLastError();
}

cudaError_t launch_transpose_f32(const float* src, long long lds, int rows, int cols, float* dst, long long ldd,
                                 cudaStream_t s) {
  dim3 grid((unsigned)cdiv(cols, 32), (unsigned)cdiv(rows, 32));
  transpose_kernel<float><<<grid, dim3(32, 8), 0, s>>>(src, lds, rows, cols, dst, ldd);
  return cudaGetLastError();
}

cudaError_t launch_sum_splits(const float* part, int splits, int w, int L, float* out, long long ldo, cudaStream_t s) {
  dim3 grid((unsigned)cdiv(L, 256), (unsigned)w);
  sum_splits_kernel<<<grid, 256, 0, s>>>(part, splits, w, L, out, ldo);
  return cudaGetLastError();
}

}  // namespace externd
