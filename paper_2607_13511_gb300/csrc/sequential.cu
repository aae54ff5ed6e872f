// The sequential algorithm (§2.3, block width 1) in one launch: a thread-block cluster keeps the whole residual
// in its shared memory and fits every component without leaving the kernel.
//
// With one component per step the method is a chain of matrix-vector products whose results feed the next
// threshold at once, so its cost is latency, not bandwidth: launched kernel by kernel it pays a launch and a
// global-memory round trip per step. Here the CS CTAs of one cluster (8) each own a slice of RPC consecutive rows
// of R (CTA c: rows c RPC .. c RPC + RPC - 1) in shared memory. Per component, with every cross-CTA sum formed
// through distributed shared memory (each CTA writes its partial, one cluster barrier, every CTA adds the CS
// partials in CTA order -- so every CTA holds the same bits, and the result does not depend on timing):
//   start   column energies h_j ||R_:j||^2 (partial over the own rows, summed over the cluster; their total is
//           ||R||_H^2, the energy after the previous component), j* = the largest (ties to the lower j), and
//           u = T_tau(R[:, j*]) (Eq. 2 over m: the sum of |R_rj*| and the largest entry summed/maxed over CTAs)
//   iters x { v = T_tau(R^T u)   (partial products over the own rows, summed: every CTA holds all of R^T u and
//                                 takes Eq. 2 over n itself, in the same order, so all hold the same v)
//             u = T_tau(R H v)   (own rows only; Eq. 2's sum and largest entry over m from the cluster) }
//   scales  d = u^T R H v / (||u||^2 v^T H v) (Prop. 1), u^T R H v and ||u||^2 summed over the cluster
//   deflate R <- R - d u v^T on the own rows; u, v, d written to B[:, i], C[i, :], D[i]
// With Prop. 2's safeguard, the best single entry of the residual is found (cluster argmax) before each fit and
// takes the component's place when it removes more (u = e_i, v = sgn(R_ij) e_j, d = |R_ij|).
// Eq. 2 is evaluated as everywhere in this library: S = sum |x| in double-float, theta = RD_float(tau S / L),
// keep |x| > theta, and the first entry of largest magnitude (sign +1 if zero) when nothing passes.
#include <cooperative_groups.h>

#include "kernels.h"

namespace externd {
namespace {

namespace cg = cooperative_groups;

constexpr int kSeqCS = 8;          // CTAs per cluster (portable cluster size)
constexpr int kSeqThreads = 256;
constexpr int kSeqWarps = kSeqThreads / 32;

// Scalars one CTA contributes to a cluster reduction: a double-float sum, a key (largest wins) with a value that
// travels with it, three float sums.
struct __align__(16) SeqPart {
  float shi, slo;
  u64 key;
  float a, b, c, kv;
};

struct SeqArgs {
  const float* A;
  const float* h;      // n importances or nullptr
  int m, n, rpc;       // rows, columns, rows per CTA
  long long k;         // components
  int iters;
  double tau;
  int8_t* B;           // m x k
  float* D;            // k
  int8_t* C;           // k x n
  double* trace;       // k energies (device) or nullptr
  double* energy;      // final energy (device)
  long long* activations;   // Prop. 2's safeguard on when not nullptr: the number of components it replaced
};

__device__ __forceinline__ F2 block_sum_f2(F2 v, F2* red) {
  v = warp_sum(v);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  F2 t;
#pragma unroll
  for (int q = 0; q < kSeqWarps; ++q) t = f2_add(t, red[q]);
  return t;
}

// An F2 sum and a maximum key over the CTA in one pass (two barriers).
__device__ __forceinline__ void block_sum_max(F2& s, u64& key, F2* redf, u64* redk) {
  s = warp_sum(s);
  key = warp_max(key);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) {
    redf[warp] = s;
    redk[warp] = key;
  }
  __syncthreads();
  F2 t;
  u64 k = 0;
#pragma unroll
  for (int q = 0; q < kSeqWarps; ++q) {
    t = f2_add(t, redf[q]);
    k = redk[q] > k ? redk[q] : k;
  }
  s = t;
  key = k;
}

__device__ __forceinline__ u64 block_max_key(u64 v, u64* red) {
  v = warp_max(v);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  u64 t = 0;
#pragma unroll
  for (int q = 0; q < kSeqWarps; ++q) t = red[q] > t ? red[q] : t;
  return t;
}

// The largest key of the CTA and the value of the thread that held it (keys are distinct or both zero).
__device__ __forceinline__ u64 block_max_key_val(u64 v, float& val, u64* red, float* redv) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const u64 t = __shfl_xor_sync(0xffffffffu, v, o);
    const float tv = __shfl_xor_sync(0xffffffffu, val, o);
    if (t > v) {
      v = t;
      val = tv;
    }
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) {
    red[warp] = v;
    redv[warp] = val;
  }
  __syncthreads();
  u64 t = 0;
  float tv = 0.f;
#pragma unroll
  for (int q = 0; q < kSeqWarps; ++q)
    if (red[q] > t) {
      t = red[q];
      tv = redv[q];
    }
  val = tv;
  return t;
}

__device__ __forceinline__ int8_t eq2(float x, float theta, bool fallback, bool is_arg) {
  if (fallback) return is_arg ? (x < 0.f ? (int8_t)-1 : (int8_t)1) : (int8_t)0;
  return ternary_of(x, theta);
}

__global__ void __launch_bounds__(kSeqThreads, 1) seq_kernel(const SeqArgs p) {
  extern __shared__ __align__(16) float smem[];
  cg::cluster_group cluster = cg::this_cluster();
  const int c = (int)cluster.block_rank();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int m = p.m, n = p.n, rpc = p.rpc;
  const int r0 = c * rpc, rows = max(0, min(rpc, m - r0));
  // shared memory: R slice, two partial vectors (cluster-read), the full vector x, v, h, u and y of the own rows
  float* Rs = smem;                                 // rpc x n
  float* pv = Rs + (size_t)rpc * n;                 // 2 x n partials (read by the cluster)
  float* x = pv + 2 * (size_t)n;                    // n: the summed vector (R^T u, or the column energies)
  float* vf = x + n;                                // n: v as float
  float* hs = vf + n;                               // n: importances (1 when unweighted)
  float* us = hs + n;                               // rpc: u of the own rows as float
  float* ys = us + rpc;                             // rpc: R H v of the own rows
  __shared__ SeqPart parts[2];                      // scalar partials (read by the cluster)
  __shared__ SeqPart total;                         // their combination
  __shared__ F2 redf[kSeqWarps];
  __shared__ u64 redk[kSeqWarps];
  __shared__ float redv[kSeqWarps];
  __shared__ double norm_a;
  // the double-precision steps (thresholds, the scale, the safeguard's decision) run on thread 0 alone -- this
  // GPU's double-precision rate is a small fraction of its single-precision one -- and reach the CTA through
  // shared memory
  __shared__ float b_th, b_d;
  __shared__ int b_fb, b_arg, b_take;
  auto threshold = [&](F2 S, u64 key, int L) {   // Eq. 2: theta = RD_float(tau S / L), fallback, its index
    if (tid == 0) {
      const float th = __double2float_rd(p.tau * (f2_value(S) / (double)L));
      b_th = th;
      b_fb = !(key_mag(key) > th);
      b_arg = (int)key_index(key);
    }
    __syncthreads();
  };
  int vbuf = 0, sbuf = 0;   // which half of pv / parts the next reduction writes
  const float* rpv[2][kSeqCS];   // the cluster's partial vectors, both halves
#pragma unroll
  for (int q = 0; q < kSeqCS; ++q) {
    rpv[0][q] = cluster.map_shared_rank(pv, q);
    rpv[1][q] = cluster.map_shared_rank(pv + n, q);
  }

  // sum over the cluster of the CTAs' n-vectors pv[vbuf] into x (CTA order)
  auto reduce_vector = [&]() {
    cluster.sync();
    const int n4 = n >> 2;   // 16-byte remote loads where the vector allows (pv rows are 16-byte aligned: n % 4 == 0)
    if ((n & 3) == 0) {
      for (int j = tid; j < n4; j += kSeqThreads) {
        float4 v[kSeqCS];
#pragma unroll
        for (int q = 0; q < kSeqCS; ++q) v[q] = reinterpret_cast<const float4*>(rpv[vbuf][q])[j];
        float4 t = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int q = 0; q < kSeqCS; ++q) {
          t.x += v[q].x;
          t.y += v[q].y;
          t.z += v[q].z;
          t.w += v[q].w;
        }
        reinterpret_cast<float4*>(x)[j] = t;
      }
    } else {
      for (int j = tid; j < n; j += kSeqThreads) {
        float v[kSeqCS];
#pragma unroll
        for (int q = 0; q < kSeqCS; ++q) v[q] = rpv[vbuf][q][j];
        float t = 0.f;
#pragma unroll
        for (int q = 0; q < kSeqCS; ++q) t += v[q];
        x[j] = t;
      }
    }
    vbuf ^= 1;
    __syncthreads();
  };
  // the cluster's combination of the CTAs' scalar partials (sums in CTA order, maximum key)
  auto reduce_scalars = [&](SeqPart mine) -> SeqPart {
    if (tid == 0) parts[sbuf] = mine;
    cluster.sync();
    if (warp == 0) {   // one warp reads the cluster's parts (lane q part q) and combines them in CTA order
      SeqPart o{};
      if (lane < kSeqCS) o = *cluster.map_shared_rank(&parts[sbuf], lane);
      SeqPart t;
      F2 s;
      t.key = 0;
      t.a = t.b = t.c = t.kv = 0.f;
#pragma unroll
      for (int q = 0; q < kSeqCS; ++q) {
        F2 f;
        f.hi = __shfl_sync(0xffffffffu, o.shi, q);
        f.lo = __shfl_sync(0xffffffffu, o.slo, q);
        s = f2_add(s, f);
        const u64 kq = __shfl_sync(0xffffffffu, o.key, q);
        const float vq = __shfl_sync(0xffffffffu, o.kv, q);
        if (kq > t.key) {
          t.key = kq;
          t.kv = vq;
        }
        t.a += __shfl_sync(0xffffffffu, o.a, q);
        t.b += __shfl_sync(0xffffffffu, o.b, q);
        t.c += __shfl_sync(0xffffffffu, o.c, q);
      }
      t.shi = s.hi;
      t.slo = s.lo;
      if (lane == 0) total = t;
    }
    __syncthreads();
    const SeqPart t = total;
    sbuf ^= 1;
    return t;
  };

  // load the own rows of A, the importances; ||A||_H^2 through the first column-energy reduction
  for (int i = tid; i < rows * n; i += kSeqThreads) Rs[i] = p.A[(size_t)r0 * n + i];
  for (int i = tid; i < (rpc - rows) * n; i += kSeqThreads) Rs[(size_t)rows * n + i] = 0.f;
  for (int j = tid; j < n; j += kSeqThreads) hs[j] = p.h != nullptr ? p.h[j] : 1.f;
  __syncthreads();

  auto column_energies = [&]() {   // x[j] = h_j sum_r R_rj^2 over the cluster; returns sum_j x[j] (F2)
    float* part = pv + (size_t)vbuf * n;
    for (int j = tid; j < n; j += kSeqThreads) {
      float s = 0.f;
      for (int r = 0; r < rows; ++r) {
        const float v = Rs[(size_t)r * n + j];
        s = fmaf(v, v, s);
      }
      part[j] = s;
    }
    reduce_vector();
    F2 tot;
    for (int j = tid; j < n; j += kSeqThreads) {
      x[j] *= hs[j];
      tot = f2_add(tot, x[j]);
    }
    __syncthreads();
    return block_sum_f2(tot, redf);
  };

  {
    const F2 a = column_energies();
    if (tid == 0) norm_a = f2_value(a);
  }
  __syncthreads();

  for (long long comp = 0; comp < p.k; ++comp) {
    // ---- Prop. 2: the best single entry of the residual this component is fitted to, by h_j R_ij^2 (|R_ij|
    // unweighted: the same order without rounding), ties to the lower row-major index
    u64 ekey = 0;
    float eval = 0.f;
    if (p.activations != nullptr) {
      for (int i = tid; i < rows * n; i += kSeqThreads) {
        const int j = i % n;
        const float v = Rs[i];
        const float sc = p.h != nullptr ? hs[j] * v * v : fabsf(v);
        const u64 key = ((u64)__float_as_uint(sc) << 32) | (u64)(0xffffffffu - (uint32_t)((size_t)r0 * n + i));
        if (key > ekey) {
          ekey = key;
          eval = v;
        }
      }
      ekey = block_max_key_val(ekey, eval, redk, redv);
      SeqPart mine{0.f, 0.f, ekey, 0.f, 0.f, 0.f, eval};
      const SeqPart tot = reduce_scalars(mine);
      ekey = tot.key;
      eval = tot.kv;
    }
    // ---- start: the column of largest energy (x holds the column energies), u = T_tau(R[:, j*])
    u64 kbest = 0;
    for (int j = tid; j < n; j += kSeqThreads) kbest = max(kbest, mag_key(x[j], (uint32_t)j));
    const int jstar = (int)key_index(block_max_key(kbest, redk));
    {
      F2 s;
      u64 key = 0;
      for (int r = tid; r < rows; r += kSeqThreads) {
        const float v = Rs[(size_t)r * n + jstar];
        s = f2_add(s, fabsf(v));
        key = max(key, mag_key(v, (uint32_t)(r0 + r)));
      }
      block_sum_max(s, key, redf, redk);
      SeqPart mine{s.hi, s.lo, key, 0.f, 0.f, 0.f, 0.f};
      const SeqPart tot = reduce_scalars(mine);
      F2 st;
      st.hi = tot.shi;
      st.lo = tot.slo;
      threshold(st, tot.key, m);
      const float th = b_th;
      const bool fb = b_fb != 0;
      const int arg = b_arg;
      for (int r = tid; r < rpc; r += kSeqThreads)
        us[r] = r < rows ? (float)eq2(Rs[(size_t)r * n + jstar], th, fb, r0 + r == arg) : 0.f;
      __syncthreads();
    }
    float d = 0.f;
    for (int it = 0; it < p.iters; ++it) {
      // ---- V-step: v = T_tau(R^T u), plain R (§2.5)
      {
        float* part = pv + (size_t)vbuf * n;
        for (int j = tid; j < n; j += kSeqThreads) {
          float s = 0.f;
          for (int r = 0; r < rows; ++r) s = fmaf(us[r], Rs[(size_t)r * n + j], s);
          part[j] = s;
        }
        reduce_vector();
        F2 s;
        u64 key = 0;
        for (int j = tid; j < n; j += kSeqThreads) {
          s = f2_add(s, fabsf(x[j]));
          key = max(key, mag_key(x[j], (uint32_t)j));
        }
        block_sum_max(s, key, redf, redk);
        threshold(s, key, n);
        const float th = b_th;
        const bool fb = b_fb != 0;
        const int arg = b_arg;
        for (int j = tid; j < n; j += kSeqThreads) vf[j] = (float)eq2(x[j], th, fb, j == arg);
        __syncthreads();
      }
      // ---- U-step: u = T_tau(R H v), the own rows (one warp per row)
      {
        for (int r = warp; r < rpc; r += kSeqWarps) {
          float s = 0.f;
          if (r < rows)
            for (int j = lane; j < n; j += 32) s = fmaf(Rs[(size_t)r * n + j], hs[j] * vf[j], s);
          s = warp_sum(s);
          if (lane == 0) ys[r] = s;
        }
        __syncthreads();
        F2 s;
        u64 key = 0;
        for (int r = tid; r < rows; r += kSeqThreads) {
          s = f2_add(s, fabsf(ys[r]));
          key = max(key, mag_key(ys[r], (uint32_t)(r0 + r)));
        }
        block_sum_max(s, key, redf, redk);
        SeqPart mine{s.hi, s.lo, key, 0.f, 0.f, 0.f, 0.f};
        const SeqPart tot = reduce_scalars(mine);
        F2 st;
        st.hi = tot.shi;
        st.lo = tot.slo;
        threshold(st, tot.key, m);
        const float th = b_th;
        const bool fb = b_fb != 0;
        const int arg = b_arg;
        for (int r = tid; r < rpc; r += kSeqThreads)
          us[r] = r < rows ? (float)eq2(ys[r], th, fb, r0 + r == arg) : 0.f;
        __syncthreads();
      }
    }
    // ---- scales (Prop. 1): d = u^T (R H v) / (||u||^2 v^T H v), with R H v from the last U-step
    {
      F2 ru, nu2;
      for (int r = tid; r < rows; r += kSeqThreads) {
        ru = f2_add(ru, us[r] * ys[r]);
        nu2 = f2_add(nu2, us[r] * us[r]);
      }
      ru = block_sum_f2(ru, redf);
      const float nu = block_sum_f2(nu2, redf).hi;   // a small integer: exact
      F2 hv;
      for (int j = tid; j < n; j += kSeqThreads) hv = f2_add(hv, hs[j] * vf[j] * vf[j]);
      hv = block_sum_f2(hv, redf);
      SeqPart mine{ru.hi, ru.lo, 0, nu, 0.f, 0.f, 0.f};
      const SeqPart tot = reduce_scalars(mine);
      const uint32_t idx = 0xffffffffu - (uint32_t)(ekey & 0xffffffffu);
      const int ei = (int)(idx / (uint32_t)n), ej = (int)(idx % (uint32_t)n);
      if (tid == 0) {
        F2 rt;
        rt.hi = tot.shi;
        rt.lo = tot.slo;
        const double den = (double)tot.a * f2_value(hv);
        const float dd = den > 0.0 ? (float)(f2_value(rt) / den) : 0.f;
        b_d = dd;
        b_take = 0;
        if (p.activations != nullptr) {
          // the component removes 2 r d - d K d (K = ||u||^2 v^T H v), the pair h_j R_ij^2: the larger one stays
          const float rf = (float)f2_value(rt), Kf = (float)den;
          const double dec = 2.0 * (double)rf * (double)dd - (double)dd * (double)Kf * (double)dd;
          const double single = (p.h != nullptr ? (double)hs[ej] : 1.0) * (double)eval * (double)eval;
          b_take = single > dec ? 1 : 0;
        }
      }
      __syncthreads();
      d = b_d;
      if (p.activations != nullptr) {
        if (b_take) {
          d = fabsf(eval);
          for (int r = tid; r < rpc; r += kSeqThreads) us[r] = (r0 + r == ei) ? 1.f : 0.f;
          for (int j = tid; j < n; j += kSeqThreads) vf[j] = (j == ej) ? (eval < 0.f ? -1.f : 1.f) : 0.f;
          if (c == 0 && tid == 0) *p.activations += 1;
        }
        __syncthreads();
      }
    }
    // ---- deflate the own rows, write the component
    for (int r = 0; r < rows; ++r) {
      const float du = -d * us[r];
      float* row = Rs + (size_t)r * n;
      for (int j = tid; j < n; j += kSeqThreads) row[j] = fmaf(du, vf[j], row[j]);
    }
    for (int r = tid; r < rows; r += kSeqThreads) p.B[(size_t)(r0 + r) * p.k + comp] = (int8_t)us[r];
    if (c == 0) {
      for (int j = tid; j < n; j += kSeqThreads) p.C[(size_t)comp * n + j] = (int8_t)vf[j];
      if (tid == 0) p.D[comp] = d;
    }
    __syncthreads();
    // ---- the next start's column energies; their total is the energy after this component
    const F2 e = column_energies();
    if (c == 0 && tid == 0) {
      const double en = 1.0 - f2_value(e) / norm_a;
      if (p.trace != nullptr) p.trace[comp] = en;
      if (comp == p.k - 1) *p.energy = en;
    }
  }
  cluster.sync();   // no CTA leaves while another may still read its shared memory
}

size_t seq_smem(int rpc, int n) { return ((size_t)rpc * n + 5 * (size_t)n + 2 * (size_t)rpc) * sizeof(float); }

}  // namespace

bool sequential_cluster_fits(long long m, long long n) {
  if (m < 1 || n < 1 || n > 4096 || m > 65536 || m * n >= (1LL << 32)) return false;
  const long long rpc = cdiv(m, kSeqCS);
  return seq_smem((int)rpc, (int)n) <= 200 * 1024;
}

cudaError_t launch_sequential_cluster(const float* A, int m, int n, long long k, int iters, double tau, const float* h,
                                      int8_t* B, float* D, int8_t* C, double* trace, double* energy,
                                      long long* activations, cudaStream_t s) {
  if (!sequential_cluster_fits(m, n)) return cudaErrorInvalidValue;
  const int rpc = (int)cdiv(m, kSeqCS);
  const size_t smem = seq_smem(rpc, n);
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(seq_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  SeqArgs a{A, h, m, n, rpc, k, iters, tau, B, D, C, trace, energy, activations};
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kSeqCS, 1, 1);
  cfg.blockDim = dim3(kSeqThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = kSeqCS;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, seq_kernel, a);
}

}  // namespace externd
