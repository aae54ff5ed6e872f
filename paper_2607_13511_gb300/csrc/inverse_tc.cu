// (G + eps I)^-1 of Eq. 3 and the Eq. 4 solve on the 5th-generation tensor cores, for blocks of 65 to 128
// components.
//
// The symmetric sweep of inv_kernel (Gauss-Jordan on an SPD matrix without pivoting, pivot blocks K of 16),
// with the 128 x 128 float32 matrix S in tensor memory (row i in lane i) instead of registers. Per step s, with
// the pivot rows Rk = S[K,:] and Q = S[K,K]^-1 in shared memory:
//   1. W = Q Rk (16 x 128) on the CUDA cores, thread j computing column j; the MMA operands A = -Rk^T and B = W,
//      split into tf32 hi + lo parts;
//   2. S[i][j] -= sum_d Rk[d][i] W[d][j] for all i, j as ONE 128 x 128 x 16 MMA of kind::tf32 (hi.hi + hi.lo +
//      lo.hi, about 22 significant bits per product, float32 accumulation in tensor memory). Meanwhile the
//      rows of the next pivot block are updated in float32 on the CUDA cores (the same fma chains as inv_kernel)
//      and the pivot warp inverts the next pivot block (warp_sweep), so neither waits for the MMA;
//   3. once the MMA is done the pivot rows and columns take their exact sweep values (column K_d of row i is
//      W[d][i] = (S[i,K] Q)_d, row K_d is W[d][.] and -Q[d][.] on the pivot block: the warp of K's lane quadrant
//      reads its 32 lanes back and rewrites them), and the rows two blocks ahead are read from tensor memory.
// After the last step S = -(G + eps I)^-1. The tensor-memory copies of a pivot block's rows before its own step
// are never used (the step rewrites them), so the pivot blocks and their inverses are float32-exact as in
// inv_kernel; the rest of S carries the MMA's ~22-bit products. Every wait on the MMA is bounded (2 s, then the
// error word and an early exit).
#include <cuda_fp16.h>

#include <cstdlib>
#include <cstring>

#include "kernels.h"
#include "sweep.cuh"
#include "umma.cuh"

namespace externd {

namespace {

constexpr int kTiN = 128;        // matrix side in tensor memory (padded with the identity)
constexpr int kTiNB = 16;        // pivot block
constexpr int kTiRows = 128;     // row threads (warps 0-3, thread i = lane i)
constexpr int kTiThreads = 192;  // + warp 4 (tensor memory, MMA issue) + warp 5 (pivot warp)
// shared memory: the MMA operands A hi, A lo, B hi, B lo (K-major, 128-byte swizzle, 128 rows of which 64 B are
// used), over which the Gram is staged first (rows of kTiP floats, 16-byte aligned: a row read as float4 runs and
// a column read as scalars both spread over all banks); then W (16 x 128), the current and next pivot rows, the
// rows two blocks ahead, Q and its transpose (two buffers each), and with MODE 1 the staged G_V.
constexpr int kTiP = 132;
constexpr uint32_t kTiOp = 16384;
constexpr uint32_t kTiStage = (uint32_t)kTiN * kTiP * 4;   // 67,584 B >= the operands' 65,536 B
constexpr uint32_t kTiRowBlk = kTiNB * kTiN * 4;           // 16 rows of 128 floats
constexpr uint32_t kTiWs = kTiStage, kTiRkA = kTiWs + kTiRowBlk, kTiRkB = kTiRkA + kTiRowBlk,
                   kTiRn = kTiRkB + kTiRowBlk, kTiQ = kTiRn + kTiRowBlk, kTiQt = kTiQ + 2 * kTiNB * kTiNB * 4,
                   kTiGV = kTiQt + 2 * kTiNB * kTiNB * 4;
constexpr size_t tc_inv_smem(int mode) { return 1024 + kTiGV + (mode == 1 ? kTiStage : 0); }

__device__ __forceinline__ void cp_async4(uint32_t dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}

// Instruction descriptor of kind::tf32: tf32 A and B, fp32 D, both K-major, M x N.
__host__ __device__ constexpr uint32_t tf32_idesc(uint32_t M, uint32_t N) {
  return (1u << 4) | (2u << 7) | (2u << 10) | ((N >> 3) << 17) | ((M >> 4) << 24);
}

__device__ __forceinline__ void mma_tf32(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, 1, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc)
      : "memory");
}

__device__ __forceinline__ uint32_t to_tf32(float x) {
  uint32_t r;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
  return r;
}

// hi + lo tf32 parts of x: hi rounds x to tf32, lo = x - hi (exact in float32) rounded to tf32 as well.
__device__ __forceinline__ void split_tf32(float x, uint32_t& hi, uint32_t& lo) {
  hi = to_tf32(x);
  lo = to_tf32(x - __uint_as_float(hi));
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&v)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(
          taddr),
      "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]), "r"(v[9]),
      "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
      : "memory");
}

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}

__device__ __forceinline__ void bar_rows() { asm volatile("bar.sync 2, 128;" ::: "memory"); }

// Row r of a 16-wide tf32 operand (hi at base, lo at base + kTiOp): the four 16-byte chunks of its first 64 bytes
// in the 128-byte swizzle.
__device__ __forceinline__ void store_operand_row(uint32_t base, int r, const float (&v)[kTiNB]) {
  const uint32_t row = (uint32_t)(r >> 3) * 1024u + (uint32_t)(r & 7) * 128u;
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    uint32_t h[4], l[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) split_tf32(v[4 * c + e], h[e], l[e]);
    const uint32_t off = row + ((uint32_t)(c ^ (r & 7)) << 4);
    st_shared_v4(base + off, h[0], h[1], h[2], h[3]);
    st_shared_v4(base + kTiOp + off, l[0], l[1], l[2], l[3]);
  }
}

// MODE 0: Ginv (out, w x w, when op is null) or its tensor-core operand image (op: hi / lo fp16 K-major, 128-byte
// swizzle, Ginv * 2^sg, then sg). MODE 1 (Eq. 4): K = G_U .* GVraw, out = d = K^-1 r. Graw (optional) receives G
// or K before the ridge. IN_INT: the Gram is the integer upper triangle Gint (reset to zero after reading), else
// the sum of `splits` float partials.
template <int MODE, bool IN_INT>
__global__ void __launch_bounds__(kTiThreads, 1) inv_tc_kernel(const float* __restrict__ Gpart, int splits, int w,
                                                              const float* __restrict__ GVraw,
                                                              const float* __restrict__ r, float* __restrict__ Graw,
                                                              float* __restrict__ out, int* Gint,
                                                              uint8_t* __restrict__ op, unsigned* err) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t sbase = (raw + 1023u) & ~1023u;
  uint8_t* const gbase = smem_raw + (sbase - raw);
  const uint32_t opA = sbase, opB = sbase + 2 * kTiOp;
  uint32_t* const Gs = reinterpret_cast<uint32_t*>(gbase);                 // staged Gram, rows of kTiP
  const float* const GVs = reinterpret_cast<const float*>(gbase + kTiGV);  // staged G_V (MODE 1)
  float* const Ws = reinterpret_cast<float*>(gbase + kTiWs);               // [16][128]
  float* RkA = reinterpret_cast<float*>(gbase + kTiRkA);                   // pivot rows of this step
  float* RkB = reinterpret_cast<float*>(gbase + kTiRkB);                   // pivot rows of the next step
  float* const Rn = reinterpret_cast<float*>(gbase + kTiRn);               // rows two blocks ahead
  float* const Qb = reinterpret_cast<float*>(gbase + kTiQ);                // [2][16][16]
  float* const Qtb = reinterpret_cast<float*>(gbase + kTiQt);              // [2][16][16], transposed
  __shared__ uint64_t mma_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ float red[4];

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const bool row_thread = tid < kTiRows;
  const int i = tid;   // the row (and tensor-memory lane) of a row thread
  if (warp == 4) {
    tmem_alloc(smem_addr(&tmem_slot), (uint32_t)kTiN);
    tmem_relinquish();
    if (lane == 0) {
      mbar_init(smem_addr(&mma_bar), 1);
      fence_barrier_init();
    }
  }
  // ---- stage the Gram (the integer upper triangle, or the float partials) and, for Eq. 4, G_V
  auto stage = [&](uint32_t* dst, const uint32_t* src) {
    // 16-byte copies where every row starts on a 16-byte boundary in global memory, else 4-byte ones
    if ((w & 3) == 0 && (reinterpret_cast<uintptr_t>(src) & 15) == 0) {
      const int q4 = w >> 2;
      for (int a = warp; a < w; a += kTiThreads / 32)
        for (int c = lane; c < q4; c += 32) cp_async16(smem_addr(dst + a * kTiP + 4 * c), src + (long long)a * w + 4 * c);
    } else {
      for (int a = warp; a < w; a += kTiThreads / 32)
        for (int b = lane; b < w; b += 32) cp_async4(smem_addr(dst + a * kTiP + b), src + (long long)a * w + b);
    }
  };
  if (IN_INT || splits == 1) {
    stage(Gs, IN_INT ? reinterpret_cast<const uint32_t*>(Gint) : reinterpret_cast<const uint32_t*>(Gpart));
  } else {
    for (int a = warp; a < w; a += kTiThreads / 32)
      for (int b = lane; b < w; b += 32) {
        float g = 0.f;
        for (int sp = 0; sp < splits; ++sp) g += Gpart[(long long)sp * w * w + (long long)a * w + b];
        Gs[a * kTiP + b] = __float_as_uint(g);
      }
  }
  if (MODE == 1) stage(reinterpret_cast<uint32_t*>(gbase + kTiGV), reinterpret_cast<const uint32_t*>(GVraw));
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
  __syncthreads();
  if (IN_INT) {
    // the lower triangle from the upper one, as float; then the Gram can be reset for the next accumulation
    for (int a = warp; a < w; a += kTiThreads / 32)
      for (int b = lane; b < w; b += 32) {
        const uint32_t g = Gs[min(a, b) * kTiP + max(a, b)];
        if (b < a) Gs[a * kTiP + b] = __float_as_uint((float)(int)g);
      }
    __syncthreads();
    for (int a = warp; a < w; a += kTiThreads / 32)
      for (int b = lane; b <= a; b += 32) Gs[b * kTiP + a] = __float_as_uint((float)(int)Gs[b * kTiP + a]);
    for (int idx = tid; idx < w * w; idx += kTiThreads) Gint[idx] = 0;
    __syncthreads();
  }
  if (MODE == 1) {   // K = G_U .* G_V
    for (int a = warp; a < w; a += kTiThreads / 32)
      for (int b = lane; b < w; b += 32) {
        float* g = reinterpret_cast<float*>(Gs + a * kTiP + b);
        *g *= GVs[a * kTiP + b];
      }
    __syncthreads();
  }
  const float* const Gf = reinterpret_cast<const float*>(Gs);
  if (Graw != nullptr) {   // G (or K) before the ridge
    for (int a = warp; a < w; a += kTiThreads / 32)
      for (int b = lane; b < w; b += 32) Graw[(long long)a * w + b] = Gf[a * kTiP + b];
  }
  if (row_thread) {
    const float sd = warp_sum(i < w ? Gf[i * kTiP + i] : 0.f);
    if (lane == 0) red[warp] = sd;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_slot;
  const uint32_t trow = tmem + ((uint32_t)(32 * (warp & 3)) << 16);   // this warp's lane quadrant
  const float eps = ((MODE == 0) || (w > 1)) ? (float)kEpsRel * (red[0] + red[1] + red[2] + red[3]) / (float)w : 0.f;

  // ---- S = G + eps I (identity on the padding) into tensor memory; rows 0..15 to RkA, rows 16..31 to Rn
  if (row_thread) {
#pragma unroll 1
    for (int c = 0; c < kTiN / 16; ++c) {
      uint32_t v[16];
#pragma unroll
      for (int e4 = 0; e4 < 4; ++e4) {
        const int j = 16 * c + 4 * e4;
        float4 g = make_float4(0.f, 0.f, 0.f, 0.f);
        if (i < w) g = *reinterpret_cast<const float4*>(Gf + i * kTiP + j);   // columns >= w are masked below
        const float gv[4] = {g.x, g.y, g.z, g.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          float x = (i < w && j + e < w) ? gv[e] : 0.f;
          if (i == j + e) x = i < w ? x + eps : 1.f;
          v[4 * e4 + e] = __float_as_uint(x);
        }
      }
      if (i < kTiNB) {
#pragma unroll
        for (int e = 0; e < 16; ++e) RkA[i * kTiN + 16 * c + e] = __uint_as_float(v[e]);
      } else if (i < 2 * kTiNB) {
#pragma unroll
        for (int e = 0; e < 16; ++e) Rn[(i - kTiNB) * kTiN + 16 * c + e] = __uint_as_float(v[e]);
      }
      tmem_st16(trow + (uint32_t)(16 * c), v);
    }
    tmem_wait_st();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const int pr = lane / 2, pc = (lane % 2) * 8;   // pivot warp: its 8 entries of the 16 x 16 block
  auto sweep_block = [&](const float* rows, int col0, int buf) {   // Q of rows[.][col0 .. col0 + 15]
    float A[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) A[e] = rows[pr * kTiN + col0 + pc + e];
    warp_sweep<kTiNB>(A, lane);
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      Qb[buf * 256 + pr * kTiNB + pc + e] = -A[e];
      Qtb[buf * 256 + (pc + e) * kTiNB + pr] = -A[e];
    }
  };
  if (warp == 5) sweep_block(RkA, 0, 0);
  __syncthreads();

  constexpr uint32_t idesc = tf32_idesc(kTiN, kTiN);
  bool ok = true;
  int step = 0;
  for (int k0 = 0; k0 < w; k0 += kTiNB, ++step) {
    const int kn = k0 + kTiNB, kn2 = kn + kTiNB, qK = k0 >> 5, cur = step & 1;
    const bool has_next = kn < w, has_next2 = kn2 < w;
    const float* const Q = Qb + cur * 256;
    const float* const Qt = Qtb + cur * 256;
    float wj[kTiNB];   // row threads: W[.][i]
    // 1. W = Q Rk, column i per row thread (fma chains over e in order, as inv_kernel); the MMA operands
    if (row_thread) {
      float rk[kTiNB];
#pragma unroll
      for (int e = 0; e < kTiNB; ++e) rk[e] = RkA[e * kTiN + i];
#pragma unroll
      for (int d = 0; d < kTiNB; ++d) wj[d] = 0.f;
#pragma unroll
      for (int e = 0; e < kTiNB; ++e) {
        const float4* qc = reinterpret_cast<const float4*>(Qt + e * kTiNB);   // Q[.][e]
#pragma unroll
        for (int d4 = 0; d4 < kTiNB / 4; ++d4) {
          const float4 q = qc[d4];
          wj[4 * d4] = fmaf(q.x, rk[e], wj[4 * d4]);
          wj[4 * d4 + 1] = fmaf(q.y, rk[e], wj[4 * d4 + 1]);
          wj[4 * d4 + 2] = fmaf(q.z, rk[e], wj[4 * d4 + 2]);
          wj[4 * d4 + 3] = fmaf(q.w, rk[e], wj[4 * d4 + 3]);
        }
      }
#pragma unroll
      for (int d = 0; d < kTiNB; ++d) Ws[d * kTiN + i] = wj[d];
      float na[kTiNB];
#pragma unroll
      for (int e = 0; e < kTiNB; ++e) na[e] = -rk[e];
      store_operand_row(opA, i, na);
      store_operand_row(opB, i, wj);
      fence_async_shared();
    }
    tc_fence_before();
    __syncthreads();
    // 2. the rank-16 update on the tensor cores; meanwhile the next pivot rows in float32
    if (warp == 4 && lane == 0) {
      tc_fence_after();
#pragma unroll
      for (int kk = 0; kk < 2; ++kk) {
        const uint64_t ah = sw128_desc(opA + 32u * kk), al = sw128_desc(opA + kTiOp + 32u * kk);
        const uint64_t bh = sw128_desc(opB + 32u * kk), bl = sw128_desc(opB + kTiOp + 32u * kk);
        mma_tf32(tmem, ah, bh, idesc);
        mma_tf32(tmem, ah, bl, idesc);
        mma_tf32(tmem, al, bh, idesc);
      }
      mma_commit(smem_addr(&mma_bar));
    }
    const bool inK = i >= k0 && i < kn;
    if (row_thread && has_next) {
      // rows kn + e after this step: column j in K is W[j - k0][kn + e] (written by thread kn + e), any other
      // column S[kn + e][j] - sum_d Rk[d][kn + e] W[d][j]
      if (!inK) {
#pragma unroll 4
        for (int e = 0; e < kTiNB; ++e) {
          float acc = Rn[e * kTiN + i];
#pragma unroll
          for (int d = 0; d < kTiNB; ++d) acc = fmaf(-RkA[d * kTiN + kn + e], wj[d], acc);
          RkB[e * kTiN + i] = acc;
        }
      }
      if (i >= kn && i < kn2) {
#pragma unroll
        for (int d = 0; d < kTiNB; ++d) RkB[(i - kn) * kTiN + k0 + d] = wj[d];
      }
    }
    __syncthreads();
    // 3. pivot warp: the next pivot block's inverse. Row threads: the exact pivot rows and columns once the MMA
    //    is done, and the rows two blocks ahead
    if (warp == 5 && has_next) sweep_block(RkB, kn, cur ^ 1);
    if (row_thread) {
      ok = mbar_wait(smem_addr(&mma_bar), (uint32_t)(step & 1), err);
      tc_fence_after();
      if (ok) {
        const int dK = i - k0;
        uint32_t colK[16];   // columns K: W[.][i], or -Q on the pivot block
#pragma unroll
        for (int e = 0; e < 16; ++e) colK[e] = __float_as_uint(inK ? -Q[dK * kTiNB + e] : wj[e]);
        tmem_st16(trow + (uint32_t)k0, colK);
        const bool aheadHere = has_next2 && (kn2 >> 5) == warp;
        if (warp == qK || aheadHere) {
          uint32_t v[kTiN / 16][16];
#pragma unroll
          for (int c = 0; c < kTiN / 16; ++c)
            if (16 * c != k0) tmem_ld16(trow + (uint32_t)(16 * c), v[c]);
          tmem_wait_ld();
          if (warp == qK) {
#pragma unroll
            for (int c = 0; c < kTiN / 16; ++c) {
              if (16 * c == k0) continue;
              if (inK) {
#pragma unroll
                for (int e = 0; e < 16; ++e) v[c][e] = __float_as_uint(Ws[dK * kTiN + 16 * c + e]);
              }
              tmem_st16(trow + (uint32_t)(16 * c), v[c]);
            }
          } else if (i >= kn2 && i < kn2 + kTiNB) {
#pragma unroll
            for (int c = 0; c < kTiN / 16; ++c) {
#pragma unroll
              for (int e = 0; e < 16; ++e)
                Rn[(i - kn2) * kTiN + 16 * c + e] = 16 * c == k0 ? wj[e] : __uint_as_float(v[c][e]);
            }
          }
        }
        tmem_wait_st();
      }
    }
    tc_fence_before();
    ok = __syncthreads_and(ok) != 0;
    tc_fence_after();
    if (!ok) break;
    float* const t = RkA;
    RkA = RkB;
    RkB = t;
  }

  // ---- outputs from -S, row i per row thread (all 128 columns read at once)
  if (ok && row_thread) {
    uint32_t v[kTiN / 16][16];
#pragma unroll
    for (int c = 0; c < kTiN / 16; ++c) tmem_ld16(trow + (uint32_t)(16 * c), v[c]);
    tmem_wait_ld();
    if (MODE == 0 && op != nullptr) {
      float mx = 0.f;
#pragma unroll
      for (int c = 0; c < kTiN / 16; ++c)
#pragma unroll
        for (int e = 0; e < 16; ++e)
          if (i < w && 16 * c + e < w) mx = fmaxf(mx, fabsf(__uint_as_float(v[c][e])));
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      if (lane == 0) red[warp] = mx;
      bar_rows();
      mx = fmaxf(fmaxf(red[0], red[1]), fmaxf(red[2], red[3]));
      const int sg = fp16_scale_exp(mx);
      const float sc = ldexpf(1.f, sg);
      // row i: the 16-byte chunk of columns k .. k + 7 (k = 0, 8, ..., 120) at k_major_offset(128, i, k)
#pragma unroll
      for (int c = 0; c < kTiN / 16; ++c) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int k = 16 * c + 8 * h;
          uint32_t hi[4], lo[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            __half h0, l0, h1, l1;
            const int j0 = k + 2 * e, j1 = j0 + 1;
            split_f16((i < w && j0 < w) ? -__uint_as_float(v[c][8 * h + 2 * e]) * sc : 0.f, h0, l0);
            split_f16((i < w && j1 < w) ? -__uint_as_float(v[c][8 * h + 2 * e + 1]) * sc : 0.f, h1, l1);
            hi[e] = (uint32_t)__half_as_ushort(h0) | ((uint32_t)__half_as_ushort(h1) << 16);
            lo[e] = (uint32_t)__half_as_ushort(l0) | ((uint32_t)__half_as_ushort(l1) << 16);
          }
          const uint32_t off = k_major_offset(128u, (uint32_t)i, (uint32_t)k);
          *reinterpret_cast<uint4*>(op + off) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
          *reinterpret_cast<uint4*>(op + 2 * 16384u + off) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
        }
      }
      if (i == 0) *reinterpret_cast<int*>(op + 4 * 16384u) = sg;
    } else if (MODE == 0) {
#pragma unroll
      for (int c = 0; c < kTiN / 16; ++c)
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          const int j = 16 * c + e;
          if (i < w && j < w) out[(long long)i * w + j] = -__uint_as_float(v[c][e]);
        }
    } else {
      F2 acc;
#pragma unroll
      for (int c = 0; c < kTiN / 16; ++c)
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          const int j = 16 * c + e;
          if (j < w) acc = f2_add(acc, -__uint_as_float(v[c][e]) * r[j]);
        }
      if (i < w) out[i] = acc.hi + acc.lo;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 4) {
    tc_fence_after();
    tmem_dealloc(tmem, (uint32_t)kTiN);
  }
}

template <int MODE, bool IN_INT>
cudaError_t launch_tc(const float* Gpart, int splits, int w, const float* GVraw, const float* r, float* Graw,
                      float* out, int* Gint, uint8_t* op, unsigned* err, cudaStream_t s) {
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(inv_tc_kernel<MODE, IN_INT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)tc_inv_smem(MODE));
    if (e != cudaSuccess) return e;
    configured = true;
  }
  inv_tc_kernel<MODE, IN_INT><<<1, kTiThreads, tc_inv_smem(MODE), s>>>(Gpart, splits, w, GVraw, r, Graw, out, Gint, op, err);
  return cudaGetLastError();
}

}  // namespace

// Off unless EXTERND_TCINV=1: on GB300 the register-tiled sweep is faster (28-31 us against ~42 us alone and
// ~55 us in the graph at w = 128). A clock64 timeline of one launch: the MMA is hidden (its wait takes ~200
// cycles), but each step still spends ~1,400 cycles on W and the operand splits, ~2,500 on the next pivot rows
// and ~2,500 on rewriting the pivot rows beside the next sweep, all on four latency-bound warps, and the
// prologue (Gram staging and mirror, tensor-memory fill, first sweep) ~23,000 cycles.
bool inverse_tc_enabled(int w) {
  static const bool enabled = [] {
    const char* e = std::getenv("EXTERND_TCINV");
    return e && std::strcmp(e, "1") == 0;
  }();
  return enabled && w > 64 && w <= 128;
}

cudaError_t launch_inverse_tc(const float* Gpart, int splits, int w, float* Graw, float* Ginv, cudaStream_t s,
                              void* op, unsigned* err) {
  return launch_tc<0, false>(Gpart, splits, w, nullptr, nullptr, Graw, Ginv, nullptr, static_cast<uint8_t*>(op),
                             err, s);
}

cudaError_t launch_inverse_tc_int(int* Gint, int w, float* Graw, float* Ginv, cudaStream_t s, void* op,
                                  unsigned* err) {
  return launch_tc<0, true>(nullptr, 0, w, nullptr, nullptr, Graw, Ginv, Gint, static_cast<uint8_t*>(op), err, s);
}

cudaError_t launch_scales_tc_int(int* GUint, const float* GVraw, const float* r, int w, float* d, cudaStream_t s,
                                 float* K, unsigned* err) {
  return launch_tc<1, true>(nullptr, 0, w, GVraw, r, K, d, GUint, nullptr, err, s);
}

cudaError_t launch_scales_tc(const float* GUpart, int splits, const float* GVraw, const float* r, int w, float* d,
                             cudaStream_t s, float* K, unsigned* err) {
  return launch_tc<1, false>(GUpart, splits, w, GVraw, r, K, d, nullptr, nullptr, err, s);
}

}  // namespace externd
