// Small dense algebra of a block: ternary Gram matrices, (G + eps I)^-1 for Eq. 3, and the joint scale solve of
// Eq. 4.
//
// Gram matrices of ternary factors are integer counts (exact in float up to 2^24); with importance weights the
// U-step Gram is sum_y h_y v_a(y) v_b(y) in float. The inverse uses the symmetric sweep operator (Gauss-Jordan
// on an SPD matrix, no pivoting needed): one 1024-thread CTA holds the w x w matrix in registers, one row per
// 1024/W_PAD threads, and sweeps the w pivots with one barrier per pivot. Sweeping every pivot of S = G turns S
// into -G^-1.
#include <cooperative_groups.h>

#include <cstdlib>
#include <cstring>

#include "kernels.h"
#include "sweep.cuh"
#include "umma.cuh"

namespace externd {

namespace {

namespace cg = cooperative_groups;

constexpr int GT = 32;     // Gram tile (a, b)
constexpr int GY = 64;     // Gram depth slice

__global__ void __launch_bounds__(256) gram_kernel(const int8_t* __restrict__ T, int ldt, int w, int L,
                                                   const float* __restrict__ h, float* __restrict__ Gpart,
                                                   int ychunk) {
  __shared__ __align__(16) int8_t Ta[GT][GY];
  __shared__ __align__(16) int8_t Tb[GT][GY];
  __shared__ float hs[GY];
  const int a0 = blockIdx.y * GT, b0 = blockIdx.x * GT;
  const int ybeg = blockIdx.z * ychunk, yend = min(L, ybeg + ychunk);
  const int tid = threadIdx.x;
  const int ia = tid >> 3, ib = (tid & 7) * 4;
  int iacc[4] = {0, 0, 0, 0};
  float facc[4] = {0.f, 0.f, 0.f, 0.f};
  for (int y0 = ybeg; y0 < yend; y0 += GY) {
    // 32 rows x 64 bytes per operand: each thread copies 8 bytes of each (rows are 16-byte aligned, zero padded)
    {
      const int row = tid >> 3, off = (tid & 7) * 8;
      const int y = y0 + off;
      unsigned long long va = 0, vb = 0;
      if (a0 + row < w && y < yend)
        va = *reinterpret_cast<const unsigned long long*>(T + (long long)(a0 + row) * ldt + y);
      if (b0 + row < w && y < yend)
        vb = *reinterpret_cast<const unsigned long long*>(T + (long long)(b0 + row) * ldt + y);
      // mask bytes past the end of this split
      const int valid = yend - y;
      if (valid < 8) {
        const unsigned long long keep = valid <= 0 ? 0ull : ((1ull << (8 * valid)) - 1ull);
        va &= keep;
        vb &= keep;
      }
      *reinterpret_cast<unsigned long long*>(&Ta[row][off]) = va;
      *reinterpret_cast<unsigned long long*>(&Tb[row][off]) = vb;
    }
    if (h != nullptr && tid < GY) hs[tid] = (y0 + tid < yend) ? __ldg(h + y0 + tid) : 0.f;
    __syncthreads();
    if (h == nullptr) {
      const int* ra = reinterpret_cast<const int*>(Ta[ia]);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int* rb = reinterpret_cast<const int*>(Tb[ib + q]);
        int s = iacc[q];
#pragma unroll
        for (int t = 0; t < GY / 4; ++t) s = __dp4a(ra[t], rb[t], s);
        iacc[q] = s;
      }
    } else {
#pragma unroll 4
      for (int t = 0; t < GY; ++t) {
        const float av = (float)Ta[ia][t] * hs[t];
#pragma unroll
        for (int q = 0; q < 4; ++q) facc[q] = fmaf(av, (float)Tb[ib + q][t], facc[q]);
      }
    }
    __syncthreads();
  }
  const int a = a0 + ia;
  if (a >= w) return;
  float* out = Gpart + (long long)blockIdx.z * w * w + (long long)a * w;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int b = b0 + ib + q;
    if (b < w) out[b] = (h == nullptr) ? (float)iacc[q] : facc[q];
  }
}

// MODE 0: Graw = sum_s Gpart[s]; Ginv = (Graw + eps I)^-1.
// MODE 1: K = (sum_s Gpart[s]) .* GVraw (+ eps I when w > 1); d = K^-1 r.
//
// Blocked symmetric sweep. Sweeping pivot k maps S to S - S[:,k] S[k,:] / p with row and column k replaced by
// S[k,:] / p and S[k][k] by -1/p (p = S[k][k]); after every pivot S = -G^-1. Sweeps compose, so NB = 8 pivots
// K are eliminated per step: with P = S[K,K] and Q = P^-1,
//   S[I,J] -= S[I,K] Q S[K,J],  S[I,K] = S[I,K] Q,  S[K,J] = Q S[K,J],  S[K,K] = -Q      (I, J outside K).
// Every intermediate S is symmetric, so S[I,K] is the transpose of the published block rows S[K,:].
//
// Layout: warp q owns the RPW = W_PAD / NWARP rows q*RPW + a; lane l owns the CPL = W_PAD / 32 columns
// l + 32 c. Row-contiguous lanes make every global load and store coalesced and every read of a row's pivot
// entries a shared-memory broadcast. Per step: the warps owning rows K publish them (barrier), warp 0 inverts the
// 8 x 8 pivot block (barrier), every thread forms t = S[i,K] Q with one FMA chain per lane and 8 shuffles per
// row, then applies the rank-8 update to its elements (barrier).
template <int W_PAD, int NWARP, int MODE>
__global__ void __launch_bounds__(NWARP * 32) sweep_kernel(const float* __restrict__ Gpart, int splits, int w,
                                                           const float* __restrict__ GVraw,
                                                           const float* __restrict__ r, float* __restrict__ Graw,
                                                           float* __restrict__ out) {
  constexpr int RPW = W_PAD / NWARP;  // rows per warp
  constexpr int CPL = W_PAD / 32;     // columns per lane
  constexpr int NB = 8;
  static_assert(RPW >= 1 && CPL >= 1 && W_PAD % NB == 0, "bad sweep shape");
  __shared__ __align__(16) float rowsK[NB][W_PAD];
  __shared__ float Qs[NB][NB];
  __shared__ float dsum[NWARP];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int r0 = warp * RPW;

  float S[RPW][CPL];
#pragma unroll
  for (int a = 0; a < RPW; ++a)
#pragma unroll
    for (int c = 0; c < CPL; ++c) S[a][c] = 0.f;
  // Sum the split Gram slices (coalesced: lanes walk a row).
  for (int sp = 0; sp < splits; ++sp) {
    const float* G = Gpart + (long long)sp * w * w;
#pragma unroll
    for (int a = 0; a < RPW; ++a) {
      const int i = r0 + a;
      if (i >= w) continue;
#pragma unroll
      for (int c = 0; c < CPL; ++c) {
        const int j = lane + 32 * c;
        if (j < w) S[a][c] += G[(long long)i * w + j];
      }
    }
  }
  float diag = 0.f;
#pragma unroll
  for (int a = 0; a < RPW; ++a) {
    const int i = r0 + a;
#pragma unroll
    for (int c = 0; c < CPL; ++c) {
      const int j = lane + 32 * c;
      float v = S[a][c];
      if (i < w && j < w) {
        if (MODE == 0) {
          Graw[(long long)i * w + j] = v;
        } else {
          v *= GVraw[(long long)i * w + j];
          if (Graw != nullptr) Graw[(long long)i * w + j] = v;
        }
        if (i == j) diag += v;
      } else {
        v = (i == j) ? 1.f : 0.f;     // identity on the padding
      }
      S[a][c] = v;
    }
  }
  // trace -> ridge (float: it only sets the ridge, whose relative size is what matters)
  const float t = warp_sum(diag);
  if (lane == 0) dsum[warp] = t;
  __syncthreads();
  float tr = 0.f;
#pragma unroll
  for (int q = 0; q < NWARP; ++q) tr += dsum[q];
  const bool ridge = (MODE == 0) || (w > 1);
  const float eps = ridge ? (float)kEpsRel * tr / (float)w : 0.f;
#pragma unroll
  for (int a = 0; a < RPW; ++a)
#pragma unroll
    for (int c = 0; c < CPL; ++c)
      if (r0 + a < w && r0 + a == lane + 32 * c) S[a][c] += eps;

  for (int k0 = 0; k0 < w; k0 += NB) {
    // 1. publish block rows K = [k0, k0 + NB)
#pragma unroll
    for (int a = 0; a < RPW; ++a) {
      const int i = r0 + a;
      if (i >= k0 && i < k0 + NB) {
#pragma unroll
        for (int c = 0; c < CPL; ++c) rowsK[i - k0][lane + 32 * c] = S[a][c];
      }
    }
    __syncthreads();
    // 2. warp 0: Q = P^-1 by the scalar symmetric sweep of the 8 x 8 block (two elements per lane)
    if (warp == 0) {
      const int e0 = 2 * lane;
      const int pr = e0 / NB, cA = e0 % NB, cB = cA + 1;
      float qa = rowsK[pr][k0 + cA], qb = rowsK[pr][k0 + cB];
      if (k0 + pr >= w || k0 + cA >= w) qa = (pr == cA) ? 1.f : 0.f;   // identity past w
      if (k0 + pr >= w || k0 + cB >= w) qb = (pr == cB) ? 1.f : 0.f;
#pragma unroll
      for (int kk = 0; kk < NB; ++kk) {
        // element e of the block lives in lane e / 2 (qa if e is even, qb if odd)
        const int ek = kk * NB + kk, ec = kk * NB + pr, ej = kk * NB + cA;
        const float pk_a = __shfl_sync(0xffffffffu, qa, ek >> 1), pk_b = __shfl_sync(0xffffffffu, qb, ek >> 1);
        const float xa = __shfl_sync(0xffffffffu, qa, ec >> 1), xb = __shfl_sync(0xffffffffu, qb, ec >> 1);
        const float pa = __shfl_sync(0xffffffffu, qa, ej >> 1), pb = __shfl_sync(0xffffffffu, qb, ej >> 1);
        // 1 / S[kk][kk] with the fast single-precision division (<= 2 ulp); the correctly rounded reciprocal
        // takes a double-precision path, slow on this GPU
        const float ip = __fdividef(1.f, (ek & 1) ? pk_b : pk_a);
        const float ci = (ec & 1) ? xb : xa;
        float na = fmaf(-ci * ip, pa, qa), nb = fmaf(-ci * ip, pb, qb);
        if (pr == kk) { na = pa * ip; nb = pb * ip; }
        if (cA == kk) na = (pr == kk) ? -ip : ci * ip;
        if (cB == kk) nb = (pr == kk) ? -ip : ci * ip;
        qa = na;
        qb = nb;
      }
      Qs[pr][cA] = -qa;                        // sweeping every pivot of P leaves -P^-1
      Qs[pr][cB] = -qb;
    }
    __syncthreads();
    // 3. update: this lane's column of Q (b = lane % 8) and the pivot-row entries of its columns
    float qcol[NB];
#pragma unroll
    for (int c = 0; c < NB; ++c) qcol[c] = Qs[c][lane & (NB - 1)];
    float rk[NB][CPL];
#pragma unroll
    for (int b = 0; b < NB; ++b)
#pragma unroll
      for (int c = 0; c < CPL; ++c) rk[b][c] = rowsK[b][lane + 32 * c];
#pragma unroll
    for (int a = 0; a < RPW; ++a) {
      const int i = r0 + a;
      if (i >= W_PAD) continue;
      const bool i_in = (i >= k0 && i < k0 + NB);        // warp-uniform
      // t[b] = sum_c S[i][k0 + c] Q[c][b]; S[i][K] = rowsK[.][i] (broadcast reads)
      float tb = 0.f;
#pragma unroll
      for (int c = 0; c < NB; ++c) tb = fmaf(rowsK[c][i], qcol[c], tb);
      float tt[NB];
#pragma unroll
      for (int b = 0; b < NB; ++b) tt[b] = __shfl_sync(0xffffffffu, tb, b);
      float qrow[NB];                                    // Q[i - k0][.] for the rows of K
      if (i_in) {
#pragma unroll
        for (int b = 0; b < NB; ++b) qrow[b] = Qs[i - k0][b];
      }
#pragma unroll
      for (int c = 0; c < CPL; ++c) {
        const int j = lane + 32 * c;
        const bool j_in = (j >= k0 && j < k0 + NB);
        float v = S[a][c];
        if (!i_in) {
          if (!j_in) {
#pragma unroll
            for (int b = 0; b < NB; ++b) v = fmaf(-tt[b], rk[b][c], v);
          } else {
#pragma unroll
            for (int b = 0; b < NB; ++b) v = (j - k0 == b) ? tt[b] : v;            // S[i,K] Q
          }
        } else {
          if (!j_in) {
            v = 0.f;                                                             // (Q S[K,J])
#pragma unroll
            for (int b = 0; b < NB; ++b) v = fmaf(qrow[b], rk[b][c], v);
          } else {
#pragma unroll
            for (int b = 0; b < NB; ++b) v = (j - k0 == b) ? -qrow[b] : v;        // -Q
          }
        }
        S[a][c] = v;
      }
    }
    __syncthreads();   // rowsK and Qs are rewritten by the next step
  }

  if (MODE == 0) {
#pragma unroll
    for (int a = 0; a < RPW; ++a) {
      const int i = r0 + a;
      if (i >= w) continue;
#pragma unroll
      for (int c = 0; c < CPL; ++c) {
        const int j = lane + 32 * c;
        if (j < w) out[(long long)i * w + j] = -S[a][c];
      }
    }
  } else {
    // d_i = -sum_j S[i][j] r_j: a warp reduction per row
#pragma unroll
    for (int a = 0; a < RPW; ++a) {
      const int i = r0 + a;
      F2 acc;
#pragma unroll
      for (int c = 0; c < CPL; ++c) {
        const int j = lane + 32 * c;
        if (j < w) acc = f2_add(acc, -S[a][c] * r[j]);
      }
      acc = warp_sum(acc);
      if (lane == 0 && i < w) out[i] = acc.hi + acc.lo;
    }
  }
}

// r_a = sum_y u_a[y] (sum_s part[s][a][y]): one CTA per component; each thread takes 4 positions at a time
// and sums their split partials in split order with a batch of loads in flight.
__global__ void __launch_bounds__(512) rvec_kernel(const int8_t* __restrict__ Ut, int ldu, int w, int L,
                                                   const float* __restrict__ part, int splits,
                                                   float* __restrict__ r) {
  constexpr int NT = 512, PY = 4, SB = 8;
  __shared__ F2 red[NT / 32];
  const int a = blockIdx.x;
  const int8_t* u = Ut + (long long)a * ldu;
  const long long sstride = (long long)w * L;
  const float* P = part + (long long)a * L;
  float acc = 0.f;
  for (int y0 = 0; y0 < L; y0 += NT * PY) {
    float p[PY];
    int uv[PY];
#pragma unroll
    for (int j = 0; j < PY; ++j) {
      const int y = y0 + j * NT + threadIdx.x;
      p[j] = 0.f;
      uv[j] = y < L ? (int)u[y] : 0;
    }
    for (int s0 = 0; s0 < splits; s0 += SB) {
      float v[SB][PY];
#pragma unroll
      for (int q = 0; q < SB; ++q)
#pragma unroll
        for (int j = 0; j < PY; ++j) {
          const int y = y0 + j * NT + threadIdx.x;
          v[q][j] = (s0 + q < splits && y < L) ? P[(s0 + q) * sstride + y] : 0.f;
        }
#pragma unroll
      for (int q = 0; q < SB; ++q)
#pragma unroll
        for (int j = 0; j < PY; ++j) p[j] += v[q][j];
    }
#pragma unroll
    for (int j = 0; j < PY; ++j) acc += uv[j] > 0 ? p[j] : (uv[j] < 0 ? -p[j] : 0.f);
  }
  F2 v;
  v.hi = acc;
  v = warp_sum(v);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
  __syncthreads();
  if (threadIdx.x == 0) {
    F2 s;
    for (int q = 0; q < NT / 32; ++q) s = f2_add(s, red[q]);
    r[a] = s.hi + s.lo;
  }
}

// Wide-block sweep for w <= 128 with lookahead: NB pivots per step. 16 tile warps (512 threads; thread (ty, tx)
// owns the RPT = W_PAD/16 rows ty*RPT + a and the CPT = W_PAD/32 columns tx + 32c in registers) and one pivot
// warp. With Q = P^-1 of the current pivot block K (computed one step ahead), per step:
//   a. tile warps: T'[i,:] = S[i,K] Q for rows outside K (S[i,K] = Rk[.,i] by symmetry), -Q[i,:] on K; the
//      owners of the next block K+ also publish S[K+,K+] as it stands before this step's update      barrier
//   b. tile warps: one uniform rank-NB update S <- D S - T' Rk (D zeroes the rows of K: outside K this is the
//      Schur complement S - S[I,K] Q S[K,J], on K it gives Q S[K,J]), then the columns of K take T'
//      (S[I,K] Q, and -Q on the pivot block); the owners of K+ publish the updated rows K+.
//      Pivot warp, meanwhile: the updated next pivot block S[K+,K+] - T'[K+,:] Rk[:,K+] (the same operations
//      in the same order as the tile owners) and its inverse by warp_sweep, for the next step          barrier
// After the last step S = -(G + eps I)^-1.
// IN_INT: the Gram comes as an integer upper triangle Gint[a * w + b] (a <= b), reset to zero after reading;
// each thread reads its upper-triangle entries and the lower ones come back mirrored through shared memory.
template <int W_PAD, int NB, int MODE, bool IN_INT>
__global__ void __launch_bounds__(544) sweep32_kernel(const float* __restrict__ Gpart, int splits, int w,
                                                      const float* __restrict__ GVraw, const float* __restrict__ r,
                                                      float* __restrict__ Graw, float* __restrict__ out, int* Gint,
                                                      uint8_t* __restrict__ op) {
  constexpr int RPT = W_PAD / 16, CPT = W_PAD / 32, EPL = NB * NB / 32, LPR = NB / EPL, TLD = NB + 4;
  static_assert(W_PAD % NB == 0 && 32 % NB == 0 && (NB * NB) % 32 == 0 && NB % 4 == 0 && RPT >= 1 && CPT >= 1,
                "bad shape");
  __shared__ __align__(16) float Rk[2][NB][W_PAD];   // published rows of the pivot block (two buffers)
  __shared__ __align__(16) float T[W_PAD][TLD];      // T' of the step (padded rows: conflict-free float4 stores)
  __shared__ __align__(16) float Qs[2][NB][NB];      // pivot-block inverses (two buffers)
  __shared__ float Pn[NB][NB];                        // next pivot block before this step's update
  __shared__ float red[16];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const bool tile = warp < 16;
  const int tx = lane, ty = tile ? warp : 0, i0 = ty * RPT;

  float S[RPT][CPT];
#pragma unroll
  for (int a = 0; a < RPT; ++a)
#pragma unroll
    for (int c = 0; c < CPT; ++c) S[a][c] = 0.f;
  if (IN_INT) {
    // stage the integer Gram in shared memory: warp q copies rows q, q + 17, ... with coalesced loads, all of a
    // thread's loads issued before its first store; then every tile thread reads its entries by symmetry
    extern __shared__ int Gs[];   // [W_PAD][W_PAD + 1]
    constexpr int NR = (W_PAD + 16) / 17, NC = W_PAD / 32, QB = 4;   // rows per warp, batches of QB rows
#pragma unroll
    for (int q0 = 0; q0 < NR; q0 += QB) {
      int v[QB][NC];
#pragma unroll
      for (int q = 0; q < QB; ++q) {
        const int i = warp + 17 * (q0 + q);
#pragma unroll
        for (int c = 0; c < NC; ++c) {
          const int j = lane + 32 * c;
          v[q][c] = (q0 + q < NR && i < w && j < w) ? Gint[(long long)i * w + j] : 0;
        }
      }
#pragma unroll
      for (int q = 0; q < QB; ++q) {
        const int i = warp + 17 * (q0 + q);
        if (q0 + q < NR && i < W_PAD) {
#pragma unroll
          for (int c = 0; c < NC; ++c) Gs[i * (W_PAD + 1) + lane + 32 * c] = v[q][c];
        }
      }
    }
    __syncthreads();
    if (tile) {
#pragma unroll
      for (int a = 0; a < RPT; ++a) {
        const int i = i0 + a;
#pragma unroll
        for (int c = 0; c < CPT; ++c) {
          const int j = tx + 32 * c;
          S[a][c] = (float)(i <= j ? Gs[i * (W_PAD + 1) + j] : Gs[j * (W_PAD + 1) + i]);
        }
      }
    }
  } else if (tile) {
    for (int sp = 0; sp < splits; ++sp) {
      const float* G = Gpart + (long long)sp * w * w;
#pragma unroll
      for (int a = 0; a < RPT; ++a) {
        const int i = i0 + a;
        if (i >= w) continue;
#pragma unroll
        for (int c = 0; c < CPT; ++c) {
          const int j = tx + 32 * c;
          if (j < w) S[a][c] += G[(long long)i * w + j];
        }
      }
    }
  }
  float diag = 0.f;
  if (tile) {
#pragma unroll
    for (int a = 0; a < RPT; ++a) {
      const int i = i0 + a;
#pragma unroll
      for (int c = 0; c < CPT; ++c) {
        const int j = tx + 32 * c;
        float v = S[a][c];
        if (i < w && j < w) {
          if (MODE == 0) {
            Graw[(long long)i * w + j] = v;
          } else {
            v *= GVraw[(long long)i * w + j];
            if (Graw != nullptr) Graw[(long long)i * w + j] = v;
          }
          if (i == j) diag += v;
        } else {
          v = (i == j) ? 1.f : 0.f;
        }
        S[a][c] = v;
      }
    }
    const float dw = warp_sum(diag);
    if (lane == 0) red[ty] = dw;
  }
  __syncthreads();
  float tr = 0.f;
#pragma unroll
  for (int q = 0; q < 16; ++q) tr += red[q];
  const float eps = ((MODE == 0) || (w > 1)) ? (float)kEpsRel * tr / (float)w : 0.f;
  if (tile) {
#pragma unroll
    for (int a = 0; a < RPT; ++a)
#pragma unroll
      for (int c = 0; c < CPT; ++c)
        if (i0 + a < w && i0 + a == tx + 32 * c) S[a][c] += eps;
  }

  // rows [kb, kb + NB) of the register tiles into Rk[buf]
  auto publish_rows = [&](int kb, int buf) {
#pragma unroll
    for (int a = 0; a < RPT; ++a) {
      const int i = i0 + a;
      if (i >= kb && i < kb + NB) {
#pragma unroll
        for (int c = 0; c < CPT; ++c) Rk[buf][i - kb][tx + 32 * c] = S[a][c];
      }
    }
  };
  // prologue: the first pivot block and its inverse
  if (tile) publish_rows(0, 0);
  __syncthreads();
  if (!tile) {
    float A[EPL];
    const int pr_ = lane / LPR, pc = (lane % LPR) * EPL;
#pragma unroll
    for (int e = 0; e < EPL; ++e) A[e] = Rk[0][pr_][pc + e];
    warp_sweep<NB>(A, lane);
#pragma unroll
    for (int e = 0; e < EPL; ++e) Qs[0][pr_][pc + e] = -A[e];
  }
  __syncthreads();

  for (int k0 = 0, step = 0; k0 < w; k0 += NB, ++step) {
    const int cur = step & 1, nxt = cur ^ 1;
    const int kn = k0 + NB;
    const bool has_next = kn < w;
    // a. T' and the next pivot block as it stands
    if (tile) {
      for (int it = tid; it < W_PAD * (NB / 4); it += 512) {
        const int i = it % W_PAD, bq = (it / W_PAD) * 4;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        if (i >= k0 && i < k0 + NB) {
          const float4 q = *reinterpret_cast<const float4*>(&Qs[cur][i - k0][bq]);
          acc = make_float4(-q.x, -q.y, -q.z, -q.w);
        } else {
#pragma unroll
          for (int c = 0; c < NB; ++c) {
            const float rv = Rk[cur][c][i];
            const float4 q = *reinterpret_cast<const float4*>(&Qs[cur][c][bq]);
            acc.x = fmaf(rv, q.x, acc.x);
            acc.y = fmaf(rv, q.y, acc.y);
            acc.z = fmaf(rv, q.z, acc.z);
            acc.w = fmaf(rv, q.w, acc.w);
          }
        }
        *reinterpret_cast<float4*>(&T[i][bq]) = acc;
      }
      if (has_next) {
#pragma unroll
        for (int a = 0; a < RPT; ++a) {
          const int i = i0 + a;
          if (i >= kn && i < kn + NB) {
#pragma unroll
            for (int c = 0; c < CPT; ++c) {
              const int j = tx + 32 * c;
              if (j >= kn && j < kn + NB) Pn[i - kn][j - kn] = S[a][c];
            }
          }
        }
      }
    }
    __syncthreads();
    // b. the update (tile warps) beside the next pivot block's inverse (pivot warp)
    if (tile) {
#pragma unroll
      for (int a = 0; a < RPT; ++a)
        if (i0 + a >= k0 && i0 + a < k0 + NB)
#pragma unroll
          for (int c = 0; c < CPT; ++c) S[a][c] = 0.f;
#pragma unroll
      for (int b = 0; b < NB; b += 4) {
        float rv[4][CPT];
#pragma unroll
        for (int q = 0; q < 4; ++q)
#pragma unroll
          for (int c = 0; c < CPT; ++c) rv[q][c] = Rk[cur][b + q][tx + 32 * c];
        if constexpr (CPT % 2 == 0) {   // column pairs on the paired FMA (each lane the same fmaf as below)
#pragma unroll
          for (int a = 0; a < RPT; ++a) {   // one row's T' at a time (a broadcast load): fewer live registers
            const float4 t = *reinterpret_cast<const float4*>(&T[i0 + a][b]);
#pragma unroll
            for (int c = 0; c < CPT; c += 2) {
              float2 s2 = make_float2(S[a][c], S[a][c + 1]);
              s2 = __ffma2_rn(make_float2(-t.x, -t.x), make_float2(rv[0][c], rv[0][c + 1]), s2);
              s2 = __ffma2_rn(make_float2(-t.y, -t.y), make_float2(rv[1][c], rv[1][c + 1]), s2);
              s2 = __ffma2_rn(make_float2(-t.z, -t.z), make_float2(rv[2][c], rv[2][c + 1]), s2);
              s2 = __ffma2_rn(make_float2(-t.w, -t.w), make_float2(rv[3][c], rv[3][c + 1]), s2);
              S[a][c] = s2.x;
              S[a][c + 1] = s2.y;
            }
          }
        } else {
          float4 tv[RPT];
#pragma unroll
          for (int a = 0; a < RPT; ++a) tv[a] = *reinterpret_cast<const float4*>(&T[i0 + a][b]);
#pragma unroll
          for (int a = 0; a < RPT; ++a)
#pragma unroll
            for (int c = 0; c < CPT; ++c) {
              S[a][c] = fmaf(-tv[a].x, rv[0][c], S[a][c]);
              S[a][c] = fmaf(-tv[a].y, rv[1][c], S[a][c]);
              S[a][c] = fmaf(-tv[a].z, rv[2][c], S[a][c]);
              S[a][c] = fmaf(-tv[a].w, rv[3][c], S[a][c]);
            }
        }
      }
      const int cK = k0 >> 5;
      const int jk = tx + 32 * cK - k0;   // this lane's column within K, when in [0, NB)
      const bool lane_in = jk >= 0 && jk < NB;
      const int jb = min(max(jk, 0), NB - 1);
#pragma unroll
      for (int a = 0; a < RPT; ++a)
#pragma unroll
        for (int c = 0; c < CPT; ++c)
          if (c == cK) {
            const float tk = T[i0 + a][jb];
            S[a][c] = lane_in ? tk : S[a][c];
          }
      if (has_next) publish_rows(kn, nxt);
    } else if (has_next) {
      float A[EPL];
      const int pr_ = lane / LPR, pc = (lane % LPR) * EPL;
#pragma unroll
      for (int e = 0; e < EPL; ++e) {
        float v = Pn[pr_][pc + e];
#pragma unroll
        for (int b = 0; b < NB; b += 4) {
          const float4 t4 = *reinterpret_cast<const float4*>(&T[kn + pr_][b]);
          v = fmaf(-t4.x, Rk[cur][b + 0][kn + pc + e], v);
          v = fmaf(-t4.y, Rk[cur][b + 1][kn + pc + e], v);
          v = fmaf(-t4.z, Rk[cur][b + 2][kn + pc + e], v);
          v = fmaf(-t4.w, Rk[cur][b + 3][kn + pc + e], v);
        }
        A[e] = v;
      }
      warp_sweep<NB>(A, lane);
#pragma unroll
      for (int e = 0; e < EPL; ++e) Qs[nxt][pr_][pc + e] = -A[e];
    }
    __syncthreads();
  }

  if (!tile) return;
  if (MODE == 0) {
#pragma unroll
    for (int a = 0; a < RPT; ++a) {
      const int i = i0 + a;
      if (i >= w) continue;
#pragma unroll
      for (int c = 0; c < CPT; ++c) {
        const int j = tx + 32 * c;
        if (j < w) out[(long long)i * w + j] = -S[a][c];
      }
    }
    if (W_PAD == 128 && op != nullptr) {
      // Ginv * 2^sg as hi / lo fp16 K-major operands (zero outside w x w) for the tensor-core decorrelation, with
      // sg from the largest magnitude; sg (int) follows the two 32 KB images.
      float mx = 0.f;
#pragma unroll
      for (int a = 0; a < RPT; ++a)
#pragma unroll
        for (int c = 0; c < CPT; ++c)
          if (i0 + a < w && tx + 32 * c < w) mx = fmaxf(mx, fabsf(S[a][c]));
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      if (lane == 0) red[warp] = mx;
      asm volatile("bar.sync 1, 512;" ::: "memory");   // the 16 tile warps (the pivot warp has left)
#pragma unroll
      for (int q = 0; q < 16; ++q) mx = fmaxf(mx, red[q]);
      const int sg = fp16_scale_exp(mx);
      const float sc = ldexpf(1.f, sg);
#pragma unroll
      for (int a = 0; a < RPT; ++a)
#pragma unroll
        for (int c = 0; c < CPT; ++c) {
          const int i = i0 + a, j = tx + 32 * c;
          __half hi, lo;
          split_f16((i < w && j < w) ? -S[a][c] * sc : 0.f, hi, lo);
          const uint32_t off = k_major_offset(128u, (uint32_t)i, (uint32_t)j);
          *reinterpret_cast<__half*>(op + off) = hi;
          *reinterpret_cast<__half*>(op + 2 * 16384u + off) = lo;
        }
      if (tid == 0) *reinterpret_cast<int*>(op + 4 * 16384u) = sg;
    }
  } else {
#pragma unroll
    for (int a = 0; a < RPT; ++a) {
      const int i = i0 + a;
      F2 acc2;
#pragma unroll
      for (int c = 0; c < CPT; ++c) {
        const int j = tx + 32 * c;
        if (j < w) acc2 = f2_add(acc2, -S[a][c] * r[j]);
      }
      acc2 = warp_sum(acc2);
      if (lane == 0 && i < w) out[i] = acc2.hi + acc2.lo;
    }
  }
  if (IN_INT) {   // every thread has read the Gram (barrier after staging): reset it for the next accumulation
    for (int idx = tid; idx < w * w; idx += 512) Gint[idx] = 0;   // tile threads (tid < 512) only
  }

}

// Register-tiled sweep for w <= 128 on one CTA: RG x CG tile threads hold the WP x WP matrix as TR x TC
// register tiles (8 x 4 over 16 warps at WP = 128, 4 x 2 over 16 warps at 64, 2 x 2 over 8 warps at 32), one
// row group per warp at WP >= 64, so every shared-memory read of a pivot row is a broadcast and every read of a
// W row covers contiguous bytes; one more warp inverts the next pivot block ahead. Thread t owns the rows
// TR * (t / CG) + a and the columns TC * (t % CG) + c. With the published rows Rk = S[K,:] of pivot block K and
// Q = S[K,K]^-1 (both ready at the start of a step):
//   A. W = Q Rk (NB x WP) into shared memory; the owners of the next block K+ also save S[K+,K+]      barrier
//   B. rows outside K: S[i,j] -= sum_d Rk[d][i] W[d][j] (S[i,K] = Rk[.,i] by symmetry; fma chains in d
//      order on the paired FMA), then the columns of K take S[i,K] Q = W[.,i]; rows of K become
//      Q S[K,J] = W[.,J] and -Q on the pivot block; the owners of K+ publish their updated rows.
//      Pivot warp, meanwhile: the updated S[K+,K+] from the saved block with the same fma chains, and its
//      inverse (warp_sweep)                                                                              barrier
// Every S stays symmetric; after the last block S = -(G + eps I)^-1. About w^3 FMAs in all. The pivot warp's
// shuffles and loads issue between the tile warps' paired FMAs, which keep the FMA pipes busy.
template <int WP>
struct InvShape {
  static constexpr int NB = WP >= 64 ? 16 : 8;   // pivot block
  static constexpr int TR = WP == 128 ? 8 : WP == 64 ? 4 : 2;
  static constexpr int TC = WP == 128 ? 4 : 2;
  static constexpr int RG = WP / TR, CG = WP / TC, NT = RG * CG;   // row groups, column groups, tile threads
  // tile warps; warps launched (at WP = 128 with the sub-partition layout of inv_role, else the tile warps then
  // the pivot warp)
  static constexpr bool REMAP = WP == 128;
  static constexpr int NW = NT / 32, NWALL = REMAP ? NW + 4 : NW + 1;
};

template <int WP>
constexpr int inv_threads() { return InvShape<WP>::NWALL * 32; }

// Warp roles of inv_kernel. Warp w runs on SM sub-partition w % 4. Warp 0 is the pivot warp; sub-partition 0
// holds only p0 tile warps beside it (warps 4, 8, ...), so the pivot warp's serial chain of shuffles and
// reciprocals is not starved of issue slots by the tile warps' FMA streams; the other tile warps fill
// sub-partitions 1-3 evenly. Returns the tile-warp index, -2 for the pivot warp, -1 for an idle warp.
template <int NW>
__device__ __forceinline__ int inv_role(int warp, int p0) {
  if (warp == 0) return -2;
  if ((warp & 3) != 0) {
    const int t = (warp >> 2) * 3 + (warp & 3) - 1;
    return t < NW - p0 ? t : -1;
  }
  const int j = warp >> 2;   // 1 .. NWALL / 4 - 1
  return j <= p0 ? NW - p0 + j - 1 : -1;
}

// The barrier of the pivot and tile warps (idle warps leave at the start).
template <int N>
__device__ __forceinline__ void inv_bar() {
  asm volatile("bar.sync 1, %0;" ::"n"(N) : "memory");
}

// Tile warps on sub-partition 0 beside the pivot warp (1 .. 4; 4 puts four tile warps on every sub-partition).
int inv_p0() {
  static const int p0 = [] {
    const char* e = std::getenv("EXTERND_INV_P0");
    const int v = e ? std::atoi(e) : 2;
    return v < 1 ? 1 : v > 4 ? 4 : v;
  }();
  return p0;
}

template <int WP>
int inv_p0_for() {   // at most the warps 4, 8, ... that the launch has on sub-partition 0
  return InvShape<WP>::REMAP ? (inv_p0() < InvShape<WP>::NWALL / 4 - 1 ? inv_p0() : InvShape<WP>::NWALL / 4 - 1) : 0;
}

template <int WP, int MODE, bool IN_INT>
__global__ void __launch_bounds__(InvShape<WP>::NWALL * 32) inv_kernel(const float* __restrict__ Gpart, int splits,
                                                                     int w, const float* __restrict__ GVraw,
                                                                     const float* __restrict__ r,
                                                                     float* __restrict__ Graw,
                                                                     float* __restrict__ out, int* Gint,
                                                                     uint8_t* __restrict__ op, int p0) {
  using SH = InvShape<WP>;
  constexpr int NB = SH::NB, TR = SH::TR, TC = SH::TC, CG = SH::CG, NT = SH::NT, NW = SH::NW;
  constexpr int EPL = NB * NB / 32, LPR = NB / EPL;
  static_assert(TR % 2 == 0 && TC % 2 == 0 && (TC == 2 || TC == 4) && NT % 32 == 0, "tile shape");
  static_assert(NB % (TR * (32 / CG)) == 0, "a warp's rows lie in one pivot block");
  __shared__ __align__(16) float Rk[2 * NB * WP];   // published rows of the pivot block (two buffers)
  __shared__ __align__(16) float Ws[NB][WP];      // W = Q Rk of the step
  __shared__ __align__(16) float Qs[2][NB][NB];   // pivot-block inverses (two buffers)
  __shared__ __align__(16) float Qt[2][NB][NB];   // the same, transposed (Qt[d][c] = Qs[c][d], bit for bit)
  __shared__ __align__(16) float Pn[NB][NB];      // next pivot block before this step's update
  __shared__ float red[NW];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tw = SH::REMAP ? inv_role<NW>(warp, p0) : warp < NW ? warp : -2;
  if (tw == -1) return;   // idle warp (never takes part in the barrier)
  const bool tile = tw >= 0;
  const int tid = tile ? tw * 32 + lane : NT + lane;   // tile threads 0 .. NT - 1, then the pivot warp
  const int tr = tile ? tid / CG : 0, tc = tid % CG, i0 = tr * TR, jb = tc * TC;
  const bool vec = (w & 3) == 0;   // rows of every w x w input and output start on 16-byte boundaries
  // a run (i, jb .. jb + TC - 1) of a w x w matrix: one vector access where it is aligned and inside
  const bool run_in = vec && jb + TC <= w;

  float S[TR][TC];
#pragma unroll
  for (int a = 0; a < TR; ++a)
#pragma unroll
    for (int c = 0; c < TC; ++c) S[a][c] = 0.f;
  if (IN_INT && tile) {
    // The run of TC columns lies wholly above the diagonal (read along the rows), wholly below it (read the
    // mirrored entries along the columns, where rows i0 .. i0 + TR - 1 are contiguous) or straddles it (entry by
    // entry); every load is issued before the first use.
    int g[TR][TC];
    const bool upper = i0 + TR - 1 <= jb, lower = i0 > jb + TC - 1;
    if (upper && run_in) {
#pragma unroll
      for (int a = 0; a < TR; ++a) {
        const int* src = Gint + (long long)(i0 + a) * w + jb;
        if (i0 + a >= w) {
#pragma unroll
          for (int c = 0; c < TC; ++c) g[a][c] = 0;
        } else if constexpr (TC == 4) {
          const int4 t = *reinterpret_cast<const int4*>(src);
          g[a][0] = t.x; g[a][1] = t.y; g[a][2] = t.z; g[a][3] = t.w;
        } else {
          const int2 t = *reinterpret_cast<const int2*>(src);
          g[a][0] = t.x; g[a][1] = t.y;
        }
      }
    } else if (lower && vec && i0 + TR <= w) {
#pragma unroll
      for (int c = 0; c < TC; ++c) {
        const int* src = Gint + (long long)(jb + c) * w + i0;
        if (jb + c >= w) {
#pragma unroll
          for (int a = 0; a < TR; ++a) g[a][c] = 0;
        } else if constexpr (TR % 4 == 0) {
#pragma unroll
          for (int a = 0; a < TR; a += 4) {
            const int4 t = *reinterpret_cast<const int4*>(src + a);
            g[a][c] = t.x; g[a + 1][c] = t.y; g[a + 2][c] = t.z; g[a + 3][c] = t.w;
          }
        } else {
#pragma unroll
          for (int a = 0; a < TR; a += 2) {
            const int2 t = *reinterpret_cast<const int2*>(src + a);
            g[a][c] = t.x; g[a + 1][c] = t.y;
          }
        }
      }
    } else {
#pragma unroll
      for (int a = 0; a < TR; ++a)
#pragma unroll
        for (int c = 0; c < TC; ++c) {
          const int i = i0 + a, j = jb + c;
          g[a][c] = (i < w && j < w) ? Gint[(long long)min(i, j) * w + max(i, j)] : 0;
        }
    }
#pragma unroll
    for (int a = 0; a < TR; ++a)
#pragma unroll
      for (int c = 0; c < TC; ++c) S[a][c] = (float)g[a][c];
  } else if (tile) {
    for (int sp = 0; sp < splits; ++sp) {
      const float* G = Gpart + (long long)sp * w * w;
#pragma unroll
      for (int a = 0; a < TR; ++a)
#pragma unroll
        for (int c = 0; c < TC; ++c) {
          const int i = i0 + a, j = jb + c;
          if (i < w && j < w) S[a][c] += G[(long long)i * w + j];
        }
    }
  }
  // loads / stores of the thread's run of row i in a w x w float matrix
  auto load_run = [&](const float* M, int i, float (&v)[TC]) {
    const float* src = M + (long long)i * w + jb;
    if (i < w && run_in) {
      if constexpr (TC == 4) {
        const float4 t = *reinterpret_cast<const float4*>(src);
        v[0] = t.x; v[1] = t.y; v[2] = t.z; v[3] = t.w;
      } else {
        const float2 t = *reinterpret_cast<const float2*>(src);
        v[0] = t.x; v[1] = t.y;
      }
    } else {
#pragma unroll
      for (int c = 0; c < TC; ++c) v[c] = (i < w && jb + c < w) ? src[c] : 0.f;
    }
  };
  auto store_run = [&](float* M, int i, const float (&v)[TC]) {
    float* dst = M + (long long)i * w + jb;
    if (i < w && run_in) {
      if constexpr (TC == 4) *reinterpret_cast<float4*>(dst) = make_float4(v[0], v[1], v[2], v[3]);
      else *reinterpret_cast<float2*>(dst) = make_float2(v[0], v[1]);
    } else {
#pragma unroll
      for (int c = 0; c < TC; ++c)
        if (i < w && jb + c < w) dst[c] = v[c];
    }
  };
  float diag = 0.f;
  if (tile) {
    if (MODE == 1) {   // K = G_U .* G_V
      float gv[TR][TC];
#pragma unroll
      for (int a = 0; a < TR; ++a) load_run(GVraw, i0 + a, gv[a]);
#pragma unroll
      for (int a = 0; a < TR; ++a)
#pragma unroll
        for (int c = 0; c < TC; ++c) S[a][c] *= gv[a][c];
    }
#pragma unroll
    for (int a = 0; a < TR; ++a)
#pragma unroll
      for (int c = 0; c < TC; ++c) {
        const int i = i0 + a, j = jb + c;
        if (i < w && j < w) {
          if (i == j) diag += S[a][c];
        } else {
          S[a][c] = (i == j) ? 1.f : 0.f;   // identity on the padding
        }
      }
    if (Graw != nullptr) {   // the Gram (MODE 0) or K (MODE 1) before the ridge
#pragma unroll
      for (int a = 0; a < TR; ++a) store_run(Graw, i0 + a, S[a]);
    }
  }
  diag = warp_sum(diag);
  if (lane == 0 && tile) red[tw] = diag;
  inv_bar<NT + 32>();
  if (IN_INT) {   // every tile thread has read its entries of the Gram: reset it for the next accumulation
    const int ww = w * w;
    if ((ww & 3) == 0) {
      for (int idx = tid; idx < ww / 4; idx += NT + 32) reinterpret_cast<int4*>(Gint)[idx] = make_int4(0, 0, 0, 0);
    } else {
      for (int idx = tid; idx < ww; idx += NT + 32) Gint[idx] = 0;
    }
  }
  float trace = 0.f;
#pragma unroll
  for (int q = 0; q < NW; ++q) trace += red[q];
  const float eps = ((MODE == 0) || (w > 1)) ? (float)kEpsRel * trace / (float)w : 0.f;
  if (tile) {
#pragma unroll
    for (int a = 0; a < TR; ++a)
#pragma unroll
      for (int c = 0; c < TC; ++c)
        if (i0 + a < w && i0 + a == jb + c) S[a][c] += eps;
  }

  // the published entry (buf, row d of the pivot block, column i)
  auto rk_at = [&](int buf, int d, int i) -> float* { return &Rk[(buf * NB + d) * WP + i]; };
  auto rk_val = [&](int buf, int d, int i) -> float { return *rk_at(buf, d, i); };
  auto publish_rows = [&](int kb, int buf) {   // rows [kb, kb + NB) of the register tiles into Rk[buf]
    if (i0 >= kb && i0 < kb + NB) {
#pragma unroll
      for (int a = 0; a < TR; ++a) {
        if constexpr (TC == 4) {
          *reinterpret_cast<float4*>(rk_at(buf, i0 + a - kb, jb)) = make_float4(S[a][0], S[a][1], S[a][2], S[a][3]);
        } else {
          *reinterpret_cast<float2*>(rk_at(buf, i0 + a - kb, jb)) = make_float2(S[a][0], S[a][1]);
        }
      }
    }
  };
  const int pr = lane / LPR, pc = (lane % LPR) * EPL;   // pivot warp: its entries of an NB x NB block
  if (tile) publish_rows(0, 0);
  inv_bar<NT + 32>();
  if (!tile) {
    float A[EPL];
#pragma unroll
    for (int e = 0; e < EPL; ++e) A[e] = rk_val(0, pr, pc + e);
    warp_sweep<NB>(A, lane);
#pragma unroll
    for (int e = 0; e < EPL; ++e) {
      Qs[0][pr][pc + e] = -A[e];
      Qt[0][pc + e][pr] = -A[e];
    }
  }
  inv_bar<NT + 32>();

  for (int k0 = 0, step = 0; k0 < w; k0 += NB, ++step) {
    const int cur = step & 1, nxt = cur ^ 1, kn = k0 + NB;
    const bool has_next = kn < w;
    const bool rowsK = i0 >= k0 && i0 < k0 + NB;          // warp-uniform: a warp's rows lie in one block
    const bool rowsN = has_next && i0 >= kn && i0 < kn + NB;
    const bool colsK = jb + TC > k0 && jb < k0 + NB;      // TC divides NB: a run is wholly in or out of K
    // A. W = Q Rk; the next pivot block as it stands. At WP = 128 four tile warps, one per sub-partition
    //    (warps 1 .. 4), form W: lane (cg, qg) of warp 1 + a the rows 4cg .. 4cg + 3 and the columns
    //    32a + 4qg .. + 3, so a warp reads each Rk row once (128 bytes) and Q as 16-byte rows of Qt; the same
    //    fma chains in d order as one output per thread.
    if constexpr (WP == 128) {
      if (warp >= 1 && warp <= 4) {
        const int c0 = 4 * (lane >> 3), q0 = 32 * (warp - 1) + 4 * (lane & 7);
        float4 acc[4];
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[c] = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int d = 0; d < NB; ++d) {
          const float4 rv = *reinterpret_cast<const float4*>(rk_at(cur, d, q0));
          const float4 qv = *reinterpret_cast<const float4*>(&Qt[cur][d][c0]);
          const float qc[4] = {qv.x, qv.y, qv.z, qv.w};
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            acc[c].x = fmaf(qc[c], rv.x, acc[c].x);
            acc[c].y = fmaf(qc[c], rv.y, acc[c].y);
            acc[c].z = fmaf(qc[c], rv.z, acc[c].z);
            acc[c].w = fmaf(qc[c], rv.w, acc[c].w);
          }
        }
#pragma unroll
        for (int c = 0; c < 4; ++c) *reinterpret_cast<float4*>(&Ws[c0 + c][q0]) = acc[c];
      }
    }
    if (tile) {
      for (int idx = WP == 128 ? NB * (WP / 4) : tid; idx < NB * (WP / 4); idx += NT) {
        const int c = idx / (WP / 4), q = (idx % (WP / 4)) * 4;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int d = 0; d < NB; ++d) {
          const float qv = Qs[cur][c][d];
          const float4 rv = *reinterpret_cast<const float4*>(rk_at(cur, d, q));
          acc.x = fmaf(qv, rv.x, acc.x);
          acc.y = fmaf(qv, rv.y, acc.y);
          acc.z = fmaf(qv, rv.z, acc.z);
          acc.w = fmaf(qv, rv.w, acc.w);
        }
        *reinterpret_cast<float4*>(&Ws[c][q]) = acc;
      }
      if (rowsN && jb >= kn && jb < kn + NB) {
#pragma unroll
        for (int a = 0; a < TR; ++a)
#pragma unroll
          for (int c = 0; c < TC; ++c) Pn[i0 + a - kn][jb + c - kn] = S[a][c];
      }
    }
    inv_bar<NT + 32>();
    // B. the update (tile warps) beside the next pivot block's inverse (pivot warp)
    if (tile) {
      if (rowsK) {
        if (colsK) {
#pragma unroll
          for (int a = 0; a < TR; ++a)
#pragma unroll
            for (int c = 0; c < TC; ++c) S[a][c] = -Qs[cur][i0 + a - k0][jb + c - k0];
        } else {
#pragma unroll
          for (int a = 0; a < TR; ++a)
#pragma unroll
            for (int c = 0; c < TC; ++c) S[a][c] = Ws[i0 + a - k0][jb + c];
        }
      } else {
#pragma unroll 4
        for (int d = 0; d < NB; ++d) {
          float rk[TR], wv[TC];
#pragma unroll
          for (int a = 0; a < TR; a += 2) {
            const float2 t = *reinterpret_cast<const float2*>(rk_at(cur, d, i0 + a));
            rk[a] = t.x;
            rk[a + 1] = t.y;
          }
          if constexpr (TC == 4) {
            const float4 t = *reinterpret_cast<const float4*>(&Ws[d][jb]);
            wv[0] = t.x; wv[1] = t.y; wv[2] = t.z; wv[3] = t.w;
          } else {
            const float2 t = *reinterpret_cast<const float2*>(&Ws[d][jb]);
            wv[0] = t.x; wv[1] = t.y;
          }
#pragma unroll
          for (int a = 0; a < TR; ++a)
#pragma unroll
            for (int c = 0; c < TC; c += 2) {   // lane-wise fma.rn, the same rounding as fmaf
              const float2 s2 = __ffma2_rn(make_float2(-rk[a], -rk[a]), make_float2(wv[c], wv[c + 1]),
                                           make_float2(S[a][c], S[a][c + 1]));
              S[a][c] = s2.x;
              S[a][c + 1] = s2.y;
            }
        }
        if (colsK) {
#pragma unroll
          for (int c = 0; c < TC; ++c)
#pragma unroll
            for (int a = 0; a < TR; ++a) S[a][c] = Ws[jb + c - k0][i0 + a];
        }
      }
      if (rowsN) publish_rows(kn, nxt);
    } else if (has_next) {
      float A[EPL];
#pragma unroll
      for (int e = 0; e < EPL; ++e) A[e] = Pn[pr][pc + e];
#pragma unroll
      for (int d = 0; d < NB; ++d) {   // the fma chains of the tile owners, in the same order
        const float rk = rk_val(cur, d, kn + pr);
        float wv[EPL];
#pragma unroll
        for (int e = 0; e < EPL; e += 2) {
          const float2 t = *reinterpret_cast<const float2*>(&Ws[d][kn + pc + e]);
          wv[e] = t.x;
          wv[e + 1] = t.y;
        }
#pragma unroll
        for (int e = 0; e < EPL; ++e) A[e] = fmaf(-rk, wv[e], A[e]);
      }
      warp_sweep<NB>(A, lane);
#pragma unroll
      for (int e = 0; e < EPL; ++e) {
        Qs[nxt][pr][pc + e] = -A[e];
        Qt[nxt][pc + e][pr] = -A[e];
      }
    }
    inv_bar<NT + 32>();
  }

  if (MODE == 0) {
    if (op == nullptr) {   // Ginv in float32 (the tensor-core decorrelation reads only the operand image below)
      if (tile) {
#pragma unroll
        for (int a = 0; a < TR; ++a) {
          float v[TC];
#pragma unroll
          for (int c = 0; c < TC; ++c) v[c] = -S[a][c];
          store_run(out, i0 + a, v);
        }
      }
    } else if constexpr (WP == 128) {
      // Ginv * 2^sg as hi / lo fp16 K-major operands (zero outside w x w) for the tensor-core decorrelation, with
      // sg from the largest magnitude; sg (int) follows the two 32 KB images.
      float mx = 0.f;
      if (tile) {
#pragma unroll
        for (int a = 0; a < TR; ++a)
#pragma unroll
          for (int c = 0; c < TC; ++c)
            if (i0 + a < w && jb + c < w) mx = fmaxf(mx, fabsf(S[a][c]));
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      if (lane == 0 && tile) red[tw] = mx;
      inv_bar<NT + 32>();
#pragma unroll
      for (int q = 0; q < NW; ++q) mx = fmaxf(mx, red[q]);
      const int sg = fp16_scale_exp(mx);
      const float sc = ldexpf(1.f, sg);
      if (tile) {   // the run of 4 columns (jb % 4 == 0) is 8 contiguous bytes of one row in the image
#pragma unroll
        for (int a = 0; a < TR; ++a) {
          const int i = i0 + a;
          __align__(8) __half hi[4];
          __align__(8) __half lo[4];
#pragma unroll
          for (int c = 0; c < 4; ++c) split_f16((i < w && jb + c < w) ? -S[a][c] * sc : 0.f, hi[c], lo[c]);
          const uint32_t off = k_major_offset(128u, (uint32_t)i, (uint32_t)jb);
          *reinterpret_cast<uint2*>(op + off) = *reinterpret_cast<const uint2*>(hi);
          *reinterpret_cast<uint2*>(op + 2 * 16384u + off) = *reinterpret_cast<const uint2*>(lo);
        }
      }
      if (tid == 0) *reinterpret_cast<int*>(op + 4 * 16384u) = sg;
    }
  } else if (tile) {
    // d_i = sum_j (-S)[i][j] r_j, double-float, over the CG threads that share the row group
    float rv[TC];
#pragma unroll
    for (int c = 0; c < TC; ++c) rv[c] = jb + c < w ? r[jb + c] : 0.f;
#pragma unroll
    for (int a = 0; a < TR; ++a) {
      const int i = i0 + a;
      F2 acc2;
#pragma unroll
      for (int c = 0; c < TC; ++c)
        if (jb + c < w) acc2 = f2_add(acc2, -S[a][c] * rv[c]);
#pragma unroll
      for (int o = CG / 2; o > 0; o >>= 1) acc2 = f2_add(acc2, f2_shfl_xor(acc2, o));
      if (tc == 0 && i < w) out[i] = acc2.hi + acc2.lo;
    }
  }
}

// Cluster sweep for 16 < w <= 128: the CS = WP / 16 CTAs of one thread-block cluster each hold one pivot block's
// 16 rows (CTA c: rows 16c .. 16c + 15) as 2 x TC register tiles; the pivot rows and inverse of each step reach
// the other CTAs through distributed shared memory. Step s (K = the rows of CTA s):
//   1. every CTA copies CTA s's published rows Rk = S[K,:] and Q = S[K,K]^-1 into its own shared memory
//   2. W = Q Rk; the next owner (CTA s + 1) saves its diagonal block                                  CTA barrier
//   3. rows outside K: S[i,j] -= sum_d Rk[d][i] W[d][j] (fma chains in d order), the columns of K take
//      W[.,i]; CTA s's rows become W and -Q on the pivot block. Meanwhile the pivot warp of CTA s + 1 forms
//      its updated diagonal block with the same fma chains and inverts it (warp_sweep); CTA s + 1 then
//      publishes its rows and that inverse                                                          cluster barrier
// The arithmetic per entry is that of inv_kernel (same operations in the same order); only the place where each
// row lives differs. Every CTA reads only its own rows of the integer Gram's mirror image and of the outputs.
// With pdl the CTAs let the next kernel of the stream launch as soon as they are all resident (programmatic
// dependent launch): the residual product then runs beside them on the other SMs.
template <int WP>
struct InvClusterShape {
  static constexpr int NB = 16, CS = WP / 16, TR = 2, TC = WP == 128 ? 4 : 2;
  static constexpr int CG = WP / TC, NT = (NB / TR) * CG;   // column groups, tile threads
};

template <int WP>
constexpr int inv_cluster_threads() { return InvClusterShape<WP>::NT + 32; }

template <int WP, int MODE, bool IN_INT>
__global__ void __launch_bounds__(InvClusterShape<WP>::NT + 32) inv_cluster_kernel(
    const float* __restrict__ Gpart, int splits, int w, const float* __restrict__ GVraw, const float* __restrict__ r,
    float* __restrict__ Graw, float* __restrict__ out, int* Gint, uint8_t* __restrict__ op, int pdl) {
  using SH = InvClusterShape<WP>;
  constexpr int NB = SH::NB, CS = SH::CS, TR = SH::TR, TC = SH::TC, CG = SH::CG, NT = SH::NT, NW = NT / 32;
  constexpr int EPL = NB * NB / 32, LPR = NB / EPL;
  static_assert(TC == 2 || TC == 4, "tile shape");
  __shared__ __align__(16) float pubR[NB][WP];   // this CTA's rows when it owns the step's pivot block
  __shared__ __align__(16) float pubQ[NB][NB];   // and the pivot block's inverse
  __shared__ __align__(16) float Rk[NB][WP];     // the step's pivot rows (copied from their owner)
  __shared__ __align__(16) float Qk[NB][NB];
  __shared__ __align__(16) float Ws[NB][WP];     // W = Q Rk
  __shared__ __align__(16) float Pn[NB][NB];     // own diagonal block before the update (next owner)
  __shared__ float red[NW + 1];
  __shared__ float cpart[2];                     // this CTA's trace part / max |Ginv| (read by the cluster)
  cg::cluster_group cluster = cg::this_cluster();
  const int c = (int)cluster.block_rank();
  if (pdl) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const bool tile = tid < NT;
  const int tr = tile ? tid / CG : 0, tc = tid % CG;
  const int lr0 = tr * TR, i0 = NB * c + lr0, jb = tc * TC;
  const bool vec = (w & 3) == 0;
  const bool run_in = vec && jb + TC <= w;

  float S[TR][TC];
#pragma unroll
  for (int a = 0; a < TR; ++a)
#pragma unroll
    for (int q = 0; q < TC; ++q) S[a][q] = 0.f;
  if (IN_INT && tile) {
    int g[TR][TC];
    const bool upper = i0 + TR - 1 <= jb, lower = i0 > jb + TC - 1;
    if (upper && run_in) {
#pragma unroll
      for (int a = 0; a < TR; ++a) {
        const int* src = Gint + (long long)(i0 + a) * w + jb;
        if (i0 + a >= w) {
#pragma unroll
          for (int q = 0; q < TC; ++q) g[a][q] = 0;
        } else if constexpr (TC == 4) {
          const int4 t = *reinterpret_cast<const int4*>(src);
          g[a][0] = t.x; g[a][1] = t.y; g[a][2] = t.z; g[a][3] = t.w;
        } else {
          const int2 t = *reinterpret_cast<const int2*>(src);
          g[a][0] = t.x; g[a][1] = t.y;
        }
      }
    } else if (lower && vec && i0 + TR <= w) {
#pragma unroll
      for (int q = 0; q < TC; ++q) {
        if (jb + q >= w) {
          g[0][q] = g[1][q] = 0;
        } else {
          const int2 t = *reinterpret_cast<const int2*>(Gint + (long long)(jb + q) * w + i0);
          g[0][q] = t.x;
          g[1][q] = t.y;
        }
      }
    } else {
#pragma unroll
      for (int a = 0; a < TR; ++a)
#pragma unroll
        for (int q = 0; q < TC; ++q) {
          const int i = i0 + a, j = jb + q;
          g[a][q] = (i < w && j < w) ? Gint[(long long)min(i, j) * w + max(i, j)] : 0;
        }
    }
#pragma unroll
    for (int a = 0; a < TR; ++a)
#pragma unroll
      for (int q = 0; q < TC; ++q) S[a][q] = (float)g[a][q];
  } else if (tile) {
    for (int sp = 0; sp < splits; ++sp) {
      const float* G = Gpart + (long long)sp * w * w;
#pragma unroll
      for (int a = 0; a < TR; ++a)
#pragma unroll
        for (int q = 0; q < TC; ++q) {
          const int i = i0 + a, j = jb + q;
          if (i < w && j < w) S[a][q] += G[(long long)i * w + j];
        }
    }
  }
  auto load_run = [&](const float* M, int i, float (&v)[TC]) {
    const float* src = M + (long long)i * w + jb;
    if (i < w && run_in) {
      if constexpr (TC == 4) {
        const float4 t = *reinterpret_cast<const float4*>(src);
        v[0] = t.x; v[1] = t.y; v[2] = t.z; v[3] = t.w;
      } else {
        const float2 t = *reinterpret_cast<const float2*>(src);
        v[0] = t.x; v[1] = t.y;
      }
    } else {
#pragma unroll
      for (int q = 0; q < TC; ++q) v[q] = (i < w && jb + q < w) ? src[q] : 0.f;
    }
  };
  auto store_run = [&](float* M, int i, const float (&v)[TC]) {
    float* dst = M + (long long)i * w + jb;
    if (i < w && run_in) {
      if constexpr (TC == 4) *reinterpret_cast<float4*>(dst) = make_float4(v[0], v[1], v[2], v[3]);
      else *reinterpret_cast<float2*>(dst) = make_float2(v[0], v[1]);
    } else {
#pragma unroll
      for (int q = 0; q < TC; ++q)
        if (i < w && jb + q < w) dst[q] = v[q];
    }
  };
  float diag = 0.f;
  if (tile) {
    if (MODE == 1) {   // K = G_U .* G_V
      float gv[TR][TC];
#pragma unroll
      for (int a = 0; a < TR; ++a) load_run(GVraw, i0 + a, gv[a]);
#pragma unroll
      for (int a = 0; a < TR; ++a)
#pragma unroll
        for (int q = 0; q < TC; ++q) S[a][q] *= gv[a][q];
    }
#pragma unroll
    for (int a = 0; a < TR; ++a)
#pragma unroll
      for (int q = 0; q < TC; ++q) {
        const int i = i0 + a, j = jb + q;
        if (i < w && j < w) {
          if (i == j) diag += S[a][q];
        } else {
          S[a][q] = (i == j) ? 1.f : 0.f;   // identity on the padding
        }
      }
    if (Graw != nullptr) {
#pragma unroll
      for (int a = 0; a < TR; ++a) store_run(Graw, i0 + a, S[a]);
    }
  }
  diag = warp_sum(diag);
  if (lane == 0) red[warp] = diag;
  __syncthreads();
  if (tid == 0) {
    float t = 0.f;
#pragma unroll
    for (int q = 0; q < NW; ++q) t += red[q];
    cpart[0] = t;
  }
  cluster.sync();
  float trace = 0.f;
#pragma unroll
  for (int q = 0; q < CS; ++q) trace += *cluster.map_shared_rank(&cpart[0], q);   // the same order everywhere
  const float eps = ((MODE == 0) || (w > 1)) ? (float)kEpsRel * trace / (float)w : 0.f;
  if (tile) {
#pragma unroll
    for (int a = 0; a < TR; ++a)
#pragma unroll
      for (int q = 0; q < TC; ++q)
        if (i0 + a < w && i0 + a == jb + q) S[a][q] += eps;
  }
  auto publish_rows = [&]() {
#pragma unroll
    for (int a = 0; a < TR; ++a) {
      if constexpr (TC == 4)
        *reinterpret_cast<float4*>(&pubR[lr0 + a][jb]) = make_float4(S[a][0], S[a][1], S[a][2], S[a][3]);
      else
        *reinterpret_cast<float2*>(&pubR[lr0 + a][jb]) = make_float2(S[a][0], S[a][1]);
    }
  };
  const int pr = lane / LPR, pc = (lane % LPR) * EPL;   // pivot warp: its entries of the 16 x 16 block
  const bool diagK = jb >= NB * c && jb < NB * c + NB;    // this thread's run lies in the own diagonal block
  if (c == 0) {
    if (tile) {
      publish_rows();
      if (diagK) {
#pragma unroll
        for (int a = 0; a < TR; ++a)
#pragma unroll
          for (int q = 0; q < TC; ++q) Pn[lr0 + a][jb + q] = S[a][q];
      }
    }
    __syncthreads();
    if (!tile) {
      float A[EPL];
#pragma unroll
      for (int e = 0; e < EPL; ++e) A[e] = Pn[pr][pc + e];
      warp_sweep<NB>(A, lane);
#pragma unroll
      for (int e = 0; e < EPL; ++e) pubQ[pr][pc + e] = -A[e];
    }
  }
  cluster.sync();

  const int nsteps = (int)cdiv(w, NB);
  for (int s = 0; s < nsteps; ++s) {
    const int k0 = NB * s, kn = k0 + NB;
    const bool owner = c == s, next = c == s + 1 && s + 1 < nsteps;
    const bool colsK = jb >= k0 && jb < k0 + NB;
    // 1. the step's pivot rows and inverse from their owner
    {
      const float4* srcR = reinterpret_cast<const float4*>(cluster.map_shared_rank(&pubR[0][0], s));
      const float4* srcQ = reinterpret_cast<const float4*>(cluster.map_shared_rank(&pubQ[0][0], s));
      for (int idx = tid; idx < NB * WP / 4 + NB * NB / 4; idx += NT + 32) {
        if (idx < NB * WP / 4) reinterpret_cast<float4*>(&Rk[0][0])[idx] = srcR[idx];
        else reinterpret_cast<float4*>(&Qk[0][0])[idx - NB * WP / 4] = srcQ[idx - NB * WP / 4];
      }
    }
    __syncthreads();
    // 2. W = Q Rk; the next owner's diagonal block as it stands
    if (tile) {
      for (int idx = tid; idx < NB * (WP / 4); idx += NT) {
        const int cc = idx / (WP / 4), q4 = (idx % (WP / 4)) * 4;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int d = 0; d < NB; ++d) {
          const float qv = Qk[cc][d];
          const float4 rv = *reinterpret_cast<const float4*>(&Rk[d][q4]);
          acc.x = fmaf(qv, rv.x, acc.x);
          acc.y = fmaf(qv, rv.y, acc.y);
          acc.z = fmaf(qv, rv.z, acc.z);
          acc.w = fmaf(qv, rv.w, acc.w);
        }
        *reinterpret_cast<float4*>(&Ws[cc][q4]) = acc;
      }
      if (next && diagK) {
#pragma unroll
        for (int a = 0; a < TR; ++a)
#pragma unroll
          for (int q = 0; q < TC; ++q) Pn[lr0 + a][jb + q - kn] = S[a][q];
      }
    }
    __syncthreads();
    // 3. the update beside the next pivot block's inverse
    if (tile) {
      if (owner) {
        if (colsK) {
#pragma unroll
          for (int a = 0; a < TR; ++a)
#pragma unroll
            for (int q = 0; q < TC; ++q) S[a][q] = -Qk[lr0 + a][jb + q - k0];
        } else {
#pragma unroll
          for (int a = 0; a < TR; ++a)
#pragma unroll
            for (int q = 0; q < TC; ++q) S[a][q] = Ws[lr0 + a][jb + q];
        }
      } else {
#pragma unroll 4
        for (int d = 0; d < NB; ++d) {
          const float2 rk = *reinterpret_cast<const float2*>(&Rk[d][i0]);
          float wv[TC];
          if constexpr (TC == 4) {
            const float4 t = *reinterpret_cast<const float4*>(&Ws[d][jb]);
            wv[0] = t.x; wv[1] = t.y; wv[2] = t.z; wv[3] = t.w;
          } else {
            const float2 t = *reinterpret_cast<const float2*>(&Ws[d][jb]);
            wv[0] = t.x; wv[1] = t.y;
          }
          const float rka[2] = {rk.x, rk.y};
#pragma unroll
          for (int a = 0; a < TR; ++a)
#pragma unroll
            for (int q = 0; q < TC; q += 2) {   // lane-wise fma.rn, the same rounding as fmaf
              const float2 s2 = __ffma2_rn(make_float2(-rka[a], -rka[a]), make_float2(wv[q], wv[q + 1]),
                                           make_float2(S[a][q], S[a][q + 1]));
              S[a][q] = s2.x;
              S[a][q + 1] = s2.y;
            }
        }
        if (colsK) {
#pragma unroll
          for (int q = 0; q < TC; ++q)
#pragma unroll
            for (int a = 0; a < TR; ++a) S[a][q] = Ws[jb + q - k0][i0 + a];
        }
      }
      if (next) publish_rows();
    } else if (next) {
      float A[EPL];
#pragma unroll
      for (int e = 0; e < EPL; ++e) A[e] = Pn[pr][pc + e];
#pragma unroll
      for (int d = 0; d < NB; ++d) {   // the fma chains of the tile owners, in the same order
        const float rk = Rk[d][kn + pr];
        float wv[EPL];
#pragma unroll
        for (int e = 0; e < EPL; e += 2) {
          const float2 t = *reinterpret_cast<const float2*>(&Ws[d][kn + pc + e]);
          wv[e] = t.x;
          wv[e + 1] = t.y;
        }
#pragma unroll
        for (int e = 0; e < EPL; ++e) A[e] = fmaf(-rk, wv[e], A[e]);
      }
      warp_sweep<NB>(A, lane);
#pragma unroll
      for (int e = 0; e < EPL; ++e) pubQ[pr][pc + e] = -A[e];
    }
    cluster.sync();   // the next owner's rows and inverse are published; Rk, Qk, Ws may be overwritten
  }

  if (MODE == 0) {
    if (op == nullptr) {
      if (tile) {
#pragma unroll
        for (int a = 0; a < TR; ++a) {
          float v[TC];
#pragma unroll
          for (int q = 0; q < TC; ++q) v[q] = -S[a][q];
          store_run(out, i0 + a, v);
        }
      }
    } else if constexpr (WP == 128) {
      // Ginv * 2^sg as hi / lo fp16 K-major operands (zero outside w x w), sg from the cluster-wide max |Ginv|
      float mx = 0.f;
      if (tile) {
#pragma unroll
        for (int a = 0; a < TR; ++a)
#pragma unroll
          for (int q = 0; q < TC; ++q)
            if (i0 + a < w && jb + q < w) mx = fmaxf(mx, fabsf(S[a][q]));
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      if (lane == 0) red[warp] = mx;
      __syncthreads();
      if (tid == 0) {
        float t = 0.f;
#pragma unroll
        for (int q = 0; q < NW; ++q) t = fmaxf(t, red[q]);
        cpart[1] = t;
      }
      cluster.sync();
#pragma unroll
      for (int q = 0; q < CS; ++q) mx = fmaxf(mx, *cluster.map_shared_rank(&cpart[1], q));
      const int sg = fp16_scale_exp(mx);
      const float sc = ldexpf(1.f, sg);
      if (tile) {
#pragma unroll
        for (int a = 0; a < TR; ++a) {
          const int i = i0 + a;
          __align__(8) __half hi[4];
          __align__(8) __half lo[4];
#pragma unroll
          for (int q = 0; q < 4; ++q) split_f16((i < w && jb + q < w) ? -S[a][q] * sc : 0.f, hi[q], lo[q]);
          const uint32_t off = k_major_offset(128u, (uint32_t)i, (uint32_t)jb);
          *reinterpret_cast<uint2*>(op + off) = *reinterpret_cast<const uint2*>(hi);
          *reinterpret_cast<uint2*>(op + 2 * 16384u + off) = *reinterpret_cast<const uint2*>(lo);
        }
      }
      if (c == 0 && tid == 0) *reinterpret_cast<int*>(op + 4 * 16384u) = sg;
    }
  } else if (tile) {
    float rv[TC];
#pragma unroll
    for (int q = 0; q < TC; ++q) rv[q] = jb + q < w ? r[jb + q] : 0.f;
#pragma unroll
    for (int a = 0; a < TR; ++a) {
      const int i = i0 + a;
      F2 acc2;
#pragma unroll
      for (int q = 0; q < TC; ++q)
        if (jb + q < w) acc2 = f2_add(acc2, -S[a][q] * rv[q]);
#pragma unroll
      for (int o = CG / 2; o > 0; o >>= 1) acc2 = f2_add(acc2, f2_shfl_xor(acc2, o));
      if (tc == 0 && i < w) out[i] = acc2.hi + acc2.lo;
    }
  }
  if (IN_INT) {   // every CTA has read its entries (the cluster barriers since): reset the own rows
    const int rows = min(NB, max(0, w - NB * c));
    int* base = Gint + (long long)NB * c * w;
    const int cnt = rows * w;
    if (vec) {
      for (int idx = tid; idx < cnt / 4; idx += NT + 32) reinterpret_cast<int4*>(base)[idx] = make_int4(0, 0, 0, 0);
    } else {
      for (int idx = tid; idx < cnt; idx += NT + 32) base[idx] = 0;
    }
  }
  cluster.sync();   // no CTA leaves while another may still read its shared memory
}

int gram_chunk(int w, int L, int* splits) {
  int sms = 152, dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int tiles = (int)(cdiv(w, GT) * cdiv(w, GT));
  int s = max(1, min((int)cdiv(sms, tiles), (int)cdiv(L, 4 * GY)));
  const int chunk = (int)round_up(cdiv(L, s), GY);
  *splits = (int)cdiv(L, chunk);
  return chunk;
}

// The register-tiled inverse (inv_kernel); EXTERND_INV=0 keeps the earlier 16-warp sweep, for comparisons.
bool tiled_inverse() {
  static const bool enabled = [] {
    const char* e = std::getenv("EXTERND_INV");
    return !(e && std::strcmp(e, "0") == 0);
  }();
  return enabled;
}

template <int W_PAD, int NB, int MODE>
cudaError_t launch_sweep_int_w(int* Gint, int w, const float* GVraw, const float* r, float* Graw, float* out,
                               cudaStream_t s, uint8_t* op) {
  const size_t smem = (size_t)W_PAD * (W_PAD + 1) * sizeof(int);   // the staged integer Gram
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(sweep32_kernel<W_PAD, NB, MODE, true>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  if (tiled_inverse())
    inv_kernel<W_PAD, MODE, true><<<1, inv_threads<W_PAD>(), 0, s>>>(nullptr, 0, w, GVraw, r, Graw, out, Gint, op,
                                                                      inv_p0_for<W_PAD>());
  else
    sweep32_kernel<W_PAD, NB, MODE, true><<<1, 544, smem, s>>>(nullptr, 0, w, GVraw, r, Graw, out, Gint, op);
  return cudaGetLastError();
}

template <int MODE>
cudaError_t launch_sweep_int(int* Gint, int w, const float* GVraw, const float* r, float* Graw, float* out,
                             cudaStream_t s, uint8_t* op = nullptr) {
  if (w <= 32) return launch_sweep_int_w<32, 8, MODE>(Gint, w, GVraw, r, Graw, out, s, nullptr);
  if (w <= 64) return launch_sweep_int_w<64, 16, MODE>(Gint, w, GVraw, r, Graw, out, s, nullptr);
  if (w <= 128) return launch_sweep_int_w<128, 16, MODE>(Gint, w, GVraw, r, Graw, out, s, op);
  return cudaErrorInvalidValue;   // callers use the float-partial Gram above 128 components
}

template <int MODE>
cudaError_t launch_sweep(const float* Gpart, int splits, int w, const float* GVraw, const float* r, float* Graw,
                         float* out, cudaStream_t s, uint8_t* op = nullptr) {
  // elements per lane RPW * CPL = W_PAD^2 / (32 * NWARP): 4 / 8 / 32 / 64
  // pivot-block sizes measured fastest on GB300: 8 up to w = 64, 16 at w = 128
  const bool tiled = tiled_inverse();
  if (w <= 32 && tiled) inv_kernel<32, MODE, false><<<1, inv_threads<32>(), 0, s>>>(Gpart, splits, w, GVraw, r, Graw, out, nullptr, nullptr, inv_p0_for<32>());
  else if (w <= 64 && tiled) inv_kernel<64, MODE, false><<<1, inv_threads<64>(), 0, s>>>(Gpart, splits, w, GVraw, r, Graw, out, nullptr, nullptr, inv_p0_for<64>());
  else if (w <= 128 && tiled) inv_kernel<128, MODE, false><<<1, inv_threads<128>(), 0, s>>>(Gpart, splits, w, GVraw, r, Graw, out, nullptr, op, inv_p0_for<128>());
  else if (w <= 32) sweep32_kernel<32, 8, MODE, false><<<1, 544, 0, s>>>(Gpart, splits, w, GVraw, r, Graw, out, nullptr, nullptr);
  else if (w <= 64) sweep32_kernel<64, 16, MODE, false><<<1, 544, 0, s>>>(Gpart, splits, w, GVraw, r, Graw, out, nullptr, nullptr);
  else if (w <= 128) sweep32_kernel<128, 16, MODE, false><<<1, 544, 0, s>>>(Gpart, splits, w, GVraw, r, Graw, out, nullptr, op);
  else sweep_kernel<256, 32, MODE><<<1, 32 * 32, 0, s>>>(Gpart, splits, w, GVraw, r, Graw, out);
  return cudaGetLastError();
}

// The cluster inverse and its launches (programmatic dependent launch of the next kernel when pdl). Off unless
// EXTERND_CLUSTER_INV=1: on this GPU the pivot rows' broadcast through distributed shared memory costs about as
// much per step as the single-CTA sweep's update, so the one-CTA inverse beside the product is faster overall.
bool cluster_inverse_enabled() {
  static const bool enabled = [] {
    const char* e = std::getenv("EXTERND_CLUSTER_INV");
    return e && std::strcmp(e, "1") == 0;
  }();
  return enabled;
}

template <int WP, int MODE, bool IN_INT>
cudaError_t launch_cluster_w(const float* Gpart, int splits, int w, const float* GVraw, const float* r, float* Graw,
                             float* out, int* Gint, uint8_t* op, bool pdl, cudaStream_t s) {
  constexpr int CS = InvClusterShape<WP>::CS;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(CS, 1, 1);
  cfg.blockDim = dim3(inv_cluster_threads<WP>(), 1, 1);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = CS;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, inv_cluster_kernel<WP, MODE, IN_INT>, Gpart, splits, w, GVraw, r, Graw, out, Gint,
                            op, pdl ? 1 : 0);
}

template <int MODE, bool IN_INT>
cudaError_t launch_cluster(const float* Gpart, int splits, int w, const float* GVraw, const float* r, float* Graw,
                           float* out, int* Gint, uint8_t* op, bool pdl, cudaStream_t s) {
  if (w <= 16 || w > 128) return cudaErrorInvalidValue;
  if (w <= 32) return launch_cluster_w<32, MODE, IN_INT>(Gpart, splits, w, GVraw, r, Graw, out, Gint, nullptr, pdl, s);
  if (w <= 64) return launch_cluster_w<64, MODE, IN_INT>(Gpart, splits, w, GVraw, r, Graw, out, Gint, nullptr, pdl, s);
  return launch_cluster_w<128, MODE, IN_INT>(Gpart, splits, w, GVraw, r, Graw, out, Gint, op, pdl, s);
}

}  // namespace

int inverse_cluster_size(int w) {
  if (!cluster_inverse_enabled() || w <= 16 || w > 128) return 0;
  return w <= 32 ? 2 : w <= 64 ? 4 : 8;
}

cudaError_t launch_inverse_cluster(const float* Gpart, int splits, int w, float* Graw, float* Ginv, cudaStream_t s,
                                   void* op, bool pdl) {
  if (op != nullptr && (w <= 64 || w > 128 || (reinterpret_cast<uintptr_t>(op) & 15) != 0)) return cudaErrorInvalidValue;
  return launch_cluster<0, false>(Gpart, splits, w, nullptr, nullptr, Graw, Ginv, nullptr, static_cast<uint8_t*>(op),
                                  pdl, s);
}

cudaError_t launch_inverse_cluster_int(int* Gint, int w, float* Graw, float* Ginv, cudaStream_t s, void* op, bool pdl) {
  if (op != nullptr && (w <= 64 || w > 128 || (reinterpret_cast<uintptr_t>(op) & 15) != 0)) return cudaErrorInvalidValue;
  return launch_cluster<0, true>(nullptr, 0, w, nullptr, nullptr, Graw, Ginv, Gint, static_cast<uint8_t*>(op), pdl,
                                 s);
}

cudaError_t launch_scales_cluster_int(int* GUint, const float* GVraw, const float* r, int w, float* d, cudaStream_t s,
                                      float* K) {
  return launch_cluster<1, true>(nullptr, 0, w, GVraw, r, K, d, GUint, nullptr, false, s);
}

int gram_splits(int w, int L) {
  int s;
  gram_chunk(w, L, &s);
  return s;
}

cudaError_t launch_gram(const int8_t* T, int ldt, int w, int L, const float* h, float* Gpart, int splits,
                        cudaStream_t s) {
  const int chunk = (int)round_up(cdiv(L, splits), GY);
  dim3 grid((unsigned)cdiv(w, GT), (unsigned)cdiv(w, GT), (unsigned)splits);   // every slice written
  gram_kernel<<<grid, 256, 0, s>>>(T, ldt, w, L, h, Gpart, chunk);
  return cudaGetLastError();
}

cudaError_t launch_inverse(const float* Gpart, int splits, int w, float* Graw, float* Ginv, cudaStream_t s,
                           void* op) {
  if (op != nullptr && (w <= 64 || w > 128 || (reinterpret_cast<uintptr_t>(op) & 15) != 0)) return cudaErrorInvalidValue;
  return launch_sweep<0>(Gpart, splits, w, nullptr, nullptr, Graw, Ginv, s, static_cast<uint8_t*>(op));
}

cudaError_t launch_inverse_int(int* Gint, int w, float* Graw, float* Ginv, cudaStream_t s, void* op) {
  if (op != nullptr && (w <= 64 || w > 128 || (reinterpret_cast<uintptr_t>(op) & 15) != 0)) return cudaErrorInvalidValue;
  return launch_sweep_int<0>(Gint, w, nullptr, nullptr, Graw, Ginv, s, static_cast<uint8_t*>(op));
}

cudaError_t launch_scales_int(int* GUint, const float* GVraw, const float* r, int w, float* d, cudaStream_t s,
                              float* K) {
  return launch_sweep_int<1>(GUint, w, GVraw, r, K, d, s);
}

cudaError_t launch_rvec(const int8_t* Ut, int ldu, int w, int L, const float* part, int splits, float* r,
                        cudaStream_t s) {
  rvec_kernel<<<(unsigned)w, 512, 0, s>>>(Ut, ldu, w, L, part, splits, r);
  return cudaGetLastError();
}

cudaError_t launch_scales(const float* GUpart, int splits, const float* GVraw, const float* r, int w, float* d,
                          cudaStream_t s, float* K) {
  return launch_sweep<1>(GUpart, splits, w, GVraw, r, K, d, s);
}

}  // namespace externd
