// Small dense algebra of a block: ternary Gram matrices, (G + eps I)^-1 for Eq. 3, and the joint scale solve of
// Eq. 4.
//
// Gram matrices of ternary factors are integer counts (exact in float up to 2^24); with importance weights the
// U-step Gram is sum_y h_y v_a(y) v_b(y) in float. The inverse uses the symmetric sweep operator (Gauss-Jordan
// on an SPD matrix, no pivoting needed): one 1024-thread CTA holds the w x w matrix in registers, one row per
// 1024/W_PAD threads, and sweeps the w pivots with one barrier per pivot. Sweeping every pivot of S = G turns S
// into -G^-1.
#include "kernels.h"
#include "umma.cuh"

namespace externd {

namespace {

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

// One warp inverts an NB x NB SPD block by the symmetric sweep: lane l holds EPL = NB^2/32 entries of row
// l / LPR (LPR = NB / EPL lanes per row), columns (l % LPR) * EPL + e. Per pivot kk every lane fetches with
// shuffles the pivot-row entries of its columns (from the lane of row kk with the same column group), the pivot,
// and its row's pivot-column entry (by symmetry the entry of row r in column kk sits at a register index that is
// the same for every lane), then updates its entries. On return A holds -P^-1.
template <int NB>
__device__ __forceinline__ void warp_sweep(float (&A)[NB * NB / 32], int lane) {
  constexpr int EPL = NB * NB / 32, LPR = NB / EPL;
  const int r = lane / LPR, cg = lane % LPR, cb = cg * EPL;
#pragma unroll
  for (int kk = 0; kk < NB; ++kk) {
    float akc[EPL];
#pragma unroll
    for (int e = 0; e < EPL; ++e) akc[e] = __shfl_sync(0xffffffffu, A[e], kk * LPR + cg);
    const float p = __shfl_sync(0xffffffffu, A[kk % EPL], kk * LPR + kk / EPL);
    const float ark0 = __shfl_sync(0xffffffffu, A[kk % EPL], r * LPR + kk / EPL);
    const float ip = __fdividef(1.f, p);
    const float ark = ark0 * ip;   // P[r][kk] / p
#pragma unroll
    for (int e = 0; e < EPL; ++e) {
      const int c = cb + e;
      float v = fmaf(-ark, akc[e], A[e]);
      v = (c == kk) ? ark : v;
      v = (r == kk) ? ((c == kk) ? -ip : akc[e] * ip) : v;
      A[e] = v;
    }
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

int gram_chunk(int w, int L, int* splits) {
  int sms = 152, dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int tiles = (int)(cdiv(w, GT) * cdiv(w, GT));
  int s = max(1, min((int)cdiv(sms, tiles), (int)cdiv(L, 4 * GY)));
  const int chunk = (int)round_up(cdiv(L, s), GY);
  *splits = (int)cdiv(L, chunk);
  return chunk;
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
  if (w <= 32) sweep32_kernel<32, 8, MODE, false><<<1, 544, 0, s>>>(Gpart, splits, w, GVraw, r, Graw, out, nullptr, nullptr);
  else if (w <= 64) sweep32_kernel<64, 16, MODE, false><<<1, 544, 0, s>>>(Gpart, splits, w, GVraw, r, Graw, out, nullptr, nullptr);
  else if (w <= 128) sweep32_kernel<128, 16, MODE, false><<<1, 544, 0, s>>>(Gpart, splits, w, GVraw, r, Graw, out, nullptr, op);
  else sweep_kernel<256, 32, MODE><<<1, 32 * 32, 0, s>>>(Gpart, splits, w, GVraw, r, Graw, out);
  return cudaGetLastError();
}

}  // namespace

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
