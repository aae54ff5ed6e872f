// Small dense algebra of a block: ternary Gram matrices, (G + eps I)^-1 for Eq. 3, and the joint scale solve of
// Eq. 4.
//
// Gram matrices of ternary factors are integer counts (exact in float up to 2^24); with importance weights the
// U-step Gram is sum_y h_y v_a(y) v_b(y) in float. The inverse uses the symmetric sweep operator (Gauss-Jordan
// on an SPD matrix, no pivoting needed): one 1024-thread CTA holds the w x w matrix in registers, one row per
// 1024/W_PAD threads, and sweeps the w pivots with one barrier per pivot. Sweeping every pivot of S = G turns S
// into -G^-1.
#include "kernels.h"

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
// Symmetric sweep: sweeping pivot k maps S to S - S[:,k] S[k,:] / p with row and column k replaced by
// S[k,:] / p and S[k][k] by -1/p (p = S[k][k]); after all pivots S = -G^-1. Every intermediate S stays
// symmetric, so the pivot column equals the pivot row: the threads that own row k publish it to shared memory
// with vector stores, every thread applies the same branch-free rank-1 update to its EPT elements, and row k
// and column k are fixed up with predicated selects. One barrier per pivot.
template <int W_PAD, int NT, int MODE>
__global__ void __launch_bounds__(NT) sweep_kernel(const float* __restrict__ Gpart, int splits, int w,
                                                   const float* __restrict__ GVraw, const double* __restrict__ r,
                                                   float* __restrict__ Graw, float* __restrict__ out) {
  constexpr int TPR = NT / W_PAD;         // threads per row
  constexpr int EPT = W_PAD / TPR;        // elements per thread (a multiple of 4)
  static_assert(EPT % 4 == 0, "EPT must allow 16-byte row stores");
  __shared__ __align__(16) float rowk[2][W_PAD];
  __shared__ double dsum[32];
  const int tid = threadIdx.x;
  const int i = tid / TPR, q = tid % TPR;
  const int j0 = q * EPT;
  float S[EPT];
  double diag = 0.0;
#pragma unroll
  for (int e = 0; e < EPT; ++e) {
    const int j = j0 + e;
    float v = (i == j) ? 1.f : 0.f;
    if (i < w && j < w) {
      float g = 0.f;
      for (int sp = 0; sp < splits; ++sp) g += Gpart[(long long)sp * w * w + (long long)i * w + j];
      if (MODE == 0) {
        Graw[(long long)i * w + j] = g;
      } else {
        g *= GVraw[(long long)i * w + j];
      }
      v = g;
      if (i == j) diag = (double)g;
    }
    S[e] = v;
  }
  // trace -> ridge
  double t = warp_sum(diag);
  if ((tid & 31) == 0) dsum[tid >> 5] = t;
  __syncthreads();
  if (tid < 32) {
    double u = warp_sum(tid < NT / 32 ? dsum[tid] : 0.0);
    if (tid == 0) dsum[0] = u;
  }
  __syncthreads();
  const bool ridge = (MODE == 0) || (w > 1);
  const float eps = ridge ? (float)(kEpsRel * dsum[0] / (double)w) : 0.f;
#pragma unroll
  for (int e = 0; e < EPT; ++e)
    if (i < w && j0 + e == i) S[e] += eps;

  for (int k = 0; k < w; ++k) {
    float* rk = rowk[k & 1];
    if (i == k) {
#pragma unroll
      for (int e = 0; e < EPT; e += 4)
        *reinterpret_cast<float4*>(&rk[j0 + e]) = make_float4(S[e], S[e + 1], S[e + 2], S[e + 3]);
    }
    __syncthreads();
    const float ip = __frcp_rn(rk[k]);
    const float ci = rk[i];           // S[i][k] = S[k][i]
    const float f = -ci * ip;
    const bool own_row = (i == k);
#pragma unroll
    for (int e = 0; e < EPT; e += 4) {
      const float4 c4 = *reinterpret_cast<const float4*>(&rk[j0 + e]);
      const float cj[4] = {c4.x, c4.y, c4.z, c4.w};
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int j = j0 + e + u;
        float v = fmaf(f, cj[u], S[e + u]);
        v = own_row ? cj[u] * ip : v;       // row k: S[k][j] / p
        v = (j == k) ? (own_row ? -ip : ci * ip) : v;   // column k: S[i][k] / p; pivot: -1/p
        S[e + u] = v;
      }
    }
  }

  if (MODE == 0) {
    if (i < w) {
#pragma unroll
      for (int e = 0; e < EPT; ++e) {
        const int j = j0 + e;
        if (j < w) out[(long long)i * w + j] = -S[e];
      }
    }
  } else {
    double acc = 0.0;
#pragma unroll
    for (int e = 0; e < EPT; ++e) {
      const int j = j0 + e;
      if (i < w && j < w) acc += -(double)S[e] * r[j];
    }
#pragma unroll
    for (int o = TPR / 2; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (q == 0 && i < w) out[i] = (float)acc;
  }
}

__global__ void __launch_bounds__(256) rvec_kernel(const int8_t* __restrict__ Ut, int ldu, int w, int L,
                                                   const float* __restrict__ part, int splits,
                                                   double* __restrict__ r) {
  __shared__ double red[8];
  const int a = blockIdx.x;
  float acc = 0.f;
  for (int y = threadIdx.x; y < L; y += 256) {
    const int8_t u = Ut[(long long)a * ldu + y];
    if (u != 0) {
      float p = 0.f;
      for (int s = 0; s < splits; ++s) p += part[((long long)s * w + a) * L + y];
      acc += (u > 0) ? p : -p;
    }
  }
  double v = warp_sum((double)acc);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
  __syncthreads();
  if (threadIdx.x == 0) {
    double s = 0.0;
    for (int q = 0; q < 8; ++q) s += red[q];
    r[a] = s;
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

template <int MODE>
cudaError_t launch_sweep(const float* Gpart, int splits, int w, const float* GVraw, const double* r, float* Graw,
                         float* out, cudaStream_t s) {
  // 16 elements per thread up to w = 128 (one barrier per pivot; the update is a branch-free rank-1 FMA)
  if (w <= 32) sweep_kernel<32, 128, MODE><<<1, 128, 0, s>>>(Gpart, splits, w, GVraw, r, Graw, out);
  else if (w <= 64) sweep_kernel<64, 256, MODE><<<1, 256, 0, s>>>(Gpart, splits, w, GVraw, r, Graw, out);
  else if (w <= 128) sweep_kernel<128, 1024, MODE><<<1, 1024, 0, s>>>(Gpart, splits, w, GVraw, r, Graw, out);
  else sweep_kernel<256, 1024, MODE><<<1, 1024, 0, s>>>(Gpart, splits, w, GVraw, r, Graw, out);
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

cudaError_t launch_inverse(const float* Gpart, int splits, int w, float* Graw, float* Ginv, cudaStream_t s) {
  return launch_sweep<0>(Gpart, splits, w, nullptr, nullptr, Graw, Ginv, s);
}

cudaError_t launch_rvec(const int8_t* Ut, int ldu, int w, int L, const float* part, int splits, double* r,
                        cudaStream_t s) {
  rvec_kernel<<<(unsigned)w, 256, 0, s>>>(Ut, ldu, w, L, part, splits, r);
  return cudaGetLastError();
}

cudaError_t launch_scales(const float* GUpart, int splits, const float* GVraw, const double* r, int w, float* d,
                          cudaStream_t s) {
  return launch_sweep<1>(GUpart, splits, w, GVraw, r, nullptr, d, s);
}

}  // namespace externd
