// The symmetric sweep of one small SPD block by one warp, shared by the Gram inverses.
#pragma once

#include <cuda_runtime.h>

namespace externd {

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

}  // namespace externd
