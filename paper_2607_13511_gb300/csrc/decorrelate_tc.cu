// Eq. 3 targets on the 5th-generation tensor cores, for blocks of 65 to 128 components:
//
//   X[a][x] = sum_b Ginv[a][b] P[b][x],   P = sum over the split-K slots of the residual product's partials,
//
// with the Eq. 2 statistics of each vector over the CTA's positions (the decorrelation's other output).
//
// One CTA per NPOS positions (16, 32 or 64; see decorrelate_tc_positions). Both operands sit in shared memory as
// fp16 hi + lo pairs, K-major with the 128-byte swizzle: A[a][b] = Ginv * 2^sg (M = 128 components) and
// B[x][b] = P * 2^sp (N = NPOS positions), the powers of two putting each operand's largest magnitude just under
// 2^14 (Ginv's over the whole matrix, P's over the CTA's tile). The Gram inverse writes A (on the side branch,
// beside the product) as the exact shared-memory image, which every CTA fetches with bulk copies while its
// threads sum the P slots. Three MMAs per 16-deep K step (hi.hi, hi.lo, lo.hi; lo.lo is below float32
// resolution) accumulate X^T in TMEM, one lane per component; in the epilogue the warp pair (q, q + 4) reads
// lane quadrant q, each warp half of the positions, and writes X and the Eq. 2 statistics of its half, which the
// pair then combines into the CTA's chunk.
#include <algorithm>

#include "grid.cuh"
#include "kernels.h"
#include "umma.cuh"

namespace externd {

namespace {

constexpr int kWp = 128;                                    // components, padded (MMA M, and K)
constexpr int kTcMinBlock = 64;   // narrower blocks keep the FMA kernels (faster there: fused targets at 2048^2)
constexpr uint32_t kAtomA = (uint32_t)kWp * 128u;           // one 64-wide K atom of A: 128 rows x 128 B
constexpr uint32_t kOpBytes = 4 * kAtomA;                   // A image: hi atoms 0, 1 then lo atoms 0, 1 (64 KB)
constexpr uint32_t kOpCopy = 16384;                         // bytes per bulk copy

template <int NPOS>
struct TcDecor {
  static constexpr uint32_t kAtomB = (uint32_t)NPOS * 128u;   // one K atom of B: NPOS rows x 128 B
  static constexpr uint32_t kSlot = (uint32_t)kWp * NPOS * 4u;  // one split-K slot of the P tile, float32
  static constexpr int kStage = NPOS == 64 ? 3 : (NPOS == 32 ? 7 : 14);   // slots staged at once (96-112 KB)
  static constexpr size_t kSmem = 1024 + kOpBytes + 2 * (2 * kAtomB) + kStage * kSlot;
  static constexpr int kPairs = NPOS / 2;                     // position pairs: the threads of one b group
  static constexpr int kBper = 128 / (256 / kPairs);          // components b per thread: 16, 8 or 4
  static constexpr uint32_t kTmemCols = NPOS < 32 ? 32u : (uint32_t)NPOS;
};

// hi / lo fp16 parts of N scaled floats, packed two per word.
template <int N>
__device__ __forceinline__ void split_pack(const float* v, float scale, uint32_t* h, uint32_t* l) {
#pragma unroll
  for (int e = 0; e < N / 2; ++e) {
    __half a0, b0, a1, b1;
    split_f16(v[2 * e] * scale, a0, b0);
    split_f16(v[2 * e + 1] * scale, a1, b1);
    h[e] = (uint32_t)__half_as_ushort(a0) | ((uint32_t)__half_as_ushort(a1) << 16);
    l[e] = (uint32_t)__half_as_ushort(b0) | ((uint32_t)__half_as_ushort(b1) << 16);
  }
}

__device__ __forceinline__ void bulk_copy(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "l"(src), "r"(bytes), "r"(bar)
               : "memory");
}

__device__ __forceinline__ void tmem_ld8(uint32_t taddr, uint32_t (&v)[8]) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
               : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7])
               : "r"(taddr));
}

// Outputs of the fused ternarization (MODE 2), as launch_apply's: T (int8, rows of ldt), its fp16 copy T16 (rows
// of ldt16; may be null), the K-major fp16 copy Tk (rows of ldk per position; may be null) and the exact Gram
// upper triangle gram[a * w + b], a <= b, added to (may be null).
struct ApplyOut {
  int8_t* T;
  long long ldt;
  __half* T16;
  long long ldt16;
  __half* Tk;
  long long ldk;
  int* gram;
  int8_t* gsc;         // with a Gram: the grid's tile Grams, gridDim.x x 128 x 128 (int8 counts, or float32)
  const float* h;      // weighted Gram T H T^T (per-position weights) into gramf instead of gram
  float* gramf;        // w x w float32, both triangles, written (not added to)
};

// MODE 0: X and the statistics; the last CTA finalizes the thresholds.
// MODE 1 (cooperative; bar: 2 zero words, left zero): every CTA finalizes its share of the thresholds after a
//   grid barrier, as in the FMA decorrelation.
// MODE 2 (cooperative; bar: 4 zero words, left zero): no X; after a second grid barrier every CTA ternarizes its
//   tile from TMEM (Eq. 2 with the finalized thresholds) into a K-major fp16 image in shared memory, from which
//   the warps write whole rows of T and T16 (the K-major copy Tk goes out position by position). With out.gram,
//   the tile's Gram T T^T is one more MMA (M = N = 128, K = NPOS) on that image, read back as int8
//   (|count| <= NPOS) and written to out.gsc in whole rows; after a third barrier CTA c adds rows c, c + G, ...
//   of all the tiles' Grams (warps over the tiles, lanes over the row, then the warps' sums in shared memory) to
//   out.gram's upper triangle (integer sums: the order does not matter). With out.h (the weighted V^T H V of
//   §2.5) the B operand is t_b(x) h(x) as a scaled fp16 hi + lo pair (two MMAs per K step), the tile Grams go to
//   out.gsc as float32, and after the third barrier the warps of the grid sum them in a fixed order (one warp per
//   16 entries of the upper triangle: 8 lane groups over the tiles, 4 entries per lane, then shuffles) into both
//   triangles of out.gramf.
template <int NPOS, int MODE>
__global__ void __launch_bounds__(256, 1) decorrelate_tc_kernel(const uint8_t* __restrict__ op, int w,
                                                                const float* __restrict__ part, int splits, int L,
                                                                float* __restrict__ X, int ldx, Stats st,
                                                                unsigned* __restrict__ bar,
                                                                unsigned* __restrict__ err, ApplyOut out) {
  using C = TcDecor<NPOS>;
  constexpr uint32_t kCols = MODE == 2 ? 256u : C::kTmemCols;   // MODE 2: the tile's Gram at column 128
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t sbase = (raw + 1023u) & ~1023u;
  uint8_t* const gbase = smem_raw + (sbase - raw);
  const uint32_t a_hi = sbase, a_lo = a_hi + 2 * kAtomA;   // the operand image: two K atoms each
  const uint32_t b_hi = a_hi + kOpBytes, b_lo = b_hi + 2 * C::kAtomB;
  uint8_t* const g_bhi = gbase + kOpBytes;
  uint8_t* const g_blo = g_bhi + 2 * C::kAtomB;
  __shared__ uint64_t op_bar, done_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ float red[8];
  __shared__ F2 half_sum[kWp];
  __shared__ u64 half_key[kWp];

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int x0 = blockIdx.x * NPOS;

  // ---- P tile: the slots go to shared memory by cp.async, kStage slots in flight at once (16, 8 or 4 bytes a
  //      copy, as L's alignment allows; positions past L zero-filled); then thread (pair xp, group bq) sums,
  //      slot by slot in order, P[kBper bq + j][x0 + 2 xp + c]
  const int sg = __ldg(reinterpret_cast<const int*>(op + kOpBytes));
  const int xp = tid % C::kPairs, bq = tid / C::kPairs;
  float pv[C::kBper][2];
#pragma unroll
  for (int j = 0; j < C::kBper; ++j) pv[j][0] = pv[j][1] = 0.f;
  {
    const uint32_t pst = sbase + kOpBytes + 4 * C::kAtomB;
    const float* const pstg = reinterpret_cast<const float*>(gbase + kOpBytes + 4 * C::kAtomB);
    const int vw = (L & 3) == 0 ? 4 : ((L & 1) == 0 ? 2 : 1);
    const int per_row = NPOS / vw, step = 256 / per_row;
    const int q = tid % per_row, r0 = tid / per_row;
    const int xq = x0 + q * vw;
    const bool xin = xq < L;
    const uint32_t nbytes = xin ? 4u * (uint32_t)vw : 0u;
    const long long sstride = (long long)w * L;
    auto stage = [&](int s0, int ns) {
      for (int u = 0; u < ns; ++u)
        for (int b = r0; b < w; b += step) {
          const float* src = part + (s0 + u) * sstride + (long long)b * L + (xin ? xq : 0);
          const uint32_t dst = pst + 4u * (uint32_t)((u * kWp + b) * NPOS + q * vw);
          if (vw == 4)
            asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(nbytes) : "memory");
          else if (vw == 2)
            asm volatile("cp.async.ca.shared.global [%0], [%1], 8, %2;" ::"r"(dst), "l"(src), "r"(nbytes) : "memory");
          else
            asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(dst), "l"(src), "r"(nbytes) : "memory");
        }
    };
    stage(0, min(C::kStage, splits));
    // the operand image, the barriers and the tensor memory while the first group is in flight
    if (tid == 0) {
      mbar_init(smem_addr(&op_bar), 1);
      mbar_init(smem_addr(&done_bar), 1);
      fence_barrier_init();
      mbar_expect_tx(smem_addr(&op_bar), kOpBytes);
#pragma unroll
      for (uint32_t c = 0; c < kOpBytes / kOpCopy; ++c)
        bulk_copy(a_hi + c * kOpCopy, op + c * kOpCopy, kOpCopy, smem_addr(&op_bar));
    }
    if (warp == 0) {
      tmem_alloc(smem_addr(&tmem_slot), kCols);
      tmem_relinquish();
    }
    for (int s0 = 0; s0 < splits; s0 += C::kStage) {
      const int ns = min(C::kStage, splits - s0);
      if (s0 > 0) stage(s0, ns);
      asm volatile("cp.async.wait_all;" ::: "memory");
      __syncthreads();
      for (int u = 0; u < ns; ++u)
#pragma unroll
        for (int j = 0; j < C::kBper; ++j) {
          const int b = C::kBper * bq + j;
          if (b < w) {
            const float2 v = *reinterpret_cast<const float2*>(pstg + (u * kWp + b) * NPOS + 2 * xp);
            pv[j][0] += v.x;
            pv[j][1] += v.y;
          }
        }
      __syncthreads();   // the stage is free for the next group
    }
  }
  // ---- 2^sp from max |P| of the tile; B row 2 xp + c, 8-byte quarter-chunk groups of 4 b
  float mp = 0.f;
#pragma unroll
  for (int j = 0; j < C::kBper; ++j) mp = fmaxf(mp, fmaxf(fabsf(pv[j][0]), fabsf(pv[j][1])));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) mp = fmaxf(mp, __shfl_xor_sync(0xffffffffu, mp, o));
  if (lane == 0) red[warp] = mp;
  __syncthreads();
  mp = red[0];
#pragma unroll
  for (int q = 1; q < 8; ++q) mp = fmaxf(mp, red[q]);
  const int sp = fp16_scale_exp(mp);
  const float scp = ldexpf(1.f, sp);
#pragma unroll
  for (int c = 0; c < 2; ++c) {
    const uint32_t xr = (uint32_t)(2 * xp + c);
#pragma unroll
    for (int e = 0; e < C::kBper / 4; ++e) {
      const int b0 = C::kBper * bq + 4 * e;
      float v[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) v[i] = pv[4 * e + i][c];
      uint32_t h[2], l[2];
      split_pack<4>(v, scp, h, l);
      const uint32_t off = (uint32_t)(b0 >> 6) * C::kAtomB + sw128_offset(xr, (uint32_t)((b0 & 63) >> 3)) +
                           8u * (uint32_t)((b0 >> 2) & 1);
      *reinterpret_cast<uint2*>(g_bhi + off) = make_uint2(h[0], h[1]);
      *reinterpret_cast<uint2*>(g_blo + off) = make_uint2(l[0], l[1]);
    }
  }
  fence_async_shared();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_slot;
  if (tid == 0) {
    if (mbar_wait(smem_addr(&op_bar), 0u, err)) {
      const uint32_t idesc = f16_idesc((uint32_t)kWp, (uint32_t)NPOS);
#pragma unroll
      for (int kk = 0; kk < kWp / 16; ++kk) {
        const uint32_t ko = (uint32_t)(kk >> 2), kb = 32u * (uint32_t)(kk & 3);
        const uint64_t ah = sw128_desc(a_hi + ko * kAtomA + kb), al = sw128_desc(a_lo + ko * kAtomA + kb);
        const uint64_t bh = sw128_desc(b_hi + ko * C::kAtomB + kb), bl = sw128_desc(b_lo + ko * C::kAtomB + kb);
        mma_f16(tmem, ah, bh, idesc, kk > 0 ? 1u : 0u);
        mma_f16(tmem, ah, bl, idesc, 1u);
        mma_f16(tmem, al, bh, idesc, 1u);
      }
    }
    mma_commit(smem_addr(&done_bar));   // arrives even when nothing was issued
  }
  __syncwarp();

  // ---- epilogue: warp q reads lane quadrant q % 4, positions (q / 4) NPOS / 2 .. + NPOS / 2 - 1
  const int quad = warp & 3, hpos = warp >> 2;
  const int a = 32 * quad + lane;
  const float ig = ldexpf(1.f, -sg), ip = ldexpf(1.f, -sp);
  const uint32_t trow = tmem + ((uint32_t)(32 * quad) << 16);   // this warp's lane quadrant
  {
    const bool ok = mbar_wait(smem_addr(&done_bar), 0u, err);
    const bool have = __all_sync(0xffffffffu, ok) != 0;
    tc_fence_after();
    AbsSum sum;
    u64 key = 0;
#pragma unroll
    for (int ch = 0; ch < NPOS / 16; ++ch) {
      const int col = hpos * (NPOS / 2) + 8 * ch;
      uint32_t d[8];
      if (have) {
        tmem_ld8(trow + (uint32_t)col, d);
        tmem_wait_ld();
      } else {
#pragma unroll
        for (int i = 0; i < 8; ++i) d[i] = 0u;
      }
      if (a < w) {
        float v[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) v[i] = __uint_as_float(d[i]) * ig * ip;
        const int xb = x0 + col;
        float* dst = X + (long long)a * ldx + xb;
        if (MODE == 2) {
        } else if (xb + 7 < L && (ldx & 3) == 0) {
          *reinterpret_cast<float4*>(dst) = make_float4(v[0], v[1], v[2], v[3]);
          *reinterpret_cast<float4*>(dst + 4) = make_float4(v[4], v[5], v[6], v[7]);
        } else {
#pragma unroll
          for (int i = 0; i < 8; ++i)
            if (xb + i < L) dst[i] = v[i];
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          if (xb + i < L) {
            sum.add(v[i]);
            const u64 kk = mag_key(v[i], (uint32_t)(xb + i));
            key = kk > key ? kk : key;
          }
        }
      }
    }
    if (hpos == 1) {
      half_sum[a] = sum.acc;
      half_key[a] = key;
    }
    tc_fence_before();
    __syncthreads();
    if (hpos == 0 && a < w) {
      const F2 s2 = f2_add(sum.acc, half_sum[a]);
      const u64 k2 = half_key[a] > key ? half_key[a] : key;
      put_stat(st, a, blockIdx.x, s2, k2);
    }
  }
  if (MODE != 2 && warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, kCols);
  }
  if (MODE == 0) {
    stats_done(st, w);
    return;
  }
  const unsigned G = gridDim.x;
  if (MODE == 1) {
    if (!grid_barrier(bar, G, err)) return;
    finalize_range(st, w, (int)blockIdx.x, (int)G);
    __syncthreads();
    if (threadIdx.x == 0) {   // exit ticket: the last CTA resets both words
      unsigned old;
      asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(old) : "l"(bar + 1) : "memory");
      if (old == G - 1u) {
        bar[0] = 0u;
        bar[1] = 0u;
      }
    }
    return;
  }
  // ---- MODE 2: thresholds of vectors blockIdx.x, blockIdx.x + G, ..., then every CTA ternarizes its tile
  bool ok = grid_barrier(bar + 0, G, err);
  if (ok) {
    finalize_range(st, w, (int)blockIdx.x, (int)G);
    ok = grid_barrier(bar + 1, G, err);
  }
  if (ok) {
    if (blockIdx.x == 0 && tid == 0) bar[0] = 0u;   // everyone has left barrier 1
    tc_fence_after();
    const float thv = a < w ? __ldcg(st.th.theta + a) : 0.f;
    const int fbv = a < w ? __ldcg(st.th.fallback + a) : 0;
    const unsigned argv = a < w ? __ldcg(st.th.arg + a) : 0u;
    uint8_t* const ts = gbase;   // the tile's trits as a K-major fp16 operand (rows a): the free A region
    uint8_t* const th_hi = gbase + 16384u;   // weighted: t h 2^sh as fp16 hi / lo, the same layout
    uint8_t* const th_lo = gbase + 32768u;
    uint8_t* const gst = gbase + 16384u;     // unweighted: the tile's int8 Gram, 128 rows x 128 B
    uint8_t* const tks = gbase + 49152u;     // Tk's position rows for the tile, NPOS x 128 fp16
    const bool wgram = out.h != nullptr, anyg = wgram || out.gram != nullptr;
    int sh = 0;
    if (wgram) {   // 2^sh from the tile's largest weight
      float hm = 0.f;
      if (tid < NPOS && x0 + tid < L) hm = fabsf(__ldg(out.h + x0 + tid));
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) hm = fmaxf(hm, __shfl_xor_sync(0xffffffffu, hm, o));
      if (lane == 0) red[warp] = hm;
      __syncthreads();
      hm = red[0];
#pragma unroll
      for (int q = 1; q < 8; ++q) hm = fmaxf(hm, red[q]);
      sh = fp16_scale_exp(hm);
    }
    const float sch = ldexpf(1.f, sh);
#pragma unroll
    for (int ch = 0; ch < NPOS / 16; ++ch) {
      const int col = hpos * (NPOS / 2) + 8 * ch, xb = x0 + col;
      uint32_t d[8];
      tmem_ld8(trow + (uint32_t)col, d);
      tmem_wait_ld();
      short t[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float v = __uint_as_float(d[i]) * ig * ip;   // as in the statistics above
        int8_t tt = 0;
        if (a < w && xb + i < L) {
          tt = ternary_of(v, thv);
          if (fbv && (uint32_t)(xb + i) == argv) tt = v < 0.f ? (int8_t)-1 : (int8_t)1;
        }
        t[i] = tt;
      }
      uint32_t h[4];
#pragma unroll
      for (int e = 0; e < 4; ++e)
        h[e] = (uint32_t)__half_as_ushort(__short2half_rn(t[2 * e])) |
               ((uint32_t)__half_as_ushort(__short2half_rn(t[2 * e + 1])) << 16);
      if (out.Tk != nullptr) {   // the K-major copy: position rows of 128 components, staged
        __half* const tr = reinterpret_cast<__half*>(tks) + col * kWp + a;
#pragma unroll
        for (int i = 0; i < 8; ++i) tr[i * kWp] = __short2half_rn(t[i]);
      }
      *reinterpret_cast<uint4*>(ts + k_major_offset(128u, (uint32_t)a, (uint32_t)col)) =
          make_uint4(h[0], h[1], h[2], h[3]);
      if (wgram) {
        float v[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) v[i] = xb + i < L ? (float)t[i] * __ldg(out.h + xb + i) : 0.f;
        uint32_t hh[4], hl[4];
        split_pack<8>(v, sch, hh, hl);
        const uint32_t off = k_major_offset(128u, (uint32_t)a, (uint32_t)col);
        *reinterpret_cast<uint4*>(th_hi + off) = make_uint4(hh[0], hh[1], hh[2], hh[3]);
        *reinterpret_cast<uint4*>(th_lo + off) = make_uint4(hl[0], hl[1], hl[2], hl[3]);
      }
    }
    fence_async_shared();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (anyg && tid == 0) {
        const uint32_t idesc = f16_idesc((uint32_t)kWp, (uint32_t)kWp);
#pragma unroll
        for (int kk = 0; kk < NPOS / 16; ++kk) {
          const uint64_t dsc = sw128_desc(sbase + 32u * (uint32_t)kk);
          if (wgram) {
            mma_f16(tmem + 128u, dsc, sw128_desc(sbase + 16384u + 32u * (uint32_t)kk), idesc, kk > 0 ? 1u : 0u);
            mma_f16(tmem + 128u, dsc, sw128_desc(sbase + 32768u + 32u * (uint32_t)kk), idesc, 1u);
          } else {
            mma_f16(tmem + 128u, dsc, dsc, idesc, kk > 0 ? 1u : 0u);
          }
        }
        mma_commit(smem_addr(&done_bar));
    }
    __syncwarp();
    {   // T and T16 rows from the staged trits, NPOS / 8 lanes per row (16 bytes of fp16 trits each): full rows
      constexpr int kCh = NPOS / 8, kRows = 32 / kCh;
      const int c = lane % kCh, xb = x0 + 8 * c;
      for (int r = warp * kRows + lane / kCh; r - lane / kCh < w; r += 8 * kRows) {
        if (r >= w || xb >= L) continue;
        const uint4 hv = *reinterpret_cast<const uint4*>(ts + k_major_offset(128u, (uint32_t)r, 8u * (uint32_t)c));
        const uint32_t hw4[4] = {hv.x, hv.y, hv.z, hv.w};
        uint32_t b[2] = {0u, 0u};
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int v = (int)__half2short_rz(__ushort_as_half((unsigned short)(hw4[i >> 1] >> (16 * (i & 1)))));
          b[i >> 2] |= (uint32_t)(uint8_t)(int8_t)v << (8 * (i & 3));
        }
        int8_t* Tr = out.T + (long long)r * out.ldt + xb;
        __half* Hr = out.T16 != nullptr ? out.T16 + (long long)r * out.ldt16 + xb : nullptr;
        if (xb + 7 < L) {
          *reinterpret_cast<uint2*>(Tr) = make_uint2(b[0], b[1]);
          if (Hr != nullptr) *reinterpret_cast<uint4*>(Hr) = hv;
        } else {
#pragma unroll
          for (int i = 0; i < 8; ++i)
            if (xb + i < L) {
              Tr[i] = (int8_t)(b[i >> 2] >> (8 * (i & 3)));
              if (Hr != nullptr) Hr[i] = __ushort_as_half((unsigned short)(hw4[i >> 1] >> (16 * (i & 1))));
            }
        }
      }
    }
    if (out.Tk != nullptr) {   // Tk rows x (components up to the next multiple of 8, zeros past w), 16 lanes a row
      const int lim = min((w + 7) & ~7, (int)min(out.ldk, (long long)kWp));
      const bool vec = (out.ldk & 7) == 0 && (reinterpret_cast<uintptr_t>(out.Tk) & 15) == 0;
      const int c8 = lane & 15;
      for (int pr = 2 * warp + (lane >> 4); pr - (lane >> 4) < NPOS; pr += 16) {
        const int x = x0 + pr;
        if (x >= L || 8 * c8 >= lim) continue;
        const uint4 v = *reinterpret_cast<const uint4*>(tks + pr * (2 * kWp) + 16 * c8);
        __half* dst = out.Tk + (long long)x * out.ldk + 8 * c8;
        if (vec && 8 * c8 + 8 <= lim) {
          *reinterpret_cast<uint4*>(dst) = v;
        } else {
          const uint32_t vv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
          for (int i = 0; i < 8; ++i)
            if (8 * c8 + i < lim) dst[i] = __ushort_as_half((unsigned short)(vv[i >> 1] >> (16 * (i & 1))));
        }
      }
    }
    if (anyg) {
      const bool gok = mbar_wait(smem_addr(&done_bar), 1u, err);
      const bool have = __all_sync(0xffffffffu, gok) != 0;
      tc_fence_after();
      if (have && wgram) {   // row a, columns 64 hpos .. + 63, unscaled, as float32
        float* dst = reinterpret_cast<float*>(out.gsc) + ((long long)blockIdx.x * kWp + a) * kWp + 64 * hpos;
        const float ih = ldexpf(1.f, -sh);
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          uint32_t g[16];
          tmem_ld16(trow + 128u + (uint32_t)(64 * hpos + 16 * c), g);
          tmem_wait_ld();
          if (a < w) {
#pragma unroll
            for (int i = 0; i < 16; i += 4)
              *reinterpret_cast<float4*>(dst + 16 * c + i) =
                  make_float4(__uint_as_float(g[i]) * ih, __uint_as_float(g[i + 1]) * ih,
                              __uint_as_float(g[i + 2]) * ih, __uint_as_float(g[i + 3]) * ih);
          }
        }
      } else if (have) {   // row a, columns 64 hpos .. + 63 of the tile's Gram as int8 in shared memory, 16-byte
        // chunks swizzled by row (the loads are warp-collective)
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          uint32_t g[16];
          tmem_ld16(trow + 128u + (uint32_t)(64 * hpos + 16 * c), g);
          tmem_wait_ld();
          uint32_t pk[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            pk[e] = 0u;
#pragma unroll
            for (int i = 0; i < 4; ++i) pk[e] |= ((uint32_t)(int)__uint_as_float(g[4 * e + i]) & 0xffu) << (8 * i);
          }
          *reinterpret_cast<uint4*>(gst + a * 128 + (((4 * hpos + c) ^ (a & 7)) << 4)) =
              make_uint4(pk[0], pk[1], pk[2], pk[3]);
        }
      }
      if (!wgram) {   // integer: the tile's Gram to out.gsc in whole rows; after a third barrier CTA c adds up rows
        // c, c + G, ... of all tiles (warp q takes tiles q, q + 8, ..., lane j entries 4j .. 4j + 3) into out.gram
        __syncthreads();
        int8_t* const gt = out.gsc + (long long)blockIdx.x * (kWp * kWp);
#pragma unroll
        for (int it = 0; it < 4; ++it) {
          const int r = 32 * it + (tid >> 3), c16 = tid & 7;
          *reinterpret_cast<uint4*>(gt + r * kWp + 16 * c16) =
              *reinterpret_cast<const uint4*>(gst + r * 128 + ((c16 ^ (r & 7)) << 4));
        }
        ok = grid_barrier(bar + 2, G, err);
        if (ok) {
          if (blockIdx.x == 0 && tid == 0) bar[1] = 0u;   // everyone has left barrier 2
          int* const rsum = reinterpret_cast<int*>(gst);   // 8 warps x 128 entries
          for (int ra = (int)blockIdx.x; ra < w; ra += (int)G) {
            int acc[4] = {0, 0, 0, 0};
            const int8_t* src = out.gsc + (long long)ra * kWp + 4 * lane;
            for (int c0 = warp; c0 < (int)G; c0 += 8 * 16) {
              unsigned v[16];
#pragma unroll
              for (int k = 0; k < 16; ++k) {
                const int c = c0 + 8 * k;
                v[k] = c < (int)G ? __ldcg(reinterpret_cast<const unsigned*>(src + (long long)c * (kWp * kWp))) : 0u;
              }
#pragma unroll
              for (int k = 0; k < 16; ++k)
#pragma unroll
                for (int i = 0; i < 4; ++i) acc[i] += (int)(int8_t)(v[k] >> (8 * i));
            }
            *reinterpret_cast<int4*>(rsum + warp * kWp + 4 * lane) = make_int4(acc[0], acc[1], acc[2], acc[3]);
            __syncthreads();
            if (tid < w && tid >= ra) {
              int tot = 0;
#pragma unroll
              for (int q = 0; q < 8; ++q) tot += rsum[q * kWp + tid];
              if (tot != 0) out.gram[(long long)ra * w + tid] += tot;
            }
            __syncthreads();
          }
        }
      } else {   // weighted: float32 tile Grams, summed in a fixed order after a third barrier
        ok = grid_barrier(bar + 2, G, err);
        if (ok) {
          if (blockIdx.x == 0 && tid == 0) bar[1] = 0u;   // everyone has left barrier 2
          // tasks: (row a, 16 columns from 16 u) for u = a / 16 .. cdiv(w, 16) - 1, rows in order; lane (q, j)
          // sums entries (a, 16 u + 4 j .. + 3) of the tiles q, q + 8, ..., 12 loads of 16 bytes in flight
          const int ng = (w + 15) >> 4, w16 = w >> 4, q = lane >> 2, j = lane & 3;
          const int ntask = ng * w - 16 * (w16 * (w16 - 1) / 2) - (w & 15) * w16;
          for (int task = (int)blockIdx.x * 8 + warp; task < ntask; task += (int)G * 8) {
            int ra = 0, t = task;
            for (; ra < w; ++ra) {
              const int n = ng - (ra >> 4);
              if (t < n) break;
              t -= n;
            }
            const int b0 = 16 * ((ra >> 4) + t) + 4 * j;
            const float* srcf = reinterpret_cast<const float*>(out.gsc) + (long long)ra * kWp + b0;
            float facc[4] = {0.f, 0.f, 0.f, 0.f};
            for (int c0 = q; c0 < (int)G; c0 += 8 * 12) {
              float4 v[12];
#pragma unroll
              for (int k = 0; k < 12; ++k) {
                const int c = c0 + 8 * k;
                v[k] = c < (int)G ? __ldcg(reinterpret_cast<const float4*>(srcf + (long long)c * kWp * kWp))
                                  : make_float4(0.f, 0.f, 0.f, 0.f);
              }
#pragma unroll
              for (int k = 0; k < 12; ++k) {
                facc[0] += v[k].x;
                facc[1] += v[k].y;
                facc[2] += v[k].z;
                facc[3] += v[k].w;
              }
            }
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              facc[i] += __shfl_xor_sync(0xffffffffu, facc[i], 4);
              facc[i] += __shfl_xor_sync(0xffffffffu, facc[i], 8);
              facc[i] += __shfl_xor_sync(0xffffffffu, facc[i], 16);
            }
            if (q == 0) {
#pragma unroll
              for (int i = 0; i < 4; ++i) {
                const int b = b0 + i;
                if (b >= ra && b < w) {
                  out.gramf[(long long)ra * w + b] = facc[i];
                  out.gramf[(long long)b * w + ra] = facc[i];
                }
              }
            }
          }
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, kCols);
  }
  if (!ok) return;
  if (tid == 0) {   // exit ticket: the last CTA resets the words still set (barrier 2 without the weighted Gram)
    unsigned old;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(old) : "l"(bar + 3) : "memory");
    if (old == G - 1u) {
      bar[1] = 0u;
      bar[2] = 0u;
      bar[3] = 0u;
    }
  }
}

// Sets the kernels' shared-memory limit (once) and returns how many CTAs of the cooperative variants the GPU
// holds at once (0 if the query failed).
template <int NPOS>
long long coop_capacity() {
  static long long cap = -1;
  if (cap < 0) {
    using C = TcDecor<NPOS>;
    cap = 0;
    int p1 = 0, p2 = 0, sms = 0, dev = 0;
    const int sm = (int)C::kSmem;
    if (cudaFuncSetAttribute(decorrelate_tc_kernel<NPOS, 0>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm) ==
            cudaSuccess &&
        cudaFuncSetAttribute(decorrelate_tc_kernel<NPOS, 1>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm) ==
            cudaSuccess &&
        cudaFuncSetAttribute(decorrelate_tc_kernel<NPOS, 2>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm) ==
            cudaSuccess &&
        cudaGetDevice(&dev) == cudaSuccess &&
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess &&
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&p1, decorrelate_tc_kernel<NPOS, 1>, 256, C::kSmem) ==
            cudaSuccess &&
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&p2, decorrelate_tc_kernel<NPOS, 2>, 256, C::kSmem) ==
            cudaSuccess)
      cap = (long long)std::min(p1, p2) * sms;
    cudaGetLastError();
  }
  return cap;
}

template <int NPOS, int MODE>
cudaError_t launch_coop(const uint8_t* op, int w, const float* part, int splits, int L, float* X, int ldx, Stats st,
                        cudaStream_t s, unsigned* bar, unsigned* err, const ApplyOut& out) {
  using C = TcDecor<NPOS>;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)cdiv(L, NPOS));
  cfg.blockDim = dim3(256);
  cfg.dynamicSmemBytes = C::kSmem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, decorrelate_tc_kernel<NPOS, MODE>, op, w, part, splits, L, X, ldx, st, bar, err,
                            out);
}

template <int NPOS>
cudaError_t launch_npos(const uint8_t* op, int w, const float* part, int splits, int L, float* X, int ldx, Stats st,
                        cudaStream_t s, unsigned* bar, unsigned* err) {
  using C = TcDecor<NPOS>;
  const long long grid = cdiv(L, NPOS);
  const ApplyOut none{};
  if (bar != nullptr && grid <= coop_capacity<NPOS>())
    return launch_coop<NPOS, 1>(op, w, part, splits, L, X, ldx, st, s, bar, err, none);
  coop_capacity<NPOS>();   // the shared-memory limit
  decorrelate_tc_kernel<NPOS, 0><<<(unsigned)grid, 256, C::kSmem, s>>>(op, w, part, splits, L, X, ldx, st, nullptr,
                                                                       err, none);
  return cudaGetLastError();
}

}  // namespace

bool decorrelate_tc_eligible(int w) { return w > kTcMinBlock && w <= kWp; }

size_t ginv_operand_bytes() { return (size_t)kOpBytes + 16; }

// The smallest tile (16, 32 or 64 positions) whose grid the GPU holds at once, so that the thresholds are
// finalized cooperatively; 64 where none is (then by the last CTA).
int decorrelate_tc_positions(int L) {
  if (cdiv(L, 16) <= coop_capacity<16>()) return 16;
  if (cdiv(L, 32) <= coop_capacity<32>()) return 32;
  return 64;
}

bool decorrelate_apply_tc_fits(int w, int L) {
  if (!decorrelate_tc_eligible(w)) return false;
  switch (decorrelate_tc_positions(L)) {
    case 16: return cdiv(L, 16) <= coop_capacity<16>();
    case 32: return cdiv(L, 32) <= coop_capacity<32>();
    default: return cdiv(L, 64) <= coop_capacity<64>();
  }
}

size_t decorrelate_apply_tc_scratch(int L) {
  return (size_t)cdiv(L, decorrelate_tc_positions(L)) * kWp * kWp * sizeof(float);
}

cudaError_t launch_decorrelate_apply_tc(const void* op, int w, const float* part, int splits, int L, Stats st,
                                        int8_t* T, long long ldt, int* gram, __half* T16, long long ldt16, __half* Tk,
                                        long long ldk, int8_t* gsc, unsigned* bar, unsigned* err, cudaStream_t s,
                                        const float* h, float* gramf) {
  const int npos = decorrelate_tc_positions(L);
  if ((h == nullptr) != (gramf == nullptr) || (h != nullptr && (gram != nullptr || gsc == nullptr)))
    return cudaErrorInvalidValue;
  if (!decorrelate_apply_tc_fits(w, L) || st.nchunk != (int)cdiv(L, npos) || op == nullptr || err == nullptr ||
      ((gram != nullptr || h != nullptr) && (gsc == nullptr || (reinterpret_cast<uintptr_t>(gsc) & 15) != 0)) ||
      bar == nullptr || T == nullptr || (reinterpret_cast<uintptr_t>(op) & 15) != 0 || (ldt & 7) != 0 ||
      (reinterpret_cast<uintptr_t>(T) & 7) != 0 ||
      (T16 != nullptr && ((ldt16 & 7) != 0 || (reinterpret_cast<uintptr_t>(T16) & 15) != 0)) ||
      (Tk != nullptr && ldk < w))
    return cudaErrorInvalidValue;
  const uint8_t* o = static_cast<const uint8_t*>(op);
  const ApplyOut out{T, ldt, T16, ldt16, Tk, ldk, gram, gsc, h, gramf};
  switch (npos) {
    case 16: return launch_coop<16, 2>(o, w, part, splits, L, nullptr, 0, st, s, bar, err, out);
    case 32: return launch_coop<32, 2>(o, w, part, splits, L, nullptr, 0, st, s, bar, err, out);
    default: return launch_coop<64, 2>(o, w, part, splits, L, nullptr, 0, st, s, bar, err, out);
  }
}

cudaError_t launch_decorrelate_tc(const void* op, int w, const float* part, int splits, int L, float* X, int ldx,
                                  Stats st, cudaStream_t s, unsigned* bar, unsigned* err) {
  const int npos = decorrelate_tc_positions(L);
  if (!decorrelate_tc_eligible(w) || st.nchunk != (int)cdiv(L, npos) || err == nullptr || op == nullptr ||
      (reinterpret_cast<uintptr_t>(op) & 15) != 0)
    return cudaErrorInvalidValue;
  const uint8_t* o = static_cast<const uint8_t*>(op);
  switch (npos) {
    case 16: return launch_npos<16>(o, w, part, splits, L, X, ldx, st, s, bar, err);
    case 32: return launch_npos<32>(o, w, part, splits, L, X, ldx, st, s, bar, err);
    default: return launch_npos<64>(o, w, part, splits, L, X, ldx, st, s, bar, err);
  }
}

}  // namespace externd
