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
// threads sum the P slots. Three MMAs per 16-deep K step (hi.hi, hi.lo,
// lo.hi; lo.lo is below float32 resolution) accumulate X^T in TMEM, one lane per component; in the epilogue the
// warp pair (q, q + 4) reads lane quadrant q, each warp half of the positions, and writes X and the Eq. 2
// statistics of its half, which the pair then combines into the CTA's chunk.
#include "grid.cuh"
#include "kernels.h"
#include "umma.cuh"

namespace externd {

namespace {

constexpr int kWp = 128;                                    // components, padded (MMA M, and K)
constexpr uint32_t kAtomA = (uint32_t)kWp * 128u;           // one 64-wide K atom of A: 128 rows x 128 B
constexpr uint32_t kOpBytes = 4 * kAtomA;                   // A image: hi atoms 0, 1 then lo atoms 0, 1 (64 KB)
constexpr uint32_t kOpCopy = 16384;                         // bytes per bulk copy

template <int NPOS>
struct TcDecor {
  static constexpr uint32_t kAtomB = (uint32_t)NPOS * 128u;   // one K atom of B: NPOS rows x 128 B
  static constexpr size_t kSmem = 1024 + kOpBytes + 2 * (2 * kAtomB);
  static constexpr int kPairs = NPOS / 2;                     // position pairs: the threads of one b group
  static constexpr int kBper = 128 / (256 / kPairs);          // components b per thread: 16, 8 or 4
  static constexpr int kSlotUnroll = 32 / kBper;              // slots loaded per round: 32 loads in flight
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

// COOP: thresholds finalized after a grid barrier by every CTA (bar: 2 zero words, left zero), as in the FMA
// decorrelation; otherwise by the last CTA.
template <int NPOS, bool COOP>
__global__ void __launch_bounds__(256, 1) decorrelate_tc_kernel(const uint8_t* __restrict__ op, int w,
                                                                const float* __restrict__ part, int splits, int L,
                                                                float* __restrict__ X, int ldx, Stats st,
                                                                unsigned* __restrict__ bar,
                                                                unsigned* __restrict__ err) {
  using C = TcDecor<NPOS>;
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
  if (tid == 0) {
    mbar_init(smem_addr(&op_bar), 1);
    mbar_init(smem_addr(&done_bar), 1);
    fence_barrier_init();
    mbar_expect_tx(smem_addr(&op_bar), kOpBytes);
#pragma unroll
    for (uint32_t c = 0; c < kOpBytes / kOpCopy; ++c) bulk_copy(a_hi + c * kOpCopy, op + c * kOpCopy, kOpCopy, smem_addr(&op_bar));
  }
  if (warp == 0) {
    tmem_alloc(smem_addr(&tmem_slot), C::kTmemCols);
    tmem_relinquish();
  }
  const int sg = __ldg(reinterpret_cast<const int*>(op + kOpBytes));

  // ---- P tile: thread (pair xp, group bq) sums, slot by slot in order, P[kBper bq + j][x0 + 2 xp + c]
  const int xp = tid % C::kPairs, bq = tid / C::kPairs;
  const int xa = x0 + 2 * xp;
  float pv[C::kBper][2];
#pragma unroll
  for (int j = 0; j < C::kBper; ++j) pv[j][0] = pv[j][1] = 0.f;
  {
    const bool vec2 = (L & 1) == 0 && xa + 1 < L;
    const long long sstride = (long long)w * L;
    for (int s0 = 0; s0 < splits; s0 += C::kSlotUnroll) {
      float2 v[C::kSlotUnroll][C::kBper];
#pragma unroll
      for (int u = 0; u < C::kSlotUnroll; ++u)
#pragma unroll
        for (int j = 0; j < C::kBper; ++j) {
          const int b = C::kBper * bq + j;
          v[u][j] = make_float2(0.f, 0.f);
          if (b < w && s0 + u < splits) {
            const float* src = part + (s0 + u) * sstride + (long long)b * L + xa;
            if (vec2) {
              v[u][j] = __ldg(reinterpret_cast<const float2*>(src));
            } else {
              v[u][j].x = xa < L ? __ldg(src) : 0.f;
              v[u][j].y = xa + 1 < L ? __ldg(src + 1) : 0.f;
            }
          }
        }
#pragma unroll
      for (int u = 0; u < C::kSlotUnroll; ++u)
#pragma unroll
        for (int j = 0; j < C::kBper; ++j) {
          pv[j][0] += v[u][j].x;
          pv[j][1] += v[u][j].y;
        }
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
  {
    const bool ok = mbar_wait(smem_addr(&done_bar), 0u, err);
    const bool have = __all_sync(0xffffffffu, ok) != 0;
    tc_fence_after();
    const float ig = ldexpf(1.f, -sg), ip = ldexpf(1.f, -sp);
    AbsSum sum;
    u64 key = 0;
#pragma unroll
    for (int ch = 0; ch < NPOS / 16; ++ch) {
      const int col = hpos * (NPOS / 2) + 8 * ch;
      uint32_t d[8];
      if (have) {
        tmem_ld8(tmem + ((uint32_t)(32 * quad) << 16) + (uint32_t)col, d);
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
        if (xb + 7 < L && (ldx & 3) == 0) {
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
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
  if (!COOP) {
    stats_done(st, w);
    return;
  }
  const unsigned G = gridDim.x;
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
}

// Sets the kernels' shared-memory limit (once) and returns how many CTAs of the cooperative variant the GPU holds
// at once (0 if the query failed).
template <int NPOS>
long long coop_capacity() {
  static long long cap = -1;
  if (cap < 0) {
    using C = TcDecor<NPOS>;
    cap = 0;
    int per_sm = 0, sms = 0, dev = 0;
    if (cudaFuncSetAttribute(decorrelate_tc_kernel<NPOS, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)C::kSmem) == cudaSuccess &&
        cudaFuncSetAttribute(decorrelate_tc_kernel<NPOS, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)C::kSmem) == cudaSuccess &&
        cudaGetDevice(&dev) == cudaSuccess &&
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess &&
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decorrelate_tc_kernel<NPOS, true>, 256, C::kSmem) ==
            cudaSuccess)
      cap = (long long)per_sm * sms;
    cudaGetLastError();
  }
  return cap;
}

template <int NPOS>
cudaError_t launch_npos(const uint8_t* op, int w, const float* part, int splits, int L, float* X, int ldx, Stats st,
                        cudaStream_t s, unsigned* bar, unsigned* err) {
  using C = TcDecor<NPOS>;
  const long long grid = cdiv(L, NPOS);
  if (bar != nullptr && grid <= coop_capacity<NPOS>()) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(256);
    cfg.dynamicSmemBytes = C::kSmem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, decorrelate_tc_kernel<NPOS, true>, op, w, part, splits, L, X, ldx, st, bar, err);
  }
  coop_capacity<NPOS>();   // the shared-memory limit
  decorrelate_tc_kernel<NPOS, false><<<(unsigned)grid, 256, C::kSmem, s>>>(op, w, part, splits, L, X, ldx, st,
                                                                           nullptr, err);
  return cudaGetLastError();
}

}  // namespace

bool decorrelate_tc_eligible(int w) { return w > 64 && w <= kWp; }

size_t ginv_operand_bytes() { return (size_t)kOpBytes + 16; }

// The smallest tile (16, 32 or 64 positions) whose grid the GPU holds at once, so that the thresholds are
// finalized cooperatively; 64 where none is (then by the last CTA).
int decorrelate_tc_positions(int L) {
  if (cdiv(L, 16) <= coop_capacity<16>()) return 16;
  if (cdiv(L, 32) <= coop_capacity<32>()) return 32;
  return 64;
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
