// Residual products on the tensor cores, fed by the Tensor Memory Accelerator (same products and accuracy scheme
// as product_tc.cu; used when R's rows are 16-byte aligned, i.e. n % 4 == 0):
//
//   V-step  part[s][a][c] = sum_{r in split s} U[r][a] R[r][c]       (§2.3 step 1, §2.4)
//   U-step  part[s][a][r] = sum_{c in split s} R[r][c] h[c] V[c][a]  (§2.3 step 1, §2.5)
//
// A CTA owns 128 output positions (MMA M) and all w components (N = w rounded up to 16), reducing over one
// split of the other dimension in stages of 64. Roles, all hand-offs through mbarriers with bounded waits:
//   R producer (1 thread)  TMA loads of the float32 R tile of a stage (128-byte swizzled boxes of 32 floats)
//                          into a ring of S32 slots; the stage's fp16 ternary tile (the MMA's B operand,
//                          128-byte swizzled K-major) goes into a ring of SB slots
//   converters (16 warps)  read a staged R tile into registers (lanes on consecutive positions) and free its
//                          slot at once, scale it by 2^s, split it into fp16 hi and lo and store the two A tiles
//                          into tensor memory (one position per lane, a ring of S16 stages); the same warps run
//                          the epilogue (TMEM -> split-K partials)
//   B producer (1 thread)  TMA loads of the ternary tiles, so that a B slot the MMAs still hold never delays R
//   MMA (one thread)       two kind::f16 MMAs per 16-deep K step (hi and lo from tensor memory against the same
//                          B in shared memory), commits that free the A stages and B slots
// R never passes through registers on its way into shared memory, and with A in tensor memory the shared memory
// holds six R stages: about 190 KB of copies in flight per SM, enough to keep the HBM queue full.
//
// Work is a sequence of units (128 positions x 64 reduction rows), tile-major. Classic plan: CTA (tile, split)
// takes one tile's units of its split, and writes partial slot `split`. Stream plan, used when tiles x splits
// would fill every SM (the w x w inverse runs beside the product on one SM, so one CTA of such a grid would wait
// for it): a 1-D grid of SMs - 1 CTAs splits all units evenly into contiguous runs; a run that crosses a tile
// boundary accumulates each tile in its own TMEM buffer (two, alternating) and writes each to the slot numbered
// by its place among the runs meeting that tile; slots a tile has no run for are written with zeros by the run
// that ends the tile. The converter warps store a finished tile's partials as soon as they have converted the
// next tile's last unit, so the MMAs keep going.
#include <cuda.h>

#include <algorithm>

#include <cstdlib>
#include <cstring>

#include "kernels.h"
#include "umma.cuh"

namespace externd {

namespace {

constexpr int kConvWarps = 16;
constexpr int kConv = kConvWarps * 32;
constexpr int kItems = 128 * 8 / kConv;   // (position, 8-deep K chunk) items per converter thread and stage
static_assert(kConv % 128 == 0 && kItems >= 1, "a converter thread keeps one position");
constexpr int kProducerWarp = kConvWarps, kMmaWarp = kConvWarps + 1, kBWarp = kConvWarps + 2;
constexpr int kThreads = (kConvWarps + 3) * 32;
constexpr int kStageK = 64;
constexpr int kS16 = 4, kSB = 4;   // A stages in tensor memory, ternary-tile slots (powers of two)
constexpr uint32_t kAcols = 64u;               // TMEM columns of one stage's A operand: 64 fp16 hi + 64 lo per row
constexpr uint32_t kStage32 = 128u * 64u * 4u;   // float32 R tile of one stage

struct TmaArgs {
  int m, n, w, wpad;
  const float* h;
  float* part;
  const float* maxabs;
  unsigned* err;
  int s32, sb, s16;
  uint32_t tmem_cols;
  uint32_t acol;       // first TMEM column of the A stages (after the accumulators)
  int nkt;             // units per tile: cdiv(Ly, 64)
  int cu;              // classic: units per split
  long long U;         // stream: all units (tiles x nkt)
  int slots;           // partial slots (classic: splits)
};


__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::
          "r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

// Byte offset of float c (0..31) of row r in a box of 128-byte rows with the 128-byte swizzle.
__device__ __forceinline__ uint32_t sw128_f32(uint32_t r, uint32_t c) {
  return r * 128u + ((((c >> 2) ^ (r & 7u)) << 4) | ((c & 3u) << 2));
}

__device__ __forceinline__ void split_pair(float x0, float x1, uint32_t& hi, uint32_t& lo) {
  const __half2 h = __floats2half2_rn(x0, x1);
  const float2 hb = __half22float2(h);
  const __half2 l = __floats2half2_rn(x0 - hb.x, x1 - hb.y);
  hi = *reinterpret_cast<const uint32_t*>(&h);
  lo = *reinterpret_cast<const uint32_t*>(&l);
}

__device__ __forceinline__ long long unit_owner(long long u, long long U, long long G) {
  return ((u + 1) * G + U - 1) / U - 1;   // the CTA whose run holds unit u (stream plan)
}

template <bool USTEP, bool STREAM>
__global__ void __launch_bounds__(kThreads, 1) product_tma_kernel(const __grid_constant__ CUtensorMap mapR,
                                                                  const __grid_constant__ CUtensorMap mapT,
                                                                  const TmaArgs p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t sbase = (raw + 1023u) & ~1023u;
  uint8_t* const gbase = smem_raw + (sbase - raw);
  const uint32_t tileB = (uint32_t)p.wpad * 128u;
  const uint32_t r32 = sbase;                                   // S32 x 32 KB
  const uint32_t rb = r32 + (uint32_t)p.s32 * kStage32;         // SB x tileB (1024-aligned: tileB = wpad * 128)
  const uint32_t bars = rb + (uint32_t)round_up((long long)kSB * tileB, 1024);
  const uint32_t full32 = bars, empty32 = full32 + 8u * p.s32;
  const uint32_t fullB = empty32 + 8u * p.s32, emptyB = fullB + 8u * kSB;
  const uint32_t full16 = emptyB + 8u * kSB, empty16 = full16 + 8u * kS16;
  const uint32_t accfull = empty16 + 8u * kS16, accempty = accfull + 16u;   // two TMEM accumulators
  const uint32_t tmem_slot = accempty + 16u;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int Lx = USTEP ? p.m : p.n;
  const int Ly = USTEP ? p.n : p.m;
  // this CTA's run of units [u0, u1)
  long long u0, u1;
  if (STREAM) {
    u0 = (long long)blockIdx.x * p.U / gridDim.x;
    u1 = ((long long)blockIdx.x + 1) * p.U / gridDim.x;
  } else {
    u0 = (long long)blockIdx.x * p.nkt + (long long)blockIdx.z * p.cu;
    u1 = min(u0 + p.cu, ((long long)blockIdx.x + 1) * p.nkt);
  }
  const int nk = (int)(u1 > u0 ? u1 - u0 : 0);

  // the power-of-two scale of the fp16 split: read by the converters once the roles split, so that the first
  // copies do not wait for this load
  float scale = 1.f, inv_scale = 1.f;
  auto load_scale = [&]() {
    float mx = __ldg(p.maxabs);
    if (USTEP && p.h != nullptr) mx *= __ldg(p.maxabs + 1);
    int ex = 0;
    if (mx > 0.f && mx <= 3.0e38f) frexpf(mx, &ex);
    const int sexp = max(-100, min(100, 14 - ex));
    scale = ldexpf(1.f, sexp);
    inv_scale = ldexpf(1.f, -sexp);
  };
  if (warp == kProducerWarp && lane == 0) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapR)) : "memory");
  } else if (warp == kBWarp && lane == 0) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapT)) : "memory");
  }

  if (tid == 0) {
    for (int s = 0; s < p.s32; ++s) {
      mbar_init(full32 + 8u * s, 1);
      mbar_init(empty32 + 8u * s, kConvWarps);
    }
    for (int s = 0; s < kSB; ++s) {
      mbar_init(fullB + 8u * s, 1);
      mbar_init(emptyB + 8u * s, 1);
    }
    for (int s = 0; s < kS16; ++s) {
      mbar_init(full16 + 8u * s, kConvWarps);
      mbar_init(empty16 + 8u * s, 1);
    }
    for (int j = 0; j < 2; ++j) {
      mbar_init(accfull + 8u * j, 1);
      mbar_init(accempty + 8u * j, kConvWarps);
    }
    fence_barrier_init();
  }
  if (warp == kMmaWarp) {
    tmem_alloc(tmem_slot, p.tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(gbase + (tmem_slot - sbase));

  bool ok = true;
  int seg = -1, seg_tile = -1;   // converters: the segment in progress and its tile
  // converter warps: partials of segment `sg` (tile `ts`) from TMEM buffer sg & 1 into its slot; false after a
  // timeout
  const int quad = warp & 3, group = warp >> 2;   // 2 warps per TMEM lane quadrant
  auto epilogue = [&](int sg, int ts) -> bool {
    const bool waited = mbar_wait(accfull + 8u * (sg & 1), (uint32_t)(sg / 2) & 1u, p.err);
    const bool have = __all_sync(0xffffffffu, waited) != 0;
    tc_fence_after();
    const int xi = ts * 128 + quad * 32 + lane;
    const long long tu0 = (long long)ts * p.nkt;
    int slot, zero_from = p.slots;
    if (STREAM) {
      const long long wf = unit_owner(tu0, p.U, gridDim.x);
      slot = (int)((long long)blockIdx.x - wf);
      if (u1 >= tu0 + p.nkt) zero_from = (int)(unit_owner(tu0 + p.nkt - 1, p.U, gridDim.x) - wf + 1);
    } else {
      slot = (int)blockIdx.z;
    }
    float* out = p.part + (long long)slot * p.w * Lx;
    for (int ch = group; ch < p.wpad / 16; ch += kConvWarps / 4) {
      uint32_t v[16];
      if (have) {
        tmem_ld16(tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)((sg & 1) * p.wpad + ch * 16), v);
        tmem_wait_ld();
      } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = 0u;
      }
      if (xi < Lx) {
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int a = ch * 16 + i;
          if (a < p.w) out[(long long)a * Lx + xi] = __uint_as_float(v[i]) * inv_scale;
        }
        for (int z = zero_from; STREAM && z < p.slots; ++z) {   // slots no run fills for this tile
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const int a = ch * 16 + i;
            if (a < p.w) p.part[((long long)z * p.w + a) * Lx + xi] = 0.f;
          }
        }
      }
    }
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(accempty + 8u * (sg & 1));
    return have;
  };
  if (warp == kProducerWarp) {
    // ------------------------------------------------------------------ TMA producer of R
    if (lane == 0) {
      int k = 0;   // stages whose R copies were issued
      int t = (int)(u0 / p.nkt), kc = (int)(u0 - (long long)t * p.nkt);   // advanced without divisions
      int s = 0, r = 0;                                                   // slot and round of stage k
      for (; k < nk; ++k) {
        if (STREAM && k > 0 && ++kc == p.nkt) {
          kc = 0;
          ++t;
        }
        const int x0 = t * 128, y0 = (STREAM ? kc : kc + k) * kStageK;   // a classic run stays in its tile
        if (r > 0 && !mbar_wait(empty32 + 8u * s, (uint32_t)(r - 1) & 1u, p.err)) break;
        mbar_expect_tx(full32 + 8u * s, kStage32);
        if (!USTEP) {
#pragma unroll
          for (int b = 0; b < 4; ++b) tma_load_2d(r32 + s * kStage32 + b * 8192u, &mapR, x0 + 32 * b, y0, full32 + 8u * s);
        } else {
#pragma unroll
          for (int b = 0; b < 2; ++b) tma_load_2d(r32 + s * kStage32 + b * 16384u, &mapR, y0 + 32 * b, x0, full32 + 8u * s);
        }
        if (++s == p.s32) {
          s = 0;
          ++r;
        }
      }
      // every copy this thread issued lands before the CTA can exit (bounded waits)
      for (int j = max(0, k - p.s32); j < k; ++j) mbar_wait(full32 + 8u * (j % p.s32), (uint32_t)(j / p.s32) & 1u, p.err);
    }
  } else if (warp == kBWarp) {
    // ------------------------------------------------------------------ TMA producer of the ternary operand
    // (its own thread, so that a B slot still held by the MMAs never holds up the next R copies)
    if (lane == 0) {
      int k = 0;
      int kc = (int)(u0 % p.nkt);
      for (; k < nk; ++k) {
        if (STREAM && k > 0 && ++kc == p.nkt) kc = 0;
        const int y0 = (STREAM ? kc : kc + k) * kStageK;
        const int sb = k & (kSB - 1);
        if (k >= kSB && !mbar_wait(emptyB + 8u * sb, (uint32_t)(k / kSB - 1) & 1u, p.err)) break;
        mbar_expect_tx(fullB + 8u * sb, tileB);
        tma_load_2d(rb + sb * tileB, &mapT, y0, 0, fullB + 8u * sb);
      }
      for (int j = max(0, k - kSB); j < k; ++j) mbar_wait(fullB + 8u * (j % kSB), (uint32_t)(j / kSB) & 1u, p.err);
    }
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = f16_idesc(128, (uint32_t)p.wpad);
      int seg = -1;
      int kc = STREAM ? (int)(u0 % p.nkt) - 1 : 0;
      for (int k = 0; k < nk; ++k) {
        if (STREAM && ++kc == p.nkt) kc = 0;
        const bool first = k == 0 || (STREAM && kc == 0);
        const bool last = k == nk - 1 || (STREAM && kc == p.nkt - 1);
        if (first) {
          ++seg;
          // a run holds at most two segments in flight: the third waits for the first one's partials
          if (seg >= 2 && !mbar_wait(accempty + 8u * (seg & 1), (uint32_t)(seg / 2 - 1) & 1u, p.err)) {
            ok = false;
            break;
          }
        }
        const int s = k & (kS16 - 1), sb = k & (kSB - 1);
        if (!mbar_wait(full16 + 8u * s, (uint32_t)(k / kS16) & 1u, p.err) ||
            !mbar_wait(fullB + 8u * sb, (uint32_t)(k / kSB) & 1u, p.err)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)((seg & 1) * p.wpad);
        // A from tensor memory: stage s holds hi in columns acol + 64 s .. + 31 and lo in the next 32, two fp16
        // (consecutive K) per column, one position per lane
        const uint32_t a_hi = tmem + p.acol + (uint32_t)s * kAcols, a_lo = a_hi + kAcols / 2, bt = rb + (uint32_t)sb * tileB;
#pragma unroll
        for (int kk = 0; kk < kStageK / 16; ++kk) {
          const uint64_t bd = sw128_desc(bt + 32u * kk);
          mma_f16_ts(d, a_hi + 8u * kk, bd, idesc, (!first || kk > 0) ? 1u : 0u);
          mma_f16_ts(d, a_lo + 8u * kk, bd, idesc, 1u);
        }
        mma_commit(empty16 + 8u * s);
        mma_commit(emptyB + 8u * sb);
        if (last) mma_commit(accfull + 8u * (seg & 1));
      }
    }
  } else {
    // ------------------------------------------------------------------ converters (and the epilogues)
    load_scale();
    // item i = tid + kConv q (q < kItems): A row x = i % 128 = tid % 128 (lanes on consecutive rows, the same
    // position for every item of a thread), K chunk o = i / 128
    const int x = tid & 127, o0 = tid >> 7;
    // V-step: float x of rows 8o + j sits at (8o + j) * 128 + (((x % 32) / 4 ^ j) * 16) + (x % 4) * 4 in box x / 32
    // (the 128-byte swizzle; 8o is a multiple of 8), the same offsets for every stage
    uint32_t voff[8];
#pragma unroll
    for (int j = 0; j < 8; ++j)
      voff[j] = (uint32_t)(x >> 5) * 8192u + (uint32_t)j * 128u + ((((uint32_t)(x & 31) >> 2) ^ (uint32_t)j) << 4) +
                ((uint32_t)(x & 3) << 2);
    // a finished segment whose partials are still to be written (stream plan), and its tile
    int pend = -1, pend_tile = -1;
    int t = (int)(u0 / p.nkt), kc = (int)(u0 - (long long)t * p.nkt);   // advanced without divisions
    int s = 0, r = 0;                                                   // R slot and round of stage k
    for (int k = 0; k < nk && ok; ++k, s = (s + 1 == p.s32) ? 0 : s + 1, r += (s == 0) ? 1 : 0) {
      if (STREAM && k > 0 && ++kc == p.nkt) {
        kc = 0;
        ++t;
      }
      if (k == 0 || (STREAM && kc == 0)) {
        if (pend >= 0) {   // (only with segments shorter than the accumulator turnaround)
          ok = epilogue(pend, pend_tile);
          pend = -1;
          if (!ok) break;
        }
        if (seg >= 0) {
          pend = seg;
          pend_tile = seg_tile;
        }
        ++seg;
        seg_tile = t;
      }
      const int s16 = k & (kS16 - 1);
      bool got = mbar_wait(full32 + 8u * s, (uint32_t)r & 1u, p.err);
      ok = __all_sync(0xffffffffu, got) != 0;
      if (!ok) break;
      // read the stage into registers and hand its slot back to the producer (the split below then overlaps the
      // next copies), then wait for the A slot the split writes into
      const uint8_t* st = gbase + (r32 - sbase) + (size_t)s * kStage32;
      const int y0 = (STREAM ? kc : kc + k) * kStageK;
      float v[kItems][8];
#pragma unroll
      for (int q = 0; q < kItems; ++q) {
        const int o = o0 + (kConv / 128) * q;
        if (!USTEP) {
          const uint8_t* bx = st + o * 1024;
#pragma unroll
          for (int j = 0; j < 8; ++j) v[q][j] = *reinterpret_cast<const float*>(bx + voff[j]);
        } else {
          // R[x0 + x][y0 + 8o .. +7]: box o / 4, row x, floats 8 (o % 4) .. +7 (two 16-byte chunks)
          const uint8_t* bx = st + (o >> 2) * 16384;
          const float4 a = *reinterpret_cast<const float4*>(bx + sw128_f32(x, 8 * (o & 3)));
          const float4 b = *reinterpret_cast<const float4*>(bx + sw128_f32(x, 8 * (o & 3) + 4));
          v[q][0] = a.x; v[q][1] = a.y; v[q][2] = a.z; v[q][3] = a.w;
          v[q][4] = b.x; v[q][5] = b.y; v[q][6] = b.z; v[q][7] = b.w;
        }
      }
      // hand the stage back: the next copy into it is an async-proxy write, so this thread's generic loads from
      // it are ordered before that write by a proxy fence (without it a lane's loads could still be in flight
      // when the copy landed, and one row of the partials took values of a later stage)
      fence_async_shared();
      __syncwarp();
      if (lane == 0) mbar_arrive(empty32 + 8u * s);
      got = k < kS16 || mbar_wait(empty16 + 8u * s16, (uint32_t)(k / kS16 - 1) & 1u, p.err);
      ok = __all_sync(0xffffffffu, got) != 0;
      if (!ok) break;
      tc_fence_after();   // the MMAs that read this A stage are complete: its columns may be rewritten
      // this warp's lanes (positions 32 (warp % 4) .. + 31) of stage s16's A columns in tensor memory
      const uint32_t a_hi = tmem + ((uint32_t)(quad * 32) << 16) + p.acol + (uint32_t)s16 * kAcols;
      const uint32_t a_lo = a_hi + kAcols / 2;
#pragma unroll
      for (int q = 0; q < kItems; ++q) {
        const int o = o0 + (kConv / 128) * q;
        const int valid = Ly - (y0 + 8 * o);   // elements of this chunk inside R
        if (USTEP && p.h != nullptr) {
          const int c = y0 + 8 * o;
#pragma unroll
          for (int j = 0; j < 8; ++j) v[q][j] *= (c + j < Ly) ? __ldg(p.h + c + j) : 0.f;
        }
        uint32_t hi[4], lo[4];
        if (valid >= 8) {
#pragma unroll
          for (int e = 0; e < 4; ++e) split_pair(v[q][2 * e] * scale, v[q][2 * e + 1] * scale, hi[e], lo[e]);
        } else {   // the last chunk of R: rows past its end enter as zeros
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float x0v = 2 * e < valid ? v[q][2 * e] * scale : 0.f;
            const float x1v = 2 * e + 1 < valid ? v[q][2 * e + 1] * scale : 0.f;
            split_pair(x0v, x1v, hi[e], lo[e]);
          }
        }
        // K chunk o (warp-uniform) is columns 4 o .. 4 o + 3: two fp16 of consecutive K per 32-bit column
        tmem_st4(a_hi + 4u * (uint32_t)o, hi[0], hi[1], hi[2], hi[3]);
        tmem_st4(a_lo + 4u * (uint32_t)o, lo[0], lo[1], lo[2], lo[3]);
      }
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(full16 + 8u * s16);
      // the previous segment's partials as soon as its MMAs have completed (checked without waiting after each
      // stage, so that the copies keep streaming meanwhile), at the latest when this segment is converted
      if (STREAM && pend >= 0) {
        const bool seg_end = k == nk - 1 || kc == p.nkt - 1;
        const bool done = __shfl_sync(0xffffffffu, lane == 0 && mbar_try_wait(accfull + 8u * (pend & 1), (uint32_t)(pend / 2) & 1u), 0);
        if (done || seg_end) {
          ok = epilogue(pend, pend_tile);
          pend = -1;
        }
      }
    }
  }
  // the last segment (or zeros after a failure, so every partial slot is written), once every role is done
  __syncthreads();
  if (warp < kConvWarps && nk > 0 && seg >= 0) epilogue(seg, seg_tile);

  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, p.tmem_cols);
  }
  // Launched early beside a w x w inverse (programmatic dependent launch): do not complete before it has, so that
  // the kernels after this one see its result. Without such a prerequisite this returns at once.
  asm volatile("griddepcontrol.wait;" ::: "memory");
}

typedef CUresult (*EncodeTiled)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiled encoder() {
  static EncodeTiled fn = [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess) {
      cudaGetLastError();
      return (EncodeTiled) nullptr;
    }
    return reinterpret_cast<EncodeTiled>(f);
  }();
  return fn;
}

struct TmaPlan {
  int wpad, s32, sb, s16;
  size_t smem;
};

TmaPlan tma_plan(int w) {
  TmaPlan t;
  t.wpad = (int)round_up(w, 16);
  const size_t tileB = (size_t)t.wpad * 128;
  // A stages live in tensor memory (4 x 64 columns beside up to 256 accumulator columns). The ternary tiles come
  // from L2 but under a saturated HBM queue still take a microsecond or more: four B slots let them be requested
  // well ahead of the MMAs, so that neither the MMAs nor (through the A stages) the converters wait for them; the
  // rest of the space holds R in flight.
  t.s16 = kS16;
  t.sb = kSB;
  const size_t budget = 227 * 1024 - 1024 - 512 - round_up((long long)t.sb * tileB, 1024);
  int s = 6;
  while (s > 1 && (size_t)s * kStage32 > budget) --s;
  t.s32 = s;
  t.smem = 1024 + (size_t)s * kStage32 + round_up((long long)t.sb * tileB, 1024) + 512;
  return t;
}

// Which plan the TMA product runs (see the header) and its partial slot count.
struct TmaWork {
  int stream, nkt, cu, slots, grid_x, grid_z;
  long long U;
};

TmaWork tma_work(int w, int Lx, int Ly) {
  int sms = 152, dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int sp, chunk;
  tc_split(w, Lx, Ly, &sp, &chunk);
  const int tiles = (int)cdiv(Lx, 128), nkt = (int)cdiv(Ly, kStageK);
  TmaWork t{0, nkt, chunk / kStageK, sp, tiles, sp, (long long)tiles * nkt};
  // SMs left to the product: the w x w inverse of the same half-step holds one (single CTA) or a cluster's worth
  const long long G = sms - std::max(1, inverse_cluster_size(w));
  static const bool stream_ok = [] {
    const char* e = std::getenv("EXTERND_STREAMK");
    return !(e && std::strcmp(e, "0") == 0);
  }();
  if (stream_ok && (long long)tiles * sp > G && G >= 1 && t.U >= G) {
    int S = 0;
    for (long long tt = 0; tt < tiles; ++tt) {
      const long long a = tt * nkt, b = a + nkt - 1;
      const long long oa = ((a + 1) * G + t.U - 1) / t.U - 1, ob = ((b + 1) * G + t.U - 1) / t.U - 1;
      S = std::max<int>(S, (int)(ob - oa + 1));
    }
    if (S <= sp + 2) {   // only where the extra partial slots stay few
      t.stream = 1;
      t.cu = 0;
      t.slots = S;
      t.grid_x = (int)G;
      t.grid_z = 1;
    }
  }
  return t;
}

template <bool USTEP>
cudaError_t launch_tma(const float* R, int m, int n, const __half* T, int ldt, int w, const float* h, float* part,
                       int splits, const float* maxabs, unsigned* err, cudaStream_t s, bool pdl) {
  EncodeTiled enc = encoder();
  if (enc == nullptr) return cudaErrorNotSupported;
  const int Lx = USTEP ? m : n, Ly = USTEP ? n : m;
  const TmaWork wk = tma_work(w, Lx, Ly);
  if (splits != wk.slots) return cudaErrorInvalidValue;
  const TmaPlan t = tma_plan(w);
  CUtensorMap mapR, mapT;
  {
    const cuuint64_t dims[2] = {(cuuint64_t)n, (cuuint64_t)m};
    const cuuint64_t strides[1] = {(cuuint64_t)n * 4};
    const cuuint32_t box[2] = {32u, USTEP ? 128u : 64u};
    const cuuint32_t es[2] = {1u, 1u};
    if (enc(&mapR, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float*>(R), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  {
    const cuuint64_t dims[2] = {(cuuint64_t)Ly, (cuuint64_t)w};
    const cuuint64_t strides[1] = {(cuuint64_t)ldt * 2};
    const cuuint32_t box[2] = {64u, (cuuint32_t)t.wpad};
    const cuuint32_t es[2] = {1u, 1u};
    if (enc(&mapT, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<__half*>(T), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  static bool configured[2] = {false, false};
  if (!configured[USTEP]) {
    cudaError_t e = cudaFuncSetAttribute(product_tma_kernel<USTEP, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         227 * 1024);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(product_tma_kernel<USTEP, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
    if (e != cudaSuccess) return e;
    configured[USTEP] = true;
  }
  // accumulators (the stream plan alternates two), then the A stages
  const uint32_t acol = (uint32_t)((wk.stream ? 2 : 1) * t.wpad);
  uint32_t cols = 32;
  while (cols < acol + (uint32_t)t.s16 * kAcols) cols <<= 1;
  TmaArgs a{m, n, w, t.wpad, h, part, maxabs, err, t.s32, t.sb, t.s16, cols, acol, wk.nkt, wk.cu, wk.U, wk.slots};
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)wk.grid_x, 1, (unsigned)wk.grid_z);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = t.smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // may start once the inverse is resident
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = pdl ? at : nullptr;
  cfg.numAttrs = pdl ? 1 : 0;
  if (wk.stream) return cudaLaunchKernelEx(&cfg, product_tma_kernel<USTEP, true>, mapR, mapT, a);
  return cudaLaunchKernelEx(&cfg, product_tma_kernel<USTEP, false>, mapR, mapT, a);
}

}  // namespace

bool tma_product_ok(const float* R, int n, const __half* T, int ldt) {
  return encoder() != nullptr && (n % 4) == 0 && ((uintptr_t)R & 15u) == 0 && ((uintptr_t)T & 15u) == 0 &&
         (ldt % 8) == 0;
}

int tma_product_slots(int w, int Lx, int Ly) { return tma_work(w, Lx, Ly).slots; }

cudaError_t launch_product_v_tma(const float* R, int m, int n, const __half* Ut, int ldu, int w, float* part,
                                 int splits, const float* maxabs, unsigned* err, cudaStream_t s, bool pdl) {
  return launch_tma<false>(R, m, n, Ut, ldu, w, nullptr, part, splits, maxabs, err, s, pdl);
}

cudaError_t launch_product_u_tma(const float* R, int m, int n, const __half* Vt, int ldv, int w, const float* h,
                                 float* part, int splits, const float* maxabs, unsigned* err, cudaStream_t s,
                                 bool pdl) {
  return launch_tma<true>(R, m, n, Vt, ldv, w, h, part, splits, maxabs, err, s, pdl);
}

}  // namespace externd
