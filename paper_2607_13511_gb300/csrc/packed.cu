// Inference with the packed factors (§2.6): y = B diag(D) (C x).
//
// Each ternary entry is stored as a 2-bit code (bit 0 set for a nonzero, bit 1 set for a negative entry) -- the
// paper's mask+sign information at a fixed position, so rows stream with coalesced 16-byte loads (the nonzero
// count the packer returns gives Eq. 5's storage of the sparse form). The codes are laid out in the register
// order of the tensor-core A fragment (mma.m16n8k16, row-major A): a 32-bit word holds the 16 codes one lane
// needs for two k-steps, placed so that (word << 2p) & 0xC000C000 is the bf16 pair of fragment register p with
// value +-2 or 0 (code bit 0 lands on the exponent's top bit, bit 1 on the sign). Decoding is thus two integer
// operations per pair of weights and the products run on the tensor cores, which keeps the product at the rate
// the packed bits stream from memory; a scalar loop over the bits would need several instructions per weight.
//
// Word layout of a rows x cols matrix: RT = ceil(rows / 16) row tiles, G = ceil(cols / 128) groups of 128
// columns, word ((rt * G + grp) * 32 + lane) * 4 + q, lane = 4 g + t. Fragment pair p (0..7) of word q is k-step
// ks = 2q + p / 4 of the group, register r = p % 4: row 16 rt + g + 8 (r & 1), columns 128 grp + 16 ks +
// 8 (r >> 1) + 2t (low half) and + 1 (high half); the low element's code sits at bits 14 - 2p, the high one's at
// 30 - 2p. Entries past rows or cols are zero.
//
// The vector is split exactly into three bf16 parts (x = hi + mid + lo: bf16 keeps fp32's exponent range and 3 x 8
// significant bits cover fp32's 24), which are the first three columns of the B fragment. Every product is exact,
// so the result differs from a float64 product only by the tensor core's fp32 accumulation and the final additions
// (three parts, then the partial sums of the warps sharing a row, each in a fixed order).
//
// Work split (stream-K): the units (pair of row tiles = 32 rows) x (group of 128 columns) are divided evenly over
// all warps of a persistent grid as contiguous runs in row-major unit order; each warp streams its run through a
// ring of cp.async stages in shared memory, six units in flight beyond the one being multiplied. When its run
// leaves a row-tile pair the warp stores its partial row sums; once the run is done it takes a ticket for each pair
// it met, and the warp holding a pair's last ticket adds the pair's partials in warp order (so the result is
// deterministic) and writes the rows. The vector's B fragments are prepared once in global memory: by a small
// kernel for x and, for the second product, by the finishing warps of the first (which own z's rows).
#include "kernels.h"
#include "umma.cuh"

#include <cuda_bf16.h>

namespace externd {

namespace {


__device__ __forceinline__ uint32_t code_of(int8_t t) { return t == 0 ? 0u : (t > 0 ? 1u : 3u); }

__global__ void __launch_bounds__(256) pack_kernel(const int8_t* __restrict__ T, long long rows, long long cols,
                                                   long long ldt, uint32_t* __restrict__ words,
                                                   unsigned long long* __restrict__ nnz) {
  const long long G = (cols + 127) / 128, RT = (rows + 15) / 16;
  const long long id = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  unsigned long long cnt = 0;
  if (id < RT * G * 128) {
    const int q = (int)(id & 3), lane = (int)((id >> 2) & 31);
    const long long tg = id >> 7, grp = tg % G, rt = tg / G;
    const int g = lane >> 2, t = lane & 3;
    uint32_t word = 0;
#pragma unroll
    for (int p = 0; p < 8; ++p) {
      const int ks = 2 * q + (p >> 2), r = p & 3;
      const long long row = 16 * rt + g + 8 * (r & 1);
      const long long col = 128 * grp + 16 * ks + 8 * (r >> 1) + 2 * t;
      if (row < rows) {
        const int8_t* src = T + row * ldt;
        if (col < cols) word |= code_of(src[col]) << (14 - 2 * p);
        if (col + 1 < cols) word |= code_of(src[col + 1]) << (30 - 2 * p);
      }
    }
    words[id] = word;
    cnt = (unsigned long long)__popc(word & 0x55555555u);
  }
  for (int o = 16; o > 0; o >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
  if ((threadIdx.x & 31) == 0 && cnt != 0) atomicAdd(nnz, cnt);
}

__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Two k-steps of one row tile: word w holds the A fragments of both, (b.x, b.y) and (b.z, b.w) the B fragments.
__device__ __forceinline__ void mma_word(float (&d)[4], uint32_t w, const uint4& b) {
  constexpr uint32_t M = 0xC000C000u;
  mma16816(d, w & M, (w << 2) & M, (w << 4) & M, (w << 6) & M, b.x, b.y);
  mma16816(d, (w << 8) & M, (w << 10) & M, (w << 12) & M, (w << 14) & M, b.z, b.w);
}

// Part `part` of the exact three-way bf16 split of x: the nearest bf16, then the nearest bf16 of each remainder.
__device__ __forceinline__ uint32_t split_part(float x, int part) {
  __nv_bfloat16 h = __float2bfloat16_rn(x);
  for (int i = 0; i < part; ++i) {
    x -= __bfloat162float(h);
    h = __float2bfloat16_rn(x);
  }
  return (uint32_t)__bfloat16_as_ushort(h);
}

// Word of the B-fragment array holding column c (its even member c & ~1) for part `part`: per group of 128 columns,
// 4 chunks q4 x 12 lanes (4 part + t) x 4 words j (k-step 2 q4 + j / 2, register j % 2).
__device__ __forceinline__ long long frag_word(long long c, int part) {
  const long long grp = c >> 7;
  const int cc = (int)(c & 127), ks = cc >> 4, kk = cc & 15;
  const int j = 2 * (ks & 1) + (kk >> 3), q4 = ks >> 1, t = (kk & 7) >> 1;
  return ((grp * 4 + q4) * 12 + 4 * part + t) * 4 + j;
}

// B fragments of a vector v of length L (zero past L) for `groups` groups of 128 columns: thread i takes columns
// 2i and 2i + 1. If zf is given, the words of its last group (the next product's vector, of length Lz) that the
// first product does not write -- columns from 32 * ceil(Lz / 32) on -- are zeroed as well.
__global__ void fragments_kernel(const float* __restrict__ v, long long L, long long groups,
                                 uint32_t* __restrict__ xf, uint32_t* __restrict__ zf, long long Lz) {
  const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  const long long c = 2 * i;
  if (zf != nullptr && i < 64) {
    const long long cz = ((Lz + 127) / 128 - 1) * 128 + 2 * i;   // a column pair of zf's last group
    if (cz >= (Lz + 31) / 32 * 32)
#pragma unroll
      for (int part = 0; part < 3; ++part) zf[frag_word(cz, part)] = 0u;
  }
  if (c >= groups * 128) return;
  const float x0 = c < L ? v[c] : 0.f, x1 = c + 1 < L ? v[c + 1] : 0.f;
#pragma unroll
  for (int part = 0; part < 3; ++part) xf[frag_word(c, part)] = split_part(x0, part) | (split_part(x1, part) << 16);
}

constexpr int kStages = 7;      // units per warp in flight + the one being multiplied
constexpr int kCtasPerSm = 2;   // 2 x 8 warps x 7 stages x 1792 B of ring per SM
constexpr int kMinRun = 4;      // units per warp at least (when the matrix is small)
constexpr int kWarpsPerCta = 8;

struct GemvArgs {
  const uint4* words;   // packed matrix
  const uint4* xf;      // B fragments of the vector
  long long rows, U, W; // rows, units, warps in the grid
  int G;                // column groups
  long long TP;         // row-tile pairs
  int segs;             // partial slots per row-tile pair (at most this many warps share one)
  const float* scale;   // row scales or NULL
  float* out;           // y (rows)
  uint32_t* zf;         // if set: B fragments of y for the next product (y's rows are its columns)
  float* partial;       // [TP][32 rows][segs]: slot s of pair tp is the s-th warp whose run meets the pair
  unsigned* ticket;     // [TP], zero and left zero
};

__device__ __forceinline__ long long unit_start(long long w, long long U, long long W) { return w * U / W; }
__device__ __forceinline__ long long unit_owner(long long u, long long U, long long W) {
  return ((u + 1) * W + U - 1) / U - 1;   // the warp whose run holds unit u
}

// This warp's partial row sums of row-tile pair tp (from its accumulators) into the pair's slot for this warp.
__device__ __forceinline__ void store_partial(const GemvArgs& a, long long wid, long long tp, const float (&acc0)[4],
                                              const float (&acc1)[4]) {
  const int lane = threadIdx.x & 31;
  // lane 4g + t holds D columns 2t, 2t + 1 of rows g and g + 8: columns 0, 1, 2 are the hi, mid, lo sums
  const float lo0 = __shfl_down_sync(0xffffffffu, acc0[0], 1), lo0b = __shfl_down_sync(0xffffffffu, acc0[2], 1);
  const float lo1 = __shfl_down_sync(0xffffffffu, acc1[0], 1), lo1b = __shfl_down_sync(0xffffffffu, acc1[2], 1);
  const long long wf = unit_owner(tp * a.G, a.U, a.W);
  float* const mine = a.partial + tp * 32 * a.segs + (wid - wf);
  if ((lane & 3) == 0) {
    const int g = lane >> 2;
    mine[(long long)g * a.segs] = (acc0[0] + acc0[1]) + lo0;
    mine[(long long)(g + 8) * a.segs] = (acc0[2] + acc0[3]) + lo0b;
    mine[(long long)(16 + g) * a.segs] = (acc1[0] + acc1[1]) + lo1;
    mine[(long long)(24 + g) * a.segs] = (acc1[2] + acc1[3]) + lo1b;
  }
}

// After the warp's run (its partials stored, no copies in flight): one ticket per row-tile pair the run met; the
// warp holding a pair's last ticket adds the pair's partials in warp order and finishes its rows.
__device__ void finish_pairs(const GemvArgs& a, long long tp_first, long long tp_last) {
  const int lane = threadIdx.x & 31;
  __syncwarp();
  for (long long tp = tp_first; tp <= tp_last; ++tp) {
    const long long wf = unit_owner(tp * a.G, a.U, a.W), wl = unit_owner(tp * a.G + a.G - 1, a.U, a.W);
    unsigned last = 0;
    if (lane == 0) {   // acquire-release at device scope: orders the warp's partial stores (ordered before it by
                       // the warp barrier) ahead of the ticket, and the finisher's reads after it
      unsigned prev;
      asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(prev) : "l"(a.ticket + tp) : "memory");
      last = prev == (unsigned)(wl - wf);
    }
    last = __shfl_sync(0xffffffffu, last, 0);
    if (!last) continue;
    __syncwarp();
    // lane = row: its slots are contiguous (segs is a multiple of 4), read 16 float4 at a time and added in order
    const float4* row = reinterpret_cast<const float4*>(a.partial + (tp * 32 + lane) * a.segs);
    const int ns = (int)(wl - wf + 1), nv = (ns + 3) >> 2;
    float y = 0.f;
    for (int v0 = 0; v0 < nv; v0 += 16) {
      float4 pv[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) pv[i] = v0 + i < nv ? __ldcg(row + v0 + i) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const int sb = 4 * (v0 + i);
        if (sb + 0 < ns) y += pv[i].x;
        if (sb + 1 < ns) y += pv[i].y;
        if (sb + 2 < ns) y += pv[i].z;
        if (sb + 3 < ns) y += pv[i].w;
      }
    }
    y *= 0.5f;                                  // the codes decode to +-2
    const long long r = 32 * tp + lane;
    if (r < a.rows) {
      if (a.scale != nullptr) y *= a.scale[r];
      a.out[r] = y;
    } else {
      y = 0.f;
    }
    if (a.zf != nullptr) {                      // fragments of y as the next product's vector (column r)
      const float y1 = __shfl_down_sync(0xffffffffu, y, 1);
      if ((lane & 1) == 0)
#pragma unroll
        for (int part = 0; part < 3; ++part)
          a.zf[frag_word(r, part)] = split_part(y, part) | (split_part(y1, part) << 16);
    }
    if (lane == 0) a.ticket[tp] = 0u;
  }
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// Per warp and stage: A of the unit's two row tiles (32 x 16 B each) and its B fragments (48 x 16 B). Every lane
// copies and later reads back only its own 16-byte chunks, so a lane's completed cp.async groups are all it waits
// for: the ring holds the in-flight units without holding registers.
constexpr int kStageChunks = 32 + 32 + 48;
size_t gemv_smem() { return (size_t)kWarpsPerCta * kStages * kStageChunks * 16; }

__global__ void __launch_bounds__(kWarpsPerCta * 32, kCtasPerSm) gemv_kernel(const GemvArgs a) {
  extern __shared__ uint4 ring[];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const long long wid = (long long)blockIdx.x * kWarpsPerCta + warp;
  if (wid >= a.W) return;
  const long long u0 = unit_start(wid, a.U, a.W), u1 = unit_start(wid + 1, a.U, a.W);
  const bool bl = lane < 12;
  const uint4 z4 = make_uint4(0u, 0u, 0u, 0u);
  const long long rtiles = (a.rows + 15) / 16;
  const int G = a.G;
  uint4* const mine = ring + (long long)warp * kStages * kStageChunks;

  // load cursor (row-tile pair, group) of the next unit to fetch, advanced without divisions
  long long ltp = u0 / G;
  int lgrp = (int)(u0 - ltp * G);
  auto issue = [&](int stage) {
    uint4* st = mine + stage * kStageChunks;
    const uint4* p0 = a.words + ((2 * ltp * G + lgrp) * 32 + lane);
    cp_async16(smem_addr(st + lane), p0, 16u);
    cp_async16(smem_addr(st + 32 + lane), 2 * ltp + 1 < rtiles ? p0 + (long long)G * 32 : p0,
               2 * ltp + 1 < rtiles ? 16u : 0u);   // a missing second tile reads as zeros
    if (bl) {
      const uint4* bq = a.xf + lgrp * 48 + lane;
#pragma unroll
      for (int q = 0; q < 4; ++q) cp_async16(smem_addr(st + 64 + 12 * q + lane), bq + 12 * q, 16u);
    }
    if (++lgrp == G) {
      lgrp = 0;
      ++ltp;
    }
  };
#pragma unroll
  for (int i = 0; i < kStages - 1; ++i) {
    if (u0 + i < u1) issue(i);
    cp_async_commit();
  }

  float acc0[4] = {0.f, 0.f, 0.f, 0.f}, acc1[4] = {0.f, 0.f, 0.f, 0.f};
  long long cur = u0 / G, ctp = cur;
  int cgrp = (int)(u0 - ctp * G);
  int stage = 0;
  for (long long uu = u0; uu < u1; ++uu) {
    const int next = stage == 0 ? kStages - 1 : stage - 1;   // the stage consumed last: free again
    if (uu + kStages - 1 < u1) issue(next);
    cp_async_commit();
    cp_async_wait<kStages - 1>();                           // this unit's copies have landed
    const uint4* st = mine + stage * kStageChunks;
    const uint4 A0 = st[lane], A1 = st[32 + lane];
    uint4 Bq[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) Bq[q] = bl ? st[64 + 12 * q + lane] : z4;
    if (ctp != cur) {
      store_partial(a, wid, cur, acc0, acc1);
#pragma unroll
      for (int e = 0; e < 4; ++e) acc0[e] = acc1[e] = 0.f;
      cur = ctp;
    }
    mma_word(acc0, A0.x, Bq[0]);
    mma_word(acc1, A1.x, Bq[0]);
    mma_word(acc0, A0.y, Bq[1]);
    mma_word(acc1, A1.y, Bq[1]);
    mma_word(acc0, A0.z, Bq[2]);
    mma_word(acc1, A1.z, Bq[2]);
    mma_word(acc0, A0.w, Bq[3]);
    mma_word(acc1, A1.w, Bq[3]);
    if (++cgrp == G) {
      cgrp = 0;
      ++ctp;
    }
    stage = stage == kStages - 1 ? 0 : stage + 1;
  }
  cp_async_wait<0>();
  store_partial(a, wid, cur, acc0, acc1);
  finish_pairs(a, u0 / G, cur);
}

struct GemvPlan {
  long long U, W, TP;
  int G, segs;
};

GemvPlan gemv_plan(long long rows, long long cols) {
  int sms = 152, dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  GemvPlan p;
  p.G = (int)cdiv(cols, 128);
  p.TP = cdiv(cdiv(rows, 16), 2);
  p.U = p.TP * p.G;
  // runs of at least kMinRun units (fewer warps share a row-tile pair), at most the resident warps
  p.W = std::max<long long>(1, std::min<long long>(p.U / kMinRun, (long long)kCtasPerSm * kWarpsPerCta * sms));
  p.segs = (int)round_up(cdiv(p.G, p.U / p.W) + 1, 4);         // runs hold at least floor(U / W) units
  return p;
}

}  // namespace

long long packed_words(long long rows, long long cols) { return cdiv(rows, 16) * cdiv(cols, 128) * 128; }

cudaError_t launch_pack_ternary(const int8_t* T, long long rows, long long cols, long long ldt, uint32_t* words,
                                unsigned long long* nnz, cudaStream_t s) {
  const long long total = packed_words(rows, cols);
  if (total == 0) return cudaSuccess;
  pack_kernel<<<(unsigned)cdiv(total, 256), 256, 0, s>>>(T, rows, cols, ldt, words, nnz);
  return cudaGetLastError();
}

long long fragment_words(long long L) { return cdiv(L, 128) * 192; }

cudaError_t launch_fragments(const float* v, long long L, uint32_t* xf, uint32_t* zf, long long Lz, cudaStream_t s) {
  const long long groups = cdiv(L, 128);
  fragments_kernel<<<(unsigned)cdiv(groups * 64, 256), 256, 0, s>>>(v, L, groups, xf, zf, Lz);
  return cudaGetLastError();
}

void gemv_scratch(long long rows, long long cols, long long* partial_floats, long long* tickets) {
  const GemvPlan p = gemv_plan(rows, cols);
  *partial_floats = p.TP * 32 * p.segs;
  *tickets = p.TP;
}

cudaError_t launch_ternary_gemv(const uint32_t* words, long long rows, long long cols, const uint32_t* xf,
                                const float* scale, float* out, uint32_t* zf, float* partial, unsigned* ticket,
                                cudaStream_t s) {
  const GemvPlan p = gemv_plan(rows, cols);
  if (partial == nullptr || ticket == nullptr) return cudaErrorInvalidValue;
  GemvArgs a{reinterpret_cast<const uint4*>(words), reinterpret_cast<const uint4*>(xf), rows, p.U, p.W, p.G, p.TP,
             p.segs, scale, out, zf, partial, ticket};
  static bool configured = false;
  if (!configured) {
    const cudaError_t e =
        cudaFuncSetAttribute(gemv_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)gemv_smem());
    if (e != cudaSuccess) return e;
    configured = true;
  }
  gemv_kernel<<<(unsigned)cdiv(p.W, kWarpsPerCta), kWarpsPerCta * 32, gemv_smem(), s>>>(a);
  return cudaGetLastError();
}

}  // namespace externd
