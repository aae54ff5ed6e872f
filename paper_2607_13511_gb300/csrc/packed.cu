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
// (three parts, then the two column parities of a CTA, then the column slices, each in a fixed order).
//
// Work split: a CTA takes 128 rows and a slice of at most 8 column groups; each warp issues all of its packed loads
// (2 row tiles x up to 4 groups) before the CTA stages the slice's B fragments, so the packed stream is in flight
// while the vector is prepared. With several slices, each CTA writes its partial rows and the last CTA of a row
// block (a per-block ticket) sums the slices in order.
#include "kernels.h"

#include <cuda_bf16.h>

namespace externd {

namespace {

constexpr int kThreads = 256;       // 8 warps: 4 row-tile pairs x 2 column parities
constexpr int kBlockRows = 128;     // rows per CTA (8 row tiles)

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

__device__ __forceinline__ uint4 ld_stream(const uint4* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
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

constexpr int kSliceGroups = 8;        // column groups per CTA: each warp takes up to 4 of one parity
constexpr int kWarpGroups = kSliceGroups / 2;

// One CTA: rows [128 rb, 128 rb + 128) x column groups [8 sl, 8 sl + 8). With S == 1 it writes
// out[r] = scale[r] * y_r itself; otherwise partial[sl * rows + r], and the last CTA of the row block writes out.
__global__ void __launch_bounds__(kThreads) gemv_kernel(const uint4* __restrict__ words, long long rows,
                                                        long long cols, int G, int S, const float* __restrict__ v,
                                                        const float* __restrict__ scale, float* __restrict__ out,
                                                        float* __restrict__ partial, unsigned* __restrict__ ticket) {
  __shared__ uint4 xf[kSliceGroups * 48];   // [group][q4][lane 0..11]: the B fragments of the slice
  __shared__ float red[2][kBlockRows];
  __shared__ bool last;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const long long rb = blockIdx.x / S;
  const int sl = (int)(blockIdx.x % S);
  const int g0 = sl * kSliceGroups, ng = min(kSliceGroups, G - g0);
  const long long c0 = 128LL * g0, c1 = min(cols, c0 + 128LL * ng);

  // this warp's packed words, all in flight before the staging below
  const int rp = warp & 3, cp = warp >> 2;
  const long long RT = (rows + 15) / 16;
  const long long rt0 = rb * 8 + 2 * rp;
  const bool rows0 = rt0 < RT, rows1 = rt0 + 1 < RT;
  const uint4 z4 = make_uint4(0u, 0u, 0u, 0u);
  uint4 a0[kWarpGroups], a1[kWarpGroups];
  {
    const uint4* p0 = words + ((rt0 * G + g0) * 32 + lane);
    const uint4* p1 = p0 + (long long)G * 32;
#pragma unroll
    for (int i = 0; i < kWarpGroups; ++i) {
      const int gl = cp + 2 * i;
      a0[i] = rows0 && gl < ng ? ld_stream(p0 + 32 * gl) : z4;
      a1[i] = rows1 && gl < ng ? ld_stream(p1 + 32 * gl) : z4;
    }
  }

  // stage the B fragments: lane 4 part + t of chunk q4 holds, for k-steps 2 q4 and 2 q4 + 1, registers 0 and 1.
  // Thread i splits columns 4i .. 4i + 3 of the slice (one coalesced load) and writes their two column pairs.
  uint32_t* xw = reinterpret_cast<uint32_t*>(xf);
  for (int i = tid; i < ng * 32; i += kThreads) {
    const long long col = c0 + 4LL * i;
    float x[4];
    if (col + 3 < c1 && (reinterpret_cast<uintptr_t>(v) & 15) == 0) {
      const float4 f = *reinterpret_cast<const float4*>(v + col);
      x[0] = f.x, x[1] = f.y, x[2] = f.z, x[3] = f.w;
    } else {
#pragma unroll
      for (int e = 0; e < 4; ++e) x[e] = col + e < c1 ? v[col + e] : 0.f;
    }
    const int gl = i >> 5, ks = (i >> 2) & 7, kk = 4 * (i & 3);        // column 128 gl + 16 ks + kk
    const int j = 2 * (ks & 1) + (kk >> 3), q4 = ks >> 1, t = (kk & 7) >> 1;
#pragma unroll
    for (int part = 0; part < 3; ++part) {
      const int w = ((gl * 4 + q4) * 12 + 4 * part + t) * 4 + j;
      xw[w] = split_part(x[0], part) | (split_part(x[1], part) << 16);
      xw[w + 4] = split_part(x[2], part) | (split_part(x[3], part) << 16);   // lane t + 1: the next column pair
    }
  }
  __syncthreads();

  float acc0[4] = {0.f, 0.f, 0.f, 0.f}, acc1[4] = {0.f, 0.f, 0.f, 0.f};
  if (rows0) {
    const bool bl = lane < 12;
#pragma unroll
    for (int i = 0; i < kWarpGroups; ++i) {
      const int gl = cp + 2 * i;
      if (gl < ng) {
        const uint4* bq = xf + gl * 48 + lane;
        uint4 b[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) b[q] = bl ? bq[12 * q] : z4;
        mma_word(acc0, a0[i].x, b[0]);
        mma_word(acc1, a1[i].x, b[0]);
        mma_word(acc0, a0[i].y, b[1]);
        mma_word(acc1, a1[i].y, b[1]);
        mma_word(acc0, a0[i].z, b[2]);
        mma_word(acc1, a1[i].z, b[2]);
        mma_word(acc0, a0[i].w, b[3]);
        mma_word(acc1, a1[i].w, b[3]);
      }
    }
  }
  // lane 4g + t holds D columns 2t, 2t + 1 of rows g and g + 8: columns 0, 1, 2 are the hi, mid, lo sums
  const float lo0 = __shfl_down_sync(0xffffffffu, acc0[0], 1), lo0b = __shfl_down_sync(0xffffffffu, acc0[2], 1);
  const float lo1 = __shfl_down_sync(0xffffffffu, acc1[0], 1), lo1b = __shfl_down_sync(0xffffffffu, acc1[2], 1);
  if ((lane & 3) == 0) {
    const int g = lane >> 2, base = 32 * rp;
    red[cp][base + g] = 0.5f * ((acc0[0] + acc0[1]) + lo0);      // the codes decode to +-2
    red[cp][base + g + 8] = 0.5f * ((acc0[2] + acc0[3]) + lo0b);
    red[cp][base + 16 + g] = 0.5f * ((acc1[0] + acc1[1]) + lo1);
    red[cp][base + 24 + g] = 0.5f * ((acc1[2] + acc1[3]) + lo1b);
  }
  __syncthreads();
  const long long r = rb * kBlockRows + tid;
  if (S == 1) {
    if (tid < kBlockRows && r < rows) {
      const float y = red[0][tid] + red[1][tid];
      out[r] = scale != nullptr ? y * scale[r] : y;
    }
    return;
  }
  if (tid < kBlockRows && r < rows) partial[(long long)sl * rows + r] = red[0][tid] + red[1][tid];
  __syncthreads();
  if (tid == 0) {
    __threadfence();
    unsigned prev;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(prev) : "l"(ticket + rb) : "memory");
    last = prev == (unsigned)(S - 1);
  }
  __syncthreads();
  if (!last) return;
  __threadfence();
  if (tid < kBlockRows && r < rows) {
    float y = 0.f;
#pragma unroll 4
    for (int s2 = 0; s2 < S; ++s2) y += __ldcg(partial + (long long)s2 * rows + r);
    out[r] = scale != nullptr ? y * scale[r] : y;
  }
  if (tid == 0) ticket[rb] = 0;
}

struct GemvPlan {
  int G, S;
  long long RB;
};

GemvPlan gemv_plan(long long rows, long long cols) {
  GemvPlan p;
  p.G = (int)cdiv(cols, 128);
  p.RB = cdiv(rows, kBlockRows);
  p.S = (int)cdiv(p.G, kSliceGroups);
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

long long gemv_partial_floats(long long rows, long long cols) {
  const GemvPlan p = gemv_plan(rows, cols);
  return p.S > 1 ? (long long)p.S * rows : 0;
}

long long gemv_tickets(long long rows) { return cdiv(rows, kBlockRows); }

cudaError_t launch_ternary_gemv(const uint32_t* words, long long rows, long long cols, const float* v,
                                const float* scale, float* out, float* partial, unsigned* ticket, cudaStream_t s) {
  const GemvPlan p = gemv_plan(rows, cols);
  if (p.S > 1 && (partial == nullptr || ticket == nullptr)) return cudaErrorInvalidValue;
  if (p.RB * p.S > 0x7fffffffLL) return cudaErrorInvalidValue;
  gemv_kernel<<<(unsigned)(p.RB * p.S), kThreads, 0, s>>>(reinterpret_cast<const uint4*>(words), rows, cols, p.G,
                                                           p.S, v, scale, out, partial, ticket);
  return cudaGetLastError();
}

}  // namespace externd
