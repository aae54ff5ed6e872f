// Residual products on the 5th-generation tensor cores (tcgen05, accumulator in tensor memory).
//
//   V-step  part[s][a][c] = sum_{r in split s} U[r][a] R[r][c]       (§2.3 step 1, §2.4; D = R^T U per tile)
//   U-step  part[s][a][r] = sum_{c in split s} R[r][c] h[c] V[c][a]  (§2.3 step 1, §2.5; D = (R H) V per tile)
//
// A CTA owns 128 output positions (the MMA's M) and all w components (N = w rounded up to 16, <= 256), and
// reduces over one split of the other dimension in stages of 64. Accuracy: the ternary operand is exact in fp16;
// the residual operand x (float32) is scaled by a power of two 2^s that puts max|x| just under 2^14 and split
// into fp16 hi = RN(x) and lo = RN(x - hi); the two MMAs hi*T and lo*T accumulate into the same fp32 TMEM
// accumulator, which the epilogue scales back by 2^-s. That keeps ~22 significant bits of every residual entry
// (the float32 product bar is 1e-5 relative), at twice the MMA count of a plain fp16 product.
//
// Warps 0-15 convert: they load float32 R with coalesced 16-byte loads, convert two values per instruction, and
// store straight into the 128-byte-swizzled K-major tiles the MMA reads (the V-step transposes on the way: its A
// rows are R's columns); the ternary factor arrives as fp16 rows written by the ternarization and is copied.
// Warp 16 allocates tensor memory and one of its threads issues the MMAs. Stages hand over through mbarriers:
// full[s] (512 producer arrivals), empty[s] (tcgen05.commit after the stage's MMAs), done (after the last).
#include "kernels.h"
#include "umma.cuh"

namespace externd {

namespace {

constexpr int kProducerWarps = 16;
constexpr int kProducers = kProducerWarps * 32;
constexpr int kThreads = kProducers + 32;   // converter/epilogue warps + 1 MMA warp
constexpr int kStageK = 64;       // reduction elements per stage: one 128-byte swizzle row of fp16
constexpr uint32_t kTileA = 128u * 128u;   // 128 rows x 64 fp16

struct TcArgs {
  const float* R;
  int m, n;
  const __half* T;        // ternary factor as fp16, component-major (w rows, ldt elements each, zero padded)
  int ldt, w, wpad;
  const float* h;         // U-step importances or nullptr
  float* part;            // split-K partials [splits][w][Lx]
  int ychunk;             // reduction elements per split (multiple of kStageK)
  const float* maxabs;    // [0] = max |R|, [1] = max h
  unsigned* err;
  int stages;
  uint32_t tmem_cols;
};

__device__ __forceinline__ void st_shared16(uint8_t* p, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  *reinterpret_cast<uint4*>(p) = make_uint4(a, b, c, d);
}

// Scaled pairs -> fp16 hi = RN(x) and lo = RN(x - hi), packed two per 32-bit word (one conversion per pair).
__device__ __forceinline__ void split_pair(float x0, float x1, uint32_t& hi, uint32_t& lo) {
  const __half2 h = __floats2half2_rn(x0, x1);
  const float2 hb = __half22float2(h);
  const __half2 l = __floats2half2_rn(x0 - hb.x, x1 - hb.y);
  hi = *reinterpret_cast<const uint32_t*>(&h);
  lo = *reinterpret_cast<const uint32_t*>(&l);
}

// Loads this thread's 16 residual values of stage k into registers (zeros outside the matrix / split).
// V-step: rows y0 + 8o + 4hf + j (j < 4) at columns x0 + 4q .. +3 -> v[4j + i], with o = lane % 8,
//         q = (warp % 8) * 4 + lane / 8, hf = warp / 8.
// U-step: rows x0 + warp * 8 + lane / 8 + 4t (t < 2) at columns y0 + 8 (lane % 8) .. +7 -> v[8t + e].
template <bool USTEP>
__device__ __forceinline__ void load_stage(const TcArgs& p, int k, int ybeg, int yend, int x0, int warp, int lane,
                                           bool vec, float (&v)[16]) {
  const int y0 = ybeg + k * kStageK;
  if (!USTEP) {
    const int o = lane & 7, q = (warp & 7) * 4 + (lane >> 3), hf = warp >> 3;
    const int c = x0 + 4 * q;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int y = y0 + 8 * o + 4 * hf + j;
      float4 t = make_float4(0.f, 0.f, 0.f, 0.f);
      if (y < yend) t = load4(p.R + (long long)y * p.n, c, p.n, vec);
      v[4 * j + 0] = t.x;
      v[4 * j + 1] = t.y;
      v[4 * j + 2] = t.z;
      v[4 * j + 3] = t.w;
    }
  } else {
    const int c = y0 + 8 * (lane & 7);
#pragma unroll
    for (int t = 0; t < 2; ++t) {
      const int r = x0 + warp * 8 + (lane >> 3) + 4 * t;
      float4 v0 = make_float4(0.f, 0.f, 0.f, 0.f), v1 = v0;
      if (r < p.m) {
        v0 = load4(p.R + (long long)r * p.n, c, yend, vec);
        v1 = load4(p.R + (long long)r * p.n, c + 4, yend, vec);
      }
      v[8 * t + 0] = v0.x;
      v[8 * t + 1] = v0.y;
      v[8 * t + 2] = v0.z;
      v[8 * t + 3] = v0.w;
      v[8 * t + 4] = v1.x;
      v[8 * t + 5] = v1.y;
      v[8 * t + 6] = v1.z;
      v[8 * t + 7] = v1.w;
    }
  }
}

// Waits for stage slot k % S to be free, converts the loaded values into the swizzled fp16 hi/lo A tiles, copies
// the fp16 ternary B tile, and arrives on full[slot]. False if the wait timed out.
template <bool USTEP>
__device__ __forceinline__ bool convert_stage(const TcArgs& p, int k, int S, uint32_t stage_bytes, uint8_t* gbase,
                                              uint32_t bars, int ybeg, int yend, int x0, int tid, int warp, int lane,
                                              bool vec, float scale, const float (&v)[16]) {
  const int s = k % S, round = k / S;
  if (round > 0 && !mbar_wait(bars + 8u * (S + s), (uint32_t)(round - 1) & 1u, p.err)) return false;
  uint8_t* a_hi = gbase + (uint32_t)s * stage_bytes;
  uint8_t* a_lo = a_hi + kTileA;
  uint8_t* bt = a_hi + 2u * kTileA;
  const int y0 = ybeg + k * kStageK;
  if (!USTEP) {
    // A row = local column 4q + i; this thread writes the 8-byte half hf of chunk o (rows 8o + 4hf .. +3)
    const int o = lane & 7, q = (warp & 7) * 4 + (lane >> 3), hf = warp >> 3;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      uint32_t h0, l0, h1, l1;
      split_pair(v[i] * scale, v[4 + i] * scale, h0, l0);
      split_pair(v[8 + i] * scale, v[12 + i] * scale, h1, l1);
      const uint32_t off = sw128_offset((uint32_t)(4 * q + i), (uint32_t)o) + 8u * hf;
      *reinterpret_cast<uint2*>(a_hi + off) = make_uint2(h0, h1);
      *reinterpret_cast<uint2*>(a_lo + off) = make_uint2(l0, l1);
    }
  } else {
    const int j = lane & 7;
    const int c = y0 + 8 * j;
    float hv[8] = {1.f, 1.f, 1.f, 1.f, 1.f, 1.f, 1.f, 1.f};
    if (p.h != nullptr) {
      const float4 h0 = load4(p.h, c, yend, vec), h1 = load4(p.h, c + 4, yend, vec);
      hv[0] = h0.x; hv[1] = h0.y; hv[2] = h0.z; hv[3] = h0.w;
      hv[4] = h1.x; hv[5] = h1.y; hv[6] = h1.z; hv[7] = h1.w;
    }
#pragma unroll
    for (int t = 0; t < 2; ++t) {
      const int row = warp * 8 + (lane >> 3) + 4 * t;
      uint32_t hi[4], lo[4];
#pragma unroll
      for (int e = 0; e < 4; ++e)
        split_pair(v[8 * t + 2 * e] * hv[2 * e] * scale, v[8 * t + 2 * e + 1] * hv[2 * e + 1] * scale, hi[e], lo[e]);
      const uint32_t off = sw128_offset((uint32_t)row, (uint32_t)j);
      st_shared16(a_hi + off, hi[0], hi[1], hi[2], hi[3]);
      st_shared16(a_lo + off, lo[0], lo[1], lo[2], lo[3]);
    }
  }
  // B rows = components: chunk oc holds reduction elements y0 + 8 oc .. +7, copied from the fp16 factor
  for (int id = tid; id < p.wpad * 8; id += kProducers) {
    const int a = id >> 3, oc = id & 7;
    const int y = y0 + 8 * oc;
    uint4 raw = make_uint4(0u, 0u, 0u, 0u);
    if (a < p.w && y < yend) {
      raw = *reinterpret_cast<const uint4*>(p.T + (long long)a * p.ldt + y);
      const int valid = yend - y;
      if (valid < 8) {   // zero the elements of the next split
        uint32_t* wv = reinterpret_cast<uint32_t*>(&raw);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          if (2 * e >= valid) wv[e] = 0u;
          else if (2 * e + 1 >= valid) wv[e] &= 0xffffu;
        }
      }
    }
    st_shared16(bt + sw128_offset((uint32_t)a, (uint32_t)oc), raw.x, raw.y, raw.z, raw.w);
  }
  fence_async_shared();
  mbar_arrive(bars + 8u * s);
  return true;
}

template <bool USTEP>
__global__ void __launch_bounds__(kThreads, 1) product_tc_kernel(const TcArgs p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t sbase = (raw + 1023u) & ~1023u;
  uint8_t* const gbase = smem_raw + (sbase - raw);
  const int S = p.stages;
  const uint32_t tileB = (uint32_t)p.wpad * 128u;
  const uint32_t stage_bytes = 2u * kTileA + tileB;
  const uint32_t bars = sbase + (uint32_t)S * stage_bytes;
  const uint32_t done_bar = bars + 16u * (uint32_t)S;
  const uint32_t tmem_slot = done_bar + 8u;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int Lx = USTEP ? p.m : p.n;
  const int Ly = USTEP ? p.n : p.m;
  const int x0 = blockIdx.x * 128;
  const int ybeg = blockIdx.z * p.ychunk;
  const int yend = min(Ly, ybeg + p.ychunk);
  const int nk = ybeg < yend ? (int)cdiv(yend - ybeg, kStageK) : 0;
  const bool vec = (p.n & 3) == 0;

  // power-of-two scale putting max |operand| just under 2^14
  float mx = __ldg(p.maxabs);
  if (USTEP && p.h != nullptr) mx *= __ldg(p.maxabs + 1);
  int ex = 0;
  if (mx > 0.f && mx <= 3.0e38f) frexpf(mx, &ex);
  const int sexp = max(-100, min(100, 14 - ex));
  const float scale = ldexpf(1.f, sexp), inv_scale = ldexpf(1.f, -sexp);

  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(bars + 8u * s, kProducers);       // full[s]
      mbar_init(bars + 8u * (S + s), 1);          // empty[s]
    }
    mbar_init(done_bar, 1);
    fence_barrier_init();
  }
  if (warp == kProducerWarps) {
    tmem_alloc(tmem_slot, p.tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(gbase + (tmem_slot - sbase));

  bool ok = true;
  if (warp < kProducerWarps) {
    // ------------------------------------------------------------------ converters
    // Loads run one stage ahead of the conversion (two rotating register buffers).
    float b0[16], b1[16];
    if (nk > 0) load_stage<USTEP>(p, 0, ybeg, yend, x0, warp, lane, vec, b0);
    for (int k = 0; k < nk && ok; k += 2) {
      if (k + 1 < nk) load_stage<USTEP>(p, k + 1, ybeg, yend, x0, warp, lane, vec, b1);
      ok = convert_stage<USTEP>(p, k, S, stage_bytes, gbase, bars, ybeg, yend, x0, tid, warp, lane, vec, scale, b0);
      if (!ok || k + 1 >= nk) break;
      if (k + 2 < nk) load_stage<USTEP>(p, k + 2, ybeg, yend, x0, warp, lane, vec, b0);
      ok = convert_stage<USTEP>(p, k + 1, S, stage_bytes, gbase, bars, ybeg, yend, x0, tid, warp, lane, vec, scale, b1);
    }
  } else if (lane == 0) {
    // ------------------------------------------------------------------ MMA issuer
    const uint32_t idesc = f16_idesc(128, (uint32_t)p.wpad);
    for (int k = 0; k < nk; ++k) {
      const int s = k % S;
      if (!mbar_wait(bars + 8u * s, (uint32_t)(k / S) & 1u, p.err)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t a_hi = sbase + (uint32_t)s * stage_bytes, a_lo = a_hi + kTileA, bt = a_hi + 2u * kTileA;
#pragma unroll
      for (int kk = 0; kk < kStageK / 16; ++kk) {
        const uint64_t bd = sw128_desc(bt + 32u * kk);
        mma_f16(tmem, sw128_desc(a_hi + 32u * kk), bd, idesc, (k > 0 || kk > 0) ? 1u : 0u);
        mma_f16(tmem, sw128_desc(a_lo + 32u * kk), bd, idesc, 1u);
      }
      mma_commit(bars + 8u * (S + s));   // frees the stage once these MMAs have read it
    }
    mma_commit(done_bar);                 // every MMA of this CTA has completed
  }

  // ------------------------------------------------------------------ epilogue (converter warps)
  const int all_ok = __syncthreads_and(ok ? 1 : 0);
  if (warp < kProducerWarps) {
    bool have = nk > 0 && all_ok;
    const bool waited = mbar_wait(done_bar, 0u, p.err);
    have = __all_sync(0xffffffffu, have && waited);
    tc_fence_after();
    const int quad = warp & 3, group = warp >> 2;   // 4 warps per TMEM lane quadrant
    const int xi = x0 + quad * 32 + lane;
    float* out = p.part + (long long)blockIdx.z * p.w * Lx;
    for (int ch = group; ch < p.wpad / 16; ch += kProducerWarps / 4) {
      uint32_t v[16];
      if (have) {
        tmem_ld16(tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)(ch * 16), v);
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
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == kProducerWarps) {
    tc_fence_after();
    tmem_dealloc(tmem, p.tmem_cols);
  }
}

struct TcPlan {
  int wpad, stages, splits, chunk;
  uint32_t tmem_cols;
  size_t smem;
};

TcPlan tc_plan(int w, int Lx, int Ly) {
  TcPlan t;
  t.wpad = (int)round_up(w, 16);
  t.tmem_cols = 32;
  while ((int)t.tmem_cols < t.wpad) t.tmem_cols <<= 1;
  const size_t stage = 2 * kTileA + (size_t)t.wpad * 128;
  const size_t budget = 227 * 1024 - 1024 - 256;
  t.stages = (int)std::min<size_t>(4, budget / stage);
  t.smem = (size_t)t.stages * stage + 1024 + 256;
  int sms = 152, dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int tiles = (int)cdiv(Lx, 128);
  // one CTA per SM (shared memory allows no second): at most one wave of tiles x splits
  int s = std::max(1, std::min(sms / tiles, (int)cdiv(Ly, 2 * kStageK)));
  t.chunk = (int)round_up(cdiv(Ly, s), kStageK);
  t.splits = (int)cdiv(Ly, t.chunk);   // no empty split
  return t;
}

template <bool USTEP>
cudaError_t launch_tc(const float* R, int m, int n, const __half* T, int ldt, int w, const float* h, float* part,
                      int splits, const float* maxabs, unsigned* err, cudaStream_t s) {
  const int Lx = USTEP ? m : n, Ly = USTEP ? n : m;
  TcPlan t = tc_plan(w, Lx, Ly);
  if (splits != t.splits) return cudaErrorInvalidValue;   // the caller planned with tc_product_splits
  static bool configured[2] = {false, false};
  if (!configured[USTEP]) {
    cudaError_t e = cudaFuncSetAttribute(product_tc_kernel<USTEP>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         227 * 1024);
    if (e != cudaSuccess) return e;
    configured[USTEP] = true;
  }
  TcArgs a{R, m, n, T, ldt, w, t.wpad, h, part, t.chunk, maxabs, err, t.stages, t.tmem_cols};
  dim3 grid((unsigned)cdiv(Lx, 128), 1, (unsigned)t.splits);
  product_tc_kernel<USTEP><<<grid, kThreads, t.smem, s>>>(a);
  return cudaGetLastError();
}

}  // namespace

int tc_product_splits(int w, int Lx, int Ly) { return tc_plan(w, Lx, Ly).splits; }

void tc_split(int w, int Lx, int Ly, int* splits, int* chunk) {
  const TcPlan t = tc_plan(w, Lx, Ly);
  *splits = t.splits;
  *chunk = t.chunk;
}

cudaError_t launch_product_v_tc(const float* R, int m, int n, const __half* Ut, int ldu, int w, float* part,
                                int splits, const float* maxabs, unsigned* err, cudaStream_t s) {
  return launch_tc<false>(R, m, n, Ut, ldu, w, nullptr, part, splits, maxabs, err, s);
}

cudaError_t launch_product_u_tc(const float* R, int m, int n, const __half* Vt, int ldv, int w, const float* h,
                                float* part, int splits, const float* maxabs, unsigned* err, cudaStream_t s) {
  return launch_tc<true>(R, m, n, Vt, ldv, w, h, part, splits, maxabs, err, s);
}

}  // namespace externd
