// Internal launch interface of the ExTernD kernels (host side). Not part of the public C ABI.
//
// Internal layouts (all row-major):
//   R      m x n float32 residual (ld n).
//   Ut     w x ldu int8: row a is component a's u (length m; ldu = round_up(m, 16), zero padded).
//   Vt     w x ldv int8: row a is component a's v (length n; ldv = round_up(n, 16), zero padded) = a block of C.
//   part   splits x w x L float32: split-K partial products; L = n for the V-step, m for the U-step.
//   X      w x ldx float32: decorrelated targets, one vector per row (the Eq. 2 input).
//   Stats  per-vector partials of the Eq. 2 statistics: part[a * nchunk + c] = {sum |x| over chunk c (double-float),
//          max magnitude key over chunk c}, 16 bytes, one chunk per producer CTA column.
#pragma once

#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"

namespace externd {

// Addresses of the caller's arrays of one decomposition, read on the device by the graph nodes that touch them
// (io.cu), so one captured graph serves every matrix of its shape.
struct IoTable {
  const float* A;
  int8_t* B;
  float* D;
  int8_t* C;
};
cudaError_t launch_io_set(IoTable* t, const float* A, int8_t* B, float* D, int8_t* C, cudaStream_t s);
// R = t->A (count floats)
cudaError_t launch_io_copy_in(const IoTable* t, float* R, long long count, cudaStream_t s);
// rows j0 .. j0 + w - 1 of t->C (k x n) = Vt's w rows (ld ldv, a multiple of 16)
cudaError_t launch_io_write_c(const int8_t* Vt, long long ldv, int w, int n, const IoTable* t, long long j0,
                              cudaStream_t s);
// t->D[j0 .. j0 + w) = d
cudaError_t launch_io_write_d(const float* d, int w, const IoTable* t, long long j0, cudaStream_t s);

// Eq. 2 thresholds of nv vectors of length L: theta = RD_float(tau * S / L), whether nothing passes, and the
// fallback index. The last CTA of the statistics producer writes them (ticket counts finished CTAs and is reset
// to zero by that CTA).
struct Thresh {
  float* theta;
  int* fallback;
  unsigned* arg;
  unsigned* ticket;
  double tau;
  int L;
};

// One chunk's partial statistics, written and read as a single 16-byte access.
struct __align__(16) StatPart {
  F2 s;
  u64 key;
};

struct Stats {
  StatPart* part;
  int nchunk;
  Thresh th;
};

__device__ __forceinline__ void put_stat(const Stats& st, int a, int c, F2 s, u64 key) {
  const uint2 sv = make_uint2(__float_as_uint(s.hi), __float_as_uint(s.lo));
  *reinterpret_cast<uint4*>(st.part + (long long)a * st.nchunk + c) =
      make_uint4(sv.x, sv.y, (unsigned)(key & 0xffffffffu), (unsigned)(key >> 32));
}

// Run by the CTA that finished last: sums every vector's chunk partials (double-float) and writes its threshold.
// G threads per vector (a power of two, as many as the CTA allows up to a warp) each take chunks g, g + G, ... in
// batches of 16 whose loads are all issued before any is used and which are summed as a pairwise tree; batches
// add in order, then the group combines with a butterfly. The order is fixed, so the result is reproducible. The
// double-precision division happens once per vector.
__device__ __forceinline__ void finalize_thresholds(const Stats& st, int nv) {
  constexpr int kBatch = 16;
  const int nt = blockDim.x;
  int G = 32;
  while (G > 1 && G * nv > nt) G >>= 1;
  const int g = threadIdx.x & (G - 1);
  for (int a0 = 0; a0 < nv; a0 += nt / G) {   // uniform across the CTA: every lane reaches the shuffles
    const int a = a0 + (int)threadIdx.x / G;
    const bool act = a < nv;
    const uint4* pp = reinterpret_cast<const uint4*>(st.part + (long long)(act ? a : 0) * st.nchunk);
    F2 s;
    u64 key = 0;
    for (int c0 = 0; c0 < st.nchunk; c0 += kBatch * G) {
      F2 sv[kBatch];
      u64 kv[kBatch];
#pragma unroll
      for (int i = 0; i < kBatch; ++i) {
        const int c = c0 + i * G + g;
        uint4 r = make_uint4(0u, 0u, 0u, 0u);
        if (act && c < st.nchunk) r = pp[c];
        sv[i].hi = __uint_as_float(r.x);
        sv[i].lo = __uint_as_float(r.y);
        kv[i] = ((u64)r.w << 32) | r.z;
      }
#pragma unroll
      for (int h = 1; h < kBatch; h <<= 1)
#pragma unroll
        for (int i = 0; i + h < kBatch; i += 2 * h) {
          sv[i] = f2_add(sv[i], sv[i + h]);
          kv[i] = kv[i + h] > kv[i] ? kv[i + h] : kv[i];
        }
      s = f2_add(s, sv[0]);
      key = kv[0] > key ? kv[0] : key;
    }
    for (int o = G >> 1; o > 0; o >>= 1) {
      s = f2_add(s, f2_shfl_xor(s, o));
      const u64 t = __shfl_xor_sync(0xffffffffu, key, o);
      key = t > key ? t : key;
    }
    if (act && g == 0) {
      const float th = __double2float_rd(st.th.tau * (f2_value(s) / (double)st.th.L));
      st.th.theta[a] = th;
      st.th.fallback[a] = !(key_mag(key) > th);
      st.th.arg[a] = key_index(key);
    }
  }
}

// Last-CTA protocol: every CTA calls this after writing its partials. After a barrier, thread 0 takes a ticket
// with an acquire-release atomic at device scope (ordering the CTA's partial writes before it and the
// finalizer's reads after it); the CTA that takes the last ticket finalizes and resets the ticket.
__device__ __forceinline__ void stats_done(const Stats& st, int nv) {
  __shared__ int s_last;
  __syncthreads();
  if (threadIdx.x == 0) {
    const unsigned total = gridDim.x * gridDim.y * gridDim.z;
    unsigned old;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(old) : "l"(st.th.ticket) : "memory");
    s_last = (old == total - 1u);
  }
  __syncthreads();
  if (s_last) {
    finalize_thresholds(st, nv);
    if (threadIdx.x == 0) *st.th.ticket = 0u;
  }
}

// ---- products (gemm.cu)
// Split-K factor of a product with Lx output positions per component and reduction length Ly.
int product_splits(int w, int Lx, int Ly);
cudaError_t launch_product_v(const float* R, int m, int n, const int8_t* Ut, int ldu, int w, float* part, int splits,
                             cudaStream_t s);
cudaError_t launch_product_u(const float* R, int m, int n, const int8_t* Vt, int ldv, int w, const float* h,
                             float* part, int splits, cudaStream_t s);
// Statistics chunks the decorrelation writes per vector of length L for a block of w components (at most
// cdiv(L, 16)).
int decorrelate_chunks(int L, int w);
// With bar (2 zero words, left zero) and err given and the grid resident at once, the grid is launched
// cooperatively and finalizes the thresholds in parallel after a grid barrier (2 s limit, err set on expiry).
// Where decorrelate_needs_operand(w) (blocks of 65 to 128 components, on the tensor cores: decorrelate_tc.cu;
// EXTERND_TCDECOR=0 keeps the FMA tiles), it reads Ginv from op, written by launch_inverse(_int), and needs err.
cudaError_t launch_decorrelate(const float* Ginv, int w, const float* part, int splits, int L, float* X, int ldx,
                               Stats st, cudaStream_t s, unsigned* bar = nullptr, unsigned* err = nullptr,
                               const void* op = nullptr);
bool decorrelate_needs_operand(int w);
// The tensor-core decorrelation (decorrelate_tc.cu): one statistics chunk per decorrelate_tc_positions(L)
// positions. Its Ginv operand (ginv_operand_bytes(), 16-byte aligned) is written by launch_inverse(_int).
bool decorrelate_tc_eligible(int w);
int decorrelate_tc_positions(int L);
size_t ginv_operand_bytes();
cudaError_t launch_decorrelate_tc(const void* op, int w, const float* part, int splits, int L, float* X, int ldx,
                                  Stats st, cudaStream_t s, unsigned* bar, unsigned* err);
// The tensor-core decorrelation followed by the ternarization of its output in one cooperative grid (the X tile
// stays in tensor memory; the tile's Gram is one more MMA), where decorrelate_apply_tc_fits(w, L). Arguments as
// launch_decorrelate_apply's, with op as launch_decorrelate's; with a Gram, gsc is scratch of
// decorrelate_apply_tc_scratch(L) bytes (16-byte aligned); bar: 4 zero words, left zero. With h (weights of the
// L positions; gram must be null) the weighted Gram T H T^T is written to both triangles of gramf (w x w float32).
bool decorrelate_apply_tc_fits(int w, int L);
size_t decorrelate_apply_tc_scratch(int L);
cudaError_t launch_decorrelate_apply_tc(const void* op, int w, const float* part, int splits, int L, Stats st,
                                        int8_t* T, long long ldt, int* gram, __half* T16, long long ldt16, __half* Tk,
                                        long long ldk, int8_t* gsc, unsigned* bar, unsigned* err, cudaStream_t s,
                                        const float* h = nullptr, float* gramf = nullptr);
// The decorrelation followed by the ternarization of its output (launch_decorrelate + launch_apply, with X kept
// on chip) in one cooperative grid, for w <= 64 and grids that fit the GPU at once; *used tells whether it ran
// (if not, nothing was launched and the caller runs the two kernels). T16 / Tk / gram as launch_apply's (gram:
// the integer upper triangle, added to). bar: 3 words, zero, left zero; err: the device error word (a barrier
// that waited 2 s sets it, and the rest of the grid's work is skipped).
bool decorrelate_apply_fits(int w, int L);
cudaError_t launch_decorrelate_apply(const float* Ginv, int w, const float* part, int splits, int L, Stats st,
                                     int8_t* T, long long ldt, int* gram, __half* T16, long long ldt16, __half* Tk,
                                     long long ldk, unsigned* bar, unsigned* err, cudaStream_t s, bool* used);
// Rout = Rin - U diag(d) V (Rout may alias Rin or be NULL); U is Ut (component-major, ldu) or, when
// u_rowmajor, an m x ldu row-major block of B. colpart: [cdiv(m,64)][n] per-tile column sums of Rout^2 (or NULL);
// normpart: [cdiv(m,64) * cdiv(n,128)] per-tile sums of h_j Rout_ij^2.
// maxpart (optional): per-tile max |Rout|.
cudaError_t launch_deflate(const float* Rin, float* Rout, int m, int n, const int8_t* U, long long ldu, bool u_rowmajor,
                           const float* d, const int8_t* Vt, long long ldv, int w, const float* h, float* colpart,
                           F2* normpart, cudaStream_t s, float* maxpart = nullptr);
int deflate_row_tiles(int m);
int deflate_tiles(int m, int n);

// ---- tensor-core products (product_tc.cu): w >= 16; the factor as fp16 rows (ld elements, 16-byte aligned, zero
// padded); maxabs = {max |R|, max h}; err = device error word
int tc_product_splits(int w, int Lx, int Ly);
cudaError_t launch_product_v_tc(const float* R, int m, int n, const __half* Ut, int ldu, int w, float* part,
                                int splits, const float* maxabs, unsigned* err, cudaStream_t s);
cudaError_t launch_product_u_tc(const float* R, int m, int n, const __half* Vt, int ldv, int w, const float* h,
                                float* part, int splits, const float* maxabs, unsigned* err, cudaStream_t s);
// ---- tensor-core deflation (deflate_tc.cu): R -= U diag(d) V^T in place with the factors as K-major fp16
// (Uk[r * ldk + a], Vk[c * ldk + a]; ldk a multiple of 8 and >= round_up(w, 16)); the statistics outputs have
// the layout of launch_deflate's (64-row x 128-column tiles).
cudaError_t launch_deflate_tc(float* R, int m, int n, const __half* Uk, const __half* Vk, long long ldk,
                              const float* d, int w, const float* h, float* colpart, F2* normpart, float* maxpart,
                              unsigned* err, cudaStream_t s);
// dst[pos * ldk + a] = (half) src[a * lda + pos * ldp] for a < w, pos < L (K-major fp16 copy of a ternary factor)
cudaError_t launch_kmajor(const int8_t* src, long long lda, long long ldp, int w, int L, __half* dst, long long ldk,
                          cudaStream_t s);
// Split plan shared by both tensor-core product kernels: split count and reduction elements per split.
void tc_split(int w, int Lx, int Ly, int* splits, int* chunk);
// TMA-fed products (product_tma.cu): same contract as the launch_product_*_tc above; usable when
// tma_product_ok (R and the factor 16-byte aligned, n % 4 == 0, factor ld a multiple of 8).
bool tma_product_ok(const float* R, int n, const __half* T, int ldt);
// Partial slots the TMA-fed product writes (its classic split count, or more under its stream plan).
int tma_product_slots(int w, int Lx, int Ly);
// pdl: launched with programmatic stream serialization behind a cluster inverse (launch_inverse_cluster*), which
// lets it start once the inverse's CTAs are resident; it completes only after the inverse has.
cudaError_t launch_product_v_tma(const float* R, int m, int n, const __half* Ut, int ldu, int w, float* part,
                                 int splits, const float* maxabs, unsigned* err, cudaStream_t s, bool pdl = false);
cudaError_t launch_product_u_tma(const float* R, int m, int n, const __half* Vt, int ldv, int w, const float* h,
                                 float* part, int splits, const float* maxabs, unsigned* err, cudaStream_t s,
                                 bool pdl = false);
// ---- packed inference (packed.cu, §2.6): 2-bit codes in tensor-core fragment order (packed_words(rows, cols)
// 32-bit words; layout in packed.cu) and the row product out[r] = scale[r] * sum_j T[r][j] v[j] (scale optional)
// with the vector given as B fragments (fragment_words(cols) words, from launch_fragments). With zf the product also
// writes the fragments of out (as the next product's vector of length rows; zf's words past 32 * ceil(rows / 32)
// must be zero). partial / ticket: gemv_scratch(rows, cols) floats / zeroed words (left zeroed).
long long packed_words(long long rows, long long cols);
cudaError_t launch_pack_ternary(const int8_t* T, long long rows, long long cols, long long ldt, uint32_t* words,
                                unsigned long long* nnz, cudaStream_t s);
long long fragment_words(long long L);
// zf (optional): zeroes the words of zf's last group past 32 * ceil(Lz / 32) columns (see launch_ternary_gemv).
cudaError_t launch_fragments(const float* v, long long L, uint32_t* xf, uint32_t* zf, long long Lz, cudaStream_t s);
void gemv_scratch(long long rows, long long cols, long long* partial_floats, long long* tickets);
cudaError_t launch_ternary_gemv(const uint32_t* words, long long rows, long long cols, const uint32_t* xf,
                                const float* scale, float* out, uint32_t* zf, float* partial, unsigned* ticket,
                                cudaStream_t s);
// dst[r][c] = (half) src[r][c] for an rows x cols int8 matrix
cudaError_t launch_i8_to_f16(const int8_t* src, long long lds, int rows, int cols, __half* dst, long long ldd,
                             cudaStream_t s);

// ---- ternarization and bookkeeping (tern.cu)
cudaError_t launch_stats(const float* X, int nv, int L, int ldx, Stats st, cudaStream_t s);
// T = T_tau(X) from finalized thresholds. If gram != NULL (requires nv <= 256) also accumulates the exact Gram
// matrix of the ternary vectors into the upper triangle gram[a * nv + b] (a <= b) with integer atomics (gram
// must hold zeros or a running sum).
// T16 (optional): the same ternary values as fp16 rows with leading dimension ldt16. Tk (optional): as fp16 in
// K-major layout, Tk[x * ldk + a] for a < nv (ldk a multiple of 8, >= round_up(nv, 8); 16-byte aligned).
// With gram (nv <= 128) the exact integer Gram is added into its upper triangle; gs then holds the per-CTA
// partials and the zero-initialized group tickets, sized by apply_gram_scratch for the vectors' length L.
constexpr int kGramGroup = 8;   // CTAs whose partials one CTA sums before the atomics
struct GramScratch {
  int* part = nullptr;
  unsigned* ticket = nullptr;
};
void apply_gram_scratch(int L, size_t* part_ints, size_t* groups);
cudaError_t launch_apply(const float* X, int nv, int L, int ldx, const Thresh& th, int8_t* T, int ldt, int* gram,
                         cudaStream_t s, __half* T16 = nullptr, long long ldt16 = 0, __half* Tk = nullptr,
                         long long ldk = 0, GramScratch gs = GramScratch{});
cudaError_t launch_gather(const float* R, int m, int n, const int* J, int w, float* Y, int ldy, Stats st,
                          cudaStream_t s);
// J = the w columns of largest h_c * sum_t colpart[t][c] (ties to the lower c), ascending; e (n floats) is scratch.
cudaError_t launch_select_with(const float* colpart, int nrt, int n, const float* h, int w, int* J, float* e,
                               cudaStream_t s);
// out[0] = sum of count partials (fixed order); if trace != NULL, trace[0] = 1 - out[0] / norm_a[0];
// if maxpart != NULL, maxout[0] = max of the count per-tile maxima.
cudaError_t launch_norm(const F2* normpart, int count, double* out, const double* norm_a, double* trace,
                        cudaStream_t s, const float* maxpart = nullptr, float* maxout = nullptr);
// out[0] = max |x_i|
cudaError_t launch_absmax(const float* x, long long n, float* out, cudaStream_t s);
// B[r][j0 + a] = Ut[a][r]; with io, B is io->B (read on the device).
cudaError_t launch_write_b(const int8_t* Ut, int ldu, int w, int m, int8_t* B, long long k, long long j0,
                           cudaStream_t s, const IoTable* io = nullptr);
// dst[c][r] = src[r][c] for an rows x cols int8 / float32 matrix (leading dims given).
cudaError_t launch_transpose_i8(const int8_t* src, long long lds, int rows, int cols, int8_t* dst, long long ldd,
                                cudaStream_t s);
cudaError_t launch_transpose_f32(const float* src, long long lds, int rows, int cols, float* dst, long long ldd,
                                 cudaStream_t s);
// out[a][x] = sum_s part[s][a][x]
cudaError_t launch_sum_splits(const float* part, int splits, int w, int L, float* out, long long ldo, cudaStream_t s);

// ---- small dense algebra (solve.cu)
int gram_splits(int w, int L);
// Gpart[s][a][b] = sum_{y in split s} T[a][y] T[b][y] (* h[y] if h)
cudaError_t launch_gram(const int8_t* T, int ldt, int w, int L, const float* h, float* Gpart, int splits,
                        cudaStream_t s);
// Graw = sum_s Gpart[s]; Ginv = (Graw + eps I)^-1 with eps = kEpsRel * trace / w. With op (65 to 128
// components), Ginv also as the tensor-core decorrelation's operand (ginv_operand_bytes(), 16-byte aligned).
cudaError_t launch_inverse(const float* Gpart, int splits, int w, float* Graw, float* Ginv, cudaStream_t s,
                           void* op = nullptr);
// Same from an integer upper-triangle Gram (as written by launch_apply), which is reset to zero after reading.
cudaError_t launch_inverse_int(int* Gint, int w, float* Graw, float* Ginv, cudaStream_t s, void* op = nullptr);
// The same inverses on a thread-block cluster of inverse_cluster_size(w) CTAs (0: not available for this width),
// which distributed shared memory connects; with pdl the next kernel on the stream may launch as soon as the
// cluster is resident (it must not read Ginv before its griddepcontrol.wait).
int inverse_cluster_size(int w);
cudaError_t launch_inverse_cluster(const float* Gpart, int splits, int w, float* Graw, float* Ginv, cudaStream_t s,
                                   void* op, bool pdl);
cudaError_t launch_inverse_cluster_int(int* Gint, int w, float* Graw, float* Ginv, cudaStream_t s, void* op, bool pdl);
// Eq. 4 on the cluster (launch_scales_int).
cudaError_t launch_scales_cluster_int(int* GUint, const float* GVraw, const float* r, int w, float* d, cudaStream_t s,
                                      float* K = nullptr);
// r[a] = sum_y Ut[a][y] * sum_s part[s][a][y]
cudaError_t launch_rvec(const int8_t* Ut, int ldu, int w, int L, const float* part, int splits, float* r,
                        cudaStream_t s);
// d solves [(sum_s GUpart[s]) .* GVraw + eps I] d = r (eps = 0 when w == 1); K (optional, w x w) receives the
// matrix without the ridge, K = G_U .* G_V of Eq. 4.
cudaError_t launch_scales(const float* GUpart, int splits, const float* GVraw, const float* r, int w, float* d,
                          cudaStream_t s, float* K = nullptr);
// Same with G_U from an integer upper-triangle Gram, reset to zero after reading.
cudaError_t launch_scales_int(int* GUint, const float* GVraw, const float* r, int w, float* d, cudaStream_t s,
                              float* K = nullptr);
// ---- the same on the tensor cores (inverse_tc.cu), for 65 to 128 components: one CTA, S in tensor memory, the
// rank-16 update of each pivot step as one tf32 MMA (split operands, ~22 significant bits per product); err is
// the device error word (a bounded wait on the MMA sets it). inverse_tc_enabled: only with EXTERND_TCINV=1 (the
// register-tiled sweep is faster on GB300).
bool inverse_tc_enabled(int w);
cudaError_t launch_inverse_tc(const float* Gpart, int splits, int w, float* Graw, float* Ginv, cudaStream_t s,
                              void* op, unsigned* err);
cudaError_t launch_inverse_tc_int(int* Gint, int w, float* Graw, float* Ginv, cudaStream_t s, void* op,
                                  unsigned* err);
cudaError_t launch_scales_tc(const float* GUpart, int splits, const float* GVraw, const float* r, int w, float* d,
                             cudaStream_t s, float* K, unsigned* err);
cudaError_t launch_scales_tc_int(int* GUint, const float* GVraw, const float* r, int w, float* d, cudaStream_t s,
                                 float* K, unsigned* err);


// ---- the sequential algorithm (§2.3, block width 1) in one launch of one thread-block cluster (sequential.cu),
// for residuals that fit the cluster's shared memory. trace (k doubles) may be nullptr; energy: one double;
// activations (one zeroed long long, or nullptr): Prop. 2's safeguard on, counting the components it replaced.
bool sequential_cluster_fits(long long m, long long n);
cudaError_t launch_sequential_cluster(const float* A, int m, int n, long long k, int iters, double tau, const float* h,
                                      int8_t* B, float* D, int8_t* C, double* trace, double* energy,
                                      long long* activations, cudaStream_t s);

// ---- extensions of the block loop (extend.cu): Prop. 2 safeguard and §2.4 refinement sweeps
struct __align__(16) EntryBest {   // a CTA's best single entry: score (|R_ij| or h_j R_ij^2), R_ij, row-major index
  float score, rij;
  unsigned long long idx;
};
struct BlockChoice {                 // the device-side decision of one block, and a running count of positive ones
  int flag, sign;
  long long row, col, count;
};
int entry_argmax_parts(int m);
cudaError_t launch_entry_argmax(const float* R, int m, int n, const float* h, EntryBest* part, cudaStream_t s);
// flag = (h_j R_ij^2 > 2 r^T d - d^T K d) for the best entry; with the flag d becomes (|R_ij|, 0, ..., 0).
cudaError_t launch_safeguard_decide(const EntryBest* part, int nparts, int n, const float* h, const float* r, float* d,
                                    const float* K, int w, BlockChoice* choice, cudaStream_t s);
// With the flag: U = e_i, V = sgn e_j as component 0 and zero components after it, in Ut / Vt and (if given) the
// K-major fp16 copies Uk / Vk.
cudaError_t launch_safeguard_replace(const BlockChoice* choice, int w, int m, int n, int8_t* Ut, long long ldm,
                                     int8_t* Vt, long long ldn, __half* Uk, __half* Vk, long long ldk,
                                     cudaStream_t s);
// flag = (2 r^T d - d^T K d >= norm_add - norm_prev).
cudaError_t launch_refine_decide(const double* norm_add, const double* norm_prev, const float* r, const float* d,
                                 const float* K, int w, BlockChoice* choice, cudaStream_t s);
// With the flag: the block (Ut, Vt, d) becomes columns / rows j0 .. j0 + w - 1 of B (m x k), C (k x n) and D.
cudaError_t launch_commit(const BlockChoice* choice, const int8_t* Ut, long long ldm, const int8_t* Vt, long long ldn,
                          const float* d, int w, int m, int n, int8_t* B, float* D, int8_t* C, long long k,
                          long long j0, cudaStream_t s);
// dst[a] = alpha * src[a]
cudaError_t launch_scale_copy(const float* src, float alpha, int w, float* dst, cudaStream_t s);
// *out = count (if out), count = 0
cudaError_t launch_count_reset(BlockChoice* choice, long long* out, cudaStream_t s);

}  // namespace externd
