/*
 * externd.h — C ABI of the GB300 ExTernD factorization library (libexternd.so).
 *
 * ExTernD (Expanded-Rank Ternary Decomposition, arxiv 2607.13511) approximates a real matrix A (m x n) as
 *     A ~ B diag(D) C,   B in {-1,0,+1}^{m x k},  C in {-1,0,+1}^{k x n},  D in R^k          (§2.1, Eq. 1)
 * with an inner rank k = mu * min(m, n) expanded past full rank, fitted greedily: components one at a time
 * (§2.3) or in blocks of b components with decorrelated targets (§2.4, Eq. 3) and jointly solved scales
 * (Eq. 4), optionally under per-column importance weights with the plain-residual V-step (§2.5).
 *
 * Conventions shared by every entry point
 *   - Matrices are C-contiguous, row-major. All array pointers are CUDA device pointers (memory that the
 *     current device can address: cudaMalloc'd, managed, or mapped pinned), owned by the caller, except where
 *     a function says "host". The library never frees caller memory.
 *   - B and the block factor U are int8 {-1,0,+1}; C and the block factor Cb are int8 {-1,0,+1}; real arrays
 *     are float32; energies are double.
 *   - Work is enqueued on the stream set with externd_set_stream (default: the legacy NULL stream). Functions
 *     that return a double through a host pointer synchronize that stream before returning; the others only
 *     enqueue work.
 *   - Return value: EXTERND_OK (0) on success, a negative EXTERND_E* code on failure; on failure the output
 *     arrays hold unspecified values. externd_strerror turns a code into a message.
 *   - The library allocates its own device workspace (kept between calls, per device); EXTERND_ENOMEM reports
 *     a failed allocation. Calls from several host threads are serialised inside the library.
 *   - Importance weights ("weights", length n) are h~ of §2.5 (the caller forms h/max(h) + lambda); every
 *     weight must be finite and > 0. NULL means unweighted (h~ = 1).
 */
#ifndef EXTERND_H
#define EXTERND_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define EXTERND_OK 0
#define EXTERND_EINVAL (-1)   /* bad size, parameter or NULL pointer                                  */
#define EXTERND_EPTR (-2)     /* a pointer that must be device memory is not accessible from the device */
#define EXTERND_ENOMEM (-3)   /* device workspace allocation failed                                   */
#define EXTERND_ECUDA (-4)    /* a CUDA call or kernel launch failed (message: externd_last_cuda_error) */
#define EXTERND_ENODEV (-5)   /* no usable CUDA device / unsupported architecture                       */
#define EXTERND_ETIMEOUT (-6) /* a kernel's bounded wait expired; it gave up and returned (results invalid) */

/* Message for a status code (static string, never NULL). */
const char *externd_strerror(int status);

/* Text of the last CUDA error seen by the library in this process (static buffer, never NULL). */
const char *externd_last_cuda_error(void);

/* Library version string. */
const char *externd_version(void);

/* Stream used by every later call (a cudaStream_t; NULL = legacy default stream). */
int externd_set_stream(void *cuda_stream);

/* §2.1: inner rank k = floor(mu * min(m, n) + 0.5) for m, n >= 1 and mu > 0 (host only). */
int externd_rank(int64_t m, int64_t n, double mu, int64_t *k);

/* §2.4: block width b = min(block, floor(min(m, n) / 8)), at least 1 (host only). */
int externd_block_width(int64_t m, int64_t n, int block, int *b);

/*
 * The whole method (§2.3 when the block width is 1, §2.4 otherwise; §2.5 when weights != NULL), for the
 * problem statement of §2.1 (Eq. 1).
 *   A        m x n float32, read only.
 *   mu > 0   rank multiplier; k = externd_rank(m, n, mu).   tau >= 0: Eq. 2 threshold scale.
 *   block >= 1 requested block width (clamped as externd_block_width; the last block is k mod b wide when
 *            that is non-zero).   iters >= 1: ALS iterations per component/block (one V-step + one U-step).
 *   weights  n float32 or NULL.
 *   B        m x k int8 out;  D  k float32 out;  C  k x n int8 out.
 *   energy   host double out, or NULL: E = 1 - ||R||^2 / ||A||^2 (weighted by h~ when weights != NULL, §2.5)
 *            from the final residual R = A - B diag(D) C kept in float32 on the device. With energy != NULL the
 *            call returns after the energy reached the host; with NULL it only enqueues the work.
 */
int externd_decompose(const float *A, int64_t m, int64_t n, double mu, double tau, int block, int iters,
                      const float *weights, int8_t *B, float *D, int8_t *C, double *energy);

/* externd_decompose that also reports the energy after every block, the E(k) curve at k = b, 2b, ..., k that
 * the rank budgets below read (greedy deflation, §2.3 / §2.4, makes it the energy of every shorter run).
 *   trace    host double[nblocks] out or NULL (nblocks = ceil(k / b)).
 * Everything else as externd_decompose; the factors are identical. */
int externd_decompose_traced(const float *A, int64_t m, int64_t n, double mu, double tau, int block, int iters,
                             const float *weights, int8_t *B, float *D, int8_t *C, double *energy, double *trace);

/* Same as externd_decompose with every array in HOST memory (pageable or pinned): the library copies A and
 * weights to the device, runs the method, and copies B, D, C back before returning. */
int externd_decompose_host(const float *A, int64_t m, int64_t n, double mu, double tau, int block, int iters,
                           const float *weights, int8_t *B, float *D, int8_t *C, double *energy);

/* Eq. 1 (weighted form of §2.5): energy = 1 - sum_ij h_j (A - B diag(D) C)_ij^2 / sum_ij h_j A_ij^2, with B
 * m x k, D k, C k x n on the device; energy is a host double. */
int externd_energy(const float *A, int64_t m, int64_t n, const int8_t *B, const float *D, const int8_t *C,
                   int64_t k, const float *weights, double *energy);

/* The paper has no counterpart to this entry point. It is externd_energy for callers that cannot allocate
 * device memory: a process whose framework has taken the whole GPU for its own caching allocator and forbids
 * raw cudaMalloc, a latency-critical path that cannot afford the implicit device synchronisation of
 * cudaMalloc/cudaFree, or a plugin that is only handed buffers. It calls no allocating routine: its scratch is
 * a static device array of EXTERND_ENERGY_NOALLOC_SCRATCH doubles (256 KiB) that every GPU loading the library
 * holds until the process exits. Arguments and result are those of externd_energy. Sizes whose
 * ceil(m/64) * ceil(n/128) + 3 exceeds EXTERND_ENERGY_NOALLOC_SCRATCH return EXTERND_EINVAL (e.g. 16384 x 16000
 * fits, 16384 x 16384 does not). The first call on each device, with that device current, looks up the
 * array's device address; make that first call before any stream capture. All calls share the array, so calls
 * whose work overlaps on the GPU (other threads, other streams) race on it. */
#define EXTERND_ENERGY_NOALLOC_SCRATCH 32768
int externd_energy_noalloc(const float *A, int64_t m, int64_t n, const int8_t *B, const float *D, const int8_t *C,
                           int64_t k, const float *weights, double *energy);

/* ---------------------------------------------------------------------------------------------------------
 * Measurement. Not part of the method: lets a caller time one kernel class inside externd_decompose with CUDA
 * events (recorded as nodes of the captured graph, on the stream the kernels run on).
 *   kind: 0 off, 1 V-step product, 2 U-step product, 3 deflation, 4 decorrelation (Eq. 3), 5 Eq. 2 apply,
 *         6 Gram matrices, 7 small solves (inverse + Eq. 4), 8 block start (select + gather), 9 both residual
 *         products (1 and 2).
 * ------------------------------------------------------------------------------------------------------- */
int externd_profile(int kind);

/* Device time (ms) summed over the instrumented launches of the last externd_decompose call, and their count.
 * Waits for that call's work to finish. */
int externd_profile_read(double *ms, int64_t *launches);

/* Number of kernels the last externd_decompose call launched (the kernel nodes of its graph). */
int externd_kernel_launches(int64_t *count);

/* ---------------------------------------------------------------------------------------------------------
 * Single steps of the method, exposed for checking each kernel on its own. U is m x w int8 (a block of B's
 * columns, row-major m x w), Cb is w x n int8 (a block of C's rows). 1 <= w <= 1024.
 * ------------------------------------------------------------------------------------------------------- */

/* Eq. 2 on every vector of X (rows x cols float32): axis = 1 ternarizes each row (length cols), axis = 0 each
 * column (length rows). T (rows x cols int8) receives T_tau: sign(x_i) * [|x_i| > tau * mean_j |x_j|], and the
 * single largest-magnitude entry (first index; +1 when it is 0) when nothing passes. */
int externd_ternarize(const float *X, int64_t rows, int64_t cols, int axis, double tau, int8_t *T);

/* §2.3 step 1 / §2.4: the V-step residual product PV = U^T R (w x n float32). Plain R even when weighted. */
int externd_vstep_product(const float *R, int64_t m, int64_t n, const int8_t *U, int64_t w, float *PV);

/* §2.3 step 1 / §2.5: the U-step residual product PU = R diag(h~) Cb^T (m x w float32). */
int externd_ustep_product(const float *R, int64_t m, int64_t n, const int8_t *Cb, int64_t w, const float *weights,
                          float *PU);

/* Eq. 3 (left): X = (U^T U + eps I)^-1 U^T R (w x n float32), eps = 1e-4 * trace(U^T U) / w. Row a of X is
 * the V target of component a (for w = 1 the product itself: T_tau is invariant to positive scaling). */
int externd_vstep_target(const float *R, int64_t m, int64_t n, const int8_t *U, int64_t w, float *X);

/* Eq. 3 (right) with §2.5: Y = R H V (V^T H V + eps I)^-1 (m x w float32), V = Cb^T, H = diag(h~),
 * eps = 1e-4 * trace(V^T H V) / w (for w = 1 the product itself). */
int externd_ustep_target(const float *R, int64_t m, int64_t n, const int8_t *Cb, int64_t w, const float *weights,
                         float *Y);

/* Eq. 4 with §2.5: d (w float32) solves [(U^T U) .* (V^T H V) + eps I] d = diag(U^T R H V); eps = 0 for w = 1
 * (Prop. 1's scale u^T R H v / (||u||^2 v^T H v)) and 1e-4 * trace / w otherwise. */
int externd_block_scales(const float *R, int64_t m, int64_t n, const int8_t *U, const int8_t *Cb, int64_t w,
                         const float *weights, float *d);

/* §2.3 step 3 / §2.4: R <- R - U diag(d) Cb in place (R m x n float32). If norm2 != NULL it receives (host)
 * sum_ij h_j R_ij^2 of the updated residual. */
int externd_deflate(float *R, int64_t m, int64_t n, const int8_t *U, const float *d, const int8_t *Cb, int64_t w,
                    const float *weights, double *norm2);

/* ---- Extensions of the block loop ------------------------------------------------------------------------- */

/* externd_decompose with the convergence safeguard of Prop. 2 (appendix): before each block is deflated, what it
 * removes from the weighted squared residual, 2 r^T d - d^T K d (r_a = u_a^T R H v_a, K = (U^T U) .* (V^T H V)), is
 * compared with what the best single-entry pair removes, max_ij h_j R_ij^2 (ties to the lower row-major index);
 * when the pair removes more, the block becomes u = e_i, v = sgn(R_ij) e_j, d = |R_ij| followed by w - 1 zero
 * components (zero columns of B, rows of C, entries of D). With b = 1 this is Prop. 2 as stated, and
 * ||R_k||^2 <= (1 - 1/(mn))^k ||A||^2 after every component. *activations (host, required) receives the number of
 * blocks replaced. Arguments and errors otherwise as externd_decompose. */
int externd_decompose_safeguarded(const float *A, int64_t m, int64_t n, double mu, double tau, int block, int iters,
                                  const float *weights, int8_t *B, float *D, int8_t *C, double *energy, double *trace,
                                  int64_t *activations);

/* Refinement sweeps (§2.4) of factors B (m x k), D (k), C (k x n) -- device memory, updated in place -- laid out
 * in blocks of b = min(block, floor(min(m, n) / 8)) components as externd_decompose writes them. Each sweep visits
 * the blocks in order: the block is added back to the residual R = A - B D C, refitted by `iters` ALS iterations
 * warm-started from its own U (no column selection), and replaced by the refit only if the refit removes at least
 * as much from the added-back residual as the block did; then the kept block is deflated. The energy therefore
 * never decreases. energy (host, or NULL): the final energy; trace (host, sweeps doubles, or NULL): the energy
 * after each sweep; replaced (host, sweeps entries, or NULL): blocks replaced per sweep. EXTERND_EINVAL for
 * k < 1, sweeps < 1 or the parameter errors of externd_decompose. Synchronous. */
int externd_refine(const float *A, int64_t m, int64_t n, double tau, int block, int iters, int sweeps,
                   const float *weights, int8_t *B, float *D, int8_t *C, int64_t k, double *energy, double *trace,
                   int64_t *replaced);

/* ---- Rank and storage budgets from the energy trace (host only; no device work) ------------------------- */

/* The inner ranks at which a run at (m, n, mu, block) finishes a block (§2.4): b, 2b, ..., k (the last one
 * capped at k), i.e. the ranks the entries of the decompose call's energy trace belong to. With ranks == NULL only
 * *count is written (the number of blocks); otherwise *count must hold the capacity of ranks and receives the
 * number written. Errors as externd_rank / externd_block_width, or EXTERND_EINVAL if the capacity is short. */
int externd_block_boundaries(int64_t m, int64_t n, double mu, int block, int64_t *ranks, int64_t *count);

/* Smallest block-boundary rank whose energy reaches target, from the trace of one run at (m, n, mu, block):
 * greedy deflation (§2.3, §2.4) makes a run at a smaller rank the prefix of this one, so the trace gives E(k) for
 * every smaller run (the equal-energy comparisons of §3 then use mu = k / min(m, n)). ntrace must equal the
 * number of blocks. *k = 0 when the run never reaches target. */
int externd_rank_for_energy(int64_t m, int64_t n, double mu, int block, const double *trace, int64_t ntrace,
                            double target, int64_t *k);

/* Per-matrix rank allocation under a storage budget (§5): matrix j has npts[j] points (k, E_j(k)) at its block
 * boundaries, stored consecutively in ks (strictly increasing per matrix) and energies; taking matrix j to rank
 * k costs costs[j] * k (> 0, e.g. (m + n) bits of mask per component); weights (or NULL for 1) scale each
 * matrix's energy. Greedy: repeatedly the next block of the matrix with the largest weighted energy gain per
 * unit cost that still fits (ties to the lower index; optimal when every curve is concave). chosen[j] receives
 * the rank of matrix j (0 for none). EXTERND_EINVAL on bad sizes, non-increasing ks or non-finite values. */
int externd_allocate_ranks(int64_t nmat, const int64_t *npts, const int64_t *ks, const double *energies,
                           const double *costs, const double *weights, double budget, int64_t *chosen);

/* ---- Inference with the factors (§2.6, Eq. 5) ----------------------------------------------------------- */

/* Packs a ternary matrix for externd_ternary_apply. T: rows x cols int8 in {-1, 0, 1}, row-major with leading
 * dimension ldt >= cols (device). Each entry becomes a 2-bit code (bit 0: nonzero, bit 1: negative), i.e. the
 * mask and sign bits of §2.6 at a fixed position, laid out for the tensor-core product: words (device,
 * caller-allocated) holds ceil(rows / 16) * ceil(cols / 128) * 128 uint32 words; word
 * ((rt * ceil(cols / 128) + grp) * 32 + lane) * 4 + q, lane = 4 g + t, carries at bits 14 - 2p (low element)
 * and 30 - 2p (high element), p = 0..7, the codes of row 16 rt + g + 8 (p & 1) and columns
 * 128 grp + 16 (2 q + p / 4) + 8 ((p & 3) >> 1) + 2 t and + 1; entries past rows or cols are zero. If nnz != NULL
 * it receives (host) the number of nonzeros, from which Eq. 5's storage of the sparse mask+sign form follows:
 * rows * cols mask bits plus nnz sign bits. Synchronous only when nnz != NULL. */
int externd_pack_ternary(const int8_t *T, int64_t rows, int64_t cols, int64_t ldt, uint32_t *words, int64_t *nnz);

/* §2.6: y = B diag(D) (C x) with B (m x k) and C (k x n) packed by externd_pack_ternary; D (k), x (n) and
 * y (m) float32, all device pointers; the intermediate D (C x) stays in the library's workspace. Each product
 * runs on the tensor cores with the vector split exactly into three bf16 parts, so the result is the exact one up
 * to fp32 accumulation. Asynchronous on the library stream. */
int externd_ternary_apply(const uint32_t *Bp, const float *D, const uint32_t *Cp, int64_t m, int64_t k, int64_t n,
                          const float *x, float *y);

#ifdef __cplusplus
}
#endif

#endif /* EXTERND_H */
