// Host side of libexternd: argument checks, device workspace, the per-block schedule of the method, CUDA-graph
// replay, and the extern "C" entry points declared in include/externd.h.
//
// Schedule of one block of w components (§2.4; w = 1 is the sequential algorithm of §2.3):
//   select    the w residual columns of largest weighted energy (start of the block; the paper leaves it open)
//   gather    Y = R[:, J], Eq. 2 statistics                 apply   U = T_tau(Y) column-wise
//   iters x { gram(U) -> (U^T U + eps I)^-1;  V-step product U^T R;  decorrelate (Eq. 3 left);  apply -> V
//             gram(V, h) -> (V^T H V + eps I)^-1;  U-step product R H V;  decorrelate (Eq. 3 right);  apply -> U }
//   gram(U), r = diag(U^T R H V), Eq. 4 solve -> d;  deflate R -= U diag(d) V^T (+ ||R||_H^2, column energies)
//   write B[:, j0:j0+w], C[j0:j0+w, :], D[j0:j0+w].
// The whole decomposition is captured once into a CUDA graph per (shape, parameters, buffers) and replayed.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <map>
#include <mutex>
#include <string>
#include <tuple>
#include <vector>

#include "../../include/externd.h"
#include "kernels.h"

using namespace externd;

namespace {

std::mutex g_mutex;
cudaStream_t g_stream = nullptr;
char g_cuda_error[512] = "no CUDA error";

int cuda_fail(cudaError_t e, const char* where) {
  std::snprintf(g_cuda_error, sizeof(g_cuda_error), "%s: %s (%s)", where, cudaGetErrorName(e), cudaGetErrorString(e));
  return EXTERND_ECUDA;
}

#define CK(call)                                              \
  do {                                                        \
    cudaError_t e_ = (call);                                  \
    if (e_ != cudaSuccess) return cuda_fail(e_, #call);       \
  } while (0)

// Grow-only device buffers, one set per device.
struct Buffer {
  void* p = nullptr;
  size_t cap = 0;
};

struct Workspace {
  std::map<std::string, Buffer> bufs;
  void* host = nullptr;        // pinned staging for results read on the host
  size_t host_cap = 0;
  cudaStream_t cap_stream = nullptr;
  cudaStream_t side = nullptr;          // second branch of the graph: Gram + inverse beside each product
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
  unsigned generation = 0;     // bumped whenever a buffer moves (invalidates captured graphs)
};

std::map<int, Workspace> g_ws;

// Event-pair instrumentation of one kernel class (externd_profile) and the kernel count of the last decompose.
struct Profile {
  int kind = 0;
  std::vector<cudaEvent_t> events;   // shared by every graph; a graph records events [0, used)
  size_t used = 0;                   // events recorded by the enqueue in progress
  size_t last_used = 0;              // events recorded by the last decompose
  long long launches = 0;            // kernels enqueued by the enqueue in progress
  long long last_launches = 0;
};
Profile g_prof;

cudaError_t prof_mark(cudaStream_t s, bool captured = true) {
  if (g_prof.used == g_prof.events.size()) {
    cudaEvent_t e;
    cudaError_t err = cudaEventCreate(&e);
    if (err != cudaSuccess) return err;
    g_prof.events.push_back(e);
  }
  // inside a stream capture the event becomes a node of the graph (external record); otherwise a plain record
  return captured ? cudaEventRecordWithFlags(g_prof.events[g_prof.used++], s, cudaEventRecordExternal)
                  : cudaEventRecord(g_prof.events[g_prof.used++], s);
}

template <typename T>
int need(Workspace& ws, const char* name, size_t count, T** out, bool zero = false) {
  Buffer& b = ws.bufs[name];
  size_t bytes = count * sizeof(T);
  if (bytes == 0) bytes = 16;
  if (b.cap < bytes) {
    if (b.p) cudaFree(b.p);
    b.p = nullptr;
    b.cap = 0;
    size_t alloc = bytes + bytes / 4;
    if (cudaMalloc(&b.p, alloc) != cudaSuccess) {
      cudaGetLastError();
      return EXTERND_ENOMEM;
    }
    b.cap = alloc;
    ++ws.generation;
    if (zero) CK(cudaMemset(b.p, 0, alloc));
  }
  *out = static_cast<T*>(b.p);
  return EXTERND_OK;
}

int need_host(Workspace& ws, size_t bytes, void** out) {
  if (ws.host_cap < bytes) {
    if (ws.host) cudaFreeHost(ws.host);
    ws.host = nullptr;
    ws.host_cap = 0;
    if (cudaMallocHost(&ws.host, bytes) != cudaSuccess) {
      cudaGetLastError();
      return EXTERND_ENOMEM;
    }
    ws.host_cap = bytes;
  }
  *out = ws.host;
  return EXTERND_OK;
}

int current_ws(Workspace** out) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    cuda_fail(e, "cudaGetDevice");
    return EXTERND_ENODEV;
  }
  Workspace& ws = g_ws[dev];
  if (ws.cap_stream == nullptr) CK(cudaStreamCreateWithFlags(&ws.cap_stream, cudaStreamNonBlocking));
  if (ws.side == nullptr) CK(cudaStreamCreateWithFlags(&ws.side, cudaStreamNonBlocking));
  if (ws.ev_fork == nullptr) CK(cudaEventCreateWithFlags(&ws.ev_fork, cudaEventDisableTiming));
  if (ws.ev_join == nullptr) CK(cudaEventCreateWithFlags(&ws.ev_join, cudaEventDisableTiming));
  *out = &ws;
  return EXTERND_OK;
}

#define TRY(x)                        \
  do {                                \
    int rc_ = (x);                    \
    if (rc_ != EXTERND_OK) return rc_; \
  } while (0)

bool is_device_ptr(const void* p) {
  if (p == nullptr) return false;
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged ||
         (at.type == cudaMemoryTypeHost && at.devicePointer != nullptr);
}

long long ld16(long long x) { return round_up(x, 16); }

// A device float holding 1: the "inverse Gram" of a one-component block, where Eq. 3's positive scalar factor
// does not change T_tau and the sequential algorithm of §2.3 ternarizes the product itself.
int get_one(Workspace& ws, float** out) {
  Buffer& one = ws.bufs["one"];
  if (one.p == nullptr) {
    if (cudaMalloc(&one.p, 256) != cudaSuccess) {
      cudaGetLastError();
      return EXTERND_ENOMEM;
    }
    one.cap = 256;
    const float v = 1.f;
    CK(cudaMemcpy(one.p, &v, sizeof(float), cudaMemcpyHostToDevice));
  }
  *out = static_cast<float*>(one.p);
  return EXTERND_OK;
}

int block_width_of(long long m, long long n, int block) {
  long long cap = std::min(m, n) / 8;
  long long b = std::min<long long>(block, cap);
  return (int)std::max<long long>(1, b);
}

// Products run on the tensor cores for blocks of 16 or more components (the float32 FMA tiles otherwise);
// EXTERND_TCGEN05=0 selects the FMA tiles everywhere, for comparisons.
bool use_tc(int w) {
  static const bool enabled = [] {
    const char* e = std::getenv("EXTERND_TCGEN05");
    return !(e && std::strcmp(e, "0") == 0);
  }();
  return enabled && w >= 16;
}
// The Gram inverse and the Eq. 4 solve: on the tensor cores for 65 to 128 components (when the products are),
// else the register-tiled sweep on one CTA.
bool tc_inverse(int w, const unsigned* err) { return err != nullptr && use_tc(w) && inverse_tc_enabled(w); }
cudaError_t inverse_int(int* Gint, int w, float* Graw, float* Ginv, cudaStream_t s, void* op, unsigned* err) {
  return tc_inverse(w, err) ? launch_inverse_tc_int(Gint, w, Graw, Ginv, s, op, err)
                            : launch_inverse_int(Gint, w, Graw, Ginv, s, op);
}
cudaError_t inverse_f(const float* Gpart, int splits, int w, float* Graw, float* Ginv, cudaStream_t s, void* op,
                      unsigned* err) {
  return tc_inverse(w, err) ? launch_inverse_tc(Gpart, splits, w, Graw, Ginv, s, op, err)
                            : launch_inverse(Gpart, splits, w, Graw, Ginv, s, op);
}
cudaError_t scales_int(int* GUint, const float* GVraw, const float* r, int w, float* d, cudaStream_t s, float* K,
                       unsigned* err) {
  return tc_inverse(w, err) ? launch_scales_tc_int(GUint, GVraw, r, w, d, s, K, err)
                            : launch_scales_int(GUint, GVraw, r, w, d, s, K);
}
cudaError_t scales_f(const float* GUpart, int splits, const float* GVraw, const float* r, int w, float* d,
                     cudaStream_t s, float* K, unsigned* err) {
  return tc_inverse(w, err) ? launch_scales_tc(GUpart, splits, GVraw, r, w, d, s, K, err)
                            : launch_scales(GUpart, splits, GVraw, r, w, d, s, K);
}
// The TMA-fed tensor-core products where the layout allows them; EXTERND_TMA=0 keeps the register-fed ones.
bool use_tma() {
  static const bool enabled = [] {
    const char* e = std::getenv("EXTERND_TMA");
    return !(e && std::strcmp(e, "0") == 0);
  }();
  return enabled;
}
// Partial slots of a product: the kernel that will run decides (product_v / product_u make the same choice).
int splits_of(int w, int Lx, int Ly, bool tma) {
  if (!use_tc(w)) return product_splits(w, Lx, Ly);
  return tma ? tma_product_slots(w, Lx, Ly) : tc_product_splits(w, Lx, Ly);
}
int splits_v(int w, int m, int n, const float* R, const __half* T16, int ld) {
  return splits_of(w, n, m, use_tma() && T16 != nullptr && tma_product_ok(R, n, T16, ld));
}
int splits_u(int w, int m, int n, const float* R, const __half* T16, int ld) {
  return splits_of(w, m, n, use_tma() && T16 != nullptr && tma_product_ok(R, n, T16, ld));
}
// The most slots either kernel can use (workspace sizing).
int splits_max(int w, int Lx, int Ly) { return std::max(splits_of(w, Lx, Ly, false), splits_of(w, Lx, Ly, true)); }

// The factor comes as int8 rows (FMA tiles) and as the same values in fp16 rows (tensor cores), both with
// leading dimension ld elements.
// The TMA-fed product of this shape and factor layout (the one that can run beside a cluster inverse).
bool tma_path(int w, const float* R, int n, const __half* T16, int ld) {
  return use_tc(w) && use_tma() && T16 != nullptr && tma_product_ok(R, n, T16, ld);
}

cudaError_t product_v(const float* R, int m, int n, const int8_t* Ut, const __half* Ut16, int ldu, int w, float* part,
                      int splits, const float* maxabs, unsigned* err, cudaStream_t s, bool pdl = false) {
  if (use_tc(w)) {
    if (use_tma() && tma_product_ok(R, n, Ut16, ldu))
      return launch_product_v_tma(R, m, n, Ut16, ldu, w, part, splits, maxabs, err, s, pdl);
    return launch_product_v_tc(R, m, n, Ut16, ldu, w, part, splits, maxabs, err, s);
  }
  return launch_product_v(R, m, n, Ut, ldu, w, part, splits, s);
}
cudaError_t product_u(const float* R, int m, int n, const int8_t* Vt, const __half* Vt16, int ldv, int w,
                      const float* h, float* part, int splits, const float* maxabs, unsigned* err, cudaStream_t s,
                      bool pdl = false) {
  if (use_tc(w)) {
    if (use_tma() && tma_product_ok(R, n, Vt16, ldv))
      return launch_product_u_tma(R, m, n, Vt16, ldv, w, h, part, splits, maxabs, err, s, pdl);
    return launch_product_u_tc(R, m, n, Vt16, ldv, w, h, part, splits, maxabs, err, s);
  }
  return launch_product_u(R, m, n, Vt, ldv, w, h, part, splits, s);
}

// Device error word of the bounded waits in the tensor-core kernels: nonzero -> EXTERND_ETIMEOUT (and reset).
int check_device_error(Workspace& ws, unsigned* err, cudaStream_t s);

// ------------------------------------------------------------------------------------------------------------
// Decomposition
// ------------------------------------------------------------------------------------------------------------
enum Mode { kPlain = 0, kSafeguard = 1, kRefine = 2 };

struct Plan {
  int m, n, b, iters, nblocks;
  long long k;
  double tau;
  int mode = kPlain;           // Prop. 2 safeguard in the block loop, or refinement sweeps of given factors
  int sweeps = 0;
  int gm, gn;                  // Gram split counts over m and n
  int nchunk_m, nchunk_n;
  long long ldm, ldn;
};

struct Bufs {
  float *R, *part, *X, *Gpart, *GrawU, *GrawV, *Ginv, *d, *one, *colpart, *colE, *maxpart, *maxabs, *theta;
  unsigned *err, *arg, *ticket, *bar;
  unsigned* gop;   // Ginv as the tensor-core decorrelation's shared-memory operand (written by the inverse)
  int8_t* gsc;     // tile Grams of the fused tensor-core decorrelation + ternarization
  int *fallback, *GintU, *GintV;
  GramScratch gram;   // per-CTA partials and group tickets of the fused Gram
  int8_t *Ut, *Vt;
  __half *Ut16, *Vt16;   // fp16 copies of Ut, Vt for the tensor-core products (nullptr when unused)
  __half *Uk16, *Vk16;   // K-major fp16 copies of the final U, V of a block for the tensor-core deflation
  long long ldk;
  StatPart* spart;
  F2* normpart;
  float* r;
  double *norm_a, *norm_r, *norm_add, *trace;
  int* J;
  float* K;               // Eq. 4's G_U .* G_V of the block (safeguard and refinement decisions)
  EntryBest* best;        // per-CTA best single entries (safeguard)
  int nbest;
  BlockChoice* choice;
  long long* counts;      // activations (safeguard) or replaced blocks per sweep (refinement)
  IoTable* io;            // the caller's A, B, D, C for this run (decompose modes; set before each replay)
};

int plan_buffers(Workspace& ws, const Plan& p, Bufs* B) {
  const long long L = std::max(p.m, p.n);
  const long long w = p.b;
  TRY(need(ws, "R", (size_t)p.m * p.n, &B->R));
  TRY(need(ws, "Ut", (size_t)w * p.ldm, &B->Ut, true));
  TRY(need(ws, "Vt", (size_t)w * p.ldn, &B->Vt, true));
  B->Ut16 = B->Vt16 = B->Uk16 = B->Vk16 = nullptr;
  B->ldk = round_up(w, 16);
  if (use_tc(p.b)) {
    TRY(need(ws, "Ut16", (size_t)w * p.ldm, &B->Ut16, true));
    TRY(need(ws, "Vt16", (size_t)w * p.ldn, &B->Vt16, true));
    TRY(need(ws, "Uk16", (size_t)p.m * B->ldk, &B->Uk16, true));
    TRY(need(ws, "Vk16", (size_t)p.n * B->ldk, &B->Vk16, true));
  }
  // split-K partials for both block widths that occur (b and the tail k mod b)
  size_t part = 0;
  for (long long wi : {(long long)p.b, p.k % p.b}) {
    if (wi < 1) continue;
    part = std::max(part, (size_t)std::max((long long)splits_max((int)wi, p.n, p.m) * wi * p.n,
                                           (long long)splits_max((int)wi, p.m, p.n) * wi * p.m));
  }
  TRY(need(ws, "part", part, &B->part));
  TRY(need(ws, "maxpart", (size_t)deflate_tiles(p.m, p.n), &B->maxpart));
  TRY(need(ws, "maxabs", 2, &B->maxabs));
  TRY(need(ws, "err", 1, &B->err, true));
  TRY(need(ws, "theta", (size_t)w, &B->theta));
  TRY(need(ws, "fallback", (size_t)w, &B->fallback));
  TRY(need(ws, "arg", (size_t)w, &B->arg));
  TRY(need(ws, "ticket", 1, &B->ticket, true));
  TRY(need(ws, "bar", 4, &B->bar, true));
  TRY(need(ws, "GintU", (size_t)w * w, &B->GintU, true));
  TRY(need(ws, "GintV", (size_t)w * w, &B->GintV, true));
  {
    size_t pm, gm, pn, gn;
    apply_gram_scratch(p.m, &pm, &gm);
    apply_gram_scratch(p.n, &pn, &gn);
    TRY(need(ws, "gram.part", std::max(pm, pn), &B->gram.part));
    TRY(need(ws, "gram.ticket", std::max(gm, gn), &B->gram.ticket, true));
  }
  TRY(need(ws, "X", (size_t)w * L, &B->X));
  TRY(need(ws, "spart", (size_t)w * std::max(p.nchunk_m, p.nchunk_n), &B->spart));
  TRY(need(ws, "Gpart", (size_t)std::max(p.gm, p.gn) * w * w, &B->Gpart));
  TRY(need(ws, "GrawU", (size_t)w * w, &B->GrawU));
  TRY(need(ws, "GrawV", (size_t)w * w, &B->GrawV));
  TRY(need(ws, "Ginv", (size_t)w * w, &B->Ginv));
  TRY(need(ws, "gop", ginv_operand_bytes() / sizeof(unsigned), &B->gop));
  B->gsc = nullptr;
  if (decorrelate_needs_operand(w))
    TRY(need(ws, "gsc", std::max(decorrelate_apply_tc_scratch(p.m), decorrelate_apply_tc_scratch(p.n)), &B->gsc));
  TRY(need(ws, "d", (size_t)w, &B->d));
  TRY(need(ws, "r", (size_t)w, &B->r));
  TRY(need(ws, "J", (size_t)w, &B->J, true));
  TRY(need(ws, "colpart", (size_t)deflate_row_tiles(p.m) * p.n, &B->colpart));
  TRY(need(ws, "colE", (size_t)p.n, &B->colE));
  TRY(need(ws, "normpart", (size_t)deflate_tiles(p.m, p.n), &B->normpart));
  TRY(need(ws, "scalars", 4, &B->norm_a));
  B->norm_r = B->norm_a + 1;
  B->norm_add = B->norm_a + 2;
  TRY(need(ws, "trace", (size_t)std::max(p.nblocks, p.sweeps), &B->trace));
  TRY(need(ws, "io", 1, &B->io, true));
  B->K = nullptr;
  B->best = nullptr;
  B->nbest = 0;
  B->choice = nullptr;
  B->counts = nullptr;
  if (p.mode != kPlain) {
    TRY(need(ws, "K", (size_t)w * w, &B->K));
    TRY(need(ws, "choice", 1, &B->choice, true));
    TRY(need(ws, "counts", (size_t)std::max(1, p.sweeps), &B->counts));
    if (p.mode == kSafeguard) {
      B->nbest = entry_argmax_parts(p.m);
      TRY(need(ws, "best", (size_t)B->nbest, &B->best));
    }
  }
  return get_one(ws, &B->one);
}

Plan make_plan(long long m, long long n, long long k, int block, int iters, double tau) {
  Plan p;
  p.m = (int)m;
  p.n = (int)n;
  p.k = k;
  p.b = block_width_of(m, n, block);
  p.iters = iters;
  p.tau = tau;
  p.nblocks = (int)cdiv(k, p.b);
  p.gm = gram_splits(p.b, p.m);
  p.gn = gram_splits(p.b, p.n);
  p.nchunk_m = (int)cdiv(p.m, 16);   // bounds every producer's chunk count (decorrelation tiles >= 16)
  p.nchunk_n = (int)cdiv(p.n, 16);
  p.ldm = ld16(m);
  p.ldn = ld16(n);
  return p;
}

#define LK(call)                                        \
  do {                                                  \
    cudaError_t e_ = (call);                            \
    if (e_ != cudaSuccess) return cuda_fail(e_, #call); \
  } while (0)

// A kernel launch of class `kind` that launches `nk` kernels: counted, and bracketed by events when profiled.
#define KLS(kind_, nk, st_, call)                           \
  do {                                                      \
    const bool prof_ = g_prof.kind != 0 && prof_match(kind_); \
    if (prof_) LK(prof_mark(st_));                          \
    LK(call);                                               \
    if (prof_) LK(prof_mark(st_));                          \
    g_prof.launches += (nk);                                \
  } while (0)
#define KL(kind_, nk, call) KLS(kind_, nk, s, call)
// Whether a launch of class kind is instrumented under the current selector.
inline bool prof_match(int kind) {
  return g_prof.kind == kind || (g_prof.kind == 9 && (kind == 1 || kind == 2));
}
// Fork the side branch from stream s / join it back into s.
#define FORK()                                              \
  do {                                                      \
    if (side == s) break;                                   \
    LK(cudaEventRecord(ws.ev_fork, s));                     \
    LK(cudaStreamWaitEvent(side, ws.ev_fork, 0));           \
  } while (0)
#define JOIN()                                              \
  do {                                                      \
    if (side == s) break;                                   \
    LK(cudaEventRecord(ws.ev_join, side));                  \
    LK(cudaStreamWaitEvent(s, ws.ev_join, 0));              \
  } while (0)

enum Kind { kVstep = 1, kUstep = 2, kDeflate = 3, kDecor = 4, kApply = 5, kGram = 6, kSolve = 7, kStart = 8,
            kProducts = 9 /* both residual products: profiling selector only */ };

// Thresholds and statistics of the Eq. 2 producers (per-block chunk counts set by fit_block).
struct Eq2 {
  Thresh th_m, th_n;
  Stats st_g, st_m, st_n;
};

Eq2 make_eq2(const Plan& p, const Bufs& B) {
  Eq2 e{Thresh{B.theta, B.fallback, B.arg, B.ticket, p.tau, p.m}, Thresh{B.theta, B.fallback, B.arg, B.ticket, p.tau, p.n},
        Stats{}, Stats{}, Stats{}};
  e.st_g = Stats{B.spart, (int)cdiv(p.m, kStatChunk), e.th_m};   // gather (block start)
  e.st_m = Stats{B.spart, 0, e.th_m};                              // U-step decorrelation
  e.st_n = Stats{B.spart, 0, e.th_n};                              // V-step decorrelation
  return e;
}

// The fused decorrelation + ternarization (one cooperative grid) where it applies; EXTERND_FUSED=0 keeps the
// two kernels everywhere, for comparisons.
bool fused_enabled() {
  static const bool enabled = [] {
    const char* e = std::getenv("EXTERND_FUSED");
    return !(e && std::strcmp(e, "0") == 0);
  }();
  return enabled;
}

// The cooperative decorrelation (parallel threshold finalize); EXTERND_COOP=0 keeps the last-CTA finalize.
bool coop_enabled() {
  static const bool enabled = [] {
    const char* e = std::getenv("EXTERND_COOP");
    return !(e && std::strcmp(e, "0") == 0);
  }();
  return enabled;
}

// Whether targets_step takes the fused tensor-core grid (65 to 128 components, co-resident).
bool fused_targets_tc(int w, int L) {
  return fused_enabled() && decorrelate_needs_operand(w) && decorrelate_apply_tc_fits(w, L);
}

// Eq. 3 targets of the product partials and Eq. 2 on them: T (and its fp16 / K-major copies, its integer Gram).
// With hw and gramf (the fused tensor-core path only: fused_targets_tc), the weighted Gram T H T^T goes to gramf.
int targets_step(const Bufs& B, const float* Ginv, int w, int splits, int L, const Stats& st, int8_t* T, int ldt,
                 int* gram, __half* T16, long long ldt16, __half* Tk, cudaStream_t s, const float* hw = nullptr,
                 float* gramf = nullptr) {
  if (fused_targets_tc(w, L)) {
    KL(kDecor, 1, launch_decorrelate_apply_tc(B.gop, w, B.part, splits, L, st, T, ldt, gram, T16, ldt16, Tk, B.ldk,
                                              B.gsc, B.bar, B.err, s, hw, gramf));
    return EXTERND_OK;
  }
  if (gramf != nullptr) return cuda_fail(cudaErrorInvalidValue, "targets_step");
  if (fused_enabled() && !decorrelate_needs_operand(w) && decorrelate_apply_fits(w, L)) {
    bool used = false;
    KL(kDecor, 1, launch_decorrelate_apply(Ginv, w, B.part, splits, L, st, T, ldt, gram, T16, ldt16, Tk, B.ldk, B.bar,
                                           B.err, s, &used));
    if (used) return EXTERND_OK;
    return cuda_fail(cudaErrorInvalidValue, "launch_decorrelate_apply");
  }
  KL(kDecor, 1, launch_decorrelate(Ginv, w, B.part, splits, L, B.X, L, st, s, coop_enabled() ? B.bar : nullptr, B.err,
                                   B.gop));
  KL(kApply, 1, launch_apply(B.X, w, L, L, st.th, T, ldt, gram, s, T16, ldt16, Tk, B.ldk, B.gram));
  return EXTERND_OK;
}

// The ALS fit of one block of w components (§2.3 for w = 1, §2.4): `iters` V-step / U-step pairs, ending with U
// in Ut (and its exact Gram where fused), V in Vt, the K-major fp16 copies for the tensor-core deflation, and the
// last U-step product in B.part. With `staged` the caller has put the starting U in Ut (and Ut16) -- a refinement
// revisit -- otherwise the block starts from the selected columns of R (§2.4, initial columns).
int fit_block(Workspace& ws, const Plan& p, const Bufs& B, Eq2& q, const float* h, int blk, int w, bool staged,
              cudaStream_t s) {
  cudaStream_t side = ws.side;
  const int m = p.m, n = p.n;
  const int nrt = deflate_row_tiles(m);
  const int sv = splits_v(w, m, n, B.R, use_tc(w) ? B.Ut16 : nullptr, (int)p.ldm);
  const int su = splits_u(w, m, n, B.R, use_tc(w) ? B.Vt16 : nullptr, (int)p.ldn);
  q.st_m.nchunk = decorrelate_chunks(m, w);
  q.st_n.nchunk = decorrelate_chunks(n, w);
  // Exact Gram matrices of unweighted ternary factors are accumulated by the apply that writes the factor
  // (integer atomics) up to 128 components; wider blocks and the weighted V^T H V use the Gram kernel.
  const bool fusedU = w <= 128, fusedV = w <= 128 && h == nullptr;
  // weighted V^T H V from the fused tensor-core targets of the V-step (into Gpart, one slice)
  const bool fusedVw = h != nullptr && w > 1 && fused_targets_tc(w, n);
  __half* const U16 = use_tc(w) ? B.Ut16 : nullptr;
  __half* const V16 = use_tc(w) ? B.Vt16 : nullptr;
  void* const gop = decorrelate_needs_operand(w) ? B.gop : nullptr;   // Ginv's tensor-core operand
  const bool cinv = inverse_cluster_size(w) > 0;                       // the cluster inverse covers this width
  if (!staged) {
    KL(kStart, 2, launch_select_with(B.colpart, nrt, n, h, w, B.J, B.colE, s));
    KL(kStart, 1, launch_gather(B.R, m, n, B.J, w, B.X, m, q.st_g, s));
    if (blk > 0) JOIN();   // the previous block's outputs (side branch) have read Ut, Vt and d
    KL(kApply, 1, launch_apply(B.X, w, m, m, q.th_m, B.Ut, (int)p.ldm, (fusedU && w > 1) ? B.GintU : nullptr, s, U16,
                               p.ldm, nullptr, 0, B.gram));
  }
  for (int it = 0; it < p.iters; ++it) {
    const bool last = it == p.iters - 1;
    // V-step: V <- T([(U^T U + eps I)^-1 U^T R]^T)   (plain R even when weighted, §2.5).
    // The Gram inverse depends only on U: it runs on the side branch while the product streams R. A staged U has
    // no integer Gram yet, so its first inverse takes the Gram kernel.
    // With a cluster inverse (the TMA product, integer Gram ready) both run on the main stream: the inverse's
    // cluster lets the product launch as soon as it is resident, and the product completes only after it.
    const bool clusterV = w > 1 && cinv && fusedU && !(staged && it == 0) && tma_path(w, B.R, n, U16, (int)p.ldm);
    if (clusterV) {
      KL(kSolve, 1, launch_inverse_cluster_int(B.GintU, w, nullptr, B.Ginv, s, gop, true));
    } else if (w > 1) {
      FORK();
      if (fusedU && !(staged && it == 0)) {
        KLS(kSolve, 1, side, inverse_int(B.GintU, w, B.GrawU, B.Ginv, side, gop, B.err));
      } else {
        KLS(kGram, 1, side, launch_gram(B.Ut, (int)p.ldm, w, m, nullptr, B.Gpart, p.gm, side));
        KLS(kSolve, 1, side, inverse_f(B.Gpart, p.gm, w, B.GrawU, B.Ginv, side, gop, B.err));
      }
    }
    KL(kVstep, 1, product_v(B.R, m, n, B.Ut, U16, (int)p.ldm, w, B.part, sv, B.maxabs, B.err, s, clusterV));
    if (w > 1 && !clusterV) JOIN();
    TRY(targets_step(B, w > 1 ? B.Ginv : B.one, w, sv, n, q.st_n, B.Vt, (int)p.ldn, fusedV ? B.GintV : nullptr, V16,
                     p.ldn, (last && use_tc(w)) ? B.Vk16 : nullptr, s, fusedVw ? h : nullptr,
                     fusedVw ? B.Gpart : nullptr));
    // U-step: U <- T(R H V (V^T H V + eps I)^-1)
    const bool clusterU = cinv && (fusedV || fusedVw) && tma_path(w, B.R, n, V16, (int)p.ldn);
    if (clusterU && fusedV) {
      KL(kSolve, 1, launch_inverse_cluster_int(B.GintV, w, B.GrawV, B.Ginv, s, gop, true));
    } else if (clusterU) {
      KL(kSolve, 1, launch_inverse_cluster(B.Gpart, 1, w, B.GrawV, B.Ginv, s, gop, true));
    } else {
      FORK();
      if (fusedV) {
        KLS(kSolve, 1, side, inverse_int(B.GintV, w, B.GrawV, B.Ginv, side, gop, B.err));
      } else if (fusedVw) {
        KLS(kSolve, 1, side, inverse_f(B.Gpart, 1, w, B.GrawV, B.Ginv, side, gop, B.err));
      } else {
        KLS(kGram, 1, side, launch_gram(B.Vt, (int)p.ldn, w, n, h, B.Gpart, p.gn, side));
        KLS(kSolve, 1, side, inverse_f(B.Gpart, p.gn, w, B.GrawV, B.Ginv, side, gop, B.err));
      }
    }
    KL(kUstep, 1, product_u(B.R, m, n, B.Vt, V16, (int)p.ldn, w, h, B.part, su, B.maxabs, B.err, s, clusterU));
    if (!clusterU) JOIN();
    // the next V-step's inverse (w > 1) or, after the last iteration, Eq. 4 consumes U's Gram
    // (the fp16 copy of U is not needed after the last iteration)
    TRY(targets_step(B, w > 1 ? B.Ginv : B.one, w, su, m, q.st_m, B.Ut, (int)p.ldm,
                     (fusedU && (w > 1 || last)) ? B.GintU : nullptr, last ? nullptr : U16, p.ldm,
                     (last && use_tc(w)) ? B.Uk16 : nullptr, s));
  }
  return EXTERND_OK;
}

// Eq. 4: [(U^T U) .* (V^T H V)] d = diag(U^T R H V), with R H V the last U-step product; K (if given) receives
// the matrix without the ridge.
int block_scales_step(const Plan& p, const Bufs& B, int w, float* K, cudaStream_t s) {
  const int m = p.m, n = p.n;
  const int su = splits_u(w, m, n, B.R, use_tc(w) ? B.Vt16 : nullptr, (int)p.ldn);
  KL(kSolve, 1, launch_rvec(B.Ut, (int)p.ldm, w, m, B.part, su, B.r, s));
  if (inverse_cluster_size(w) > 0) {
    KL(kSolve, 1, launch_scales_cluster_int(B.GintU, B.GrawV, B.r, w, B.d, s, K));
  } else if (w <= 128) {
    KL(kSolve, 1, scales_int(B.GintU, B.GrawV, B.r, w, B.d, s, K, B.err));
  } else {
    KL(kGram, 1, launch_gram(B.Ut, (int)p.ldm, w, m, nullptr, B.Gpart, p.gm, s));
    KL(kSolve, 1, scales_f(B.Gpart, p.gm, B.GrawV, B.r, w, B.d, s, K, B.err));
  }
  return EXTERND_OK;
}

// R <- R - U diag(d) V^T with the block in (Ut, Vt, d) / (Uk16, Vk16, d), statistics for the next selection, and
// the squared norm into *norm (and the energy into *trace if given).
int deflate_step(const Plan& p, const Bufs& B, const float* h, int w, double* norm, double* trace, cudaStream_t s) {
  const int m = p.m, n = p.n;
  if (use_tc(w)) {
    KL(kDeflate, 1, launch_deflate_tc(B.R, m, n, B.Uk16, B.Vk16, B.ldk, B.d, w, h, B.colpart, B.normpart, B.maxpart,
                                      B.err, s));
  } else {
    KL(kDeflate, 1, launch_deflate(B.R, B.R, m, n, B.Ut, p.ldm, false, B.d, B.Vt, p.ldn, w, h, B.colpart, B.normpart,
                                   s, B.maxpart));
  }
  KL(0, 1, launch_norm(B.normpart, deflate_tiles(m, n), norm, trace != nullptr ? B.norm_a : nullptr, trace, s,
                       B.maxpart, B.maxabs));
  return EXTERND_OK;
}

// R = A with column energies, ||A||_H^2 and the fp16 scaling scalars. A == nullptr: A is B.io->A, copied first.
int start_residual(const Plan& p, const Bufs& B, const float* A, const float* h, cudaStream_t s) {
  const int m = p.m, n = p.n;
  if (A == nullptr) {
    KL(0, 1, launch_io_copy_in(B.io, B.R, (long long)m * n, s));
    A = B.R;
  }
  KL(kDeflate, 1, launch_deflate(A, B.R, m, n, nullptr, 0, false, nullptr, nullptr, 0, 0, h, B.colpart, B.normpart, s,
                                 B.maxpart));
  KL(0, 1, launch_norm(B.normpart, deflate_tiles(m, n), B.norm_a, nullptr, nullptr, s, B.maxpart, B.maxabs));
  if (h != nullptr) KL(0, 1, launch_absmax(h, n, B.maxabs + 1, s));
  return EXTERND_OK;
}

// Enqueues the whole decomposition on stream s (with Prop. 2's safeguard when p.mode == kSafeguard). The caller's
// A, B, D, C are not named here: the graph reads them from B.io, set on the stream before each run.
int enqueue_decompose(Workspace& ws, const Plan& p, const Bufs& B, const float* h, cudaStream_t s) {
  cudaStream_t side = ws.side;
  const int m = p.m, n = p.n;
  Eq2 q = make_eq2(p, B);
  g_prof.used = 0;
  g_prof.launches = 0;
  TRY(start_residual(p, B, nullptr, h, s));
  const bool guard = p.mode == kSafeguard;
  for (int blk = 0; blk < p.nblocks; ++blk) {
    const long long j0 = (long long)blk * p.b;
    const int w = (int)std::min<long long>(p.b, p.k - j0);
    // Prop. 2: the best single entry of the residual this block is fitted to
    if (guard) KL(0, 1, launch_entry_argmax(B.R, m, n, h, B.best, s));
    TRY(fit_block(ws, p, B, q, h, blk, w, false, s));
    if (!guard) {
      // The block's outputs leave on the side branch: B from the final U and C from the final V now, D after the
      // scales; the next block joins before it overwrites Ut.
      FORK();
      KLS(0, 1, side, launch_write_b(B.Ut, (int)p.ldm, w, m, nullptr, p.k, j0, side, B.io));
      KLS(0, 1, side, launch_io_write_c(B.Vt, p.ldn, w, p.n, B.io, j0, side));
    }
    TRY(block_scales_step(p, B, w, guard ? B.K : nullptr, s));
    if (guard) {
      KL(0, 1, launch_safeguard_decide(B.best, B.nbest, n, h, B.r, B.d, B.K, w, B.choice, s));
      KL(0, 1, launch_safeguard_replace(B.choice, w, m, n, B.Ut, p.ldm, B.Vt, p.ldn, use_tc(w) ? B.Uk16 : nullptr,
                                        use_tc(w) ? B.Vk16 : nullptr, B.ldk, s));
      FORK();
      KLS(0, 1, side, launch_write_b(B.Ut, (int)p.ldm, w, m, nullptr, p.k, j0, side, B.io));
      KLS(0, 1, side, launch_io_write_c(B.Vt, p.ldn, w, p.n, B.io, j0, side));
    } else {
      FORK();
    }
    KLS(0, 1, side, launch_io_write_d(B.d, w, B.io, j0, side));
    TRY(deflate_step(p, B, h, w, B.norm_r, B.trace + blk, s));
  }
  if (p.nblocks > 0) JOIN();
  if (guard) KL(0, 1, launch_count_reset(B.choice, B.counts, s));
  return EXTERND_OK;
}

// Block j0 .. j0 + w - 1 of the factors (B m x k, C k x n, D) into the internal layouts: Ut (and its fp16 copy
// when `u16`), Vt, the K-major fp16 copies for the tensor-core deflation, and sign * D into B.d.
int stage_block(const Plan& p, const Bufs& B, const int8_t* Bf, const float* Df, const int8_t* Cf, long long j0, int w,
                float sign, bool u16, cudaStream_t s) {
  const int m = p.m, n = p.n;
  KL(0, 1, launch_transpose_i8(Bf + j0, p.k, m, w, B.Ut, p.ldm, s));
  LK(cudaMemcpy2DAsync(B.Vt, (size_t)p.ldn, Cf + j0 * n, (size_t)n, (size_t)n, (size_t)w, cudaMemcpyDeviceToDevice, s));
  if (use_tc(w)) {
    if (u16) KL(0, 1, launch_i8_to_f16(B.Ut, p.ldm, w, m, B.Ut16, p.ldm, s));
    KL(0, 1, launch_kmajor(B.Ut, p.ldm, 1, w, m, B.Uk16, B.ldk, s));
    KL(0, 1, launch_kmajor(B.Vt, p.ldn, 1, w, n, B.Vk16, B.ldk, s));
  }
  KL(0, 1, launch_scale_copy(Df + j0, sign, w, B.d, s));
  return EXTERND_OK;
}

// Enqueues p.sweeps refinement sweeps (§2.4) of the factors in (Bf, Df, Cf), updated in place: R = A - B D C,
// then for every block in order: add it back, refit it from its own U, keep the refit if it removes at least as
// much, deflate the kept block. trace[s] = energy after sweep s; counts[s] = blocks replaced in sweep s.
int enqueue_refine(Workspace& ws, const Plan& p, const Bufs& B, const float* A, const float* h, int8_t* Bf, float* Df,
                   int8_t* Cf, cudaStream_t s) {
  const int m = p.m, n = p.n;
  Eq2 q = make_eq2(p, B);
  g_prof.used = 0;
  g_prof.launches = 0;
  TRY(start_residual(p, B, A, h, s));
  for (int blk = 0; blk < p.nblocks; ++blk) {
    const long long j0 = (long long)blk * p.b;
    const int w = (int)std::min<long long>(p.b, p.k - j0);
    TRY(stage_block(p, B, Bf, Df, Cf, j0, w, 1.f, false, s));
    TRY(deflate_step(p, B, h, w, B.norm_r, nullptr, s));
  }
  for (int sw = 0; sw < p.sweeps; ++sw) {
    for (int blk = 0; blk < p.nblocks; ++blk) {
      const long long j0 = (long long)blk * p.b;
      const int w = (int)std::min<long long>(p.b, p.k - j0);
      TRY(stage_block(p, B, Bf, Df, Cf, j0, w, -1.f, true, s));
      TRY(deflate_step(p, B, h, w, B.norm_add, nullptr, s));              // add back: R_add = R + U D V^T
      TRY(fit_block(ws, p, B, q, h, blk, w, true, s));
      TRY(block_scales_step(p, B, w, B.K, s));
      KL(0, 1, launch_refine_decide(B.norm_add, B.norm_r, B.r, B.d, B.K, w, B.choice, s));
      KL(0, 1, launch_commit(B.choice, B.Ut, p.ldm, B.Vt, p.ldn, B.d, w, m, n, Bf, Df, Cf, p.k, j0, s));
      TRY(stage_block(p, B, Bf, Df, Cf, j0, w, 1.f, false, s));           // the kept block
      TRY(deflate_step(p, B, h, w, B.norm_r, blk == p.nblocks - 1 ? B.trace + sw : nullptr, s));
    }
    KL(0, 1, launch_count_reset(B.choice, B.counts + sw, s));
  }
  return EXTERND_OK;
}

struct GraphKey {
  const void *A, *h, *B, *D, *C;
  long long m, n, k;
  int b, iters;
  double tau;
  unsigned gen;
  int prof, mode, sweeps;
  bool operator<(const GraphKey& o) const {
    return std::tie(A, h, B, D, C, m, n, k, b, iters, tau, gen, prof, mode, sweeps) <
           std::tie(o.A, o.h, o.B, o.D, o.C, o.m, o.n, o.k, o.b, o.iters, o.tau, o.gen, o.prof, o.mode, o.sweeps);
  }
};

struct CachedGraph {
  cudaGraphExec_t exec;
  size_t events;        // profiling events the graph records
  long long launches;   // kernel nodes
};

std::map<int, std::map<GraphKey, CachedGraph>> g_graphs;

bool graphs_enabled() {
  const char* e = std::getenv("EXTERND_GRAPHS");
  return !(e && std::strcmp(e, "0") == 0);
}

// Runs the block loop of plan p on the library stream: captured once per configuration into a CUDA graph and
// replayed (EXTERND_GRAPHS=0 enqueues it directly). Then reads `ntrace` trace entries and, in the safeguard and
// refinement modes, `ncounts` counts back to the host.
int run_plan(const Plan& p, const float* A, const float* h, int8_t* Bout, float* Dout, int8_t* Cout, double* energy,
             double* trace, int ntrace, long long* counts, int ncounts) {
  Workspace* ws;
  TRY(current_ws(&ws));
  Bufs B;
  TRY(plan_buffers(*ws, p, &B));
  int dev;
  CK(cudaGetDevice(&dev));
  cudaStream_t s = g_stream;
  // The decompose modes read the caller's arrays through B.io, so their graphs serve every A, B, D, C of a shape;
  // refinement updates the factors in place at many nodes and keeps them in its graph.
  const bool via_io = p.mode != kRefine;
  auto enqueue = [&](cudaStream_t st) {
    return p.mode == kRefine ? enqueue_refine(*ws, p, B, A, h, Bout, Dout, Cout, st)
                             : enqueue_decompose(*ws, p, B, h, st);
  };
  if (via_io) LK(launch_io_set(B.io, A, Bout, Dout, Cout, s));
  if (graphs_enabled()) {
    GraphKey key{via_io ? nullptr : A, h, via_io ? nullptr : Bout, via_io ? nullptr : Dout, via_io ? nullptr : Cout,
                 p.m, p.n, p.k, p.b, p.iters, p.tau, ws->generation, g_prof.kind, p.mode, p.sweeps};
    auto& cache = g_graphs[dev];
    auto it = cache.find(key);
    if (it == cache.end()) {
      if (cache.size() >= 16) {
        for (auto& kv : cache) cudaGraphExecDestroy(kv.second.exec);
        cache.clear();
      }
      cudaGraph_t graph;
      CK(cudaStreamBeginCapture(ws->cap_stream, cudaStreamCaptureModeThreadLocal));
      int rc = enqueue(ws->cap_stream);
      cudaError_t ec = cudaStreamEndCapture(ws->cap_stream, &graph);
      if (rc != EXTERND_OK) return rc;
      if (ec != cudaSuccess) return cuda_fail(ec, "cudaStreamEndCapture");
      cudaGraphExec_t exec;
      cudaError_t ei = cudaGraphInstantiate(&exec, graph, 0);
      cudaGraphDestroy(graph);
      if (ei != cudaSuccess) return cuda_fail(ei, "cudaGraphInstantiate");
      it = cache.emplace(key, CachedGraph{exec, g_prof.used, g_prof.launches}).first;
    }
    CK(cudaGraphLaunch(it->second.exec, s));
    g_prof.last_used = it->second.events;
    g_prof.last_launches = it->second.launches + (via_io ? 1 : 0);
  } else {
    TRY(enqueue(s));
    g_prof.last_used = g_prof.used;
    g_prof.last_launches = g_prof.launches + (via_io ? 1 : 0);
  }
  if (energy != nullptr || trace != nullptr || counts != nullptr) {
    const size_t tb = sizeof(double) * (size_t)ntrace, cb = sizeof(long long) * (size_t)ncounts;
    void* hbuf;
    TRY(need_host(*ws, tb + cb + 16, &hbuf));
    if (ntrace > 0) CK(cudaMemcpyAsync(hbuf, B.trace, tb, cudaMemcpyDeviceToHost, s));
    if (ncounts > 0) CK(cudaMemcpyAsync(static_cast<char*>(hbuf) + tb, B.counts, cb, cudaMemcpyDeviceToHost, s));
    CK(cudaStreamSynchronize(s));
    const double* tr = static_cast<const double*>(hbuf);
    if (energy && ntrace > 0) *energy = tr[ntrace - 1];
    if (trace && ntrace > 0) std::memcpy(trace, tr, tb);
    if (counts && ncounts > 0) std::memcpy(counts, static_cast<char*>(hbuf) + tb, cb);
    TRY(check_device_error(*ws, B.err, s));
  }
  CK(cudaGetLastError());
  return EXTERND_OK;
}

// The one-launch cluster kernel for block width 1 where the residual fits its shared memory;
// EXTERND_SEQ=0 keeps the kernel-by-kernel schedule, for comparisons.
bool sequential_cluster_enabled() {
  static const bool enabled = [] {
    const char* e = std::getenv("EXTERND_SEQ");
    return !(e && std::strcmp(e, "0") == 0);
  }();
  return enabled;
}

// §2.3 in one cluster launch (sequential.cu): the components, the energy after each, the final energy.
int run_sequential(const Plan& p, const float* A, const float* h, int8_t* Bout, float* Dout, int8_t* Cout,
                   double* energy, double* trace, long long* activations) {
  Workspace* ws;
  TRY(current_ws(&ws));
  double *tr, *en;
  long long* act = nullptr;
  TRY(need(*ws, "trace", (size_t)p.k, &tr));
  TRY(need(*ws, "seq.energy", 1, &en));
  cudaStream_t s = g_stream;
  if (activations != nullptr) {
    TRY(need(*ws, "seq.act", 1, &act));
    LK(cudaMemsetAsync(act, 0, sizeof(long long), s));
  }
  g_prof.used = 0;
  const bool prof = g_prof.kind == kSolve;   // the whole fit is one kernel: timed as the solve class
  if (prof) LK(prof_mark(s, false));
  LK(launch_sequential_cluster(A, p.m, p.n, p.k, p.iters, p.tau, h, Bout, Dout, Cout, tr, en, act, s));
  if (prof) LK(prof_mark(s, false));
  g_prof.last_used = g_prof.used;
  g_prof.last_launches = 1;
  if (energy != nullptr || trace != nullptr || activations != nullptr) {
    const size_t tb = sizeof(double) * (size_t)(trace != nullptr ? p.k : 0);
    void* hbuf;
    TRY(need_host(*ws, tb + 16, &hbuf));
    CK(cudaMemcpyAsync(hbuf, en, sizeof(double), cudaMemcpyDeviceToHost, s));
    if (act) CK(cudaMemcpyAsync(static_cast<char*>(hbuf) + 8, act, sizeof(long long), cudaMemcpyDeviceToHost, s));
    if (tb > 0) CK(cudaMemcpyAsync(static_cast<char*>(hbuf) + 16, tr, tb, cudaMemcpyDeviceToHost, s));
    CK(cudaStreamSynchronize(s));
    if (energy) *energy = *static_cast<const double*>(hbuf);
    if (activations) *activations = *reinterpret_cast<const long long*>(static_cast<char*>(hbuf) + 8);
    if (tb > 0) std::memcpy(trace, static_cast<char*>(hbuf) + 16, tb);
  }
  CK(cudaGetLastError());
  return EXTERND_OK;
}

int run_decompose(const float* A, long long m, long long n, double mu, double tau, int block, int iters,
                  const float* h, int8_t* Bout, float* Dout, int8_t* Cout, double* energy, double* trace,
                  long long* activations = nullptr) {
  int64_t k;
  TRY(externd_rank(m, n, mu, &k));
  Plan p = make_plan(m, n, k, block, iters, tau);
  p.mode = activations != nullptr ? kSafeguard : kPlain;
  if (p.b == 1 && sequential_cluster_enabled() && sequential_cluster_fits(m, n))
    return run_sequential(p, A, h, Bout, Dout, Cout, energy, trace, activations);
  return run_plan(p, A, h, Bout, Dout, Cout, energy, trace, p.nblocks, activations, activations ? 1 : 0);
}

int check_device_error(Workspace& ws, unsigned* err, cudaStream_t s) {
  void* hb;
  TRY(need_host(ws, sizeof(double), &hb));
  CK(cudaMemcpyAsync(hb, err, sizeof(unsigned), cudaMemcpyDeviceToHost, s));
  CK(cudaStreamSynchronize(s));
  if (*static_cast<unsigned*>(hb) != 0u) {
    CK(cudaMemsetAsync(err, 0, sizeof(unsigned), s));
    auto bar = ws.bufs.find("bar");   // a grid that gave up may have left its barrier counters set
    if (bar != ws.bufs.end() && bar->second.p != nullptr) CK(cudaMemsetAsync(bar->second.p, 0, bar->second.cap, s));
    CK(cudaStreamSynchronize(s));
    return EXTERND_ETIMEOUT;
  }
  return EXTERND_OK;
}

// Sizes the kernels' grids cover: rows of R tile by 64 in gridDim.y (<= 65535 tiles), columns by 128 in gridDim.x.
constexpr long long kMaxRows = 65535LL * 64;
constexpr long long kMaxCols = 1LL << 30;

int check_common(long long m, long long n) {
  if (m < 1 || n < 1 || m > kMaxRows || n > kMaxCols || m * n > (1LL << 40)) return EXTERND_EINVAL;
  return EXTERND_OK;
}

int check_params(double mu, double tau, int block, int iters) {
  if (!(mu > 0) || !std::isfinite(mu) || !(tau >= 0) || !std::isfinite(tau)) return EXTERND_EINVAL;
  if (block < 1 || block > kMaxBlock || iters < 1) return EXTERND_EINVAL;
  return EXTERND_OK;
}

int check_dev(const void* p) { return is_device_ptr(p) ? EXTERND_OK : (p ? EXTERND_EPTR : EXTERND_EINVAL); }

// Per-step helpers: the fp16 scaling scalars {max |R|, max h} and the error word for a tensor-core product.
int step_scalars(Workspace& ws, const float* R, long long count, const float* h, long long n, float** mx,
                 unsigned** err) {
  TRY(need(ws, "step.maxabs", 2, mx));
  TRY(need(ws, "err", 1, err, true));
  LK(launch_absmax(R, count, *mx, g_stream));
  if (h != nullptr) LK(launch_absmax(h, n, *mx + 1, g_stream));
  return EXTERND_OK;
}

// Per-step helpers: bring a caller's m x w U into the internal Ut layout, and a w x n Cb into Vt; with T16 given,
// also the fp16 copy the tensor-core products read (nullptr when the FMA tiles run).
int stage_u(Workspace& ws, const int8_t* U, long long m, int w, int8_t** Ut, __half** T16 = nullptr) {
  TRY(need(ws, "Ut", (size_t)w * ld16(m), Ut, true));
  LK(launch_transpose_i8(U, w, (int)m, w, *Ut, ld16(m), g_stream));
  if (T16 != nullptr) {
    *T16 = nullptr;
    if (use_tc(w)) {
      TRY(need(ws, "Ut16", (size_t)w * ld16(m), T16, true));
      LK(launch_i8_to_f16(*Ut, ld16(m), w, (int)m, *T16, ld16(m), g_stream));
    }
  }
  return EXTERND_OK;
}

int stage_v(Workspace& ws, const int8_t* Cb, long long n, int w, int8_t** Vt, __half** T16 = nullptr) {
  TRY(need(ws, "Vt", (size_t)w * ld16(n), Vt, true));
  LK(cudaMemcpy2DAsync(*Vt, (size_t)ld16(n), Cb, (size_t)n, (size_t)n, (size_t)w, cudaMemcpyDeviceToDevice, g_stream));
  if (T16 != nullptr) {
    *T16 = nullptr;
    if (use_tc(w)) {
      TRY(need(ws, "Vt16", (size_t)w * ld16(n), T16, true));
      LK(launch_i8_to_f16(Cb, n, w, (int)n, *T16, ld16(n), g_stream));
    }
  }
  return EXTERND_OK;
}

int read_double(Workspace& ws, const double* dptr, double* out) {
  void* hb;
  TRY(need_host(ws, sizeof(double), &hb));
  CK(cudaMemcpyAsync(hb, dptr, sizeof(double), cudaMemcpyDeviceToHost, g_stream));
  CK(cudaStreamSynchronize(g_stream));
  *out = *static_cast<double*>(hb);
  return EXTERND_OK;
}

}  // namespace

// ==============================================================================================================
extern "C" {

const char* externd_strerror(int status) {
  switch (status) {
    case EXTERND_OK: return "ok";
    case EXTERND_EINVAL: return "invalid argument (size, parameter or NULL pointer)";
    case EXTERND_EPTR: return "pointer is not accessible from the CUDA device";
    case EXTERND_ENOMEM: return "device workspace allocation failed";
    case EXTERND_ECUDA: return "CUDA error (see externd_last_cuda_error)";
    case EXTERND_ENODEV: return "no usable CUDA device";
    case EXTERND_ETIMEOUT: return "a bounded device wait expired (a kernel gave up and returned)";
    default: return "unknown status";
  }
}

const char* externd_last_cuda_error(void) { return g_cuda_error; }

const char* externd_version(void) { return "externd-gb300 0.1 (sm_103a)"; }

int externd_set_stream(void* cuda_stream) {
  std::lock_guard<std::mutex> lock(g_mutex);
  g_stream = static_cast<cudaStream_t>(cuda_stream);
  return EXTERND_OK;
}

int externd_profile(int kind) {
  std::lock_guard<std::mutex> lock(g_mutex);
  if (kind < 0 || kind > 9) return EXTERND_EINVAL;
  g_prof.kind = kind;
  return EXTERND_OK;
}

int externd_profile_read(double* ms, int64_t* launches) {
  std::lock_guard<std::mutex> lock(g_mutex);
  if (ms == nullptr || launches == nullptr) return EXTERND_EINVAL;
  double total = 0.0;
  const size_t n = g_prof.last_used;
  if (n >= 2) CK(cudaEventSynchronize(g_prof.events[n - 1]));
  for (size_t i = 0; i + 1 < n; i += 2) {
    float t = 0.f;
    CK(cudaEventElapsedTime(&t, g_prof.events[i], g_prof.events[i + 1]));
    total += t;
  }
  *ms = total;
  *launches = (int64_t)(n / 2);
  return EXTERND_OK;
}

int externd_kernel_launches(int64_t* count) {
  std::lock_guard<std::mutex> lock(g_mutex);
  if (count == nullptr) return EXTERND_EINVAL;
  *count = g_prof.last_launches;
  return EXTERND_OK;
}

int externd_rank(int64_t m, int64_t n, double mu, int64_t* k) {
  if (k == nullptr || m < 1 || n < 1 || !(mu > 0) || !std::isfinite(mu)) return EXTERND_EINVAL;
  const double v = std::floor(mu * (double)std::min(m, n) + 0.5);
  if (v < 1 || v > 1e12) return EXTERND_EINVAL;
  *k = (int64_t)v;
  return EXTERND_OK;
}

int externd_block_width(int64_t m, int64_t n, int block, int* b) {
  if (b == nullptr || m < 1 || n < 1 || block < 1 || block > kMaxBlock) return EXTERND_EINVAL;
  *b = block_width_of(m, n, block);
  return EXTERND_OK;
}

int externd_decompose(const float* A, int64_t m, int64_t n, double mu, double tau, int block, int iters,
                      const float* weights, int8_t* B, float* D, int8_t* C, double* energy) {
  return externd_decompose_traced(A, m, n, mu, tau, block, iters, weights, B, D, C, energy, nullptr);
}

int externd_decompose_traced(const float* A, int64_t m, int64_t n, double mu, double tau, int block, int iters,
                             const float* weights, int8_t* B, float* D, int8_t* C, double* energy, double* trace) {
  std::lock_guard<std::mutex> lock(g_mutex);
  TRY(check_common(m, n));
  TRY(check_params(mu, tau, block, iters));
  // with energy == trace == NULL the results still land in B, D, C and nothing is read back
  TRY(check_dev(A));
  TRY(check_dev(B));
  TRY(check_dev(D));
  TRY(check_dev(C));
  if (weights != nullptr) TRY(check_dev(weights));
  return run_decompose(A, m, n, mu, tau, block, iters, weights, B, D, C, energy, trace);
}

int externd_decompose_safeguarded(const float* A, int64_t m, int64_t n, double mu, double tau, int block, int iters,
                                  const float* weights, int8_t* B, float* D, int8_t* C, double* energy, double* trace,
                                  int64_t* activations) {
  std::lock_guard<std::mutex> lock(g_mutex);
  TRY(check_common(m, n));
  TRY(check_params(mu, tau, block, iters));
  if (activations == nullptr) return EXTERND_EINVAL;
  TRY(check_dev(A));
  TRY(check_dev(B));
  TRY(check_dev(D));
  TRY(check_dev(C));
  if (weights != nullptr) TRY(check_dev(weights));
  long long act = 0;
  TRY(run_decompose(A, m, n, mu, tau, block, iters, weights, B, D, C, energy, trace, &act));
  *activations = act;
  return EXTERND_OK;
}

int externd_refine(const float* A, int64_t m, int64_t n, double tau, int block, int iters, int sweeps,
                   const float* weights, int8_t* B, float* D, int8_t* C, int64_t k, double* energy, double* trace,
                   int64_t* replaced) {
  std::lock_guard<std::mutex> lock(g_mutex);
  TRY(check_common(m, n));
  if (k < 1 || k > (1LL << 31) || sweeps < 1 || sweeps > 1000000) return EXTERND_EINVAL;
  TRY(check_params(1.0, tau, block, iters));
  TRY(check_dev(A));
  TRY(check_dev(B));
  TRY(check_dev(D));
  TRY(check_dev(C));
  if (weights != nullptr) TRY(check_dev(weights));
  Plan p = make_plan(m, n, k, block, iters, tau);
  p.mode = kRefine;
  p.sweeps = sweeps;
  std::vector<long long> counts((size_t)sweeps);
  TRY(run_plan(p, A, weights, B, D, C, energy, trace, sweeps, counts.data(), sweeps));
  if (replaced != nullptr)
    for (int i = 0; i < sweeps; ++i) replaced[i] = counts[(size_t)i];
  return EXTERND_OK;
}

int externd_decompose_host(const float* A, int64_t m, int64_t n, double mu, double tau, int block, int iters,
                           const float* weights, int8_t* B, float* D, int8_t* C, double* energy) {
  std::lock_guard<std::mutex> lock(g_mutex);
  TRY(check_common(m, n));
  TRY(check_params(mu, tau, block, iters));
  if (A == nullptr || B == nullptr || D == nullptr || C == nullptr) return EXTERND_EINVAL;
  int64_t k;
  TRY(externd_rank(m, n, mu, &k));
  Workspace* ws;
  TRY(current_ws(&ws));
  float *dA, *dh = nullptr, *dD;
  int8_t *dB, *dC;
  TRY(need(*ws, "host.A", (size_t)m * n, &dA));
  TRY(need(*ws, "host.B", (size_t)m * k, &dB));
  TRY(need(*ws, "host.C", (size_t)k * n, &dC));
  TRY(need(*ws, "host.D", (size_t)k, &dD));
  if (weights) TRY(need(*ws, "host.h", (size_t)n, &dh));
  cudaStream_t s = g_stream;
  CK(cudaMemcpyAsync(dA, A, sizeof(float) * m * n, cudaMemcpyHostToDevice, s));
  if (weights) CK(cudaMemcpyAsync(dh, weights, sizeof(float) * n, cudaMemcpyHostToDevice, s));
  TRY(run_decompose(dA, m, n, mu, tau, block, iters, dh, dB, dD, dC, energy, nullptr));
  CK(cudaMemcpyAsync(B, dB, (size_t)m * k, cudaMemcpyDeviceToHost, s));
  CK(cudaMemcpyAsync(C, dC, (size_t)k * n, cudaMemcpyDeviceToHost, s));
  CK(cudaMemcpyAsync(D, dD, sizeof(float) * k, cudaMemcpyDeviceToHost, s));
  CK(cudaStreamSynchronize(s));
  return EXTERND_OK;
}

int externd_energy(const float* A, int64_t m, int64_t n, const int8_t* B, const float* D, const int8_t* C, int64_t k,
                   const float* weights, double* energy) {
  std::lock_guard<std::mutex> lock(g_mutex);
  TRY(check_common(m, n));
  if (k < 1 || k > (1LL << 31) || energy == nullptr) return EXTERND_EINVAL;
  TRY(check_dev(A));
  TRY(check_dev(B));
  TRY(check_dev(D));
  TRY(check_dev(C));
  if (weights != nullptr) TRY(check_dev(weights));
  Workspace* ws;
  TRY(current_ws(&ws));
  F2* part;
  double* sc;
  TRY(need(*ws, "energy.part", (size_t)deflate_tiles((int)m, (int)n), &part));
  TRY(need(*ws, "energy.sc", 4, &sc));
  const int tiles = deflate_tiles((int)m, (int)n);
  LK(launch_deflate(A, nullptr, (int)m, (int)n, nullptr, 0, false, nullptr, nullptr, 0, 0, weights, nullptr, part,
                    g_stream));
  LK(launch_norm(part, tiles, sc, nullptr, nullptr, g_stream));
  LK(launch_deflate(A, nullptr, (int)m, (int)n, B, k, true, D, C, n, (int)k, weights, nullptr, part, g_stream));
  LK(launch_norm(part, tiles, sc + 1, sc, sc + 2, g_stream));
  return read_double(*ws, sc + 2, energy);
}

int externd_ternarize(const float* X, int64_t rows, int64_t cols, int axis, double tau, int8_t* T) {
  std::lock_guard<std::mutex> lock(g_mutex);
  TRY(check_common(rows, cols));
  if ((axis != 0 && axis != 1) || !(tau >= 0) || !std::isfinite(tau)) return EXTERND_EINVAL;
  TRY(check_dev(X));
  TRY(check_dev(T));
  Workspace* ws;
  TRY(current_ws(&ws));
  const long long nv = axis == 1 ? rows : cols, L = axis == 1 ? cols : rows;
  if (nv > 65535) return EXTERND_EINVAL;   // one grid row per vector
  const int nchunk = (int)cdiv(L, kStatChunk);
  StatPart* sp;
  float* theta;
  int* fb;
  unsigned *arg, *ticket;
  TRY(need(*ws, "tern.spart", (size_t)nv * nchunk, &sp));
  TRY(need(*ws, "tern.theta", (size_t)nv, &theta));
  TRY(need(*ws, "tern.fallback", (size_t)nv, &fb));
  TRY(need(*ws, "tern.arg", (size_t)nv, &arg));
  TRY(need(*ws, "ticket", 1, &ticket, true));
  const Thresh th{theta, fb, arg, ticket, tau, (int)L};
  Stats st{sp, nchunk, th};
  if (axis == 1) {
    LK(launch_stats(X, (int)nv, (int)L, (int)L, st, g_stream));
    LK(launch_apply(X, (int)nv, (int)L, L, th, T, (int)L, nullptr, g_stream));
  } else {
    float* Xt;
    int8_t* Tt;
    TRY(need(*ws, "tern.X", (size_t)nv * L, &Xt));
    TRY(need(*ws, "tern.T", (size_t)nv * L, &Tt));
    LK(launch_transpose_f32(X, cols, (int)rows, (int)cols, Xt, L, g_stream));
    LK(launch_stats(Xt, (int)nv, (int)L, (int)L, st, g_stream));
    LK(launch_apply(Xt, (int)nv, (int)L, L, th, Tt, (int)L, nullptr, g_stream));
    LK(launch_transpose_i8(Tt, L, (int)nv, (int)L, T, cols, g_stream));
  }
  CK(cudaGetLastError());
  return EXTERND_OK;
}

#define STEP_CHECKS(R_, w_)                                  \
  TRY(check_common(m, n));                                   \
  if ((w_) < 1 || (w_) > kMaxBlock) return EXTERND_EINVAL;   \
  TRY(check_dev(R_));

int externd_vstep_product(const float* R, int64_t m, int64_t n, const int8_t* U, int64_t w, float* PV) {
  std::lock_guard<std::mutex> lock(g_mutex);
  STEP_CHECKS(R, w);
  TRY(check_dev(U));
  TRY(check_dev(PV));
  Workspace* ws;
  TRY(current_ws(&ws));
  int8_t* Ut;
  __half* U16;
  float *part, *mx;
  unsigned* err;
  TRY(stage_u(*ws, U, m, (int)w, &Ut, &U16));
  TRY(step_scalars(*ws, R, m * n, nullptr, 0, &mx, &err));
  const int sv = splits_v((int)w, (int)m, (int)n, R, U16, (int)ld16(m));
  TRY(need(*ws, "part", (size_t)sv * w * n, &part));
  LK(product_v(R, (int)m, (int)n, Ut, U16, (int)ld16(m), (int)w, part, sv, mx, err, g_stream));
  LK(launch_sum_splits(part, sv, (int)w, (int)n, PV, n, g_stream));
  return check_device_error(*ws, err, g_stream);
}

int externd_ustep_product(const float* R, int64_t m, int64_t n, const int8_t* Cb, int64_t w, const float* weights,
                          float* PU) {
  std::lock_guard<std::mutex> lock(g_mutex);
  STEP_CHECKS(R, w);
  TRY(check_dev(Cb));
  TRY(check_dev(PU));
  if (weights) TRY(check_dev(weights));
  Workspace* ws;
  TRY(current_ws(&ws));
  int8_t* Vt;
  __half* V16;
  float *part, *X, *mx;
  unsigned* err;
  TRY(stage_v(*ws, Cb, n, (int)w, &Vt, &V16));
  TRY(step_scalars(*ws, R, m * n, weights, n, &mx, &err));
  const int su = splits_u((int)w, (int)m, (int)n, R, V16, (int)ld16(n));
  TRY(need(*ws, "part", (size_t)su * w * m, &part));
  TRY(need(*ws, "X", (size_t)w * m, &X));
  LK(product_u(R, (int)m, (int)n, Vt, V16, (int)ld16(n), (int)w, weights, part, su, mx, err, g_stream));
  LK(launch_sum_splits(part, su, (int)w, (int)m, X, m, g_stream));
  LK(launch_transpose_f32(X, m, (int)w, (int)m, PU, w, g_stream));
  return check_device_error(*ws, err, g_stream);
}

namespace {
int step_target(bool vstep, const float* R, long long m, long long n, const int8_t* F, int w, const float* h,
                float* out) {
  Workspace* ws;
  TRY(current_ws(&ws));
  const long long L = vstep ? n : m;
  const int nchunk = decorrelate_chunks((int)L, w);
  int8_t* T;
  __half* T16;
  float *part, *X, *Gpart, *Graw, *Ginv, *one;
  StatPart* sp;
  if (vstep) TRY(stage_u(*ws, F, m, w, &T, &T16));
  else TRY(stage_v(*ws, F, n, w, &T, &T16));
  const long long ldt = vstep ? ld16(m) : ld16(n);
  const long long Lred = vstep ? m : n;
  float* mx;
  unsigned* err;
  TRY(step_scalars(*ws, R, m * n, vstep ? nullptr : h, n, &mx, &err));
  const int splits = vstep ? splits_v(w, (int)m, (int)n, R, T16, (int)ldt) : splits_u(w, (int)m, (int)n, R, T16, (int)ldt);
  const int gs = gram_splits(w, (int)Lred);
  TRY(need(*ws, "part", (size_t)splits * w * L, &part));
  TRY(need(*ws, "X", (size_t)w * L, &X));
  TRY(need(*ws, "Gpart", (size_t)gs * w * w, &Gpart));
  TRY(need(*ws, "GrawV", (size_t)w * w, &Graw));
  TRY(need(*ws, "Ginv", (size_t)w * w, &Ginv));
  TRY(need(*ws, "spart", (size_t)w * nchunk, &sp));
  TRY(get_one(*ws, &one));
  if (vstep) LK(product_v(R, (int)m, (int)n, T, T16, (int)ldt, w, part, splits, mx, err, g_stream));
  else LK(product_u(R, (int)m, (int)n, T, T16, (int)ldt, w, h, part, splits, mx, err, g_stream));
  unsigned* gop = nullptr;
  if (decorrelate_needs_operand(w)) TRY(need(*ws, "gop", ginv_operand_bytes() / sizeof(unsigned), &gop));
  if (w > 1) {
    LK(launch_gram(T, (int)ldt, w, (int)Lred, vstep ? nullptr : h, Gpart, gs, g_stream));
    LK(inverse_f(Gpart, gs, w, Graw, Ginv, g_stream, gop, err));
  }
  float* theta;
  int* fb;
  unsigned *arg, *ticket;
  TRY(need(*ws, "theta", (size_t)w, &theta));
  TRY(need(*ws, "fallback", (size_t)w, &fb));
  TRY(need(*ws, "arg", (size_t)w, &arg));
  TRY(need(*ws, "ticket", 1, &ticket, true));
  Stats st{sp, nchunk, Thresh{theta, fb, arg, ticket, 0.0, (int)L}};
  if (vstep) {
    LK(launch_decorrelate(w > 1 ? Ginv : one, w, part, splits, (int)L, out, (int)L, st, g_stream, nullptr, err, gop));
  } else {
    LK(launch_decorrelate(w > 1 ? Ginv : one, w, part, splits, (int)L, X, (int)L, st, g_stream, nullptr, err, gop));
    LK(launch_transpose_f32(X, L, w, (int)L, out, w, g_stream));
  }
  return check_device_error(*ws, err, g_stream);
}
}  // namespace

int externd_vstep_target(const float* R, int64_t m, int64_t n, const int8_t* U, int64_t w, float* X) {
  std::lock_guard<std::mutex> lock(g_mutex);
  STEP_CHECKS(R, w);
  TRY(check_dev(U));
  TRY(check_dev(X));
  return step_target(true, R, m, n, U, (int)w, nullptr, X);
}

int externd_ustep_target(const float* R, int64_t m, int64_t n, const int8_t* Cb, int64_t w, const float* weights,
                         float* Y) {
  std::lock_guard<std::mutex> lock(g_mutex);
  STEP_CHECKS(R, w);
  TRY(check_dev(Cb));
  TRY(check_dev(Y));
  if (weights) TRY(check_dev(weights));
  return step_target(false, R, m, n, Cb, (int)w, weights, Y);
}

int externd_block_scales(const float* R, int64_t m, int64_t n, const int8_t* U, const int8_t* Cb, int64_t w,
                         const float* weights, float* d) {
  std::lock_guard<std::mutex> lock(g_mutex);
  STEP_CHECKS(R, w);
  TRY(check_dev(U));
  TRY(check_dev(Cb));
  TRY(check_dev(d));
  if (weights) TRY(check_dev(weights));
  Workspace* ws;
  TRY(current_ws(&ws));
  int8_t *Ut, *Vt;
  __half* V16;
  float *part, *Gpart, *GrawV, *Ginv, *mx;
  unsigned* err;
  float* r;
  TRY(stage_u(*ws, U, m, (int)w, &Ut));
  TRY(stage_v(*ws, Cb, n, (int)w, &Vt, &V16));
  TRY(step_scalars(*ws, R, m * n, weights, n, &mx, &err));
  const int su = splits_u((int)w, (int)m, (int)n, R, V16, (int)ld16(n));
  const int gm = gram_splits((int)w, (int)m), gn = gram_splits((int)w, (int)n);
  TRY(need(*ws, "part", (size_t)su * w * m, &part));
  TRY(need(*ws, "Gpart", (size_t)std::max(gm, gn) * w * w, &Gpart));
  TRY(need(*ws, "GrawV", (size_t)w * w, &GrawV));
  TRY(need(*ws, "Ginv", (size_t)w * w, &Ginv));
  TRY(need(*ws, "r", (size_t)w, &r));
  LK(product_u(R, (int)m, (int)n, Vt, V16, (int)ld16(n), (int)w, weights, part, su, mx, err, g_stream));
  LK(launch_gram(Vt, (int)ld16(n), (int)w, (int)n, weights, Gpart, gn, g_stream));
  LK(inverse_f(Gpart, gn, (int)w, GrawV, Ginv, g_stream, nullptr, err));
  LK(launch_gram(Ut, (int)ld16(m), (int)w, (int)m, nullptr, Gpart, gm, g_stream));
  LK(launch_rvec(Ut, (int)ld16(m), (int)w, (int)m, part, su, r, g_stream));
  LK(scales_f(Gpart, gm, GrawV, r, (int)w, d, g_stream, nullptr, err));
  return check_device_error(*ws, err, g_stream);
}

int externd_deflate(float* R, int64_t m, int64_t n, const int8_t* U, const float* d, const int8_t* Cb, int64_t w,
                    const float* weights, double* norm2) {
  std::lock_guard<std::mutex> lock(g_mutex);
  STEP_CHECKS(R, w);
  TRY(check_dev(U));
  TRY(check_dev(d));
  TRY(check_dev(Cb));
  if (weights) TRY(check_dev(weights));
  Workspace* ws;
  TRY(current_ws(&ws));
  F2* part;
  double* sc;
  const int tiles = deflate_tiles((int)m, (int)n);
  TRY(need(*ws, "energy.part", (size_t)tiles, &part));
  TRY(need(*ws, "energy.sc", 4, &sc));
  if (use_tc((int)w)) {
    const long long ldk = round_up(w, 16);
    __half *Uk, *Vk;
    unsigned* err;
    TRY(need(*ws, "step.Uk16", (size_t)m * ldk, &Uk, true));
    TRY(need(*ws, "step.Vk16", (size_t)n * ldk, &Vk, true));
    TRY(need(*ws, "err", 1, &err, true));
    LK(launch_kmajor(U, 1, w, (int)w, (int)m, Uk, ldk, g_stream));    // U is m x w row-major
    LK(launch_kmajor(Cb, n, 1, (int)w, (int)n, Vk, ldk, g_stream));   // Cb is w x n row-major
    LK(launch_deflate_tc(R, (int)m, (int)n, Uk, Vk, ldk, d, (int)w, weights, nullptr, part, nullptr, err,
                         g_stream));
    LK(launch_norm(part, tiles, sc, nullptr, nullptr, g_stream));
    TRY(check_device_error(*ws, err, g_stream));
  } else {
    int8_t *Ut, *Vt;
    TRY(stage_u(*ws, U, m, (int)w, &Ut));
    TRY(stage_v(*ws, Cb, n, (int)w, &Vt));
    LK(launch_deflate(R, R, (int)m, (int)n, Ut, ld16(m), false, d, Vt, ld16(n), (int)w, weights, nullptr, part,
                      g_stream));
    LK(launch_norm(part, tiles, sc, nullptr, nullptr, g_stream));
  }
  if (norm2 != nullptr) return read_double(*ws, sc, norm2);
  return EXTERND_OK;
}

int externd_pack_ternary(const int8_t* T, int64_t rows, int64_t cols, int64_t ldt, uint32_t* words, int64_t* nnz) {
  std::lock_guard<std::mutex> lock(g_mutex);
  if (rows < 1 || cols < 1 || ldt < cols || rows > (1LL << 31) || cols > (1LL << 31) ||
      packed_words(rows, cols) > (1LL << 36))
    return EXTERND_EINVAL;
  TRY(check_dev(T));
  TRY(check_dev(words));
  Workspace* ws;
  TRY(current_ws(&ws));
  unsigned long long* cnt;
  TRY(need(*ws, "pack.nnz", 1, &cnt));
  LK(cudaMemsetAsync(cnt, 0, sizeof(unsigned long long), g_stream));
  LK(launch_pack_ternary(T, rows, cols, ldt, words, cnt, g_stream));
  if (nnz != nullptr) {
    void* hb;
    TRY(need_host(*ws, sizeof(unsigned long long), &hb));
    CK(cudaMemcpyAsync(hb, cnt, sizeof(unsigned long long), cudaMemcpyDeviceToHost, g_stream));
    CK(cudaStreamSynchronize(g_stream));
    *nnz = (int64_t)(*static_cast<unsigned long long*>(hb));
  }
  return EXTERND_OK;
}

int externd_ternary_apply(const uint32_t* Bp, const float* D, const uint32_t* Cp, int64_t m, int64_t k, int64_t n,
                          const float* x, float* y) {
  std::lock_guard<std::mutex> lock(g_mutex);
  if (m < 1 || k < 1 || n < 1 || m > (1LL << 31) || k > (1LL << 31) || n > (1LL << 31)) return EXTERND_EINVAL;
  TRY(check_dev(Bp));
  TRY(check_dev(D));
  TRY(check_dev(Cp));
  TRY(check_dev(x));
  TRY(check_dev(y));
  Workspace* ws;
  TRY(current_ws(&ws));
  // z = D (.) (C x) goes straight into the fragments of the second product's vector
  float *z, *part;
  uint32_t *xf, *zf;
  unsigned* ticket;
  long long pc, tc, pb, tb;
  gemv_scratch(k, n, &pc, &tc);
  gemv_scratch(m, k, &pb, &tb);
  TRY(need(*ws, "apply.z", (size_t)k, &z));
  TRY(need(*ws, "apply.xf", (size_t)fragment_words(n), &xf));
  TRY(need(*ws, "apply.zf", (size_t)fragment_words(k), &zf, true));
  TRY(need(*ws, "apply.part", (size_t)std::max(pc, pb), &part));
  TRY(need(*ws, "apply.ticket", (size_t)std::max(tc, tb), &ticket, true));
  // x's fragments; the first product writes z's up to 32 * ceil(k / 32) columns, the rest of the last group is zeroed
  LK(launch_fragments(x, n, xf, zf, k, g_stream));
  LK(launch_ternary_gemv(Cp, k, n, xf, D, z, zf, part, ticket, g_stream));
  LK(launch_ternary_gemv(Bp, m, k, zf, nullptr, y, nullptr, part, ticket, g_stream));
  return EXTERND_OK;
}

}  // extern "C"

// Accessors for other translation units of the library (the stream, lock and error text above).
namespace externd {
cudaStream_t library_stream() { return g_stream; }
std::mutex& library_mutex() { return g_mutex; }
int record_cuda_error(cudaError_t e, const char* where) { return cuda_fail(e, where); }
}  // namespace externd
