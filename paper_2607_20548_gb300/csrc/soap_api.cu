// libsoap: the C ABI of include/soap.h.
//
// Memory plan. The optimizer state proper is all that stays resident: per matrix M_hat and v
// (rows x cols), the factors L and R as packed lower-triangular tiles (half of a full matrix),
// and the bases Q_L, Q_R. Matrices with the same (rows, cols, sides) form a class, whose state
// sits in contiguous arenas ([count][...]). Everything a step forms from that state -- the
// gradient copy G and G^T, every tensor-core operand's tf32 lo part, Q^T, the unpacked
// factors, the QR's workspace and the rotation intermediates -- lives in one workspace arena.
// A step walks the classes in slices (runs of consecutive matrices of one class) grouped into
// waves: a wave's slices are laid out side by side in the arena, and the next wave reuses it.
// When the whole model fits, there is one wave holding every class whole; otherwise the waves
// are cut to the free device memory (or to the caller's workspace limit).
//
// Within a wave, the slices' own launches go to the caller's stream (prepared largest factor
// first, rotated smallest first); the QR refreshes of the wave are regrouped by factor size, one
// batched QR per size on its own pair of streams, forked as soon as the last slice feeding it is
// prepared and joined by events before the slices whose bases it refreshes are rotated.
//
// Per slice, the step (Alg. 1 with the standard factor EMAs of section 2) is:
//   M_hat <- b1 M_hat + (1-b1) G, Gc <- G                 momentum in the original basis
//   L <- b L + (1-b) Gc Gc^T, R <- b R + (1-b) Gc^T Gc     S1 (on the unpacked factors, then packed)
//   P = L Q_L -> Q_L = QR(P).Q; same for R                 S2, S3 (when t mod F == 0)
//   X1 = Q_L^T Gc, X2 = Q_L^T M_hat                        S5, S4 (re-projected m)
//   G' = X1 Q_R, m = X2 Q_R
//   v <- b2 v + (1-b2) G'^2, N = m / (sqrt(v) + eps)        S6
//   X1 = Q_L N; W <- (1 - lr wd) W - lr X1 Q_R^T           S7, S8 (fused in the GEMM epilogue)
// With hparams.stale, S1 moves to the end of the step (the refresh sees the earlier gradients
// only). With hparams.kl, S1 takes Alg. 1's KL-Shampoo form instead: each factor's EMA term is
// weighed by the other factor's inverse, Q diag(1/(lam + eps)) Q^T with lam = diag(Q^T F Q)
// (an identity side as lam = 1); see accumulate_factors.
#include <algorithm>
#include <cstdio>
#include <cstring>
#include <map>
#include <string>
#include <tuple>
#include <vector>

#include "profile.h"
#include "soap_internal.h"

namespace {

struct ClassState {
  int64_t rows = 0, cols = 0;
  bool left = false, right = false;
  int count = 0;
  std::vector<int> members;
  size_t ptr_offset = 0;  // index of this class's params pointers in the pointer table
  // tensor-core path (both dimensions multiples of 4): operand copies with lo parts in the
  // workspace, factors packed; otherwise CUDA cores with full factors
  bool tc = false;
  // working orientation transposed: a class preconditioned on its left only runs as the
  // right-only problem of G^T, and keeps M_hat and v as M_hat^T and v^T
  bool tr = false;
  // persistent state
  float* Mhat = nullptr;  // first moment in the original basis, in the working orientation
  float* V = nullptr;
  float* L = nullptr;     // tc: [count][packed_floats(rows)]; CUDA cores: [count][rows][rows]
  float* QL = nullptr;    // [count][rows][rows]
  float* R = nullptr;
  float* QR = nullptr;
  uint8_t* skipL = nullptr;
  uint8_t* skipR = nullptr;
  // KL-Shampoo factor form, two-sided classes: the approximate eigenvalues of the last step
  float* lamL = nullptr;  // [count][rows]
  float* lamR = nullptr;  // [count][cols]
  int64_t lpk() const { return tc ? soap::packed_floats((int)rows) : rows * rows; }
  int64_t rpk() const { return tc ? soap::packed_floats((int)cols) : cols * cols; }
};

// `count` consecutive matrices of one class, starting at slot `first`: the persistent state
// offset to that slot, and the slice's operands in the workspace.
struct View {
  int cls = 0, first = 0, count = 0;
  // persistent state of the slice
  float *Mhat = nullptr, *V = nullptr, *L = nullptr, *QL = nullptr, *R = nullptr, *QR = nullptr;
  uint8_t *skipL = nullptr, *skipR = nullptr;
  float *lamL = nullptr, *lamR = nullptr;
  // workspace: [G | M_hat copy] (or G alone if tr) and [G^T] (or [G^T | M_hat^T copy]), lo parts
  float *Gc = nullptr, *Gc_lo = nullptr, *Gt = nullptr, *Gt_lo = nullptr;
  float *Mc = nullptr, *Mc_lo = nullptr;  // the M_hat copy inside Gc or Gt
  // workspace: unpacked factors with lo parts, and the bases' lo parts and transposes
  float *Lf = nullptr, *Lf_lo = nullptr, *QL_lo = nullptr, *QLt = nullptr, *QLt_lo = nullptr;
  float *Rf = nullptr, *Rf_lo = nullptr, *QR_lo = nullptr, *QRt = nullptr, *QRt_lo = nullptr;
};

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

// View of matrices [first, first + count) of class `cls` with its workspace at `base` (null
// base: only the size is computed); returns the workspace bytes.
size_t make_view(const ClassState& c, int cls, int first, int count, char* base, View* v) {
  View w;
  w.cls = cls;
  w.first = first;
  w.count = count;
  const int64_t m = c.rows, n = c.cols, mn = m * n;
  w.Mhat = c.Mhat ? c.Mhat + first * mn : nullptr;
  w.V = c.V ? c.V + first * mn : nullptr;
  if (c.left) {
    w.L = c.L ? c.L + first * c.lpk() : nullptr;
    w.QL = c.QL ? c.QL + first * m * m : nullptr;
    w.skipL = c.skipL ? c.skipL + first * m : nullptr;
    w.lamL = c.lamL ? c.lamL + first * m : nullptr;
  }
  if (c.right) {
    w.R = c.R ? c.R + first * c.rpk() : nullptr;
    w.QR = c.QR ? c.QR + first * n * n : nullptr;
    w.skipR = c.skipR ? c.skipR + first * n : nullptr;
    w.lamR = c.lamR ? c.lamR + first * n : nullptr;
  }
  size_t off = 0;
  auto take = [&](size_t floats) -> float* {
    const size_t o = off;
    off += align256(floats * sizeof(float));
    return base ? reinterpret_cast<float*>(base + o) : nullptr;
  };
  const size_t cmn = (size_t)count * mn, cmm = (size_t)count * m * m, cnn = (size_t)count * n * n;
  if (!c.tc) {
    w.Gc = take(cmn);  // the gradient copy; M_hat stays where it is
    w.Lf = w.L;
    w.Rf = w.R;
  } else {
    const size_t ga = c.tr ? cmn : 2 * cmn, ta = c.tr ? 2 * cmn : cmn;
    w.Gc = take(ga);
    w.Gc_lo = take(ga);
    w.Gt = take(ta);
    w.Gt_lo = take(ta);
    if (base) {
      w.Mc = c.tr ? w.Gt + cmn : w.Gc + cmn;
      w.Mc_lo = c.tr ? w.Gt_lo + cmn : w.Gc_lo + cmn;
    }
    if (c.left) {
      w.Lf = take(cmm);
      w.Lf_lo = take(cmm);
      w.QL_lo = take(cmm);
      w.QLt = take(cmm);
      w.QLt_lo = take(cmm);
    }
    if (c.right) {
      w.Rf = take(cnn);
      w.Rf_lo = take(cnn);
      w.QR_lo = take(cnn);
      w.QRt = take(cnn);
      w.QRt_lo = take(cnn);
    }
  }
  if (v) *v = w;
  return off;
}

// One preconditioned side of one slice: `count` factors of size n in a QR group.
struct QrJob {
  int slice;
  bool left;
  int offset;  // first batch index of this job inside its group
};

// All factors of one size in a wave, refreshed by one batched QR on their own streams.
struct QrGroup {
  int n = 0;
  int batch = 0;
  std::vector<QrJob> jobs;
  size_t ws_off = 0, ws_bytes = 0, skip_off = 0;  // in the arena
  int slot = 0;                                   // which stream pair and events
};

struct Slice {
  int cls = 0, first = 0, count = 0;
  size_t off = 0;  // workspace offset in the arena
};

struct Wave {
  std::vector<Slice> slices;
  std::vector<int> prep_order;               // slices, largest factor first
  std::vector<int> update_order;             // slices, smallest largest-factor first
  std::vector<std::vector<int>> fork_after;  // per slice: groups whose last feeding slice it is
  std::vector<std::vector<int>> groups_of;   // per slice: the groups its bases come from
  std::vector<QrGroup> groups;
  size_t bytes = 0;    // arena bytes the wave uses
  size_t base = 0;     // where its half of the arena starts (waves alternate between two halves)
  int slot_base = 0;   // its groups' stream pairs are slots slot_base + g.slot
};

// Streams and events of one QR group slot (reused by every wave).
struct GroupStreams {
  cudaStream_t stream = nullptr;  // panels and the rows that gate them (high priority)
  cudaStream_t far = nullptr;     // the rest of each block's trailing update (low priority)
  cudaEvent_t ev_vt = nullptr, ev_far = nullptr, ev_vq[2] = {nullptr, nullptr};
  cudaEvent_t done = nullptr;
  cudaEvent_t fork = nullptr;  // recorded on the caller's stream once the group's inputs are ready
};

struct DeviceGuard {
  int prev = -1;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
    if (prev != dev) cudaSetDevice(dev);
  }
  ~DeviceGuard() {
    int cur = -1;
    if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
  }
};

}  // namespace

struct soap_s {
  int device = 0;
  soap_hparams hp{};
  float lr = 0.f, wd = 0.f;
  int64_t t = 0;
  std::vector<soap_shape> shapes;
  std::vector<std::pair<int, int>> loc;  // matrix index -> (class, slot)
  std::vector<ClassState> classes;
  std::vector<Wave> waves;
  bool pipelined = false;  // waves alternate between two halves of the arena
  std::vector<GroupStreams> slots;
  char* arena = nullptr;  // workspace of one wave at a time
  size_t arena_bytes = 0;
  size_t state_bytes = 0;
  // rotation intermediates, shared by the slices of a wave (their rotations run one after
  // another on the caller's stream)
  float* X1 = nullptr;
  float* X2 = nullptr;
  float* Gp = nullptr;   // [G' | m'] for the tensor-core path: Gp .. Gp + 2 * ws_mat
  float* Mp = nullptr;   // m' for the CUDA-core path (Gp + ws_mat)
  float* YMt = nullptr;  // (G Q_R)^T and (M_hat Q_R)^T
  float* YMt_lo = nullptr;
  float* N_lo = nullptr;
  float* Zt = nullptr;   // (N Q_R^T)^T
  float* Zt_lo = nullptr;
  float* lam_ws = nullptr;  // Q^T F of the KL form's eigenvalue estimate (two-sided classes)
  size_t ws_mat = 0;
  size_t rot_bytes = 0;
  int* d_status = nullptr;
  int* h_status = nullptr;  // pinned mirror, refreshed after every step
  cudaEvent_t status_ev = nullptr;
  bool status_pending = false;
  cudaEvent_t step_done = nullptr;  // the last enqueued step's end (steps share the workspace)
  bool step_recorded = false;
  void** d_ptrs = nullptr;  // params/grads pointer table, [class][params..., grads...]
  size_t nptrs = 0;
  std::vector<void*> last_ptrs;
  std::vector<void*> allocs;
  soap::Profiler prof;
  std::string err;
};

namespace {

soap_status_t fail(soap_handle h, soap_status_t code, const std::string& msg) {
  if (h) h->err = msg;
  return code;
}

soap_status_t cuda_fail(soap_handle h, cudaError_t e, const char* what) {
  std::string m = std::string(what) + ": " + cudaGetErrorString(e);
  if (e == cudaErrorMemoryAllocation) return fail(h, SOAP_ERR_OOM, m);
  return fail(h, SOAP_ERR_CUDA, m);
}

#define SOAP_CUDA(h, expr)                              \
  do {                                                  \
    cudaError_t e_ = (expr);                            \
    if (e_ != cudaSuccess) return cuda_fail(h, e_, #expr); \
  } while (0)

// Report the cause: a product whose wait gave up leaves its output unwritten, which can make
// later values non-finite, and a non-finite gradient also makes the QR of that step break down.
soap_status_t status_code(int bits) {
  if (bits & soap::kStatusTimeout) return SOAP_ERR_TIMEOUT;
  if (bits & soap::kStatusNonFinite) return SOAP_ERR_NONFINITE;
  if (bits & soap::kStatusQrBreakdown) return SOAP_ERR_QR_BREAKDOWN;
  return SOAP_OK;
}

cudaError_t dalloc(soap_handle h, void** p, size_t bytes) {
  *p = nullptr;
  if (bytes == 0) return cudaSuccess;
  cudaError_t e = cudaMalloc(p, bytes);
  if (e == cudaSuccess) h->allocs.push_back(*p);
  return e;
}

void free_all(soap_handle h) {
  if (soap::t_profiler == &h->prof) soap::t_profiler = nullptr;
  for (cudaEvent_t ev : h->prof.events) cudaEventDestroy(ev);
  h->prof.events.clear();
  for (void* p : h->allocs) cudaFree(p);
  h->allocs.clear();
  if (h->h_status) cudaFreeHost(h->h_status);
  if (h->status_ev) cudaEventDestroy(h->status_ev);
  if (h->step_done) cudaEventDestroy(h->step_done);
  for (auto& g : h->slots) {
    if (g.stream) cudaStreamDestroy(g.stream);
    if (g.far) cudaStreamDestroy(g.far);
    for (cudaEvent_t ev : {g.done, g.fork, g.ev_vt, g.ev_far, g.ev_vq[0], g.ev_vq[1]})
      if (ev) cudaEventDestroy(ev);
  }
  h->slots.clear();
  h->h_status = nullptr;
  h->status_ev = h->step_done = nullptr;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

soap::TcOperand opnd(const float* hi, const float* lo, int64_t ld, int64_t stride, int batch) {
  return soap::TcOperand{hi, lo, ld, stride, batch};
}

soap::TcEpilogue epi(soap_handle h, float* C, int64_t ldc, int64_t c_stride, float* C_lo, int transpose, float alpha,
                     float beta) {
  return soap::TcEpilogue{C, nullptr, ldc, c_stride, C_lo, ldc, c_stride, transpose, alpha, beta, h->d_status};
}

View view_of(soap_handle h, const Wave& w, const Slice& sl) {
  View v;
  make_view(h->classes[sl.cls], sl.cls, sl.first, sl.count, h->arena + w.base + sl.off, &v);
  return v;
}

// A slice's step in three phases, so that the QR refreshes of a wave can be batched by size:
//   A  operand preparation and S1 (per slice, caller's stream)
//   B  S2 + S3 for every preconditioned side, one batched QR per size group (refresh_group)
//   C  S5-S8: rotations, Adam in the basis, back-rotation and update (per slice)
//
// Two-sided slices run every contraction as a tcgen05 product C = A B^T of K-major operands:
//   S1  L <- b L + (1-b) G G^T       A = G,     B = G
//       R <- b R + (1-b) G^T G       A = G^T,   B = G^T
//   S2  P^T = Q_L^T L                A = Q_L^T, B = L (symmetric)  -> QR -> Q_L, Q_L^T
//   S5  Y^T = ([G | M_hat] Q_R)^T    A = [G|M], B = Q_R^T    (transposed epilogue)
//       [G' | m'] = Q_L^T Y          A = Q_L^T, B = Y^T
//   S6  N = Adam(G', m', v)
//   S7  Z^T = (N Q_R^T)^T            A = N,     B = Q_R      (transposed epilogue)
//   S8  W <- (1 - lr wd) W - lr Q_L Z  A = Q_L, B = Z^T      (epilogue into W)
// One-sided slices take the same route with one rotation on each side of Adam (a left-only
// class as the right-only problem of G^T). Classes whose rows or columns are not a multiple
// of 4 (rows of an operand must be 16-byte multiples for TMA) run on CUDA cores.
soap_status_t prepare(soap_handle h, const ClassState& c, const View& v, const float* const* d_grads, bool refresh,
                      cudaStream_t s) {
  const soap_hparams& hp = h->hp;
  const int B = v.count, m = (int)c.rows, n = (int)c.cols;
  const int64_t mn = (int64_t)m * n;
  if (!c.tc) {
    SOAP_CUDA(h, soap::momentum_and_copy(d_grads, v.Gc, v.Mhat, mn, B, hp.beta1, h->d_status, s));
    return SOAP_OK;
  }
  SOAP_CUDA(h, soap::momentum_split(d_grads, v.Gc, v.Gc_lo, v.Gt, v.Gt_lo, v.Mhat, v.Mc, v.Mc_lo, m, n, B, hp.beta1,
                                    c.tr, h->d_status, s));
  // the factors' lo parts are read before S1 rewrites them by the KL form's eigenvalue product
  // and by the stale variant's refresh
  const bool lo = hp.kl || hp.stale;
  // Q^T and its lo part feed S2 (and the KL eigenvalues); Q's own lo part only the rotations,
  // for which a refresh writes it anew
  if (c.left) {
    SOAP_CUDA(h, soap::basis_split(v.QL, refresh ? nullptr : v.QL_lo, v.QLt, v.QLt_lo, m, B, s));
    SOAP_CUDA(h, soap::unpack_sym(v.L, v.Lf, lo ? v.Lf_lo : nullptr, m, B, s));
  }
  if (c.right) {
    SOAP_CUDA(h, soap::basis_split(v.QR, refresh ? nullptr : v.QR_lo, v.QRt, v.QRt_lo, n, B, s));
    SOAP_CUDA(h, soap::unpack_sym(v.R, v.Rf, lo ? v.Rf_lo : nullptr, n, B, s));
  }
  return SOAP_OK;
}

// S1 for one slice (after prepare): the standard factor EMAs, or Alg. 1's KL form, on the
// unpacked factors, which are then packed back into the state.
soap_status_t accumulate_factors(soap_handle h, const ClassState& c, const View& v, cudaStream_t s) {
  const soap_hparams& hp = h->hp;
  const int B = v.count, m = (int)c.rows, n = (int)c.cols;
  const int64_t mn = (int64_t)m * n, mm = (int64_t)m * m, nn = (int64_t)n * n;
  const float fb = hp.factor_beta;
  // S1 weights. Standard form: 1 - b. KL form with an identity side (S = I, lambda = 1):
  // (1 - b) / (other dimension * (1 + eps)); a two-sided KL class weighs G's columns (rows)
  // by the other factor's eigenvalues instead (below).
  const float aL = hp.kl ? (float)((1.0 - fb) / ((double)n * (1.0 + hp.eps))) : 1.f - fb;
  const float aR = hp.kl ? (float)((1.0 - fb) / ((double)m * (1.0 + hp.eps))) : 1.f - fb;
  using soap::strided;
  using soap::strided_mut;
  if (!c.tc) {
    if (c.left)  // S1: L <- b L + (1-b) G G^T
      SOAP_CUDA(h, soap::gemm(false, true, m, m, n, aL, strided(v.Gc, n, mn), strided(v.Gc, n, mn), fb,
                              strided_mut(v.L, m, mm), B, s));
    if (c.right)  // S1: R <- b R + (1-b) G^T G
      SOAP_CUDA(h, soap::gemm(true, false, n, n, m, aR, strided(v.Gc, n, mn), strided(v.Gc, n, mn), fb,
                              strided_mut(v.R, n, nn), B, s));
    return SOAP_OK;
  }
  if (hp.kl && c.left && c.right) {
    // KL-Shampoo factor form (Alg. 1), from the factors and bases held before this step:
    //   lam_L = diag(Q_L^T L Q_L), lam_R = diag(Q_R^T R Q_R)       (C = Q^T F, then row dots)
    //   Y = G Q_R diag(sqrt(w_R)),  w_R = (1-b) / (cols (lam_R + eps))
    //   X = G^T Q_L diag(sqrt(w_L)), w_L = (1-b) / (rows (lam_L + eps))
    //   L <- b L + Y Y^T,  R <- b R + X X^T
    // Y and X (with their lo parts) live in the rotation workspace, free until phase C.
    const int64_t cls = (int64_t)B * mn;
    float* C = h->lam_ws;
    SOAP_CUDA(h, soap::gemm_tc_nt(m, m, m, B, opnd(v.QLt, v.QLt_lo, m, mm, B), opnd(v.Lf, v.Lf_lo, m, mm, B),
                                  epi(h, C, m, mm, nullptr, 0, 1.f, 0.f), s));
    SOAP_CUDA(h, soap::diag_dot(C, v.QLt, v.lamL, m, B, s));
    SOAP_CUDA(h, soap::gemm_tc_nt(n, n, n, B, opnd(v.QRt, v.QRt_lo, n, nn, B), opnd(v.Rf, v.Rf_lo, n, nn, B),
                                  epi(h, C, n, nn, nullptr, 0, 1.f, 0.f), s));
    SOAP_CUDA(h, soap::diag_dot(C, v.QRt, v.lamR, n, B, s));
    float* Y = h->YMt;
    float* Y_lo = h->YMt_lo;
    float* X = h->YMt + cls;
    float* X_lo = h->YMt_lo + cls;
    SOAP_CUDA(h, soap::gemm_tc_nt(m, n, n, B, opnd(v.Gc, v.Gc_lo, n, mn, B), opnd(v.QRt, v.QRt_lo, n, nn, B),
                                  epi(h, Y, n, mn, nullptr, 0, 1.f, 0.f), s));
    SOAP_CUDA(h, soap::scale_cols_split(Y, Y_lo, v.lamR, m, n, B, (float)((1.0 - fb) / n), hp.eps, s));
    SOAP_CUDA(h, soap::gemm_tc_nt(n, m, m, B, opnd(v.Gt, v.Gt_lo, m, mn, B), opnd(v.QLt, v.QLt_lo, m, mm, B),
                                  epi(h, X, m, mn, nullptr, 0, 1.f, 0.f), s));
    SOAP_CUDA(h, soap::scale_cols_split(X, X_lo, v.lamL, n, m, B, (float)((1.0 - fb) / m), hp.eps, s));
    SOAP_CUDA(h, soap::gemm_tc_syrk(m, n, B, opnd(Y, Y_lo, n, mn, B), epi(h, v.Lf, m, mm, v.Lf_lo, 0, 1.f, fb), s));
    SOAP_CUDA(h, soap::gemm_tc_syrk(n, m, B, opnd(X, X_lo, m, mn, B), epi(h, v.Rf, n, nn, v.Rf_lo, 0, 1.f, fb), s));
  } else {
    // S1 as symmetric products: the lower tiles of G G^T (G^T G), mirrored
    if (c.left)
      SOAP_CUDA(h, soap::gemm_tc_syrk(m, n, B, opnd(v.Gc, v.Gc_lo, n, mn, B), epi(h, v.Lf, m, mm, v.Lf_lo, 0, aL, fb),
                                      s));
    if (c.right)
      SOAP_CUDA(h, soap::gemm_tc_syrk(n, m, B, opnd(v.Gt, v.Gt_lo, m, mn, B), epi(h, v.Rf, n, nn, v.Rf_lo, 0, aR, fb),
                                      s));
  }
  if (c.left) SOAP_CUDA(h, soap::pack_sym(v.Lf, v.L, m, B, s));
  if (c.right) SOAP_CUDA(h, soap::pack_sym(v.Rf, v.R, n, B, s));
  return SOAP_OK;
}

// S2 + S3 for the preconditioned sides of one size group of a wave: P^T = Q^T F for each member
// (F the unpacked factor, symmetric) into one batched input, one QR, then Q (into the state),
// Q^T and the lo parts (into the slices' workspace) and the zero-column flags. The group runs
// on its own streams from the moment its members' factors are updated on the caller's stream,
// concurrently with other groups.
soap_status_t refresh_group(soap_handle h, const Wave& w, const QrGroup& g, cudaStream_t s) {
  const soap_hparams& hp = h->hp;
  using soap::strided;
  using soap::strided_mut;
  GroupStreams& gs = h->slots[w.slot_base + g.slot];
  SOAP_CUDA(h, cudaEventRecord(gs.fork, s));
  SOAP_CUDA(h, cudaStreamWaitEvent(gs.stream, gs.fork, 0));
  const int n = g.n;
  const int64_t nn = (int64_t)n * n;
  void* ws = h->arena + w.base + g.ws_off;
  uint8_t* skip = reinterpret_cast<uint8_t*>(h->arena + w.base + g.skip_off);
  float* At;
  soap::qr_input_buffers(ws, n, g.batch, &At);
  for (const QrJob& j : g.jobs) {
    const Slice& sl = w.slices[j.slice];
    const ClassState& c = h->classes[sl.cls];
    const View v = view_of(h, w, sl);
    float* at = At + (int64_t)j.offset * nn;
    if (c.tc) {
      SOAP_CUDA(h, soap::gemm_tc_nt(n, n, n, v.count, opnd(j.left ? v.QLt : v.QRt, j.left ? v.QLt_lo : v.QRt_lo, n, nn,
                                                           v.count),
                                    opnd(j.left ? v.Lf : v.Rf, j.left ? v.Lf_lo : v.Rf_lo, n, nn, v.count),
                                    epi(h, at, n, nn, nullptr, 0, 1.f, 0.f), gs.stream));
    } else {
      SOAP_CUDA(h, soap::gemm(true, false, n, n, n, 1.f, strided(j.left ? v.QL : v.QR, n, nn),
                              strided(j.left ? v.L : v.R, n, nn), 0.f, strided_mut(at, n, nn), v.count, gs.stream));
    }
  }
  // the Q accumulation ends with Q^T in the input buffers
  const soap::QrLookahead la{gs.far, gs.ev_vt, gs.ev_far, {gs.ev_vq[0], gs.ev_vq[1]}};
  SOAP_CUDA(h, soap::qr_q_t(n, g.batch, nullptr, nullptr, nullptr, nullptr, skip, hp.qr_tol, ws, g.ws_bytes,
                            h->d_status, gs.stream, &la));
  for (const QrJob& j : g.jobs) {
    const Slice& sl = w.slices[j.slice];
    const ClassState& c = h->classes[sl.cls];
    const View v = view_of(h, w, sl);
    const float* qt = At + (int64_t)j.offset * nn;
    float* Q = j.left ? v.QL : v.QR;
    if (c.tc)
      SOAP_CUDA(h, soap::basis_from_qt(qt, nullptr, j.left ? v.QLt : v.QRt, j.left ? v.QLt_lo : v.QRt_lo, Q,
                                       j.left ? v.QL_lo : v.QR_lo, n, v.count, gs.stream));
    else
      SOAP_CUDA(h, soap::basis_from_qt(qt, nullptr, nullptr, nullptr, Q, nullptr, n, v.count, gs.stream));
    SOAP_CUDA(h, cudaMemcpyAsync(j.left ? v.skipL : v.skipR, skip + (int64_t)j.offset * n, (size_t)v.count * n,
                                 cudaMemcpyDeviceToDevice, gs.stream));
  }
  SOAP_CUDA(h, cudaEventRecord(gs.done, gs.stream));
  return SOAP_OK;
}

soap_status_t rotate_update(soap_handle h, const ClassState& c, const View& v, float* const* d_params, float bc1,
                            float bc2, cudaStream_t s) {
  const soap_hparams& hp = h->hp;
  const int B = v.count, m = (int)c.rows, n = (int)c.cols;
  const int64_t mn = (int64_t)m * n, mm = (int64_t)m * m, nn = (int64_t)n * n;
  using soap::strided;
  using soap::strided_mut;
  if (c.tc && !(c.left && c.right)) {
    // one preconditioned side, as a right-sided problem in the working orientation: the
    // rr x cc matrices X = G (or G^T) with basis Q = Q_R (or Q_L)
    //   [G' | m'] = [X | M_hat] Q    A = [X | M_hat],  B = Q^T   (batch 2B)
    //   N = Adam(G', m', v)
    //   W <- (1 - lr wd) W - lr N Q^T  A = N,  B = Q   (epilogue into W, transposed if c.tr)
    const int rr = c.tr ? n : m, cc = c.tr ? m : n;
    const int64_t cls = (int64_t)B * mn, qq = (int64_t)cc * cc;
    const float* X = c.tr ? v.Gt : v.Gc;
    const float* X_lo = c.tr ? v.Gt_lo : v.Gc_lo;
    const float* Q = c.tr ? v.QL : v.QR;
    const float* Q_lo = c.tr ? v.QL_lo : v.QR_lo;
    const float* Qt = c.tr ? v.QLt : v.QRt;
    const float* Qt_lo = c.tr ? v.QLt_lo : v.QRt_lo;
    SOAP_CUDA(h, soap::gemm_tc_nt(rr, cc, cc, 2 * B, opnd(X, X_lo, cc, mn, 2 * B), opnd(Qt, Qt_lo, cc, qq, B),
                                  epi(h, h->Gp, cc, mn, nullptr, 0, 1.f, 0.f), s));
    const uint8_t* skip = hp.guard ? (c.tr ? v.skipL : v.skipR) : nullptr;
    SOAP_CUDA(h, soap::adam_in_basis(h->Gp, h->Gp + cls, v.V, rr, cc, B, hp.beta1, hp.beta2, hp.eps, bc1, bc2, nullptr,
                                     skip, h->N_lo, h->d_status, s));
    soap::TcEpilogue ew = epi(h, nullptr, n, 0, nullptr, c.tr ? 1 : 0, -h->lr, 1.f - h->lr * h->wd);
    ew.C_ptrs = d_params;
    SOAP_CUDA(h, soap::gemm_tc_nt(rr, cc, cc, B, opnd(h->Gp, h->N_lo, cc, mn, B), opnd(Q, Q_lo, cc, qq, B), ew, s));
    return SOAP_OK;
  }
  if (c.tc) {
    const int64_t cls = (int64_t)B * mn;
    // rotations of the gradient and of the momentum in one launch each (batch 2B)
    SOAP_CUDA(h, soap::gemm_tc_nt(m, n, n, 2 * B, opnd(v.Gc, v.Gc_lo, n, mn, 2 * B), opnd(v.QRt, v.QRt_lo, n, nn, B),
                                  epi(h, h->YMt, m, mn, h->YMt_lo, 1, 1.f, 0.f), s));
    SOAP_CUDA(h, soap::gemm_tc_nt(m, n, m, 2 * B, opnd(v.QLt, v.QLt_lo, m, mm, B),
                                  opnd(h->YMt, h->YMt_lo, m, mn, 2 * B), epi(h, h->Gp, n, mn, nullptr, 0, 1.f, 0.f), s));
    SOAP_CUDA(h, soap::adam_in_basis(h->Gp, h->Gp + cls, v.V, m, n, B, hp.beta1, hp.beta2, hp.eps, bc1, bc2,
                                     hp.guard ? v.skipL : nullptr, hp.guard ? v.skipR : nullptr, h->N_lo, h->d_status,
                                     s));
    SOAP_CUDA(h, soap::gemm_tc_nt(m, n, n, B, opnd(h->Gp, h->N_lo, n, mn, B), opnd(v.QR, v.QR_lo, n, nn, B),
                                  epi(h, h->Zt, m, mn, h->Zt_lo, 1, 1.f, 0.f), s));
    soap::TcEpilogue ew = epi(h, nullptr, n, 0, nullptr, 0, -h->lr, 1.f - h->lr * h->wd);
    ew.C_ptrs = d_params;
    SOAP_CUDA(h, soap::gemm_tc_nt(m, n, m, B, opnd(v.QL, v.QL_lo, m, mm, B), opnd(h->Zt, h->Zt_lo, m, mn, B), ew, s));
    return SOAP_OK;
  }
  // S5 and the re-projected first moment: G' = Q_L^T G Q_R, m = Q_L^T M_hat Q_R
  const float* xg = v.Gc;
  const float* xm = v.Mhat;
  if (c.left) {
    SOAP_CUDA(h, soap::gemm(true, false, m, n, m, 1.f, strided(v.QL, m, mm), strided(v.Gc, n, mn), 0.f,
                            strided_mut(h->X1, n, mn), B, s));
    SOAP_CUDA(h, soap::gemm(true, false, m, n, m, 1.f, strided(v.QL, m, mm), strided(v.Mhat, n, mn), 0.f,
                            strided_mut(h->X2, n, mn), B, s));
    xg = h->X1;
    xm = h->X2;
  }
  float* gp;
  const float* mp;
  if (c.right) {
    SOAP_CUDA(h, soap::gemm(false, false, m, n, n, 1.f, strided(xg, n, mn), strided(v.QR, n, nn), 0.f,
                            strided_mut(h->Gp, n, mn), B, s));
    SOAP_CUDA(h, soap::gemm(false, false, m, n, n, 1.f, strided(xm, n, mn), strided(v.QR, n, nn), 0.f,
                            strided_mut(h->Mp, n, mn), B, s));
    gp = h->Gp;
    mp = h->Mp;
  } else {
    gp = const_cast<float*>(xg);  // X1, or the gradient copy when no side rotates
    mp = xm;
  }
  // S6
  SOAP_CUDA(h, soap::adam_in_basis(gp, mp, v.V, m, n, B, hp.beta1, hp.beta2, hp.eps, bc1, bc2,
                                   (hp.guard && c.left) ? v.skipL : nullptr, (hp.guard && c.right) ? v.skipR : nullptr,
                                   nullptr, h->d_status, s));
  // S7 + S8: W <- (1 - lr wd) W - lr Q_L N Q_R^T
  const float keep = 1.f - h->lr * h->wd;
  soap::MutOperand W{nullptr, d_params, 0, 0, n};
  if (c.left && c.right) {
    SOAP_CUDA(h, soap::gemm(false, false, m, n, m, 1.f, strided(v.QL, m, mm), strided(gp, n, mn), 0.f,
                            strided_mut(h->X1, n, mn), B, s));
    SOAP_CUDA(h, soap::gemm(false, true, m, n, n, -h->lr, strided(h->X1, n, mn), strided(v.QR, n, nn), keep, W, B, s));
  } else if (c.left) {
    SOAP_CUDA(h, soap::gemm(false, false, m, n, m, -h->lr, strided(v.QL, m, mm), strided(gp, n, mn), keep, W, B, s));
  } else if (c.right) {
    SOAP_CUDA(h, soap::gemm(false, true, m, n, n, -h->lr, strided(gp, n, mn), strided(v.QR, n, nn), keep, W, B, s));
  } else {
    SOAP_CUDA(h, soap::weight_update(d_params, gp, mn, B, h->lr, h->wd, s));
  }
  return SOAP_OK;
}

// ---- the wave plan ---------------------------------------------------------------------

int largest_side(const ClassState& c) {
  return (int)std::max(c.left ? c.rows : (int64_t)0, c.right ? c.cols : (int64_t)0);
}

// Rotation intermediates (floats) that a slice of `count` matrices of class c needs.
struct RotSizes {
  size_t mat = 0, tc = 0, two = 0, x = 0, lam = 0;
  void grow(const RotSizes& o) {
    mat = std::max(mat, o.mat);
    tc = std::max(tc, o.tc);
    two = std::max(two, o.two);
    x = std::max(x, o.x);
    lam = std::max(lam, o.lam);
  }
  size_t bytes() const { return 4 * (2 * mat + tc + 4 * two + 2 * two + 2 * x + lam) + 16 * 256; }
};
RotSizes rot_sizes(const ClassState& c, int count, bool kl) {
  RotSizes r;
  const size_t mn = (size_t)count * c.rows * c.cols;
  r.mat = mn;
  if (c.tc) r.tc = mn;
  if (c.tc && c.left && c.right) r.two = mn;
  // X1/X2: a CUDA-core slice's intermediates, or one matrix (state reads and writes)
  r.x = c.tc ? (size_t)(c.rows * c.cols) : mn;
  if (kl && c.tc && c.left && c.right) r.lam = (size_t)count * std::max(c.rows * c.rows, c.cols * c.cols);
  return r;
}

// Lays out one wave: its slices' workspaces and its QR groups in the arena (offsets from 0).
void layout_wave(soap_handle h, Wave& w) {
  size_t off = 0;
  for (Slice& sl : w.slices) {
    sl.off = off;
    off += make_view(h->classes[sl.cls], sl.cls, sl.first, sl.count, nullptr, nullptr);
  }
  // QR groups: every preconditioned side of the wave's slices, grouped by size, largest first
  w.groups.clear();
  std::map<int, int, std::greater<int>> by_n;
  for (const Slice& sl : w.slices) {
    const ClassState& c = h->classes[sl.cls];
    if (c.left) by_n.emplace((int)c.rows, 0);
    if (c.right) by_n.emplace((int)c.cols, 0);
  }
  for (auto& kv : by_n) {
    kv.second = (int)w.groups.size();
    QrGroup g;
    g.n = kv.first;
    g.slot = kv.second;
    w.groups.push_back(g);
  }
  for (int si = 0; si < (int)w.slices.size(); ++si) {
    const Slice& sl = w.slices[si];
    const ClassState& c = h->classes[sl.cls];
    for (int side = 0; side < 2; ++side) {
      if (side == 0 ? !c.left : !c.right) continue;
      QrGroup& g = w.groups[by_n[(int)(side == 0 ? c.rows : c.cols)]];
      g.jobs.push_back(QrJob{si, side == 0, g.batch});
      g.batch += sl.count;
    }
  }
  for (QrGroup& g : w.groups) {
    g.ws_bytes = soap::qr_workspace_bytes(g.n, g.batch, true);
    g.ws_off = off;
    off += align256(g.ws_bytes);
    g.skip_off = off;
    off += align256((size_t)g.batch * g.n);
  }
  w.bytes = off;
  // step order: see soap_step
  const int ns = (int)w.slices.size();
  auto largest = [&](int si) { return largest_side(h->classes[w.slices[si].cls]); };
  w.prep_order.resize(ns);
  for (int si = 0; si < ns; ++si) w.prep_order[si] = si;
  w.update_order = w.prep_order;
  std::stable_sort(w.prep_order.begin(), w.prep_order.end(), [&](int x, int y) { return largest(x) > largest(y); });
  std::stable_sort(w.update_order.begin(), w.update_order.end(), [&](int x, int y) { return largest(x) < largest(y); });
  w.fork_after.assign(ns, {});
  w.groups_of.assign(ns, {});
  std::vector<int> pos(ns);
  for (int q = 0; q < ns; ++q) pos[w.prep_order[q]] = q;
  for (int gi = 0; gi < (int)w.groups.size(); ++gi) {
    int last = -1;
    for (const QrJob& j : w.groups[gi].jobs) {
      w.groups_of[j.slice].push_back(gi);
      if (last < 0 || pos[j.slice] > pos[last]) last = j.slice;
    }
    if (last >= 0) w.fork_after[last].push_back(gi);
  }
}

// Largest slice a wave (or a product launch) may hold: batched launches index matrices in a
// 16-bit grid dimension, and the rotations run [G | M_hat] as one batch of twice the slice.
constexpr int kMaxSlice = 32767;

// Cuts the classes into waves whose workspace (arena + rotation intermediates) fits `budget`
// bytes. Returns false if some class cannot fit even one matrix.
bool plan_waves(soap_handle h, size_t budget, bool single_ok, std::vector<Wave>* out, RotSizes* rot,
                bool* pipelined) {
  *pipelined = false;
  const int nc = (int)h->classes.size();
  std::vector<int> order(nc);
  for (int ci = 0; ci < nc; ++ci) order[ci] = ci;
  std::stable_sort(order.begin(), order.end(),
                   [&](int x, int y) { return largest_side(h->classes[x]) > largest_side(h->classes[y]); });
  const bool kl = h->hp.kl != 0;
  if (single_ok) {
    // every class whole in one wave
    Wave w;
    RotSizes r;
    bool fits = true;
    for (int ci : order) {
      const ClassState& c = h->classes[ci];
      if (c.count > kMaxSlice) fits = false;
      w.slices.push_back(Slice{ci, 0, c.count, 0});
      r.grow(rot_sizes(c, c.count, kl));
    }
    layout_wave(h, w);
    for (const QrGroup& g : w.groups)
      if (g.batch > 65535) fits = false;
    if (fits && w.bytes + r.bytes() <= budget) {
      out->assign(1, w);
      *rot = r;
      return true;
    }
  }
  // waves cut to the budget: a slice costs its workspace, its share of its QR groups and (as if
  // every slice needed its own) its rotation intermediates per matrix, so the sum is an upper bound
  auto per_matrix = [&](const ClassState& c) {
    size_t b = make_view(c, 0, 0, 1, nullptr, nullptr) + rot_sizes(c, 1, kl).bytes();
    if (c.left) b += soap::qr_workspace_bytes((int)c.rows, 1, true) + (size_t)c.rows + 64 * 256;
    if (c.right) b += soap::qr_workspace_bytes((int)c.cols, 1, true) + (size_t)c.cols + 64 * 256;
    return b + 8 * 256;
  };
  auto cut = [&](size_t wave_budget, std::vector<Wave>* waves) -> bool {
    waves->clear();
    Wave cur;
    size_t used = 0;
    for (int ci : order) {
      const ClassState& c = h->classes[ci];
      const size_t pm = per_matrix(c);
      if (pm > wave_budget) return false;
      int first = 0;
      while (first < c.count) {
        int k = (int)std::min<size_t>((size_t)(c.count - first), (wave_budget - used) / pm);
        k = std::min(k, kMaxSlice);
        if (k <= 0) {
          waves->push_back(cur);
          cur = Wave();
          used = 0;
          continue;
        }
        cur.slices.push_back(Slice{ci, first, k, 0});
        used += (size_t)k * pm;
        first += k;
      }
    }
    if (!cur.slices.empty()) waves->push_back(cur);
    return true;
  };
  // Waves are pipelined where the budget allows (a wave's preparation and factor update run while
  // the previous wave's QR does): two waves hold the arena at a time, each in its half; else they
  // run one after another in the whole budget.
  std::vector<Wave> waves;
  *pipelined = cut(budget / 2, &waves) && waves.size() > 1;
  if (!*pipelined && !cut(budget, &waves)) return false;
  RotSizes r;
  size_t half = 0, groups = 0;
  for (Wave& w : waves) {
    layout_wave(h, w);
    half = std::max(half, align256(w.bytes));
    groups = std::max(groups, w.groups.size());
    for (const Slice& sl : w.slices) r.grow(rot_sizes(h->classes[sl.cls], sl.count, kl));
  }
  if (*pipelined)
    for (size_t wi = 0; wi < waves.size(); ++wi) {
      waves[wi].base = (wi & 1) ? half : 0;
      waves[wi].slot_base = (wi & 1) ? (int)groups : 0;
    }
  *out = waves;
  *rot = r;
  return true;
}

}  // namespace

extern "C" {

void soap_default_hparams(soap_hparams* hp) {
  if (!hp) return;
  hp->lr = 3e-3f;
  hp->beta1 = 0.95f;
  hp->beta2 = 0.95f;
  hp->factor_beta = 0.95f;
  hp->eps = 1e-8f;
  hp->weight_decay = 0.1f;
  hp->eig_every = 1;
  hp->bias_correction = 0;
  hp->qr_tol = 2e-5f;
  hp->guard = 1;
  hp->kl = 0;
  hp->stale = 0;
}

soap_status_t soap_create_ex(const soap_shape* shapes, int32_t n, const soap_hparams* hp, int32_t device,
                             size_t workspace_limit, soap_handle* out) {
  if (!out) return SOAP_ERR_INVALID_ARG;
  *out = nullptr;
  if (!shapes || n <= 0 || !hp) return SOAP_ERR_INVALID_ARG;
  if (hp->eig_every < 1 || !(hp->eps >= 0.f) || !(hp->qr_tol >= 0.f)) return SOAP_ERR_INVALID_ARG;
  if (hp->kl != 0 && hp->kl != 1) return SOAP_ERR_INVALID_ARG;
  if (hp->kl && !(hp->eps > 0.f)) return SOAP_ERR_INVALID_ARG;
  if ((hp->stale != 0 && hp->stale != 1) || (hp->stale && (hp->kl || hp->guard))) return SOAP_ERR_INVALID_ARG;
  for (int i = 0; i < n; ++i) {
    const soap_shape& s = shapes[i];
    if (s.rows < 1 || s.cols < 1 || s.rows > (1 << 20) || s.cols > (1 << 20)) return SOAP_ERR_INVALID_ARG;
    if (s.rows * s.cols > (int64_t(1) << 31) - 1) return SOAP_ERR_INVALID_ARG;
    if ((s.precond_left && s.rows > 8192) || (s.precond_right && s.cols > 8192)) return SOAP_ERR_INVALID_ARG;
    // the QR's tensor-core products read the factors with TMA: 16-byte rows
    if ((s.precond_left && (s.rows & 3)) || (s.precond_right && (s.cols & 3))) return SOAP_ERR_INVALID_ARG;
  }
  int ndev = 0;
  if (cudaGetDeviceCount(&ndev) != cudaSuccess || device < 0 || device >= ndev) return SOAP_ERR_CUDA;
  DeviceGuard g(device);
  soap_handle h = new soap_s();
  h->device = device;
  h->hp = *hp;
  h->lr = hp->lr;
  h->wd = hp->weight_decay;
  h->shapes.assign(shapes, shapes + n);
  h->loc.resize(n);

  std::map<std::tuple<int64_t, int64_t, bool, bool>, int> index;
  for (int i = 0; i < n; ++i) {
    const soap_shape& s = shapes[i];
    auto key = std::make_tuple(s.rows, s.cols, s.precond_left != 0, s.precond_right != 0);
    auto it = index.find(key);
    int ci;
    if (it == index.end()) {
      ci = (int)h->classes.size();
      index[key] = ci;
      ClassState c;
      c.rows = s.rows;
      c.cols = s.cols;
      c.left = s.precond_left != 0;
      c.right = s.precond_right != 0;
      h->classes.push_back(c);
    } else {
      ci = it->second;
    }
    h->loc[i] = {ci, h->classes[ci].count};
    h->classes[ci].members.push_back(i);
    h->classes[ci].count++;
  }

  // persistent state
  size_t off = 0;
  cudaError_t e = cudaSuccess;
  auto take = [&](void** p, size_t bytes) {
    if (e == cudaSuccess) e = dalloc(h, p, bytes);
    if (e == cudaSuccess) h->state_bytes += bytes;
  };
  for (auto& c : h->classes) {
    const size_t mn = (size_t)c.count * c.rows * c.cols;
    c.ptr_offset = off;
    off += 2 * (size_t)c.count;
    // tensor-core operands are read with TMA: rows of both G and G^T must be 16-byte multiples
    c.tc = (c.left || c.right) && (c.rows % 4 == 0) && (c.cols % 4 == 0);
    c.tr = c.tc && c.left && !c.right;
    take((void**)&c.Mhat, mn * 4);
    take((void**)&c.V, mn * 4);
    if (c.left) {
      take((void**)&c.L, (size_t)c.count * c.lpk() * 4);
      take((void**)&c.QL, (size_t)c.count * c.rows * c.rows * 4);
      take((void**)&c.skipL, (size_t)c.count * c.rows);
    }
    if (c.right) {
      take((void**)&c.R, (size_t)c.count * c.rpk() * 4);
      take((void**)&c.QR, (size_t)c.count * c.cols * c.cols * 4);
      take((void**)&c.skipR, (size_t)c.count * c.cols);
    }
    if (hp->kl && c.left && c.right) {
      take((void**)&c.lamL, (size_t)c.count * c.rows * 4);
      take((void**)&c.lamR, (size_t)c.count * c.cols * 4);
    }
  }
  h->nptrs = off;
  take((void**)&h->d_status, sizeof(int));
  take((void**)&h->d_ptrs, h->nptrs * sizeof(void*));
  if (e == cudaSuccess) e = cudaMallocHost((void**)&h->h_status, sizeof(int));
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->status_ev, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->step_done, cudaEventDisableTiming);

  // the workspace: one wave holding every class if that fits (within the limit, or leaving a
  // reserve of free memory), else waves cut to what is available
  RotSizes rot;
  if (e == cudaSuccess) {
    size_t free_b = 0, total_b = 0;
    e = cudaMemGetInfo(&free_b, &total_b);
    const size_t reserve = (size_t(1) << 30) + total_b / 100;
    const size_t avail = free_b > reserve ? free_b - reserve : 0;
    const size_t budget = workspace_limit ? std::min(workspace_limit, avail) : avail;
    if (e == cudaSuccess && !plan_waves(h, budget, true, &h->waves, &rot, &h->pipelined))
      e = cudaErrorMemoryAllocation;
  }
  if (e == cudaSuccess) {
    for (const Wave& w : h->waves) h->arena_bytes = std::max(h->arena_bytes, w.base + w.bytes);
    e = dalloc(h, (void**)&h->arena, h->arena_bytes);
  }
  size_t nslots = 0;
  for (const Wave& w : h->waves) nslots = std::max(nslots, (size_t)w.slot_base + w.groups.size());
  h->slots.resize(nslots);
  for (GroupStreams& gs : h->slots) {
    // the panel chain is latency-bound: its stream goes first when SMs free up
    int prio_lo = 0, prio_hi = 0;
    if (e == cudaSuccess) e = cudaDeviceGetStreamPriorityRange(&prio_lo, &prio_hi);
    if (e == cudaSuccess) e = cudaStreamCreateWithPriority(&gs.stream, cudaStreamNonBlocking, prio_hi);
    if (e == cudaSuccess) e = cudaStreamCreateWithPriority(&gs.far, cudaStreamNonBlocking, prio_lo);
    for (cudaEvent_t* ev : {&gs.done, &gs.fork, &gs.ev_vt, &gs.ev_far, &gs.ev_vq[0], &gs.ev_vq[1]})
      if (e == cudaSuccess) e = cudaEventCreateWithFlags(ev, cudaEventDisableTiming);
  }
  // rotation intermediates: [G' | m'] for every slice; N's lo part for tensor-core slices; the
  // intermediate products of two-sided tensor-core slices; X1/X2 for CUDA-core slices and for
  // single-matrix state reads and writes; Q^T F for the KL form's eigenvalues
  h->ws_mat = rot.mat;
  h->rot_bytes = rot.bytes();
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->X1, rot.x * 4);
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->X2, rot.x * 4);
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->Gp, 2 * rot.mat * 4);
  h->Mp = h->Gp ? h->Gp + rot.mat : nullptr;
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->N_lo, rot.tc * 4);
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->YMt, 2 * rot.two * 4);
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->YMt_lo, 2 * rot.two * 4);
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->Zt, rot.two * 4);
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->Zt_lo, rot.two * 4);
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->lam_ws, rot.lam * 4);
  if (e != cudaSuccess) {
    soap_status_t code = e == cudaErrorMemoryAllocation ? SOAP_ERR_OOM : SOAP_ERR_CUDA;
    free_all(h);
    delete h;
    cudaGetLastError();
    return code;
  }
  *h->h_status = 0;
  // initial state: L = R = 0, Q = I, M_hat = v = 0
  for (auto& c : h->classes) {
    const size_t mn = (size_t)c.count * c.rows * c.cols;
    if (e == cudaSuccess) e = cudaMemset(c.Mhat, 0, mn * 4);
    if (e == cudaSuccess) e = cudaMemset(c.V, 0, mn * 4);
    if (c.left) {
      if (e == cudaSuccess) e = cudaMemset(c.L, 0, (size_t)c.count * c.lpk() * 4);
      if (e == cudaSuccess) e = soap::set_identity(c.QL, (int)c.rows, c.count, 0);
      if (e == cudaSuccess) e = cudaMemset(c.skipL, 0, (size_t)c.count * c.rows);
    }
    if (c.right) {
      if (e == cudaSuccess) e = cudaMemset(c.R, 0, (size_t)c.count * c.rpk() * 4);
      if (e == cudaSuccess) e = soap::set_identity(c.QR, (int)c.cols, c.count, 0);
      if (e == cudaSuccess) e = cudaMemset(c.skipR, 0, (size_t)c.count * c.cols);
    }
    if (c.lamL && e == cudaSuccess) e = cudaMemset(c.lamL, 0, (size_t)c.count * c.rows * 4);
    if (c.lamR && e == cudaSuccess) e = cudaMemset(c.lamR, 0, (size_t)c.count * c.cols * 4);
  }
  if (e == cudaSuccess) e = cudaMemset(h->d_status, 0, sizeof(int));
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    free_all(h);
    delete h;
    cudaGetLastError();
    return SOAP_ERR_CUDA;
  }
  h->last_ptrs.assign(h->nptrs, nullptr);
  *out = h;
  return SOAP_OK;
}

soap_status_t soap_create(const soap_shape* shapes, int32_t n, const soap_hparams* hp, int32_t device,
                          soap_handle* out) {
  return soap_create_ex(shapes, n, hp, device, 0, out);
}

soap_status_t soap_plan_info(soap_handle h, int32_t* waves, int32_t* pipelined, size_t* workspace_bytes,
                             size_t* state_bytes) {
  if (!h) return SOAP_ERR_INVALID_ARG;
  if (waves) *waves = (int32_t)h->waves.size();
  if (pipelined) *pipelined = h->pipelined ? 1 : 0;
  if (workspace_bytes) *workspace_bytes = h->arena_bytes + h->rot_bytes;
  if (state_bytes) *state_bytes = h->state_bytes;
  return SOAP_OK;
}

soap_status_t soap_set_lr(soap_handle h, float lr, float weight_decay) {
  if (!h || !(lr >= 0.f) || !(weight_decay >= 0.f)) return SOAP_ERR_INVALID_ARG;
  h->lr = lr;
  h->wd = weight_decay;
  return SOAP_OK;
}

soap_status_t soap_step(soap_handle h, float* const* params, const float* const* grads,
                        soap_stream_t stream_) {
  if (!h) return SOAP_ERR_INVALID_ARG;
  if (!params || !grads) return fail(h, SOAP_ERR_INVALID_ARG, "soap_step: null pointer array");
  const int n = (int)h->shapes.size();
  for (int i = 0; i < n; ++i) {
    if (!params[i] || !grads[i] || !aligned16(params[i]) || !aligned16(grads[i]))
      return fail(h, SOAP_ERR_INVALID_ARG, "soap_step: matrix " + std::to_string(i) +
                                               " has a null or non-16-byte-aligned pointer");
  }
  DeviceGuard g(h->device);
  cudaStream_t s = (cudaStream_t)stream_;
  // sticky status from a finished earlier step
  if (h->status_pending && cudaEventQuery(h->status_ev) == cudaSuccess) {
    h->status_pending = false;
    soap_status_t st = status_code(*h->h_status);
    if (st != SOAP_OK) return fail(h, st, "soap_step: sticky device status from an earlier step");
  }
  // steps share the workspace: a step on another stream starts after the previous one ends
  if (h->step_recorded) SOAP_CUDA(h, cudaStreamWaitEvent(s, h->step_done, 0));
  // pointer table: [class][params..., grads...], written on the stream through kernel
  // parameters when it changed (nothing on the host waits)
  bool changed = false;
  for (auto& c : h->classes) {
    for (int j = 0; j < c.count; ++j) {
      const int m = c.members[j];
      void* pp = params[m];
      void* gp = const_cast<float*>(grads[m]);
      if (h->last_ptrs[c.ptr_offset + j] != pp || h->last_ptrs[c.ptr_offset + c.count + j] != gp) changed = true;
      h->last_ptrs[c.ptr_offset + j] = pp;
      h->last_ptrs[c.ptr_offset + c.count + j] = gp;
    }
  }
  if (changed) SOAP_CUDA(h, soap::put_ptrs(h->d_ptrs, h->last_ptrs.data(), (int64_t)h->nptrs, s));

  h->t += 1;
  const int64_t t = h->t;
  const soap_hparams& hp = h->hp;
  const bool refresh = (t % hp.eig_every) == 0;
  const float bc1 = hp.bias_correction ? 1.f - powf(hp.beta1, (float)t) : 1.f;
  const float bc2 = hp.bias_correction ? 1.f - powf(hp.beta2, (float)t) : 1.f;
  auto params_of = [&](const Slice& sl) {
    return reinterpret_cast<float* const*>(h->d_ptrs + h->classes[sl.cls].ptr_offset + sl.first);
  };
  auto grads_of = [&](const Slice& sl) {
    const ClassState& c = h->classes[sl.cls];
    return reinterpret_cast<const float* const*>(h->d_ptrs + c.ptr_offset + c.count + sl.first);
  };
  // Per wave: phase A slice by slice, each size group's refresh forked as soon as the last
  // slice feeding it is prepared (slices with the largest factors first, so the longest refresh
  // starts earliest); phase C slice by slice, each waiting only for the groups its bases come
  // from (slices with the smallest factors first, whose refreshes finish earliest). Pipelined
  // waves run on the caller's stream as A0, A1, C0, A2, C1, ...: the next wave's preparation
  // and factor update run while this wave's QR does, in the other half of the arena; a wave
  // reuses a half only after the wave before it in that half has finished (its phase C, which
  // joined its groups, precedes on the stream). The stale variant refreshes from the factors
  // as they stand and accumulates G_t into them after the wave's updates.
  auto phase_a = [&](const Wave& w) -> soap_status_t {
    for (int si : w.prep_order) {
      const Slice& sl = w.slices[si];
      const ClassState& c = h->classes[sl.cls];
      const View v = view_of(h, w, sl);
      soap_status_t st = prepare(h, c, v, grads_of(sl), refresh, s);
      if (st == SOAP_OK && !hp.stale) st = accumulate_factors(h, c, v, s);
      if (st != SOAP_OK) return st;
      if (refresh)
        for (int gi : w.fork_after[si]) {
          st = refresh_group(h, w, w.groups[gi], s);
          if (st != SOAP_OK) return st;
        }
    }
    return SOAP_OK;
  };
  auto phase_c = [&](const Wave& w) -> soap_status_t {
    std::vector<bool> joined(w.groups.size(), !refresh);
    for (int si : w.update_order) {
      for (int gi : w.groups_of[si])
        if (!joined[gi]) {
          SOAP_CUDA(h, cudaStreamWaitEvent(s, h->slots[w.slot_base + w.groups[gi].slot].done, 0));
          joined[gi] = true;
        }
      const Slice& sl = w.slices[si];
      soap_status_t st = rotate_update(h, h->classes[sl.cls], view_of(h, w, sl), params_of(sl), bc1, bc2, s);
      if (st != SOAP_OK) return st;
    }
    for (size_t gi = 0; gi < w.groups.size(); ++gi)
      if (!joined[gi]) SOAP_CUDA(h, cudaStreamWaitEvent(s, h->slots[w.slot_base + w.groups[gi].slot].done, 0));
    if (hp.stale)
      for (int si : w.prep_order) {
        const Slice& sl = w.slices[si];
        soap_status_t st = accumulate_factors(h, h->classes[sl.cls], view_of(h, w, sl), s);
        if (st != SOAP_OK) return st;
      }
    return SOAP_OK;
  };
  const size_t nw = h->waves.size();
  if (h->pipelined) {
    soap_status_t st = phase_a(h->waves[0]);
    if (st != SOAP_OK) return st;
    for (size_t wi = 0; wi < nw; ++wi) {
      st = wi + 1 < nw ? phase_a(h->waves[wi + 1]) : SOAP_OK;
      if (st == SOAP_OK) st = phase_c(h->waves[wi]);
      if (st != SOAP_OK) return st;
    }
  } else {
    for (size_t wi = 0; wi < nw; ++wi) {
      soap_status_t st = phase_a(h->waves[wi]);
      if (st == SOAP_OK) st = phase_c(h->waves[wi]);
      if (st != SOAP_OK) return st;
    }
  }
  SOAP_CUDA(h, cudaMemcpyAsync(h->h_status, h->d_status, sizeof(int), cudaMemcpyDeviceToHost, s));
  SOAP_CUDA(h, cudaEventRecord(h->status_ev, s));
  SOAP_CUDA(h, cudaEventRecord(h->step_done, s));
  h->status_pending = true;
  h->step_recorded = true;
  return SOAP_OK;
}

size_t soap_state_bytes(soap_handle h, int32_t idx, int32_t which) {
  if (!h || idx < 0 || idx >= (int)h->shapes.size()) return 0;
  const soap_shape& s = h->shapes[idx];
  switch (which) {
    case SOAP_STATE_M:
    case SOAP_STATE_V:
    case SOAP_STATE_MHAT: return (size_t)s.rows * s.cols * 4;
    case SOAP_STATE_L:
    case SOAP_STATE_QL: return s.precond_left ? (size_t)s.rows * s.rows * 4 : 0;
    case SOAP_STATE_R:
    case SOAP_STATE_QR: return s.precond_right ? (size_t)s.cols * s.cols * 4 : 0;
    case SOAP_STATE_SKIP_L: return s.precond_left ? (size_t)s.rows : 0;
    case SOAP_STATE_SKIP_R: return s.precond_right ? (size_t)s.cols : 0;
    case SOAP_STATE_LAMBDA_L:
      return h->hp.kl && s.precond_left && s.precond_right ? (size_t)s.rows * 4 : 0;
    case SOAP_STATE_LAMBDA_R:
      return h->hp.kl && s.precond_left && s.precond_right ? (size_t)s.cols * 4 : 0;
    default: return 0;
  }
}

}  // extern "C"

namespace {
// One matrix of the state as a slice of its own, with its workspace at the start of the arena
// (state reads and writes are ordered with the steps, which use the same arena).
View single_view(soap_handle h, int idx) {
  const auto [ci, slot] = h->loc[idx];
  View v;
  make_view(h->classes[ci], ci, slot, 1, h->arena, &v);
  return v;
}

// Address of a piece kept as it is handed out (not SOAP_STATE_M, which is derived, nor a
// packed factor).
void* state_ptr(const View& v, int which) {
  switch (which) {
    case SOAP_STATE_V: return v.V;
    case SOAP_STATE_MHAT: return v.Mhat;
    case SOAP_STATE_QL: return v.QL;
    case SOAP_STATE_QR: return v.QR;
    case SOAP_STATE_SKIP_L: return v.skipL;
    case SOAP_STATE_SKIP_R: return v.skipR;
    case SOAP_STATE_LAMBDA_L: return v.lamL;
    case SOAP_STATE_LAMBDA_R: return v.lamR;
    default: return nullptr;
  }
}

soap_status_t state_get_impl(soap_handle h, int32_t idx, int32_t which, void* dst, soap_stream_t stream_) {
  const size_t bytes = soap_state_bytes(h, idx, which);
  if (bytes == 0 || !dst) return fail(h, SOAP_ERR_INVALID_ARG, "soap_state_get: no such state piece");
  DeviceGuard g(h->device);
  cudaStream_t s = (cudaStream_t)stream_;
  const ClassState& c = h->classes[h->loc[idx].first];
  const View v = single_view(h, idx);
  const int m = (int)c.rows, nc = (int)c.cols;
  const int64_t mn = (int64_t)m * nc;
  if (c.tr && (which == SOAP_STATE_V || which == SOAP_STATE_MHAT)) {
    // stored transposed (n x m): hand out the m x n matrix
    SOAP_CUDA(h, soap::transpose((const float*)state_ptr(v, which), h->X1, nc, m, 1, s));
    SOAP_CUDA(h, cudaMemcpyAsync(dst, h->X1, bytes, cudaMemcpyDefault, s));
    return SOAP_OK;
  }
  if (which == SOAP_STATE_L || which == SOAP_STATE_R) {
    const bool left = which == SOAP_STATE_L;
    const float* F = left ? v.L : v.R;
    if (c.tc) {
      SOAP_CUDA(h, soap::unpack_sym(F, left ? v.Lf : v.Rf, nullptr, left ? m : nc, 1, s));
      F = left ? v.Lf : v.Rf;
    }
    SOAP_CUDA(h, cudaMemcpyAsync(dst, F, bytes, cudaMemcpyDefault, s));
    return SOAP_OK;
  }
  if (which != SOAP_STATE_M) {
    SOAP_CUDA(h, cudaMemcpyAsync(dst, state_ptr(v, which), bytes, cudaMemcpyDefault, s));
    return SOAP_OK;
  }
  // m = Q_L^T M_hat Q_R, computed into the workspace with the operands and products of the step
  const float* x = v.Mhat;
  if (c.tc) {
    if (c.left) SOAP_CUDA(h, soap::basis_split(v.QL, v.QL_lo, v.QLt, v.QLt_lo, m, 1, s));
    if (c.right) SOAP_CUDA(h, soap::basis_split(v.QR, v.QR_lo, v.QRt, v.QRt_lo, nc, 1, s));
    float* x_lo = v.Mc_lo;
    SOAP_CUDA(h, soap::split_tf32(x, nullptr, x_lo, mn, s));
    if (!(c.left && c.right)) {
      // the step's product [X | M_hat] Q for this matrix alone (bit-identical), written in the
      // original orientation
      const int rr = c.tr ? nc : m, cc = c.tr ? m : nc;
      const int64_t qq = (int64_t)cc * cc;
      SOAP_CUDA(h, soap::gemm_tc_nt(rr, cc, cc, 1, opnd(x, x_lo, cc, mn, 1),
                                    opnd(c.tr ? v.QLt : v.QRt, c.tr ? v.QLt_lo : v.QRt_lo, cc, qq, 1),
                                    epi(h, h->Gp, c.tr ? rr : cc, mn, nullptr, c.tr ? 1 : 0, 1.f, 0.f), s));
      SOAP_CUDA(h, cudaMemcpyAsync(dst, h->Gp, bytes, cudaMemcpyDefault, s));
      return SOAP_OK;
    }
    // the same tensor-core products, on the same operands, as the step's rotation of M_hat:
    // bit-identical to the m the last step used
    const int64_t mm = (int64_t)m * m, nn = (int64_t)nc * nc;
    SOAP_CUDA(h, soap::gemm_tc_nt(m, nc, nc, 1, opnd(x, x_lo, nc, mn, 1), opnd(v.QRt, v.QRt_lo, nc, nn, 1),
                                  epi(h, h->X1, m, mn, h->X2, 1, 1.f, 0.f), s));
    SOAP_CUDA(h, soap::gemm_tc_nt(m, nc, m, 1, opnd(v.QLt, v.QLt_lo, m, mm, 1), opnd(h->X1, h->X2, m, mn, 1),
                                  epi(h, h->Gp, nc, mn, nullptr, 0, 1.f, 0.f), s));
    SOAP_CUDA(h, cudaMemcpyAsync(dst, h->Gp, bytes, cudaMemcpyDefault, s));
    return SOAP_OK;
  }
  using soap::strided;
  using soap::strided_mut;
  if (c.left) {
    SOAP_CUDA(h, soap::gemm(true, false, m, nc, m, 1.f, strided(v.QL, m, 0), strided(x, nc, 0), 0.f,
                            strided_mut(h->X1, nc, 0), 1, s));
    x = h->X1;
  }
  if (c.right) {
    SOAP_CUDA(h, soap::gemm(false, false, m, nc, nc, 1.f, strided(x, nc, 0), strided(v.QR, nc, 0), 0.f,
                            strided_mut(h->Gp, nc, 0), 1, s));
    x = h->Gp;
  }
  SOAP_CUDA(h, cudaMemcpyAsync(dst, x, bytes, cudaMemcpyDefault, s));
  return SOAP_OK;
}

soap_status_t state_set_impl(soap_handle h, int32_t idx, int32_t which, const void* src, soap_stream_t stream_) {
  const size_t bytes = soap_state_bytes(h, idx, which);
  if (bytes == 0 || !src) return fail(h, SOAP_ERR_INVALID_ARG, "soap_state_set: no such state piece");
  if (which == SOAP_STATE_LAMBDA_L || which == SOAP_STATE_LAMBDA_R)
    return fail(h, SOAP_ERR_INVALID_ARG, "soap_state_set: the KL eigenvalue estimates are read-only");
  DeviceGuard g(h->device);
  cudaStream_t s = (cudaStream_t)stream_;
  const ClassState& c = h->classes[h->loc[idx].first];
  const View v = single_view(h, idx);
  const int m = (int)c.rows, nc = (int)c.cols;
  if (which == SOAP_STATE_L || which == SOAP_STATE_R) {
    const bool left = which == SOAP_STATE_L;
    if (!c.tc) {
      SOAP_CUDA(h, cudaMemcpyAsync(left ? v.L : v.R, src, bytes, cudaMemcpyDefault, s));
      return SOAP_OK;
    }
    // the lower triangle is kept (the factor is symmetric)
    float* F = left ? v.Lf : v.Rf;
    SOAP_CUDA(h, cudaMemcpyAsync(F, src, bytes, cudaMemcpyDefault, s));
    SOAP_CUDA(h, soap::pack_sym(F, left ? v.L : v.R, left ? m : nc, 1, s));
    return SOAP_OK;
  }
  if (which != SOAP_STATE_M) {
    if (c.tr && (which == SOAP_STATE_V || which == SOAP_STATE_MHAT)) {
      // stored transposed (n x m)
      SOAP_CUDA(h, cudaMemcpyAsync(h->X1, src, bytes, cudaMemcpyDefault, s));
      SOAP_CUDA(h, soap::transpose(h->X1, (float*)state_ptr(v, which), m, nc, 1, s));
    } else {
      SOAP_CUDA(h, cudaMemcpyAsync(state_ptr(v, which), src, bytes, cudaMemcpyDefault, s));
    }
    return SOAP_OK;
  }
  // M_hat = Q_L m Q_R^T
  using soap::strided;
  using soap::strided_mut;
  float* dstm = v.Mhat;
  SOAP_CUDA(h, cudaMemcpyAsync(h->Gp, src, bytes, cudaMemcpyDefault, s));
  const float* x = h->Gp;
  if (c.left) {
    float* out = (c.right || c.tr) ? h->X1 : dstm;
    SOAP_CUDA(h, soap::gemm(false, false, m, nc, m, 1.f, strided(v.QL, m, 0), strided(x, nc, 0), 0.f,
                            strided_mut(out, nc, 0), 1, s));
    x = out;
  }
  if (c.right) {
    SOAP_CUDA(h, soap::gemm(false, true, m, nc, nc, 1.f, strided(x, nc, 0), strided(v.QR, nc, 0), 0.f,
                            strided_mut(dstm, nc, 0), 1, s));
  } else if (c.tr) {
    SOAP_CUDA(h, soap::transpose(x, dstm, m, nc, 1, s));
  } else if (!c.left) {
    SOAP_CUDA(h, cudaMemcpyAsync(dstm, x, bytes, cudaMemcpyDeviceToDevice, s));
  }
  return SOAP_OK;
}

// State reads and writes use the step's workspace: each is ordered after the last enqueued
// step (or state access), and the next step after it, whatever streams they come on.
soap_status_t ordered_state_op(soap_handle h, cudaStream_t s, soap_status_t (*op)(soap_handle, int32_t, int32_t, void*,
                                                                                 soap_stream_t),
                               int32_t idx, int32_t which, void* buf) {
  DeviceGuard g(h->device);
  if (h->step_recorded) SOAP_CUDA(h, cudaStreamWaitEvent(s, h->step_done, 0));
  soap_status_t st = op(h, idx, which, buf, (soap_stream_t)s);
  cudaError_t e = cudaEventRecord(h->step_done, s);
  if (e == cudaSuccess) h->step_recorded = true;
  if (st == SOAP_OK && e != cudaSuccess) return cuda_fail(h, e, "cudaEventRecord(step_done)");
  return st;
}

soap_status_t state_set_void(soap_handle h, int32_t idx, int32_t which, void* src, soap_stream_t s) {
  return state_set_impl(h, idx, which, src, s);
}

}  // namespace

extern "C" {

soap_status_t soap_state_get(soap_handle h, int32_t idx, int32_t which, void* dst, soap_stream_t stream) {
  if (!h) return SOAP_ERR_INVALID_ARG;
  return ordered_state_op(h, (cudaStream_t)stream, state_get_impl, idx, which, dst);
}

soap_status_t soap_state_set(soap_handle h, int32_t idx, int32_t which, const void* src, soap_stream_t stream) {
  if (!h) return SOAP_ERR_INVALID_ARG;
  return ordered_state_op(h, (cudaStream_t)stream, state_set_void, idx, which, const_cast<void*>(src));
}

int64_t soap_get_step(soap_handle h) { return h ? h->t : -1; }

soap_status_t soap_set_step(soap_handle h, int64_t t) {
  if (!h || t < 0) return SOAP_ERR_INVALID_ARG;
  h->t = t;
  return SOAP_OK;
}

soap_status_t soap_status(soap_handle h, soap_stream_t stream_) {
  if (!h) return SOAP_ERR_INVALID_ARG;
  DeviceGuard g(h->device);
  SOAP_CUDA(h, cudaStreamSynchronize((cudaStream_t)stream_));
  int bits = 0;
  SOAP_CUDA(h, cudaMemcpy(&bits, h->d_status, sizeof(int), cudaMemcpyDeviceToHost));
  soap_status_t st = status_code(bits);
  if (st != SOAP_OK) h->err = "device status word " + std::to_string(bits);
  return st;
}

soap_status_t soap_clear_status(soap_handle h, soap_stream_t stream_) {
  if (!h) return SOAP_ERR_INVALID_ARG;
  DeviceGuard g(h->device);
  SOAP_CUDA(h, cudaMemsetAsync(h->d_status, 0, sizeof(int), (cudaStream_t)stream_));
  h->status_pending = false;
  *h->h_status = 0;
  return SOAP_OK;
}

const char* soap_last_error(soap_handle h) { return h ? h->err.c_str() : "null handle"; }

void soap_destroy(soap_handle h) {
  if (!h) return;
  DeviceGuard g(h->device);
  cudaDeviceSynchronize();
  free_all(h);
  delete h;
}

soap_status_t soap_profile_begin(soap_handle h, int64_t max_launches) {
  return soap_profile_begin_ex(h, max_launches, 0);
}

soap_status_t soap_profile_begin_ex(soap_handle h, int64_t max_launches, int32_t flags) {
  if (!h || max_launches < 1 || max_launches > (int64_t(1) << 22) || (flags & ~SOAP_PROFILE_SERIAL))
    return SOAP_ERR_INVALID_ARG;
  DeviceGuard g(h->device);
  soap::Profiler& p = h->prof;
  while ((int64_t)p.events.size() < 2 * max_launches) {
    cudaEvent_t ev;
    SOAP_CUDA(h, cudaEventCreate(&ev));
    p.events.push_back(ev);
  }
  p.capacity = (size_t)max_launches;
  p.recs.clear();
  p.overflow = false;
  p.serial = (flags & SOAP_PROFILE_SERIAL) != 0;
  soap::t_profiler = &p;
  return SOAP_OK;
}

soap_status_t soap_profile_end(soap_handle h, soap_stream_t stream, soap_kernel_stats* out, int32_t* overflow) {
  if (!h || !out) return SOAP_ERR_INVALID_ARG;
  DeviceGuard g(h->device);
  if (soap::t_profiler == &h->prof) soap::t_profiler = nullptr;
  SOAP_CUDA(h, cudaStreamSynchronize((cudaStream_t)stream));
  SOAP_CUDA(h, cudaDeviceSynchronize());
  for (int f = 0; f < soap::kNumFamilies; ++f) out[f] = soap_kernel_stats{f, 0, 0.0, 0.0, 0.0};
  const soap::Profiler& p = h->prof;
  for (size_t i = 0; i < p.recs.size(); ++i) {
    float ms = 0.f;
    SOAP_CUDA(h, cudaEventElapsedTime(&ms, p.events[2 * i], p.events[2 * i + 1]));
    soap_kernel_stats& o = out[p.recs[i].family];
    o.launches += 1;
    o.ms += ms;
    o.flops += p.recs[i].flops;
    o.bytes += p.recs[i].bytes;
  }
  if (overflow) *overflow = p.overflow ? 1 : 0;
  h->prof.recs.clear();
  return SOAP_OK;
}

soap_status_t soap_profile_records(soap_handle h, soap_launch_record* out, int64_t max, int64_t* count) {
  if (!h || !count || max < 0 || (max > 0 && !out)) return SOAP_ERR_INVALID_ARG;
  DeviceGuard g(h->device);
  SOAP_CUDA(h, cudaDeviceSynchronize());
  const soap::Profiler& p = h->prof;
  const int64_t n = std::min<int64_t>(max, (int64_t)p.recs.size());
  for (int64_t i = 0; i < n; ++i) {
    float t0 = 0.f, t1 = 0.f;
    SOAP_CUDA(h, cudaEventElapsedTime(&t0, p.events[0], p.events[2 * i]));
    SOAP_CUDA(h, cudaEventElapsedTime(&t1, p.events[0], p.events[2 * i + 1]));
    out[i] = soap_launch_record{p.recs[i].family, (double)t0, (double)t1, p.recs[i].flops, p.recs[i].bytes};
  }
  *count = n;
  return SOAP_OK;
}

soap_status_t soap_layerwise_assign(const soap_shape* shapes, int32_t n, int32_t world, int32_t policy,
                                    int32_t* owner, double* load) {
  if (!shapes || !owner || n < 1 || world < 1 || (policy != 0 && policy != 1)) return SOAP_ERR_INVALID_ARG;
  for (int i = 0; i < n; ++i)
    if (shapes[i].rows < 1 || shapes[i].cols < 1) return SOAP_ERR_INVALID_ARG;
  // the step's FLOPs for one matrix (2 per multiply-add): S1 as a symmetric product, the power
  // step, Householder QR with explicit Q, and the rotations of G, m and N per preconditioned side
  auto cost = [&](const soap_shape& s) {
    const double m = (double)s.rows, c = (double)s.cols;
    double f = 0.0;
    if (s.precond_left) f += m * m * c + 2 * m * m * m + (8.0 / 3.0) * m * m * m + 8 * m * m * c;
    if (s.precond_right) f += c * c * m + 2 * c * c * c + (8.0 / 3.0) * c * c * c + 8 * m * c * c;
    return f + 10 * m * c;  // the elementwise work
  };
  std::vector<int> order(n);
  for (int i = 0; i < n; ++i) order[i] = i;
  std::stable_sort(order.begin(), order.end(), [&](int a, int b) {
    return shapes[a].rows * shapes[a].cols > shapes[b].rows * shapes[b].cols;
  });
  std::vector<double> l(world, 0.0);
  for (int q = 0; q < n; ++q) {
    const int i = order[q];
    int r = q % world;
    if (policy == 1) {
      r = 0;
      for (int k = 1; k < world; ++k)
        if (l[k] < l[r]) r = k;
    }
    owner[i] = r;
    l[r] += cost(shapes[i]);
  }
  if (load)
    for (int r = 0; r < world; ++r) load[r] = l[r];
  return SOAP_OK;
}

size_t soap_qr_workspace_bytes(int32_t n, int32_t batch) {
  if (n <= 0 || batch <= 0) return 0;
  return soap::qr_workspace_bytes(n, batch) + 256;
}

soap_status_t soap_qr(int32_t n, int32_t batch, const float* P, float* Q, uint8_t* skip, float tol, void* workspace,
                      size_t workspace_bytes, int32_t* status, soap_stream_t stream) {
  if (n <= 0 || n > 8192 || (n & 3) || batch <= 0 || batch > 65535 || !P || !Q || !skip || !workspace ||
      !(tol >= 0.f))
    return SOAP_ERR_INVALID_ARG;
  if (!aligned16(P) || !aligned16(Q) || (reinterpret_cast<uintptr_t>(workspace) & 255) ||
      (reinterpret_cast<uintptr_t>(status) & 3))
    return SOAP_ERR_INVALID_ARG;
  if (workspace_bytes < soap_qr_workspace_bytes(n, batch)) return SOAP_ERR_INVALID_ARG;
  cudaStream_t s = (cudaStream_t)stream;
  // the kernels OR their status bits into the caller's word, or else into the last 256 bytes of
  // the workspace
  const size_t qb = soap::qr_workspace_bytes(n, batch);
  int* word = status ? reinterpret_cast<int*>(status) : reinterpret_cast<int*>(static_cast<char*>(workspace) + qb);
  if (cudaMemsetAsync(word, 0, sizeof(int), s) != cudaSuccess) return SOAP_ERR_CUDA;
  cudaError_t e = soap::qr_q(n, batch, P, Q, skip, tol, workspace, qb, word, s);
  return e == cudaSuccess ? SOAP_OK : SOAP_ERR_CUDA;
}

soap_status_t soap_gemm(int32_t trans_a, int32_t trans_b, int32_t M, int32_t N, int32_t K, float alpha,
                        const float* A, int64_t lda, int64_t stride_a, const float* B, int64_t ldb, int64_t stride_b,
                        float beta, float* C, int64_t ldc, int64_t stride_c, int32_t batch, soap_stream_t stream) {
  if (M < 0 || N < 0 || K < 0 || batch < 0 || batch > 65535) return SOAP_ERR_INVALID_ARG;
  if (M == 0 || N == 0 || batch == 0) return SOAP_OK;
  if (!C || (K > 0 && (!A || !B))) return SOAP_ERR_INVALID_ARG;
  const int64_t a_rows = trans_a ? K : M, a_cols = trans_a ? M : K;
  const int64_t b_rows = trans_b ? N : K, b_cols = trans_b ? K : N;
  if ((K > 0 && (lda < a_cols || ldb < b_cols)) || ldc < N) return SOAP_ERR_INVALID_ARG;
  (void)a_rows;
  (void)b_rows;
  cudaError_t e = soap::gemm(trans_a != 0, trans_b != 0, M, N, K, alpha, soap::strided(A, lda, stride_a),
                             soap::strided(B, ldb, stride_b), beta, soap::strided_mut(C, ldc, stride_c), batch,
                             (cudaStream_t)stream);
  return e == cudaSuccess ? SOAP_OK : SOAP_ERR_CUDA;
}

soap_status_t soap_gemm_tf32x4(int32_t M, int32_t N, int32_t K, int32_t batch, const float* A_hi, const float* A_lo,
                               int64_t lda, int64_t stride_a, const float* B_hi, const float* B_lo, int64_t ldb,
                               int64_t stride_b, int32_t b_batch, float alpha, float beta, float* C, int64_t ldc,
                               int64_t stride_c, int32_t transpose_c, float* C_lo, int32_t* status,
                               soap_stream_t stream) {
  if (M < 0 || N < 0 || K < 0 || batch < 0 || batch > 65535 || b_batch < 0) return SOAP_ERR_INVALID_ARG;
  if (M == 0 || N == 0 || batch == 0) return SOAP_OK;
  if (!A_hi || !A_lo || !B_hi || !B_lo || !C) return SOAP_ERR_INVALID_ARG;
  // A and B are read by TMA: 16-byte aligned bases, rows and batch strides in multiples of 16 bytes
  const void* ptrs[4] = {A_hi, A_lo, B_hi, B_lo};
  for (const void* p : ptrs)
    if (!aligned16(p)) return SOAP_ERR_INVALID_ARG;
  if ((lda | ldb | stride_a | stride_b) & 3) return SOAP_ERR_INVALID_ARG;
  if (lda < K || ldb < K || ldc < (transpose_c ? M : N)) return SOAP_ERR_INVALID_ARG;
  soap::TcOperand A{A_hi, A_lo, lda, stride_a, batch};
  soap::TcOperand B{B_hi, B_lo, ldb, stride_b, b_batch > 0 ? b_batch : batch};
  soap::TcEpilogue ep{C, nullptr, ldc, stride_c, C_lo, ldc, stride_c, transpose_c, alpha, beta,
                      reinterpret_cast<int*>(status)};
  cudaError_t e = soap::gemm_tc_nt(M, N, K, batch, A, B, ep, (cudaStream_t)stream);
  return e == cudaSuccess ? SOAP_OK : (e == cudaErrorInvalidValue ? SOAP_ERR_INVALID_ARG : SOAP_ERR_CUDA);
}

soap_status_t soap_wait_limit(uint64_t limit_ns, const int32_t* hold) {
  if ((reinterpret_cast<uintptr_t>(hold) & 3) != 0) return SOAP_ERR_INVALID_ARG;
  soap::set_wait_limit(limit_ns, reinterpret_cast<const int*>(hold));
  return SOAP_OK;
}

soap_status_t soap_split_tf32(const float* x, float* hi, float* lo, int64_t n, soap_stream_t stream) {
  if (n < 0 || (n > 0 && (!x || !lo))) return SOAP_ERR_INVALID_ARG;
  return soap::split_tf32(x, hi, lo, n, (cudaStream_t)stream) == cudaSuccess ? SOAP_OK : SOAP_ERR_CUDA;
}

}  // extern "C"
