// libsoap: the C ABI of include/soap.h.
//
// Plan: matrices with the same (rows, cols, sides) form a class; each class keeps
// its state in contiguous arenas ([count][rows][cols], [count][rows][rows], ...)
// so every contraction of the step is one batched GEMM per class. The classes' own
// launches go to the caller's stream (prepared largest factor first, rotated smallest
// first) and share one workspace sized for the largest class; the QR refreshes are
// regrouped by factor size, one batched QR per size on its own pair of streams, forked
// as soon as the last class feeding it is prepared and joined by events before the
// classes whose bases it refreshes are rotated.
//
// Per class, the step (Alg. 1 with the standard factor EMAs of section 2) is:
//   M_hat <- b1 M_hat + (1-b1) G, Gc <- G                 momentum in the original basis
//   L <- b L + (1-b) Gc Gc^T, R <- b R + (1-b) Gc^T Gc     S1
//   P = L Q_L -> Q_L = QR(P).Q; same for R                 S2, S3 (when t mod F == 0)
//   X1 = Q_L^T Gc, X2 = Q_L^T M_hat                        S5, S4 (re-projected m)
//   G' = X1 Q_R, m = X2 Q_R
//   v <- b2 v + (1-b2) G'^2, N = m / (sqrt(v) + eps)        S6
//   X1 = Q_L N; W <- (1 - lr wd) W - lr X1 Q_R^T           S7, S8 (fused in the GEMM epilogue)
// With hparams.stale, S1 moves to the end of the step (the refresh sees the earlier gradients
// only). With hparams.kl, S1 takes Alg. 1's KL-Shampoo form instead: each factor's EMA term is
// weighed by the other factor's inverse, Q diag(1/(lam + eps)) Q^T with lam = diag(Q^T F Q)
// (an identity side as lam = 1); see prepare_class.
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
  float* Gc = nullptr;    // G (copy of the caller's gradient); [G | M_hat] unless `tr`
  float* Mhat = nullptr;  // first moment in the original basis, in the working orientation
  float* V = nullptr;
  float* L = nullptr;
  float* QL = nullptr;
  float* R = nullptr;
  float* QR = nullptr;
  uint8_t* skipL = nullptr;
  uint8_t* skipR = nullptr;
  size_t ptr_offset = 0;  // index of this class's params pointers in the pointer table
  // tensor-core path: operand copies and their lo parts
  bool tc = false;
  // working orientation transposed: a class preconditioned on its left only runs as the
  // right-only problem of G^T, and keeps M_hat and v as M_hat^T and v^T
  bool tr = false;
  float* Gc_lo = nullptr;  // lo parts of the Gc arena
  float* Gt = nullptr;     // G^T; [G^T | M_hat^T] if `tr`
  float* Gt_lo = nullptr;
  float* Mhat_lo = nullptr;
  float* L_lo = nullptr;
  float* R_lo = nullptr;
  float* QL_lo = nullptr;
  float* QLt = nullptr;
  float* QLt_lo = nullptr;
  float* QR_lo = nullptr;
  float* QRt = nullptr;
  float* QRt_lo = nullptr;
  bool basis_dirty = true;  // Q^T and lo parts must be rebuilt from Q before use
  // KL-Shampoo factor form, two-sided classes: the approximate eigenvalues of the last step
  float* lamL = nullptr;  // [count][rows]
  float* lamR = nullptr;  // [count][cols]
};

// One preconditioned side of one class: `count` factors of size n in a QR group.
struct QrJob {
  int cls;
  bool left;
  int offset;  // first batch index of this job inside its group
};

// All factors of one size, refreshed by one batched QR on their own stream.
struct QrGroup {
  int n = 0;
  int batch = 0;
  std::vector<QrJob> jobs;
  void* ws = nullptr;
  size_t ws_bytes = 0;
  uint8_t* skip = nullptr;  // [batch][n]
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
  std::vector<QrGroup> groups;  // largest n first
  std::vector<int> prep_order;               // classes, largest factor first
  std::vector<int> update_order;             // classes, smallest largest-factor first
  std::vector<std::vector<int>> fork_after;  // per class: groups whose last feeding class it is
  std::vector<std::vector<int>> groups_of;   // per class: the groups its bases come from
  int* d_status = nullptr;
  int* h_status = nullptr;          // pinned mirror, refreshed after every step
  cudaEvent_t status_ev = nullptr;
  bool status_pending = false;
  void** h_ptrs = nullptr;          // pinned staging for the params/grads pointer table
  void** d_ptrs = nullptr;
  size_t nptrs = 0;
  cudaEvent_t stage_ev = nullptr;
  bool stage_pending = false;
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

// A non-finite gradient also makes the QR of that step break down; report the cause.
soap_status_t status_code(int bits) {
  if (bits & soap::kStatusNonFinite) return SOAP_ERR_NONFINITE;
  if (bits & soap::kStatusQrBreakdown) return SOAP_ERR_QR_BREAKDOWN;
  if (bits & soap::kStatusTimeout) return SOAP_ERR_TIMEOUT;
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
  if (h->h_ptrs) cudaFreeHost(h->h_ptrs);
  if (h->status_ev) cudaEventDestroy(h->status_ev);
  if (h->stage_ev) cudaEventDestroy(h->stage_ev);
  for (auto& g : h->groups) {
    if (g.stream) cudaStreamDestroy(g.stream);
    if (g.far) cudaStreamDestroy(g.far);
    if (g.done) cudaEventDestroy(g.done);
    if (g.fork) cudaEventDestroy(g.fork);
    g.fork = nullptr;
    if (g.ev_vt) cudaEventDestroy(g.ev_vt);
    if (g.ev_far) cudaEventDestroy(g.ev_far);
    for (cudaEvent_t& ev : g.ev_vq) {
      if (ev) cudaEventDestroy(ev);
      ev = nullptr;
    }
    g.stream = g.far = nullptr;
    g.done = g.ev_vt = g.ev_far = nullptr;
  }
  h->h_status = nullptr;
  h->h_ptrs = nullptr;
  h->status_ev = h->stage_ev = nullptr;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

soap::TcOperand opnd(const float* hi, const float* lo, int64_t ld, int64_t stride, int batch) {
  return soap::TcOperand{hi, lo, ld, stride, batch};
}

soap::TcEpilogue epi(soap_handle h, float* C, int64_t ldc, int64_t c_stride, float* C_lo, int transpose, float alpha,
                     float beta) {
  return soap::TcEpilogue{C, nullptr, ldc, c_stride, C_lo, ldc, c_stride, transpose, alpha, beta, h->d_status};
}

// A class's step in three phases, so that the QR refreshes of all classes can be batched by size:
//   A  operand preparation and S1 (per class, caller's stream)
//   B  S2 + S3 for every preconditioned side, one batched QR per size group (refresh_bases)
//   C  S5-S8: rotations, Adam in the basis, back-rotation and update (per class)
//
// Two-sided classes run every contraction as a tcgen05 product C = A B^T of K-major operands:
//   S1  L <- b L + (1-b) G G^T       A = G,     B = G
//       R <- b R + (1-b) G^T G       A = G^T,   B = G^T
//   S2  P^T = Q_L^T L                A = Q_L^T, B = L (symmetric)  -> QR -> Q_L, Q_L^T
//   S5  Y^T = ([G | M_hat] Q_R)^T    A = [G|M], B = Q_R^T    (transposed epilogue)
//       [G' | m'] = Q_L^T Y          A = Q_L^T, B = Y^T
//   S6  N = Adam(G', m', v)
//   S7  Z^T = (N Q_R^T)^T            A = N,     B = Q_R      (transposed epilogue)
//   S8  W <- (1 - lr wd) W - lr Q_L Z  A = Q_L, B = Z^T      (epilogue into W)
// One-sided classes take the same route with one rotation on each side of Adam (a left-only
// class as the right-only problem of G^T). Classes whose rows or columns are not a multiple
// of 4 (rows of an operand must be 16-byte multiples for TMA) run on CUDA cores.
soap_status_t prepare_class(soap_handle h, ClassState& c, const float* const* d_grads, cudaStream_t s) {
  const soap_hparams& hp = h->hp;
  const int B = c.count, m = (int)c.rows, n = (int)c.cols;
  const int64_t mn = (int64_t)m * n;
  if (!c.tc) {
    SOAP_CUDA(h, soap::momentum_and_copy(d_grads, c.Gc, c.Mhat, mn, B, hp.beta1, h->d_status, s));
    return SOAP_OK;
  }
  SOAP_CUDA(h, soap::momentum_split(d_grads, c.Gc, c.Gc_lo, c.Gt, c.Gt_lo, c.Mhat, c.Mhat_lo, m, n, B, hp.beta1, c.tr,
                                    h->d_status, s));
  if (c.basis_dirty) {
    if (c.left) SOAP_CUDA(h, soap::basis_split(c.QL, c.QL_lo, c.QLt, c.QLt_lo, m, B, s));
    if (c.right) SOAP_CUDA(h, soap::basis_split(c.QR, c.QR_lo, c.QRt, c.QRt_lo, n, B, s));
    c.basis_dirty = false;
  }
  return SOAP_OK;
}

// S1 for one class (after prepare_class): the standard factor EMAs, or Alg. 1's KL form.
soap_status_t accumulate_factors(soap_handle h, ClassState& c, cudaStream_t s) {
  const soap_hparams& hp = h->hp;
  const int B = c.count, m = (int)c.rows, n = (int)c.cols;
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
      SOAP_CUDA(h, soap::gemm(false, true, m, m, n, aL, strided(c.Gc, n, mn), strided(c.Gc, n, mn), fb,
                              strided_mut(c.L, m, mm), B, s));
    if (c.right)  // S1: R <- b R + (1-b) G^T G
      SOAP_CUDA(h, soap::gemm(true, false, n, n, m, aR, strided(c.Gc, n, mn), strided(c.Gc, n, mn), fb,
                              strided_mut(c.R, n, nn), B, s));
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
    SOAP_CUDA(h, soap::gemm_tc_nt(m, m, m, B, opnd(c.QLt, c.QLt_lo, m, mm, B), opnd(c.L, c.L_lo, m, mm, B),
                                  epi(h, C, m, mm, nullptr, 0, 1.f, 0.f), s));
    SOAP_CUDA(h, soap::diag_dot(C, c.QLt, c.lamL, m, B, s));
    SOAP_CUDA(h, soap::gemm_tc_nt(n, n, n, B, opnd(c.QRt, c.QRt_lo, n, nn, B), opnd(c.R, c.R_lo, n, nn, B),
                                  epi(h, C, n, nn, nullptr, 0, 1.f, 0.f), s));
    SOAP_CUDA(h, soap::diag_dot(C, c.QRt, c.lamR, n, B, s));
    float* Y = h->YMt;
    float* Y_lo = h->YMt_lo;
    float* X = h->YMt + cls;
    float* X_lo = h->YMt_lo + cls;
    SOAP_CUDA(h, soap::gemm_tc_nt(m, n, n, B, opnd(c.Gc, c.Gc_lo, n, mn, B), opnd(c.QRt, c.QRt_lo, n, nn, B),
                                  epi(h, Y, n, mn, nullptr, 0, 1.f, 0.f), s));
    SOAP_CUDA(h, soap::scale_cols_split(Y, Y_lo, c.lamR, m, n, B, (float)((1.0 - fb) / n), hp.eps, s));
    SOAP_CUDA(h, soap::gemm_tc_nt(n, m, m, B, opnd(c.Gt, c.Gt_lo, m, mn, B), opnd(c.QLt, c.QLt_lo, m, mm, B),
                                  epi(h, X, m, mn, nullptr, 0, 1.f, 0.f), s));
    SOAP_CUDA(h, soap::scale_cols_split(X, X_lo, c.lamL, n, m, B, (float)((1.0 - fb) / m), hp.eps, s));
    SOAP_CUDA(h, soap::gemm_tc_nt(m, m, n, B, opnd(Y, Y_lo, n, mn, B), opnd(Y, Y_lo, n, mn, B),
                                  epi(h, c.L, m, mm, c.L_lo, 0, 1.f, fb), s));
    SOAP_CUDA(h, soap::gemm_tc_nt(n, n, m, B, opnd(X, X_lo, m, mn, B), opnd(X, X_lo, m, mn, B),
                                  epi(h, c.R, n, nn, c.R_lo, 0, 1.f, fb), s));
    return SOAP_OK;
  }
  if (c.left)
    SOAP_CUDA(h, soap::gemm_tc_nt(m, m, n, B, opnd(c.Gc, c.Gc_lo, n, mn, B), opnd(c.Gc, c.Gc_lo, n, mn, B),
                                  epi(h, c.L, m, mm, c.L_lo, 0, aL, fb), s));
  if (c.right)
    SOAP_CUDA(h, soap::gemm_tc_nt(n, n, m, B, opnd(c.Gt, c.Gt_lo, m, mn, B), opnd(c.Gt, c.Gt_lo, m, mn, B),
                                  epi(h, c.R, n, nn, c.R_lo, 0, aR, fb), s));
  return SOAP_OK;
}

// S2 + S3 for the preconditioned sides of one size group: P^T = Q^T F for each member (F the
// factor, symmetric) into one batched input, one QR, then Q^T, Q (and lo parts) and the
// zero-column flags back to the classes. The group runs on its own stream from the moment
// its members' factors are updated on the caller's stream, concurrently with other groups.
soap_status_t refresh_group(soap_handle h, QrGroup& g, cudaStream_t s) {
  const soap_hparams& hp = h->hp;
  using soap::strided;
  using soap::strided_mut;
  SOAP_CUDA(h, cudaEventRecord(g.fork, s));
  {
    cudaStream_t gs = g.stream;
    SOAP_CUDA(h, cudaStreamWaitEvent(gs, g.fork, 0));
    const int n = g.n;
    const int64_t nn = (int64_t)n * n;
    float* At;
    soap::qr_input_buffers(g.ws, n, g.batch, &At);
    for (const QrJob& j : g.jobs) {
      ClassState& c = h->classes[j.cls];
      float* F = j.left ? c.L : c.R;
      float* at = At + (int64_t)j.offset * nn;
      if (c.tc) {
        SOAP_CUDA(h, soap::gemm_tc_nt(n, n, n, c.count, opnd(j.left ? c.QLt : c.QRt, j.left ? c.QLt_lo : c.QRt_lo, n, nn,
                                                             c.count),
                                      opnd(F, j.left ? c.L_lo : c.R_lo, n, nn, c.count),
                                      epi(h, at, n, nn, nullptr, 0, 1.f, 0.f), gs));
      } else {
        SOAP_CUDA(h, soap::gemm(true, false, n, n, n, 1.f, strided(j.left ? c.QL : c.QR, n, nn), strided(F, n, nn), 0.f,
                                strided_mut(at, n, nn), c.count, gs));
      }
    }
    // the Q accumulation ends with Q^T and its lo part in the input buffers
    const soap::QrLookahead la{g.far, g.ev_vt, g.ev_far, {g.ev_vq[0], g.ev_vq[1]}};
    SOAP_CUDA(h, soap::qr_q_t(n, g.batch, nullptr, nullptr, nullptr, nullptr, g.skip, hp.qr_tol, g.ws, g.ws_bytes,
                              h->d_status, gs, &la));
    for (const QrJob& j : g.jobs) {
      ClassState& c = h->classes[j.cls];
      const float* qt = At + (int64_t)j.offset * nn;
      float* Q = j.left ? c.QL : c.QR;
      if (c.tc)
        SOAP_CUDA(h, soap::basis_from_qt(qt, nullptr, j.left ? c.QLt : c.QRt, j.left ? c.QLt_lo : c.QRt_lo, Q,
                                         j.left ? c.QL_lo : c.QR_lo, n, c.count, gs));
      else
        SOAP_CUDA(h, soap::basis_from_qt(qt, nullptr, nullptr, nullptr, Q, nullptr, n, c.count, gs));
      SOAP_CUDA(h, cudaMemcpyAsync(j.left ? c.skipL : c.skipR, g.skip + (int64_t)j.offset * n, (size_t)c.count * n,
                                   cudaMemcpyDeviceToDevice, gs));
    }
    SOAP_CUDA(h, cudaEventRecord(g.done, gs));
  }
  return SOAP_OK;
}

soap_status_t rotate_update_class(soap_handle h, ClassState& c, float* const* d_params, float bc1, float bc2,
                                  cudaStream_t s) {
  const soap_hparams& hp = h->hp;
  const int B = c.count, m = (int)c.rows, n = (int)c.cols;
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
    const float* X = c.tr ? c.Gt : c.Gc;
    const float* X_lo = c.tr ? c.Gt_lo : c.Gc_lo;
    const float* Q = c.tr ? c.QL : c.QR;
    const float* Q_lo = c.tr ? c.QL_lo : c.QR_lo;
    const float* Qt = c.tr ? c.QLt : c.QRt;
    const float* Qt_lo = c.tr ? c.QLt_lo : c.QRt_lo;
    SOAP_CUDA(h, soap::gemm_tc_nt(rr, cc, cc, 2 * B, opnd(X, X_lo, cc, mn, 2 * B), opnd(Qt, Qt_lo, cc, qq, B),
                                  epi(h, h->Gp, cc, mn, nullptr, 0, 1.f, 0.f), s));
    const uint8_t* skip = hp.guard ? (c.tr ? c.skipL : c.skipR) : nullptr;
    SOAP_CUDA(h, soap::adam_in_basis(h->Gp, h->Gp + cls, c.V, rr, cc, B, hp.beta1, hp.beta2, hp.eps, bc1, bc2, nullptr,
                                     skip, h->N_lo, h->d_status, s));
    soap::TcEpilogue ew = epi(h, nullptr, n, 0, nullptr, c.tr ? 1 : 0, -h->lr, 1.f - h->lr * h->wd);
    ew.C_ptrs = d_params;
    SOAP_CUDA(h, soap::gemm_tc_nt(rr, cc, cc, B, opnd(h->Gp, h->N_lo, cc, mn, B), opnd(Q, Q_lo, cc, qq, B), ew, s));
    return SOAP_OK;
  }
  if (c.tc) {
    const int64_t cls = (int64_t)B * mn;
    // rotations of the gradient and of the momentum in one launch each (batch 2B)
    SOAP_CUDA(h, soap::gemm_tc_nt(m, n, n, 2 * B, opnd(c.Gc, c.Gc_lo, n, mn, 2 * B), opnd(c.QRt, c.QRt_lo, n, nn, B),
                                  epi(h, h->YMt, m, mn, h->YMt_lo, 1, 1.f, 0.f), s));
    SOAP_CUDA(h, soap::gemm_tc_nt(m, n, m, 2 * B, opnd(c.QLt, c.QLt_lo, m, mm, B),
                                  opnd(h->YMt, h->YMt_lo, m, mn, 2 * B), epi(h, h->Gp, n, mn, nullptr, 0, 1.f, 0.f), s));
    SOAP_CUDA(h, soap::adam_in_basis(h->Gp, h->Gp + cls, c.V, m, n, B, hp.beta1, hp.beta2, hp.eps, bc1, bc2,
                                     hp.guard ? c.skipL : nullptr, hp.guard ? c.skipR : nullptr, h->N_lo, h->d_status,
                                     s));
    SOAP_CUDA(h, soap::gemm_tc_nt(m, n, n, B, opnd(h->Gp, h->N_lo, n, mn, B), opnd(c.QR, c.QR_lo, n, nn, B),
                                  epi(h, h->Zt, m, mn, h->Zt_lo, 1, 1.f, 0.f), s));
    soap::TcEpilogue ew = epi(h, nullptr, n, 0, nullptr, 0, -h->lr, 1.f - h->lr * h->wd);
    ew.C_ptrs = d_params;
    SOAP_CUDA(h, soap::gemm_tc_nt(m, n, m, B, opnd(c.QL, c.QL_lo, m, mm, B), opnd(h->Zt, h->Zt_lo, m, mn, B), ew, s));
    return SOAP_OK;
  }
  // S5 and the re-projected first moment: G' = Q_L^T G Q_R, m = Q_L^T M_hat Q_R
  const float* xg = c.Gc;
  const float* xm = c.Mhat;
  if (c.left) {
    SOAP_CUDA(h, soap::gemm(true, false, m, n, m, 1.f, strided(c.QL, m, mm), strided(c.Gc, n, mn), 0.f,
                            strided_mut(h->X1, n, mn), B, s));
    SOAP_CUDA(h, soap::gemm(true, false, m, n, m, 1.f, strided(c.QL, m, mm), strided(c.Mhat, n, mn), 0.f,
                            strided_mut(h->X2, n, mn), B, s));
    xg = h->X1;
    xm = h->X2;
  }
  float* gp;
  const float* mp;
  if (c.right) {
    SOAP_CUDA(h, soap::gemm(false, false, m, n, n, 1.f, strided(xg, n, mn), strided(c.QR, n, nn), 0.f,
                            strided_mut(h->Gp, n, mn), B, s));
    SOAP_CUDA(h, soap::gemm(false, false, m, n, n, 1.f, strided(xm, n, mn), strided(c.QR, n, nn), 0.f,
                            strided_mut(h->Mp, n, mn), B, s));
    gp = h->Gp;
    mp = h->Mp;
  } else {
    gp = const_cast<float*>(xg);  // X1, or the gradient arena copy when no side rotates
    mp = xm;
  }
  // S6
  SOAP_CUDA(h, soap::adam_in_basis(gp, mp, c.V, m, n, B, hp.beta1, hp.beta2, hp.eps, bc1, bc2,
                                   (hp.guard && c.left) ? c.skipL : nullptr, (hp.guard && c.right) ? c.skipR : nullptr,
                                   nullptr, h->d_status, s));
  // S7 + S8: W <- (1 - lr wd) W - lr Q_L N Q_R^T
  const float keep = 1.f - h->lr * h->wd;
  soap::MutOperand W{nullptr, d_params, 0, 0, n};
  if (c.left && c.right) {
    SOAP_CUDA(h, soap::gemm(false, false, m, n, m, 1.f, strided(c.QL, m, mm), strided(gp, n, mn), 0.f,
                            strided_mut(h->X1, n, mn), B, s));
    SOAP_CUDA(h, soap::gemm(false, true, m, n, n, -h->lr, strided(h->X1, n, mn), strided(c.QR, n, nn), keep, W, B, s));
  } else if (c.left) {
    SOAP_CUDA(h, soap::gemm(false, false, m, n, m, -h->lr, strided(c.QL, m, mm), strided(gp, n, mn), keep, W, B, s));
  } else if (c.right) {
    SOAP_CUDA(h, soap::gemm(false, true, m, n, n, -h->lr, strided(gp, n, mn), strided(c.QR, n, nn), keep, W, B, s));
  } else {
    SOAP_CUDA(h, soap::weight_update(d_params, gp, mn, B, h->lr, h->wd, s));
  }
  return SOAP_OK;
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
  hp->qr_tol = 1e-4f;
  hp->guard = 1;
  hp->kl = 0;
  hp->stale = 0;
}

soap_status_t soap_create(const soap_shape* shapes, int32_t n, const soap_hparams* hp,
                          int32_t device, soap_handle* out) {
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
  for (auto& c : h->classes) {
    if (c.count > 65535) {
      delete h;
      return SOAP_ERR_INVALID_ARG;
    }
  }

  size_t ws_mat = 0;
  size_t off = 0;
  cudaError_t e = cudaSuccess;
  for (auto& c : h->classes) {
    const size_t mn = (size_t)c.count * c.rows * c.cols;
    c.ptr_offset = off;
    off += 2 * (size_t)c.count;
    // tensor-core operands are read with TMA: rows of both G and G^T must be 16-byte multiples
    c.tc = (c.left || c.right) && (c.rows % 4 == 0) && (c.cols % 4 == 0);
    c.tr = c.tc && c.left && !c.right;
    // the arena holding M_hat directly after G (or G^T), so that one batch-2B product rotates both
    const size_t ga = c.tr ? mn : 2 * mn, ta = c.tr ? 2 * mn : mn;
    if (e == cudaSuccess) e = dalloc(h, (void**)&c.Gc, (c.tc ? ga : 2 * mn) * 4);
    if (e == cudaSuccess) e = dalloc(h, (void**)&c.V, mn * 4);
    if (c.tc) {
      if (e == cudaSuccess) e = dalloc(h, (void**)&c.Gc_lo, ga * 4);
      if (e == cudaSuccess) e = dalloc(h, (void**)&c.Gt, ta * 4);
      if (e == cudaSuccess) e = dalloc(h, (void**)&c.Gt_lo, ta * 4);
    }
    if (e == cudaSuccess) {
      c.Mhat = c.tr ? c.Gt + mn : c.Gc + mn;
      c.Mhat_lo = !c.tc ? nullptr : c.tr ? c.Gt_lo + mn : c.Gc_lo + mn;
    }
    if (c.left) {
      const size_t mm = (size_t)c.count * c.rows * c.rows;
      if (e == cudaSuccess) e = dalloc(h, (void**)&c.L, mm * 4);
      if (e == cudaSuccess) e = dalloc(h, (void**)&c.QL, mm * 4);
      if (e == cudaSuccess) e = dalloc(h, (void**)&c.skipL, (size_t)c.count * c.rows);
      if (c.tc) {
        if (e == cudaSuccess) e = dalloc(h, (void**)&c.L_lo, mm * 4);
        if (e == cudaSuccess) e = dalloc(h, (void**)&c.QL_lo, mm * 4);
        if (e == cudaSuccess) e = dalloc(h, (void**)&c.QLt, mm * 4);
        if (e == cudaSuccess) e = dalloc(h, (void**)&c.QLt_lo, mm * 4);
      }
    }
    if (c.right) {
      const size_t nn = (size_t)c.count * c.cols * c.cols;
      if (e == cudaSuccess) e = dalloc(h, (void**)&c.R, nn * 4);
      if (e == cudaSuccess) e = dalloc(h, (void**)&c.QR, nn * 4);
      if (e == cudaSuccess) e = dalloc(h, (void**)&c.skipR, (size_t)c.count * c.cols);
      if (c.tc) {
        if (e == cudaSuccess) e = dalloc(h, (void**)&c.R_lo, nn * 4);
        if (e == cudaSuccess) e = dalloc(h, (void**)&c.QR_lo, nn * 4);
        if (e == cudaSuccess) e = dalloc(h, (void**)&c.QRt, nn * 4);
        if (e == cudaSuccess) e = dalloc(h, (void**)&c.QRt_lo, nn * 4);
      }
    }
    if (hp->kl && c.left && c.right) {
      if (e == cudaSuccess) e = dalloc(h, (void**)&c.lamL, (size_t)c.count * c.rows * 4);
      if (e == cudaSuccess) e = dalloc(h, (void**)&c.lamR, (size_t)c.count * c.cols * 4);
      if (e == cudaSuccess) e = cudaMemset(c.lamL, 0, (size_t)c.count * c.rows * 4);
      if (e == cudaSuccess) e = cudaMemset(c.lamR, 0, (size_t)c.count * c.cols * 4);
    }
    ws_mat = std::max(ws_mat, mn);
  }
  // QR groups: every preconditioned side, grouped by size
  {
    std::map<int, int, std::greater<int>> by_n;
    for (int ci = 0; ci < (int)h->classes.size(); ++ci) {
      const ClassState& c = h->classes[ci];
      for (int side = 0; side < 2; ++side) {
        if (side == 0 ? !c.left : !c.right) continue;
        const int n = (int)(side == 0 ? c.rows : c.cols);
        auto it = by_n.find(n);
        if (it == by_n.end()) it = by_n.emplace(n, (int)by_n.size()).first;
        (void)it;
      }
    }
    for (auto& kv : by_n) {
      QrGroup g;
      g.n = kv.first;
      h->groups.push_back(g);
    }
    for (int ci = 0; ci < (int)h->classes.size(); ++ci) {
      const ClassState& c = h->classes[ci];
      for (int side = 0; side < 2; ++side) {
        if (side == 0 ? !c.left : !c.right) continue;
        const int n = (int)(side == 0 ? c.rows : c.cols);
        for (auto& g : h->groups)
          if (g.n == n) {
            g.jobs.push_back(QrJob{ci, side == 0, g.batch});
            g.batch += c.count;
          }
      }
    }
    for (auto& g : h->groups) {
      if (g.batch > 65535) e = cudaErrorInvalidValue;
      g.ws_bytes = soap::qr_workspace_bytes(g.n, g.batch, true);
      if (e == cudaSuccess) e = dalloc(h, &g.ws, g.ws_bytes);
      if (e == cudaSuccess) e = dalloc(h, (void**)&g.skip, (size_t)g.batch * g.n);
      // the panel chain is latency-bound: its stream goes first when SMs free up
      int prio_lo = 0, prio_hi = 0;
      if (e == cudaSuccess) e = cudaDeviceGetStreamPriorityRange(&prio_lo, &prio_hi);
      if (e == cudaSuccess) e = cudaStreamCreateWithPriority(&g.stream, cudaStreamNonBlocking, prio_hi);
      if (e == cudaSuccess) e = cudaStreamCreateWithPriority(&g.far, cudaStreamNonBlocking, prio_lo);
      if (e == cudaSuccess) e = cudaEventCreateWithFlags(&g.done, cudaEventDisableTiming);
      if (e == cudaSuccess) e = cudaEventCreateWithFlags(&g.fork, cudaEventDisableTiming);
      if (e == cudaSuccess) e = cudaEventCreateWithFlags(&g.ev_vt, cudaEventDisableTiming);
      if (e == cudaSuccess) e = cudaEventCreateWithFlags(&g.ev_far, cudaEventDisableTiming);
      for (cudaEvent_t& ev : g.ev_vq)
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming);
    }
    // step order: see soap_step
    const int nc = (int)h->classes.size();
    auto largest = [&](int ci) {
      const ClassState& c = h->classes[ci];
      return std::max(c.left ? c.rows : (int64_t)0, c.right ? c.cols : (int64_t)0);
    };
    h->prep_order.resize(nc);
    for (int ci = 0; ci < nc; ++ci) h->prep_order[ci] = ci;
    h->update_order = h->prep_order;
    std::stable_sort(h->prep_order.begin(), h->prep_order.end(), [&](int x, int y) { return largest(x) > largest(y); });
    std::stable_sort(h->update_order.begin(), h->update_order.end(),
                     [&](int x, int y) { return largest(x) < largest(y); });
    h->fork_after.assign(nc, {});
    h->groups_of.assign(nc, {});
    std::vector<int> pos(nc);
    for (int q = 0; q < nc; ++q) pos[h->prep_order[q]] = q;
    for (int gi = 0; gi < (int)h->groups.size(); ++gi) {
      int last = -1;
      for (const QrJob& j : h->groups[gi].jobs) {
        h->groups_of[j.cls].push_back(gi);
        if (last < 0 || pos[j.cls] > pos[last]) last = j.cls;
      }
      if (last >= 0) h->fork_after[last].push_back(gi);
    }
  }
  h->nptrs = off;
  // workspaces: [G' | m'] for every class; N's lo part for tensor-core classes; the
  // intermediate products of two-sided tensor-core classes; X1/X2 for CUDA-core classes and
  // for single-matrix state reads and writes
  size_t ws_tc = 0, ws_two = 0, ws_x = 0, ws_lam = 0;
  for (auto& c : h->classes) {
    const size_t mn = (size_t)c.count * c.rows * c.cols;
    if (c.tc) ws_tc = std::max(ws_tc, mn);
    if (c.tc && c.left && c.right) ws_two = std::max(ws_two, mn);
    if (hp->kl && c.left && c.right)
      ws_lam = std::max(ws_lam, (size_t)c.count * std::max(c.rows * c.rows, c.cols * c.cols));
    ws_x = std::max(ws_x, c.tc ? (size_t)(c.rows * c.cols) : mn);
  }
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->X1, ws_x * 4);
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->X2, ws_x * 4);
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->Gp, 2 * ws_mat * 4);
  h->Mp = h->Gp ? h->Gp + ws_mat : nullptr;
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->N_lo, ws_tc * 4);
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->YMt, 2 * ws_two * 4);
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->YMt_lo, 2 * ws_two * 4);
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->Zt, ws_two * 4);
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->Zt_lo, ws_two * 4);
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->lam_ws, ws_lam * 4);
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->d_status, sizeof(int));
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->d_ptrs, h->nptrs * sizeof(void*));
  if (e == cudaSuccess) e = cudaMallocHost((void**)&h->h_status, sizeof(int));
  if (e == cudaSuccess) e = cudaMallocHost((void**)&h->h_ptrs, h->nptrs * sizeof(void*));
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->status_ev, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->stage_ev, cudaEventDisableTiming);
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
    if (c.tc && e == cudaSuccess) e = cudaMemset(c.Mhat_lo, 0, mn * 4);
    if (e == cudaSuccess) e = cudaMemset(c.V, 0, mn * 4);
    if (c.left) {
      if (e == cudaSuccess) e = cudaMemset(c.L, 0, (size_t)c.count * c.rows * c.rows * 4);
      if (c.tc && e == cudaSuccess) e = cudaMemset(c.L_lo, 0, (size_t)c.count * c.rows * c.rows * 4);
      if (e == cudaSuccess) e = soap::set_identity(c.QL, (int)c.rows, c.count, 0);
      if (e == cudaSuccess) e = cudaMemset(c.skipL, 0, (size_t)c.count * c.rows);
    }
    if (c.right) {
      if (e == cudaSuccess) e = cudaMemset(c.R, 0, (size_t)c.count * c.cols * c.cols * 4);
      if (c.tc && e == cudaSuccess) e = cudaMemset(c.R_lo, 0, (size_t)c.count * c.cols * c.cols * 4);
      if (e == cudaSuccess) e = soap::set_identity(c.QR, (int)c.cols, c.count, 0);
      if (e == cudaSuccess) e = cudaMemset(c.skipR, 0, (size_t)c.count * c.cols);
    }
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
  // pointer table: [class][params..., grads...], uploaded only when it changed
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
  if (changed) {
    if (h->stage_pending) SOAP_CUDA(h, cudaEventSynchronize(h->stage_ev));
    std::memcpy(h->h_ptrs, h->last_ptrs.data(), h->nptrs * sizeof(void*));
    SOAP_CUDA(h, cudaMemcpyAsync(h->d_ptrs, h->h_ptrs, h->nptrs * sizeof(void*), cudaMemcpyHostToDevice, s));
    SOAP_CUDA(h, cudaEventRecord(h->stage_ev, s));
    h->stage_pending = true;
  }

  h->t += 1;
  const int64_t t = h->t;
  const soap_hparams& hp = h->hp;
  const bool refresh = (t % hp.eig_every) == 0;
  const float bc1 = hp.bias_correction ? 1.f - powf(hp.beta1, (float)t) : 1.f;
  const float bc2 = hp.bias_correction ? 1.f - powf(hp.beta2, (float)t) : 1.f;
  auto params_of = [&](const ClassState& c) { return reinterpret_cast<float* const*>(h->d_ptrs + c.ptr_offset); };
  auto grads_of = [&](const ClassState& c) {
    return reinterpret_cast<const float* const*>(h->d_ptrs + c.ptr_offset + c.count);
  };
  // Phase A class by class, each size group's refresh forked as soon as the last class feeding
  // it is prepared (classes with the largest factors first, so the longest refresh starts
  // earliest); phase C class by class, each waiting only for the groups its bases come from
  // (classes with the smallest factors first, whose refreshes finish earliest).
  // The stale variant refreshes from the factors as they stand and accumulates G_t into them
  // at the end of the step.
  for (int ci : h->prep_order) {
    soap_status_t st = prepare_class(h, h->classes[ci], grads_of(h->classes[ci]), s);
    if (st == SOAP_OK && !hp.stale) st = accumulate_factors(h, h->classes[ci], s);
    if (st != SOAP_OK) return st;
    if (refresh)
      for (int gi : h->fork_after[ci]) {
        st = refresh_group(h, h->groups[gi], s);
        if (st != SOAP_OK) return st;
      }
  }
  std::vector<bool> joined(h->groups.size(), !refresh);
  for (int ci : h->update_order) {
    for (int gi : h->groups_of[ci])
      if (!joined[gi]) {
        SOAP_CUDA(h, cudaStreamWaitEvent(s, h->groups[gi].done, 0));
        joined[gi] = true;
      }
    soap_status_t st = rotate_update_class(h, h->classes[ci], params_of(h->classes[ci]), bc1, bc2, s);
    if (st != SOAP_OK) return st;
  }
  for (size_t gi = 0; gi < h->groups.size(); ++gi)
    if (!joined[gi]) SOAP_CUDA(h, cudaStreamWaitEvent(s, h->groups[gi].done, 0));
  if (hp.stale)
    for (auto& c : h->classes) {
      soap_status_t st = accumulate_factors(h, c, s);
      if (st != SOAP_OK) return st;
    }
  SOAP_CUDA(h, cudaMemcpyAsync(h->h_status, h->d_status, sizeof(int), cudaMemcpyDeviceToHost, s));
  SOAP_CUDA(h, cudaEventRecord(h->status_ev, s));
  h->status_pending = true;
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

namespace {
// Address of a stored state piece (not SOAP_STATE_M, which is derived).
void* state_ptr(soap_handle h, int idx, int which) {
  const auto [ci, slot] = h->loc[idx];
  ClassState& c = h->classes[ci];
  const size_t mn = (size_t)c.rows * c.cols, mm = (size_t)c.rows * c.rows, nn = (size_t)c.cols * c.cols;
  switch (which) {
    case SOAP_STATE_V: return c.V + slot * mn;
    case SOAP_STATE_MHAT: return c.Mhat + slot * mn;
    case SOAP_STATE_L: return c.L ? c.L + slot * mm : nullptr;
    case SOAP_STATE_QL: return c.QL ? c.QL + slot * mm : nullptr;
    case SOAP_STATE_R: return c.R ? c.R + slot * nn : nullptr;
    case SOAP_STATE_QR: return c.QR ? c.QR + slot * nn : nullptr;
    case SOAP_STATE_SKIP_L: return c.skipL ? c.skipL + slot * c.rows : nullptr;
    case SOAP_STATE_SKIP_R: return c.skipR ? c.skipR + slot * c.cols : nullptr;
    case SOAP_STATE_LAMBDA_L: return c.lamL ? c.lamL + slot * c.rows : nullptr;
    case SOAP_STATE_LAMBDA_R: return c.lamR ? c.lamR + slot * c.cols : nullptr;
    default: return nullptr;
  }
}
}  // namespace

soap_status_t soap_state_get(soap_handle h, int32_t idx, int32_t which, void* dst, soap_stream_t stream_) {
  if (!h) return SOAP_ERR_INVALID_ARG;
  const size_t bytes = soap_state_bytes(h, idx, which);
  if (bytes == 0 || !dst) return fail(h, SOAP_ERR_INVALID_ARG, "soap_state_get: no such state piece");
  DeviceGuard g(h->device);
  cudaStream_t s = (cudaStream_t)stream_;
  const auto [ci, slot] = h->loc[idx];
  ClassState& c = h->classes[ci];
  const int m = (int)c.rows, nc = (int)c.cols;
  const int64_t mn = (int64_t)m * nc;
  if (c.tr && (which == SOAP_STATE_V || which == SOAP_STATE_MHAT)) {
    // stored transposed (n x m): hand out the m x n matrix
    SOAP_CUDA(h, soap::transpose((const float*)state_ptr(h, idx, which), h->X1, nc, m, 1, s));
    SOAP_CUDA(h, cudaMemcpyAsync(dst, h->X1, bytes, cudaMemcpyDefault, s));
    return SOAP_OK;
  }
  if (which != SOAP_STATE_M) {
    SOAP_CUDA(h, cudaMemcpyAsync(dst, state_ptr(h, idx, which), bytes, cudaMemcpyDefault, s));
    return SOAP_OK;
  }
  // m = Q_L^T M_hat Q_R, computed into the workspace
  const float* x = c.Mhat + slot * mn;
  if (c.tc && c.basis_dirty) {
    if (c.left) SOAP_CUDA(h, soap::basis_split(c.QL, c.QL_lo, c.QLt, c.QLt_lo, m, c.count, s));
    if (c.right) SOAP_CUDA(h, soap::basis_split(c.QR, c.QR_lo, c.QRt, c.QRt_lo, nc, c.count, s));
    c.basis_dirty = false;
  }
  if (c.tc && !(c.left && c.right)) {
    // the step's product [X | M_hat] Q for this matrix alone (bit-identical), written in the
    // original orientation
    const int rr = c.tr ? nc : m, cc = c.tr ? m : nc;
    const int64_t qq = (int64_t)cc * cc;
    const float* Qt = (c.tr ? c.QLt : c.QRt) + slot * qq;
    const float* Qt_lo = (c.tr ? c.QLt_lo : c.QRt_lo) + slot * qq;
    SOAP_CUDA(h, soap::gemm_tc_nt(rr, cc, cc, 1, opnd(x, c.Mhat_lo + slot * mn, cc, mn, 1), opnd(Qt, Qt_lo, cc, qq, 1),
                                  epi(h, h->Gp, c.tr ? rr : cc, mn, nullptr, c.tr ? 1 : 0, 1.f, 0.f), s));
    SOAP_CUDA(h, cudaMemcpyAsync(dst, h->Gp, bytes, cudaMemcpyDefault, s));
    return SOAP_OK;
  }
  if (c.tc) {
    // the same tensor-core products, on the same operands, as the step's rotation of M_hat:
    // bit-identical to the m the last step used
    const int64_t mm = (int64_t)m * m, nn = (int64_t)nc * nc;
    SOAP_CUDA(h, soap::gemm_tc_nt(m, nc, nc, 1, opnd(x, c.Mhat_lo + slot * mn, nc, mn, 1),
                                  opnd(c.QRt + slot * nn, c.QRt_lo + slot * nn, nc, nn, 1),
                                  epi(h, h->X1, m, mn, h->X2, 1, 1.f, 0.f), s));
    SOAP_CUDA(h, soap::gemm_tc_nt(m, nc, m, 1, opnd(c.QLt + slot * mm, c.QLt_lo + slot * mm, m, mm, 1),
                                  opnd(h->X1, h->X2, m, mn, 1), epi(h, h->Gp, nc, mn, nullptr, 0, 1.f, 0.f), s));
    SOAP_CUDA(h, cudaMemcpyAsync(dst, h->Gp, bytes, cudaMemcpyDefault, s));
    return SOAP_OK;
  }
  using soap::strided;
  using soap::strided_mut;
  if (c.left) {
    SOAP_CUDA(h, soap::gemm(true, false, m, nc, m, 1.f, strided(c.QL + (int64_t)slot * m * m, m, 0), strided(x, nc, 0),
                            0.f, strided_mut(h->X1, nc, 0), 1, s));
    x = h->X1;
  }
  if (c.right) {
    SOAP_CUDA(h, soap::gemm(false, false, m, nc, nc, 1.f, strided(x, nc, 0), strided(c.QR + (int64_t)slot * nc * nc, nc, 0),
                            0.f, strided_mut(h->Gp, nc, 0), 1, s));
    x = h->Gp;
  }
  SOAP_CUDA(h, cudaMemcpyAsync(dst, x, bytes, cudaMemcpyDefault, s));
  return SOAP_OK;
}

soap_status_t soap_state_set(soap_handle h, int32_t idx, int32_t which, const void* src, soap_stream_t stream_) {
  if (!h) return SOAP_ERR_INVALID_ARG;
  const size_t bytes = soap_state_bytes(h, idx, which);
  if (bytes == 0 || !src) return fail(h, SOAP_ERR_INVALID_ARG, "soap_state_set: no such state piece");
  if (which == SOAP_STATE_LAMBDA_L || which == SOAP_STATE_LAMBDA_R)
    return fail(h, SOAP_ERR_INVALID_ARG, "soap_state_set: the KL eigenvalue estimates are read-only");
  DeviceGuard g(h->device);
  cudaStream_t s = (cudaStream_t)stream_;
  const auto [ci, slot] = h->loc[idx];
  ClassState& c = h->classes[ci];
  const int m = (int)c.rows, nc = (int)c.cols;
  const int64_t mn = (int64_t)m * nc;
  float* dstm = c.Mhat + slot * mn;
  if (which != SOAP_STATE_M) {
    if (c.tr && (which == SOAP_STATE_V || which == SOAP_STATE_MHAT)) {
      // stored transposed (n x m)
      SOAP_CUDA(h, cudaMemcpyAsync(h->X1, src, bytes, cudaMemcpyDefault, s));
      SOAP_CUDA(h, soap::transpose(h->X1, (float*)state_ptr(h, idx, which), m, nc, 1, s));
    } else {
      SOAP_CUDA(h, cudaMemcpyAsync(state_ptr(h, idx, which), src, bytes, cudaMemcpyDefault, s));
    }
    if (which == SOAP_STATE_QL || which == SOAP_STATE_QR) c.basis_dirty = true;
    if (which == SOAP_STATE_MHAT && c.tc)
      SOAP_CUDA(h, soap::split_tf32(dstm, nullptr, c.Mhat_lo + slot * mn, mn, s));
    // the factors' lo parts: the KL form reads them (lambda = diag(Q^T F Q)) before S1 rewrites them
    if (which == SOAP_STATE_L && c.tc)
      SOAP_CUDA(h, soap::split_tf32(c.L + slot * (int64_t)m * m, nullptr, c.L_lo + slot * (int64_t)m * m,
                                    (int64_t)m * m, s));
    if (which == SOAP_STATE_R && c.tc)
      SOAP_CUDA(h, soap::split_tf32(c.R + slot * (int64_t)nc * nc, nullptr, c.R_lo + slot * (int64_t)nc * nc,
                                    (int64_t)nc * nc, s));
    return SOAP_OK;
  }
  // M_hat = Q_L m Q_R^T
  using soap::strided;
  using soap::strided_mut;
  SOAP_CUDA(h, cudaMemcpyAsync(h->Gp, src, bytes, cudaMemcpyDefault, s));
  const float* x = h->Gp;
  if (c.left) {
    float* out = (c.right || c.tr) ? h->X1 : dstm;
    SOAP_CUDA(h, soap::gemm(false, false, m, nc, m, 1.f, strided(c.QL + (int64_t)slot * m * m, m, 0), strided(x, nc, 0),
                            0.f, strided_mut(out, nc, 0), 1, s));
    x = out;
  }
  if (c.right) {
    SOAP_CUDA(h, soap::gemm(false, true, m, nc, nc, 1.f, strided(x, nc, 0), strided(c.QR + (int64_t)slot * nc * nc, nc, 0),
                            0.f, strided_mut(dstm, nc, 0), 1, s));
  } else if (c.tr) {
    SOAP_CUDA(h, soap::transpose(x, dstm, m, nc, 1, s));
  } else if (!c.left) {
    SOAP_CUDA(h, cudaMemcpyAsync(dstm, x, bytes, cudaMemcpyDeviceToDevice, s));
  }
  if (c.tc) SOAP_CUDA(h, soap::split_tf32(dstm, nullptr, c.Mhat_lo + slot * mn, mn, s));
  return SOAP_OK;
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
  if (!h || max_launches < 1 || max_launches > (int64_t(1) << 22)) return SOAP_ERR_INVALID_ARG;
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
    out[i] = soap_launch_record{p.recs[i].family, (double)t0, (double)t1};
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
                      size_t workspace_bytes, soap_stream_t stream) {
  if (n <= 0 || n > 8192 || (n & 3) || batch <= 0 || batch > 65535 || !P || !Q || !skip || !workspace ||
      !(tol >= 0.f))
    return SOAP_ERR_INVALID_ARG;
  if (!aligned16(P) || !aligned16(Q) || (reinterpret_cast<uintptr_t>(workspace) & 255))
    return SOAP_ERR_INVALID_ARG;
  if (workspace_bytes < soap_qr_workspace_bytes(n, batch)) return SOAP_ERR_INVALID_ARG;
  cudaStream_t s = (cudaStream_t)stream;
  // the status word lives in the last 256 bytes of the caller's workspace
  const size_t qb = soap::qr_workspace_bytes(n, batch);
  int* status = reinterpret_cast<int*>(static_cast<char*>(workspace) + qb);
  if (cudaMemsetAsync(status, 0, sizeof(int), s) != cudaSuccess) return SOAP_ERR_CUDA;
  cudaError_t e = soap::qr_q(n, batch, P, Q, skip, tol, workspace, qb, status, s);
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

soap_status_t soap_split_tf32(const float* x, float* hi, float* lo, int64_t n, soap_stream_t stream) {
  if (n < 0 || (n > 0 && (!x || !lo))) return SOAP_ERR_INVALID_ARG;
  return soap::split_tf32(x, hi, lo, n, (cudaStream_t)stream) == cudaSuccess ? SOAP_OK : SOAP_ERR_CUDA;
}

}  // extern "C"
