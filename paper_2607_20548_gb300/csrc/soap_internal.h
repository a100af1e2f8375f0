// Internal declarations shared by the libsoap translation units (not part of the ABI).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/soap.h"
#include "profile.h"

namespace soap {

// Sticky device status bits (combined with atomicOr by the kernels).
enum : int {
  kStatusNonFinite = 1,
  kStatusQrBreakdown = 2,
  kStatusTimeout = 4,
};

// A batched matrix operand: matrix b starts at (ptrs ? ptrs[b] : base + b * stride) + offset.
struct Operand {
  const float* base;
  const float* const* ptrs;  // device array of per-matrix pointers, or nullptr
  int64_t stride;
  int64_t offset;
  int64_t ld;
};

struct MutOperand {
  float* base;
  float* const* ptrs;
  int64_t stride;
  int64_t offset;
  int64_t ld;
};

inline Operand strided(const float* base, int64_t ld, int64_t stride, int64_t offset = 0) {
  return Operand{base, nullptr, stride, offset, ld};
}
inline MutOperand strided_mut(float* base, int64_t ld, int64_t stride, int64_t offset = 0) {
  return MutOperand{base, nullptr, stride, offset, ld};
}

// C_b = alpha * op(A_b) op(B_b) + beta * C_b for b < batch (fp32-accurate).
// Returns a cudaError_t from the launch.
cudaError_t gemm(bool trans_a, bool trans_b, int M, int N, int K, float alpha, Operand A,
                 Operand B, float beta, MutOperand C, int batch, cudaStream_t stream);

// CUDA-core fp32 engine (exact fp32 FMAs); any shape.
cudaError_t gemm_simt(bool trans_a, bool trans_b, int M, int N, int K, float alpha, Operand A,
                      Operand B, float beta, MutOperand C, int batch, cudaStream_t stream);

// ---- tcgen05 fp32 engine (four TF32 products): C_b = alpha * A_b B_(b mod B.batch)^T + beta * C_b
// An operand is `batch` row-major (rows x K) matrices split as hi = trunc_tf32(x) (the fp32
// array itself may serve: the tensor core drops the 13 low mantissa bits) and lo = x - hi.
struct TcOperand {
  const float* hi;
  const float* lo;
  int64_t ld;      // elements between rows
  int64_t stride;  // elements between matrices
  int batch;       // distinct matrices (0: one per launch batch entry)
};
struct TcEpilogue {
  float* C;              // output (or nullptr), offset b * c_stride ...
  float* const* C_ptrs;  // ... or a device array of per-matrix output pointers
  int64_t ldc;
  int64_t c_stride;
  float* C_lo;           // optional: also write out - tf32(out) here (same layout, ld_lo)
  int64_t ld_lo;
  int64_t lo_stride;
  int transpose;         // write C^T (C_b is then N x M with leading dimension ldc)
  float alpha, beta;     // beta != 0 reads C
  int* status;           // device status word for a timed-out wait (may be nullptr)
  // set by gemm_tc_nt from the library's wait settings (soap_wait_limit), not by callers:
  uint64_t wait_ns = 0;       // bounded waits give up after this long
  const int* hold = nullptr;  // testing the timeout path: the epilogue first waits for *hold != 0
};
// `family` tags the launch for the library's profiler. With a split workspace (room for
// ksplit * batch * M * N floats) a launch of few tiles and long K may split K over more CTAs
// and add the partial sums in a second kernel (row-major C with beta = 0 only).
cudaError_t gemm_tc_nt(int M, int N, int K, int batch, const TcOperand& A, const TcOperand& B,
                       const TcEpilogue& ep, cudaStream_t stream, int family = kFamGemmTc,
                       float* split_ws = nullptr, size_t split_ws_floats = 0);
// Bound of the tensor-core products' device waits (0: 2 s) and, for testing the timeout path, a
// device flag their epilogues first wait for (nullptr: none); applies to later launches.
void set_wait_limit(uint64_t ns, const int* hold);
// Symmetric product C_b = alpha A_b A_b^T + beta C_b (M x M, A_b M x K): only the 128 x 128 tiles on
// or below the diagonal are computed, each below it also stored (with its lo part) in the mirror
// position. Needs a row-major, 16-byte aligned C with its lo part; other forms go to gemm_tc_nt.
cudaError_t gemm_tc_syrk(int M, int K, int batch, const TcOperand& A, const TcEpilogue& ep, cudaStream_t stream,
                         int family = kFamGemmTc);
// hi = trunc_tf32(x), lo = x - hi (exact), elementwise over n values.
cudaError_t split_tf32(const float* x, float* hi, float* lo, int64_t n, cudaStream_t stream);

// Householder QR (explicit Q) of `batch` contiguous n x n matrices (n a multiple of 4).
// Workspace of qr_q / qr_q_t; `lookahead` adds the buffers of the two-stream schedule.
size_t qr_workspace_bytes(int n, int batch, bool lookahead = false);
// P read only; Q written. Uses the tensor-core QR on P^T (staged in the workspace).
cudaError_t qr_q(int n, int batch, const float* P, float* Q, uint8_t* skip, float tol,
                 void* workspace, size_t workspace_bytes, int* status, cudaStream_t stream);
// Where the factored matrix P^T must be placed before qr_q_t.
void qr_input_buffers(void* workspace, int n, int batch, float** At);
// QR of P whose transpose is already in qr_input_buffers(). Writes Q^T into Qt (or, if Qt is
// nullptr, into the workspace) and, if Q is given, Q and (if Q_lo is given) its lo part.
// Qt_lo is not written.
// The look-ahead schedule of qr_q_t: a second (low-priority) stream and its events.
struct QrLookahead {
  cudaStream_t far;     // trailing updates beyond the next block, and V T for the Q accumulation
  cudaEvent_t vt;       // this block's V T^T and the next block's rows are ready (caller's stream)
  cudaEvent_t far_done; // the far update of the previous block is done (recorded on `far`)
  cudaEvent_t vq[2];    // V T of the block using buffer 0 / 1 is done (recorded on `far`)
};
// With `la` (all members set, and a workspace sized with lookahead) the trailing update of each
// 128-column block, except the next block's rows, and the block's V T run on la->far and
// overlap the next block's panels; everything is joined back on `stream` before return.
cudaError_t qr_q_t(int n, int batch, float* Qt, float* Qt_lo, float* Q, float* Q_lo, uint8_t* skip,
                   float tol, void* workspace, size_t workspace_bytes, int* status,
                   cudaStream_t stream, const QrLookahead* la = nullptr);

// bf16 tensor-core product out_b = alpha A_b B_b^T + beta Cin_b (A_b M x K, B_b N x K, bf16
// row-major; fp32 accumulation). Outputs (any may be null): out (bf16, ld, stride; Cin has the
// same layout), out_t (bf16, transposed: element (r, c) at c * ld_t + r) and out_f32.
// N and K must be multiples of 8.
struct Bf16Epilogue {
  __nv_bfloat16* out;
  int64_t ld, stride;
  const __nv_bfloat16* cin;
  __nv_bfloat16* out_t;
  int64_t ld_t, stride_t;
  float* out_f32;
  int64_t ld_f32, stride_f32;
  float alpha, beta;
  int* status;
};
cudaError_t gemm_bf16_nt(int M, int N, int K, int batch, const __nv_bfloat16* A, int64_t lda, int64_t a_stride,
                         const __nv_bfloat16* B, int64_t ldb, int64_t b_stride, const Bf16Epilogue& ep,
                         cudaStream_t stream);

// Muon's elementwise kernels (batched over `batch` rows x cols matrices of a class).
// M <- beta1 M + (1 - beta1) G and norm2[b] += ||M_b||_F^2 (norm2 zeroed by the caller);
// non-finite gradients set kStatusNonFinite.
cudaError_t muon_momentum(const float* const* grads, float* M, double* norm2, int64_t elems, int batch, float beta1,
                          int* status, cudaStream_t stream);
// X_0 = M / max(||M||_F, eps) in bf16, as X (r x c) and X^T (c x r) with (r, c) = (rows, cols),
// or, if `transposed`, (r, c) = (cols, rows) and X = M^T scaled.
cudaError_t muon_init_x(const float* M, const double* norm2, float eps, __nv_bfloat16* X, __nv_bfloat16* Xt,
                        int rows, int cols, int batch, bool transposed, cudaStream_t stream);
// W <- (1 - lr wd) W - lr scale O, O bf16 rows x cols.
cudaError_t muon_update(float* const* params, const __nv_bfloat16* O, int64_t elems, int batch, float lr, float wd,
                        float scale, cudaStream_t stream);

// Elementwise kernels of the step.
// M_hat <- b1 M_hat + (1-b1) G and Gc <- G for each matrix of a class.
cudaError_t momentum_and_copy(const float* const* grads, float* Gc, float* Mhat, int64_t elems,
                              int batch, float beta1, int* status, cudaStream_t stream);
// v <- b2 v + (1-b2) G'^2; N = m' / (sqrt(v) + eps) (bias-corrected if t > 0 given),
// written over Gp; guard rows/cols zeroed.
cudaError_t adam_in_basis(float* Gp, const float* Mp, float* V, int rows, int cols, int batch,
                          float beta1, float beta2, float eps, float bc1, float bc2,
                          const uint8_t* skipL, const uint8_t* skipR, float* N_lo, int* status,
                          cudaStream_t stream);
// Tensor-core operand preparation: G and G^T with their lo parts, and the momentum EMA
// M_hat <- b1 M_hat + (1-b1) G in place, with a copy of the new M_hat and its lo part
// (Mcopy, Mcopy_lo); M_hat is stored in G's orientation or (if mhat_transposed) as M_hat^T,
// and so is its copy.
cudaError_t momentum_split(const float* const* grads, float* Gn, float* Gn_lo, float* Gt, float* Gt_lo,
                           float* Mhat, float* Mcopy, float* Mcopy_lo, int rows, int cols, int batch, float beta1,
                           bool mhat_transposed, int* status, cudaStream_t stream);
// Packed symmetric storage: the lower-triangular 32 x 32 tiles of an n x n matrix, tile (I, J)
// (I >= J) at tile index I (I + 1) / 2 + J, each row-major; packed_floats(n) per matrix.
int64_t packed_floats(int n);
// F_b (full, n x n) and, if F_lo is given, its lo part from the packed tiles P_b.
cudaError_t unpack_sym(const float* P, float* F, float* F_lo, int n, int batch, cudaStream_t stream);
// P_b from the lower triangle of F_b.
cudaError_t pack_sym(const float* F, float* P, int n, int batch, cudaStream_t stream);
// Device pointer table written from a host array through kernel parameters (no host buffer
// has to outlive the call, and nothing waits on the host).
constexpr int kPtrChunk = 480;
struct PtrChunk {
  void* p[kPtrChunk];
};
cudaError_t put_ptrs(void** dst, void* const* src, int64_t n, cudaStream_t stream);
// dst_b = src_b^T for `batch` contiguous rows x cols matrices.
cudaError_t transpose(const float* src, float* dst, int rows, int cols, int batch, cudaStream_t stream);
// From Q^T: a copy of it with its lo part, and Q with its lo part (any output may be null;
// the lo parts are formed from the values, Qt_lo is not read).
cudaError_t basis_from_qt(const float* Qt, const float* Qt_lo, float* Qt_out, float* Qt_lo_out, float* Q,
                          float* Q_lo, int n, int batch, cudaStream_t stream);
// Q -> lo part, Q^T, lo part of Q^T for `batch` n x n bases.
cudaError_t basis_split(const float* Q, float* Q_lo, float* Qt, float* Qt_lo, int n, int batch,
                        cudaStream_t stream);
// W <- (1 - lr*wd) W - lr * D (both sides identity).
cudaError_t weight_update(float* const* params, const float* D, int64_t elems, int batch,
                          float lr, float wd, cudaStream_t stream);
// KL-Shampoo factor form: lam[b][i] = sum_k C[b][i][k] Qt[b][i][k], the diagonal of Q^T F Q
// from C = Q^T F (n a multiple of 4).
cudaError_t diag_dot(const float* C, const float* Qt, float* lam, int n, int batch, cudaStream_t stream);
// X[b][:, j] *= sqrt(coef / (max(lam[b][j], 0) + eps)) in place, with the lo part into X_lo
// (cols a multiple of 4).
cudaError_t scale_cols_split(float* X, float* X_lo, const float* lam, int rows, int cols, int batch,
                             float coef, float eps, cudaStream_t stream);
// Sets `batch` n x n matrices to the identity.
cudaError_t set_identity(float* Q, int n, int batch, cudaStream_t stream);

}  // namespace soap
