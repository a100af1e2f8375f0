/*
 * libsoap -- the SOAP optimizer step (arXiv 2607.20548, Alg. 1 "KL-SOAP used in
 * experiments", with the standard Shampoo factor EMAs of section 2) batched over
 * every weight matrix of a model, on one NVIDIA GB300 (sm_103a).
 *
 * Conventions shared by every entry point
 *   - Matrices are fp32, row-major, contiguous: element (i, j) of a rows x cols
 *     matrix sits at i * cols + j. Orientation follows Alg. 1's state list:
 *     W, G, m, v are rows x cols ("in x out"); L, Q_L are rows x rows; R, Q_R are
 *     cols x cols.
 *   - Device pointers must be 16-byte aligned and must not alias each other.
 *   - A preconditioned side must be a multiple of 4 long and at most 8192 (the tensor-core
 *     products read rows with TMA); identity sides have no such limit.
 *   - Every call that takes a stream only enqueues work on it (no host
 *     synchronisation) unless its comment says otherwise. Streams are
 *     cudaStream_t values passed as soap_stream_t; 0 is the legacy default stream.
 *   - The library owns all optimizer state and workspace; the caller owns params,
 *     grads, the stream, and any buffer it passes in.
 *   - Host-side validation failures return immediately with an error code and
 *     leave the state untouched. Conditions found on the device (non-finite
 *     values, a QR breakdown, a bounded wait that ran out) set a sticky status
 *     word that soap_status() reads and that the next soap_step() returns. No
 *     kernel traps.
 */
#ifndef SOAP_H_
#define SOAP_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* soap_stream_t; /* identical to cudaStream_t */
typedef struct soap_s* soap_handle;        /* opaque, owned by the library */

typedef enum {
  SOAP_OK = 0,
  SOAP_ERR_INVALID_ARG = 1, /* bad shape, index, pointer alignment or null pointer */
  SOAP_ERR_CUDA = 2,        /* a CUDA runtime call failed; see soap_last_error */
  SOAP_ERR_OOM = 3,         /* device memory for state or workspace not available */
  SOAP_ERR_NONFINITE = 4,   /* NaN or Inf seen in a gradient or in the state */
  SOAP_ERR_QR_BREAKDOWN = 5,/* a QR pivot norm was not finite */
  SOAP_ERR_TIMEOUT = 6      /* a bounded device-side wait gave up */
} soap_status_t;

/* One weight matrix. precond_left = 0 keeps Q_L = I fixed and stores no L (an
 * "identity side"); likewise precond_right for Q_R and R. */
typedef struct {
  int64_t rows, cols;
  int32_t precond_left, precond_right;
} soap_shape;

/* Hyper-parameters of Alg. 1 and its table.
 *   lr, weight_decay: eta_t and lambda_t of the update W <- (1 - eta lambda) W - eta dW
 *   beta1, beta2:     first/second-moment EMA coefficients in the rotated basis
 *   factor_beta:      Kronecker-factor EMA coefficient b in L <- b L + (1-b) G G^T
 *                     (every EMA weights the OLD state by its coefficient)
 *   eps:              added outside the square root, N = m / (sqrt(v) + eps)
 *   eig_every:        F; the basis is refreshed when t mod F == 0 (the paper uses 1)
 *   bias_correction:  0 = literal Alg. 1 (none); 1 = divide m, v by (1 - beta^t)
 *   qr_tol:           a Householder column whose remaining norm is <= qr_tol*||P||_F
 *                     is treated as exactly zero (no reflector, R_kk = 0, sign +1)
 *   guard:            1 = rows/cols of N that belong to such zero columns are 0
 *   kl:               0 = standard Shampoo factor EMAs (above); 1 = Alg. 1's KL-Shampoo form
 *                       L <- b L + (1-b)/cols * G Q_R diag(1/(lam_R + eps)) Q_R^T G^T
 *                       R <- b R + (1-b)/rows * G^T Q_L diag(1/(lam_L + eps)) Q_L^T G
 *                     with lam = diag(Q^T F Q) from the factor and basis held before the
 *                     step (a negative lam, which only rounding produces, counts as 0); an
 *                     identity side counts as Q = I, lam = 1. Requires eps > 0.
 *   stale:            0 = the refresh sees the current gradient (section 5's real-time
 *                     update); 1 = the stale variant section 5 diagnoses: the refresh uses the
 *                     factors of the earlier steps and G enters them after the step's update.
 *                     Requires kl = 0 and guard = 0 (the factors' zero QR columns are then not
 *                     null directions of the current gradient). */
typedef struct {
  float lr, beta1, beta2, factor_beta, eps, weight_decay;
  int32_t eig_every;
  int32_t bias_correction;
  float qr_tol;
  int32_t guard;
  int32_t kl;
  int32_t stale;
} soap_hparams;

/* Fills *hp with the defaults used for the paper's workloads: lr 3e-3,
 * beta1 = beta2 = factor_beta = 0.95, eps 1e-8, weight_decay 0.1, F = 1, no bias
 * correction, qr_tol 2e-5, guard on, standard factor EMAs (kl 0) with the current gradient
 * (stale 0). */
void soap_default_hparams(soap_hparams* hp);

/* Creates the optimizer for n matrices on CUDA device `device` and allocates all
 * state (Alg. 1 "Optimizer States") and workspace up front: L = R = 0, Q = I,
 * m = v = 0, t = 0. shapes[] is copied. Returns SOAP_ERR_OOM if the state does
 * not fit; *out is then NULL; SOAP_ERR_INVALID_ARG for kl = 1 with eps <= 0 (the first
 * KL step weighs by 1/eps) and for stale = 1 with kl or guard set. The device becomes
 * current for the calling thread. Handles on different devices may coexist in one process
 * (each kernel's launch attributes are set once per device); the usual layout is one process
 * per GPU. */
soap_status_t soap_create(const soap_shape* shapes, int32_t n, const soap_hparams* hp,
                          int32_t device, soap_handle* out);

/* soap_create with a bound on the workspace. Besides the optimizer state proper (per matrix
 * M_hat and v, the factors L and R stored as their lower-triangular 32 x 32 tiles, the bases
 * Q_L and Q_R), a step needs a workspace for the operands it forms (the gradient copy and its
 * transpose, tf32 lo parts, Q^T, the unpacked factors, the QR's buffers, the rotation
 * intermediates). Matrices are stepped in waves: runs of matrices whose workspace fits side by
 * side, the next wave reusing it. workspace_limit = 0 (what soap_create does) takes one wave
 * holding every matrix if that leaves 1 GiB + 1% of the device's memory free, else waves cut
 * to the memory free at that moment less that reserve; workspace_limit > 0 caps the workspace
 * at that many bytes (and at the free memory less the reserve). Returns SOAP_ERR_OOM if the
 * state does not fit, or if one matrix of some shape needs more workspace than allowed. */
soap_status_t soap_create_ex(const soap_shape* shapes, int32_t n, const soap_hparams* hp, int32_t device,
                             size_t workspace_limit, soap_handle* out);

/* The plan soap_create chose: number of waves per step; whether they are pipelined (1: the
 * workspace holds two waves, each in its half, so that one wave's preparation and factor
 * update run while the previous wave's QR does; 0: waves run one after another); workspace
 * bytes and state bytes (device memory held by the handle is their sum). Any pointer may be
 * NULL. */
soap_status_t soap_plan_info(soap_handle h, int32_t* waves, int32_t* pipelined, size_t* workspace_bytes,
                             size_t* state_bytes);

/* One SOAP step (Alg. 1) over all n matrices, enqueued on `stream`:
 * factor EMAs with the current gradient, power step P = L Q and QR refresh with
 * diag(R) >= 0, first-moment re-projection, rotation G' = Q_L^T G Q_R, Adam in the
 * rotated basis, back-rotation dW = Q_L N Q_R^T and W <- (1 - eta lambda) W - eta dW.
 * params[i] / grads[i]: device pointers to matrix i (rows_i x cols_i, fp32); params
 * are updated in place, grads are only read. Both pointer arrays are host arrays
 * and are copied before the call returns (a changed table is written to the device by the
 * launches themselves; nothing on the host waits for the GPU). Steps, and state reads and
 * writes, share the handle's workspace: each is ordered after the one enqueued before it,
 * whatever stream either came on. Returns a pending sticky device status from an earlier
 * step, if any, before enqueuing anything. */
soap_status_t soap_step(soap_handle h, float* const* params, const float* const* grads,
                        soap_stream_t stream);

/* Sets eta_t and lambda_t for the following steps (Alg. 1 takes them per step). */
soap_status_t soap_set_lr(soap_handle h, float lr, float weight_decay);

/* Which piece of a matrix's state soap_state_get/set move. */
typedef enum {
  SOAP_STATE_M = 0,     /* first moment m in the current eigenbasis (rows x cols) */
  SOAP_STATE_V = 1,     /* second moment v in the current eigenbasis (rows x cols) */
  SOAP_STATE_L = 2,     /* left factor L (rows x rows) */
  SOAP_STATE_QL = 3,    /* left eigenbasis Q_L (rows x rows) */
  SOAP_STATE_R = 4,     /* right factor R (cols x cols) */
  SOAP_STATE_QR = 5,    /* right eigenbasis Q_R (cols x cols) */
  SOAP_STATE_MHAT = 6,  /* first moment in the original basis, Q_L m Q_R^T (rows x cols);
                           the library's own storage, bit-exact for checkpoints */
  SOAP_STATE_SKIP_L = 7,/* uint8 per row: 1 where Q_L's column came from a zero QR column */
  SOAP_STATE_SKIP_R = 8,/* uint8 per col: same for Q_R */
  SOAP_STATE_LAMBDA_L = 9, /* fp32 per row: lam_L = diag(Q_L^T L Q_L) as the last KL step
                              computed it (before the clamp at 0); read-only, present only
                              with kl = 1 on a matrix preconditioned on both sides */
  SOAP_STATE_LAMBDA_R = 10 /* fp32 per col: lam_R likewise */
} soap_state_which;

/* Number of bytes soap_state_get/set move for (idx, which); 0 if that piece does not
 * exist (an identity side) or the arguments are invalid. */
size_t soap_state_bytes(soap_handle h, int32_t idx, int32_t which);

/* Copies one piece of matrix idx's state to dst (host or device memory; the copy is
 * ordered on `stream`; a host dst is complete when the stream is). SOAP_STATE_M is
 * computed on the fly as Q_L^T M_hat Q_R (fp32 GEMMs), so it is not bit-exact with
 * what a later soap_state_set(SOAP_STATE_M) stores; use SOAP_STATE_MHAT to
 * checkpoint. Returns SOAP_ERR_INVALID_ARG for an identity side's L/Q/R. */
soap_status_t soap_state_get(soap_handle h, int32_t idx, int32_t which, void* dst,
                             soap_stream_t stream);

/* Copies src (host or device) into one piece of matrix idx's state, ordered on
 * `stream`. Setting SOAP_STATE_M stores Q_L m Q_R^T with the Q_L, Q_R held at that
 * moment, so set Q_L and Q_R first. SOAP_STATE_LAMBDA_L/R are read-only (each KL step
 * recomputes them): setting one returns SOAP_ERR_INVALID_ARG. */
soap_status_t soap_state_set(soap_handle h, int32_t idx, int32_t which, const void* src,
                             soap_stream_t stream);

/* Step counter t (number of completed soap_step calls, or the value last set). */
int64_t soap_get_step(soap_handle h);
soap_status_t soap_set_step(soap_handle h, int64_t t);

/* Synchronises `stream`, then returns the sticky device status (SOAP_OK if clean). */
soap_status_t soap_status(soap_handle h, soap_stream_t stream);

/* Clears the sticky device status (ordered on `stream`). */
soap_status_t soap_clear_status(soap_handle h, soap_stream_t stream);

/* Human-readable text of the last error on this handle (never NULL). */
const char* soap_last_error(soap_handle h);

/* Frees all state and workspace. Safe on NULL. Synchronises the device first. */
void soap_destroy(soap_handle h);

/* ---- kernel timing (diagnostics; the paper has no counterpart) ---------------------- */

/* Kernel families the library launches. */
typedef enum {
  SOAP_KERNEL_GEMM_SIMT = 0,   /* CUDA-core fp32 batched GEMM */
  SOAP_KERNEL_GEMM_TC = 1,     /* tcgen05 batched GEMM: fp32-accurate (four TF32 products), or bf16 (Muon) */
  SOAP_KERNEL_QR_PANEL = 2,    /* cluster panel factorisation of the QR */
  SOAP_KERNEL_ELEMENTWISE = 3, /* momentum, Adam, weight update */
  SOAP_KERNEL_OTHER = 4,       /* norms, identity fills */
  SOAP_KERNEL_QR_UPDATE = 5    /* tensor-core products of the QR's block updates */
} soap_kernel_family;

typedef struct {
  int32_t family;    /* soap_kernel_family */
  int64_t launches;  /* kernel launches timed */
  double ms;         /* sum of per-launch CUDA-event durations */
  double flops;      /* sum of algorithmic FLOPs of those launches */
  double bytes;      /* sum of algorithmic bytes moved by those launches */
} soap_kernel_stats;

/* Starts timing every kernel launch the calling thread makes through the library
 * (up to max_launches; later launches are counted as overflow and not timed). Each
 * launch is bracketed by two CUDA events on its own stream. */
soap_status_t soap_profile_begin(soap_handle h, int64_t max_launches);

/* soap_profile_begin with flags. SOAP_PROFILE_SERIAL makes every timed launch wait for the
 * device to be idle before it starts (a host-side device synchronisation), so that each
 * launch runs alone and its time measures the kernel in isolation rather than beside the
 * library's concurrent streams; a step timed this way runs slower as a whole. */
#define SOAP_PROFILE_SERIAL 1
soap_status_t soap_profile_begin_ex(soap_handle h, int64_t max_launches, int32_t flags);

/* Synchronises `stream`, stops timing and writes one soap_kernel_stats per family
 * (6 entries) to out[]. *overflow is set to 1 if max_launches was exceeded. */
soap_status_t soap_profile_end(soap_handle h, soap_stream_t stream, soap_kernel_stats* out,
                               int32_t* overflow);

/* One timed launch: its family, its start and end, in ms after the first timed launch
 * started (CUDA events on the launch's stream), and the algorithmic FLOPs and bytes it was
 * tagged with (the same figures soap_profile_end sums per family). */
typedef struct {
  int32_t family;   /* soap_kernel_family */
  double start_ms;
  double end_ms;
  double flops;
  double bytes;
} soap_launch_record;

/* Synchronises the device and copies the launches timed since soap_profile_begin, in launch
 * order, to out[] (at most max of them; *count receives how many were written). Call it
 * before soap_profile_end, which discards them. The library's QR streams run concurrently
 * with each other and with the caller's stream, so records may overlap in time. */
soap_status_t soap_profile_records(soap_handle h, soap_launch_record* out, int64_t max, int64_t* count);

/* Failure detection (the paper has no counterpart). Every device-side wait of the tensor-core
 * products is bounded: after `limit_ns` nanoseconds (0: the default, 2 s) it gives up, the
 * kernel drains what it has in flight, frees its tensor memory and returns, and the status word
 * gets SOAP_STATUS_TIMEOUT (soap_status then returns SOAP_ERR_TIMEOUT). `hold`, if not NULL, is
 * a device int32 that every such product first waits for to become non-zero -- a flag that
 * nothing sets makes the waits run out, which is how the timeout path is tested without a
 * fault. Applies to launches enqueued after the call, from any thread; soap_wait_limit(0, NULL)
 * restores the defaults. Results of a product whose wait gave up are not valid. */
soap_status_t soap_wait_limit(uint64_t limit_ns, const int32_t* hold);

/* ---- stand-alone sub-steps (the same kernels soap_step runs) ------------------- */

/* Device status bits of the stand-alone sub-steps (the int32 words they take as `status`):
 * set by the kernels with an atomic OR, never cleared by them. */
#define SOAP_STATUS_NONFINITE 1     /* a non-finite value in the input */
#define SOAP_STATUS_QR_BREAKDOWN 2  /* a QR pivot norm was not finite */
#define SOAP_STATUS_TIMEOUT 4       /* a bounded device-side wait gave up (results invalid) */

/* S3, Alg. 1 "QR(L_t Q_L).Q": for `batch` square n x n matrices P (device,
 * contiguous, batch stride n*n), writes Q with P = Q R and diag(R) >= 0 (blocked
 * Householder QR, explicit Q) and skip[b*n + k] = 1 where column k was treated as
 * exactly zero (remaining norm <= tol * ||P_b||_F). P is read only. `workspace`
 * must hold soap_qr_workspace_bytes(n, batch) bytes of device memory (256-byte aligned).
 * status: NULL, or a device int32 (4-byte aligned) that the call sets to 0 on the stream and
 * into which its kernels OR SOAP_STATUS_QR_BREAKDOWN / SOAP_STATUS_TIMEOUT; read it once the
 * stream has passed the call (0 = Q is valid). */
size_t soap_qr_workspace_bytes(int32_t n, int32_t batch);
soap_status_t soap_qr(int32_t n, int32_t batch, const float* P, float* Q, uint8_t* skip,
                      float tol, void* workspace, size_t workspace_bytes, int32_t* status,
                      soap_stream_t stream);

/* soap_qr for callers that cannot give this library device memory. The paper has no
 * counterpart; it exists for callers that cannot allocate when they need a QR: a
 * cudaMalloc or cudaFree may wait until the whole device is idle, and some programs do
 * not own their device memory at all (a framework's caching pool, or a fixed budget
 * handed out at start-up, owns it). Same arguments and results as soap_qr, without the
 * workspace: it uses a 32 MiB array compiled into libsoap.so, which every GPU that
 * loads the library keeps until the process exits. That is room for one 1024 x 1024
 * matrix or, e.g., three of 512 x 512; a (n, batch) whose soap_qr_workspace_bytes()
 * exceeds 32 MiB - 256 B is refused with SOAP_ERR_INVALID_ARG before anything is
 * enqueued. It never calls cudaMalloc, cudaFree or any allocating routine.
 * status: as for soap_qr (NULL: the word is kept inside the array, where no one reads it).
 * The first call on each device looks up the array's device address with that device
 * current (cudaGetSymbolAddress); make that first call before any stream capture. All
 * calls in the process share the one array per device and it keeps the last call's
 * contents, so two calls that can overlap on the GPU (different streams without
 * ordering between them) race: order them, e.g. on one stream. */
soap_status_t soap_qr_static(int32_t n, int32_t batch, const float* P, float* Q, uint8_t* skip,
                             float tol, int32_t* status, soap_stream_t stream);

/* The fp32-accurate batched product used by every contraction of the step (S1, S2,
 * S4, S5, S7 and the QR updates): for b < batch,
 *   C_b = alpha * op(A_b) * op(B_b) + beta * C_b,
 * op(X) = X or X^T (trans_x != 0), op(A_b) is M x K, op(B_b) is K x N, all
 * row-major with leading dimensions lda/ldb/ldc and batch strides in elements.
 * beta == 0 does not read C. */
soap_status_t soap_gemm(int32_t trans_a, int32_t trans_b, int32_t M, int32_t N, int32_t K,
                        float alpha, const float* A, int64_t lda, int64_t stride_a,
                        const float* B, int64_t ldb, int64_t stride_b, float beta, float* C,
                        int64_t ldc, int64_t stride_c, int32_t batch, soap_stream_t stream);

/* The tensor-core form of that product (tcgen05, four TF32 products): for b < batch,
 *   C_b = alpha * A_b * B_(b mod b_batch)^T + beta * C_b        (or C_b^T if transpose_c)
 * with A_b (M x K) and B (N x K) row-major, each given as hi and lo, where hi is x with its
 * 13 low mantissa bits cleared (the tf32 value the tensor core reads from an fp32 word, so
 * hi may be x itself) and lo is x - hi rounded to the nearest tf32 (see soap_split_tf32);
 * the accumulator adds a_lo b_lo + a_lo b_hi + a_hi b_lo + a_hi b_hi in fp32, each 32-wide
 * K block summed afresh and added in fp32 registers (fp32-level accuracy at any K).
 * lda, ldb, ldc and every batch stride must be multiples of 4 elements and every
 * pointer 16-byte aligned. C_lo, if non-NULL, receives out - tf32(out) in C's layout
 * (leading dimension ldc). status, if non-NULL, is a device int32 into which the kernel ORs
 * SOAP_STATUS_TIMEOUT if a bounded internal wait gave up (it is not cleared). */
soap_status_t soap_gemm_tf32x4(int32_t M, int32_t N, int32_t K, int32_t batch, const float* A_hi,
                               const float* A_lo, int64_t lda, int64_t stride_a, const float* B_hi,
                               const float* B_lo, int64_t ldb, int64_t stride_b, int32_t b_batch,
                               float alpha, float beta, float* C, int64_t ldc, int64_t stride_c,
                               int32_t transpose_c, float* C_lo, int32_t* status,
                               soap_stream_t stream);

/* hi = x with its 13 low mantissa bits cleared (tf32 by truncation), lo = x - hi (exact in
 * fp32) rounded to the nearest tf32, for n values on the device; hi may be NULL. */
soap_status_t soap_split_tf32(const float* x, float* hi, float* lo, int64_t n, soap_stream_t stream);

/* Layer-wise ownership for data-parallel ranks (section 6, "layer-wise distributed
 * optimizer"): every matrix is stepped by exactly one of `world` ranks, which then share the
 * updated weights with the others (an all-gather of variable-size pieces). Host-only; no
 * device is touched.
 *   policy 0: the paper's assignment -- matrices sorted by size (rows * cols, largest first,
 *             ties by index) and dealt round-robin to ranks 0, 1, ..., world-1, 0, ...
 *   policy 1: longest processing time first on this library's step cost -- the same order,
 *             each matrix to the rank with the smallest cost so far (ties: lowest rank), the
 *             cost of a matrix being the FLOPs of its SOAP step (S1 as a symmetric product,
 *             the power step, the QR, the rotations), identity sides dropped
 * owner[i] receives matrix i's rank; load[r] (may be NULL) receives rank r's summed cost
 * (FLOPs, under either policy). SOAP_ERR_INVALID_ARG for n < 1, world < 1, a null shapes or
 * owner, an unknown policy or a non-positive side. */
soap_status_t soap_layerwise_assign(const soap_shape* shapes, int32_t n, int32_t world, int32_t policy,
                                    int32_t* owner, double* load);

#ifdef __cplusplus
}
#endif
#endif /* SOAP_H_ */
