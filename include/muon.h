/*
 * libsoap's Muon entry points -- the paper's Alg. "Muon" (momentum orthogonalized by
 * Newton-Schulz, with decoupled weight decay) batched over every weight matrix of a model,
 * on one NVIDIA GB300 (sm_103a), in the same library as the SOAP step (include/soap.h).
 *
 * Per matrix W (rows x cols, "in x out") with gradient G, step t:
 *   M <- beta1 M + (1 - beta1) G                      momentum EMA (fp32)
 *   X_0 = M / max(||M||_F, eps)                        normalised momentum
 *   X_i = a_i X + (b_i A + c_i A^2) X,  A = X X^T       Newton-Schulz, i = 1..n, in bf16 (bf16
 *                                                      operands, fp32 accumulation, bf16
 *                                                      results), as the paper's iterations run
 *   W <- (1 - lr wd) W - lr sqrt(max(rows, cols)) X_n  update RMS matching and weight decay
 * A matrix with rows > cols is orthogonalized as its transpose (X^T X in place of X X^T gives
 * the same X_n for these odd polynomial steps), so every A is min(rows, cols) square.
 *
 * Conventions: those of include/soap.h (fp32 row-major contiguous matrices, 16-byte aligned
 * device pointers, stream-ordered calls, a sticky device status word, no kernel traps), and
 * the same status codes. rows and cols must be multiples of 8 (the bf16 operands are read
 * with TMA in 16-byte rows).
 */
#ifndef MUON_H_
#define MUON_H_

#include <stddef.h>
#include <stdint.h>

#include "soap.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef struct muon_s* muon_handle; /* opaque, owned by the library */

/* Hyper-parameters of Alg. Muon and its table.
 *   lr, weight_decay: eta_t and lambda_t
 *   beta1:            momentum EMA coefficient (weights the old momentum)
 *   eps:              lower bound of the Frobenius norm in the normalisation
 *   ns_steps:         n, the number of Newton-Schulz iterations (1 .. 64)
 *   coeffs:           host array of 3 * ns_steps floats (a_1, b_1, c_1, a_2, ...), copied by
 *                     muon_create; NULL selects the quintic Newton-Schulz polynomial
 *                     (15 - 10 x + 3 x^2) / 8 of X^T X for every step, which converges to
 *                     the polar factor from ||X_0||_2 <= 1. */
typedef struct {
  float lr, beta1, weight_decay, eps;
  int32_t ns_steps;
  const float* coeffs;
} muon_hparams;

/* Fills *hp with the table's values: lr 3e-3, beta1 0.9, weight_decay 0.1, eps 1e-7,
 * ns_steps 16, coeffs NULL. */
void muon_default_hparams(muon_hparams* hp);

/* Creates the optimizer for n matrices (shapes[i].rows x shapes[i].cols; the precond_* flags
 * are ignored) on CUDA device `device`; allocates the momentum (zero) and the bf16 workspace.
 * SOAP_ERR_INVALID_ARG for a side that is not a positive multiple of 8 or for ns_steps
 * outside 1 .. 64; SOAP_ERR_OOM if the state does not fit (*out is then NULL). */
soap_status_t muon_create(const soap_shape* shapes, int32_t n, const muon_hparams* hp, int32_t device,
                          muon_handle* out);

/* One Muon step over all n matrices, enqueued on `stream`; params[i] / grads[i] are device
 * pointers (host pointer arrays, copied before return). Returns a pending sticky device
 * status from an earlier step, if any, before enqueuing anything. */
soap_status_t muon_step(muon_handle h, float* const* params, const float* const* grads, soap_stream_t stream);

/* Sets eta_t and lambda_t for the following steps. */
soap_status_t muon_set_lr(muon_handle h, float lr, float weight_decay);

/* Copies matrix idx's momentum M (rows x cols fp32) to dst / from src (host or device),
 * ordered on `stream`. */
soap_status_t muon_state_get(muon_handle h, int32_t idx, void* dst, soap_stream_t stream);
soap_status_t muon_state_set(muon_handle h, int32_t idx, const void* src, soap_stream_t stream);

/* Synchronises `stream` and returns the sticky device status (SOAP_OK if none). */
soap_status_t muon_status(muon_handle h, soap_stream_t stream);

/* Per-launch kernel timing, as soap_profile_begin / soap_profile_end (include/soap.h) for this
 * handle: the bf16 tensor-core products count as SOAP_KERNEL_GEMM_TC, the momentum, the
 * normalisation and the update as SOAP_KERNEL_ELEMENTWISE. */
soap_status_t muon_profile_begin(muon_handle h, int64_t max_launches);
soap_status_t muon_profile_end(muon_handle h, soap_stream_t stream, soap_kernel_stats* out, int32_t* overflow);

/* Human-readable description of the last error on this handle ("" if none). */
const char* muon_last_error(muon_handle h);

/* Frees all device memory of the handle (synchronises the device first). */
void muon_destroy(muon_handle h);

#ifdef __cplusplus
}
#endif

#endif /* MUON_H_ */
