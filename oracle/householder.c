/*
 * Oracle QR for the SOAP eigenbasis refresh -- TEST INFRASTRUCTURE ONLY.
 *
 * Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline leg may load
 * this code. The CUDA path shares nothing with it.
 *
 * What it computes (KL-SOAP, Alg. 1, "Eigenbasis Re-computation" block, and the
 * appendix "SOAP Eigenbasis Update Frequency"): the orthogonal factor Q of the QR
 * decomposition P = Q R of a square matrix P = L_t Q_old, with the sign convention
 * diag(R) >= 0 so that Q is unique when P has full rank.
 *
 * Algorithm: plain unblocked Householder QR as in Golub & Van Loan, "Matrix
 * Computations", 4th ed., Alg. 5.2.1, with the LAPACK reflector convention
 * (beta = -sign(alpha) * ||x||, v(1) = 1, tau = (beta - alpha) / beta), followed by
 * backward accumulation of Q = H_1 H_2 ... H_n (Golub & Van Loan section 5.1.6), and
 * finally the sign fix: column k of Q is negated wherever R_kk < 0.
 *
 * Reading for rank-deficient P (the paper is silent): in exact arithmetic a
 * Householder step whose sub-column x is zero uses no reflector (H_k = I, R_kk = 0).
 * In finite precision x is rounding noise instead of zero, so a column is treated
 * as exactly zero when ||x||_2 <= tol * ||P||_F. Such a column is reported in
 * skipped[k] = 1, keeps sign +1, and Q's column k becomes H_1 ... H_{k-1} e_k.
 * tol <= 0 keeps only the exact-arithmetic rule (skip when ||x|| == 0).
 *
 * Row-major storage, element (i, j) at i * n + j. Work is O(n^3) with no blocking;
 * OpenMP splits each rank-1 update over column ranges only.
 */
#include <math.h>
#include <stdlib.h>
#include <string.h>

#define DEFINE_HOUSEHOLDER_Q(T, NAME, SQRT)                                          \
  int NAME(int n, const T* P, T* Q, unsigned char* skipped, T* rdiag, double tol) {  \
    if (n <= 0) return 0;                                                           \
    size_t nn = (size_t)n * (size_t)n;                                               \
    T* A = (T*)malloc(nn * sizeof(T));                                               \
    T* V = (T*)malloc(nn * sizeof(T));  /* row k holds reflector k (entries k..n-1) */ \
    T* tau = (T*)malloc((size_t)n * sizeof(T));                                      \
    if (!A || !V || !tau) { free(A); free(V); free(tau); return -1; }                \
    memcpy(A, P, nn * sizeof(T));                                                    \
    /* ||P||_F, the scale for the rank-deficiency reading */                       \
    T pn2 = 0;                                                                       \
    for (size_t e = 0; e < nn; ++e) pn2 += A[e] * A[e];                              \
    T thresh = (T)(tol > 0 ? tol : 0) * SQRT(pn2);                                   \
    for (int k = 0; k < n; ++k) {                                                    \
      /* x = A(k:n, k) */                                                            \
      T alpha = A[(size_t)k * n + k];                                                \
      T sigma = 0;                                                                   \
      for (int i = k + 1; i < n; ++i) sigma += A[(size_t)i * n + k] * A[(size_t)i * n + k]; \
      T xnorm = SQRT(alpha * alpha + sigma);                                         \
      T* v = V + (size_t)k * n;                                                      \
      if (xnorm == 0 || xnorm <= thresh) {                                           \
        /* zero sub-column: H_k = I, R_kk = 0 */                                     \
        tau[k] = 0;                                                                  \
        skipped[k] = 1;                                                              \
        rdiag[k] = 0;                                                                \
        for (int i = k; i < n; ++i) v[i] = 0;                                        \
        v[k] = 1;                                                                    \
        continue;                                                                    \
      }                                                                              \
      skipped[k] = 0;                                                                \
      T beta = alpha >= 0 ? -xnorm : xnorm; /* beta = -sign(alpha) ||x|| */         \
      T v0 = alpha - beta;                  /* no cancellation: same sign as alpha */\
      tau[k] = (beta - alpha) / beta;                                                \
      v[k] = 1;                                                                      \
      for (int i = k + 1; i < n; ++i) v[i] = A[(size_t)i * n + k] / v0;              \
      A[(size_t)k * n + k] = beta;                                                   \
      for (int i = k + 1; i < n; ++i) A[(size_t)i * n + k] = 0;                      \
      rdiag[k] = beta;                                                               \
      /* A(k:n, k+1:n) <- (I - tau v v^T) A(k:n, k+1:n) */                           \
      T tk = tau[k];                                                                 \
      _Pragma("omp parallel for schedule(static) if (n - k > 512)")                   \
      for (int jb = k + 1; jb < n; jb += 64) {                                       \
        int je = jb + 64 < n ? jb + 64 : n;                                          \
        T acc[64];                                                                   \
        for (int j = jb; j < je; ++j) acc[j - jb] = 0;                               \
        for (int i = k; i < n; ++i) {                                                \
          T vi = v[i];                                                               \
          const T* row = A + (size_t)i * n;                                          \
          for (int j = jb; j < je; ++j) acc[j - jb] += vi * row[j];                  \
        }                                                                            \
        for (int i = k; i < n; ++i) {                                                \
          T s = tk * v[i];                                                           \
          T* row = A + (size_t)i * n;                                                \
          for (int j = jb; j < je; ++j) row[j] -= s * acc[j - jb];                   \
        }                                                                            \
      }                                                                              \
    }                                                                                \
    /* Q = H_1 ... H_n I, accumulated backwards: Q(k:n, k:n) <- H_k Q(k:n, k:n) */   \
    memset(Q, 0, nn * sizeof(T));                                                    \
    for (int i = 0; i < n; ++i) Q[(size_t)i * n + i] = 1;                            \
    for (int k = n - 1; k >= 0; --k) {                                               \
      if (tau[k] == 0) continue;                                                     \
      const T* v = V + (size_t)k * n;                                                \
      T tk = tau[k];                                                                 \
      _Pragma("omp parallel for schedule(static) if (n - k > 512)")                   \
      for (int jb = k; jb < n; jb += 64) {                                           \
        int je = jb + 64 < n ? jb + 64 : n;                                          \
        T acc[64];                                                                   \
        for (int j = jb; j < je; ++j) acc[j - jb] = 0;                               \
        for (int i = k; i < n; ++i) {                                                \
          T vi = v[i];                                                               \
          const T* row = Q + (size_t)i * n;                                          \
          for (int j = jb; j < je; ++j) acc[j - jb] += vi * row[j];                  \
        }                                                                            \
        for (int i = k; i < n; ++i) {                                                \
          T s = tk * v[i];                                                           \
          T* row = Q + (size_t)i * n;                                                \
          for (int j = jb; j < je; ++j) row[j] -= s * acc[j - jb];                   \
        }                                                                            \
      }                                                                              \
    }                                                                                \
    /* sign convention diag(R) >= 0: negate column k of Q where R_kk < 0 */          \
    for (int k = 0; k < n; ++k) {                                                    \
      if (rdiag[k] < 0) {                                                            \
        for (int i = 0; i < n; ++i) Q[(size_t)i * n + k] = -Q[(size_t)i * n + k];    \
        rdiag[k] = -rdiag[k];                                                        \
      }                                                                              \
    }                                                                                \
    free(A); free(V); free(tau);                                                     \
    return 0;                                                                        \
  }

DEFINE_HOUSEHOLDER_Q(double, oracle_householder_q_f64, sqrt)
DEFINE_HOUSEHOLDER_Q(float, oracle_householder_q_f32, sqrtf)
