// Dispatch of the batched fp32-accurate GEMM used by every contraction of the step.
#include "profile.h"
#include "soap_internal.h"

namespace soap {

cudaError_t gemm(bool ta, bool tb, int M, int N, int K, float alpha, Operand A, Operand B, float beta,
                 MutOperand C, int batch, cudaStream_t s) {
  const double flops = 2.0 * M * N * (double)K * batch;
  const double bytes = 4.0 * batch * ((double)M * K + (double)K * N + (double)M * N * (beta != 0.f ? 2 : 1));
  ProfScope prof(kFamGemmSimt, flops, bytes, s);
  return gemm_simt(ta, tb, M, N, K, alpha, A, B, beta, C, batch, s);
}

}  // namespace soap
