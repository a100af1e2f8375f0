// Batched fp32 GEMM on the CUDA cores: C_b = alpha * op(A_b) op(B_b) + beta * C_b.
//
// Exact fp32 FMAs, so it is the accuracy reference for the tensor-core path and
// the engine where the tcgen05 path does not apply: the whole step of a class with a
// side that is not a multiple of 4 (TMA copies 16-byte rows), and the basis changes
// of the first moment in soap_state_get/set.
//
// Tiling: BM x BN output tile per 256-thread CTA, BK = 8, each thread owns a
// (BM/16) x (BN/16) micro-tile at rows ty + 16 i and columns tx + 16 j, operands
// double-buffered through shared memory (k-major, padded to avoid bank conflicts).
#include "soap_internal.h"

namespace soap {
namespace {

constexpr int kBK = 8;
constexpr int kThreads = 256;

__device__ __forceinline__ const float* resolve(const Operand& o, int b) {
  return (o.ptrs ? o.ptrs[b] : o.base + (int64_t)b * o.stride) + o.offset;
}
__device__ __forceinline__ float* resolve(const MutOperand& o, int b) {
  return (o.ptrs ? o.ptrs[b] : o.base + (int64_t)b * o.stride) + o.offset;
}

template <bool TA, bool TB, int BM, int BN>
__global__ void __launch_bounds__(kThreads) gemm_simt_kernel(int M, int N, int K, float alpha,
                                                             Operand A, Operand B, float beta,
                                                             MutOperand C) {
  constexpr int TM = BM / 16, TN = BN / 16;
  constexpr int A_PER = BM * kBK / kThreads;
  constexpr int B_PER = BN * kBK / kThreads;
  __shared__ float As[2][kBK][BM + 4];
  __shared__ float Bs[2][kBK][BN + 4];

  const int b = blockIdx.z;
  const int m0 = blockIdx.y * BM, n0 = blockIdx.x * BN;
  const float* Ab = resolve(A, b);
  const float* Bb = resolve(B, b);
  float* Cb = resolve(C, b);
  const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;

  float ra[A_PER], rb[B_PER];
  // op(A) element (mm, kk): A stored M x K (row mm) or, transposed, K x M (row kk).
  // The fastest-varying index follows the stored row so global reads coalesce.
  auto a_coord = [](int e, int& mm, int& kk) {
    if (!TA) { mm = e / kBK; kk = e % kBK; } else { kk = e / BM; mm = e % BM; }
  };
  auto b_coord = [](int e, int& kk, int& nn) {
    if (!TB) { kk = e / BN; nn = e % BN; } else { nn = e / kBK; kk = e % kBK; }
  };
  auto load = [&](int k0) {
#pragma unroll
    for (int i = 0; i < A_PER; ++i) {
      int mm, kk;
      a_coord(tid + i * kThreads, mm, kk);
      const int gm = m0 + mm, gk = k0 + kk;
      float v = 0.f;
      if (gm < M && gk < K) v = TA ? Ab[(int64_t)gk * A.ld + gm] : Ab[(int64_t)gm * A.ld + gk];
      ra[i] = v;
    }
#pragma unroll
    for (int i = 0; i < B_PER; ++i) {
      int kk, nn;
      b_coord(tid + i * kThreads, kk, nn);
      const int gk = k0 + kk, gn = n0 + nn;
      float v = 0.f;
      if (gk < K && gn < N) v = TB ? Bb[(int64_t)gn * B.ld + gk] : Bb[(int64_t)gk * B.ld + gn];
      rb[i] = v;
    }
  };
  auto store = [&](int buf) {
#pragma unroll
    for (int i = 0; i < A_PER; ++i) {
      int mm, kk;
      a_coord(tid + i * kThreads, mm, kk);
      As[buf][kk][mm] = ra[i];
    }
#pragma unroll
    for (int i = 0; i < B_PER; ++i) {
      int kk, nn;
      b_coord(tid + i * kThreads, kk, nn);
      Bs[buf][kk][nn] = rb[i];
    }
  };

  float acc[TM][TN];
#pragma unroll
  for (int i = 0; i < TM; ++i)
#pragma unroll
    for (int j = 0; j < TN; ++j) acc[i][j] = 0.f;

  const int nk = (K + kBK - 1) / kBK;
  if (nk > 0) {
    load(0);
    store(0);
  }
  __syncthreads();
  for (int t = 0; t < nk; ++t) {
    const int cur = t & 1;
    if (t + 1 < nk) load((t + 1) * kBK);
#pragma unroll
    for (int kk = 0; kk < kBK; ++kk) {
      float a[TM], bv[TN];
#pragma unroll
      for (int i = 0; i < TM; ++i) a[i] = As[cur][kk][ty + 16 * i];
#pragma unroll
      for (int j = 0; j < TN; ++j) bv[j] = Bs[cur][kk][tx + 16 * j];
#pragma unroll
      for (int i = 0; i < TM; ++i)
#pragma unroll
        for (int j = 0; j < TN; ++j) acc[i][j] = fmaf(a[i], bv[j], acc[i][j]);
    }
    if (t + 1 < nk) store(cur ^ 1);
    __syncthreads();
  }

#pragma unroll
  for (int i = 0; i < TM; ++i) {
    const int gm = m0 + ty + 16 * i;
    if (gm >= M) continue;
#pragma unroll
    for (int j = 0; j < TN; ++j) {
      const int gn = n0 + tx + 16 * j;
      if (gn >= N) continue;
      float* c = Cb + (int64_t)gm * C.ld + gn;
      float v = alpha * acc[i][j];
      if (beta != 0.f) v = fmaf(beta, *c, v);
      *c = v;
    }
  }
}

template <int BM, int BN>
cudaError_t launch_tile(bool ta, bool tb, int M, int N, int K, float alpha, Operand A, Operand B,
                        float beta, MutOperand C, int batch, cudaStream_t s) {
  dim3 grid((N + BN - 1) / BN, (M + BM - 1) / BM, batch);
  if (!ta && !tb) gemm_simt_kernel<false, false, BM, BN><<<grid, kThreads, 0, s>>>(M, N, K, alpha, A, B, beta, C);
  else if (!ta && tb) gemm_simt_kernel<false, true, BM, BN><<<grid, kThreads, 0, s>>>(M, N, K, alpha, A, B, beta, C);
  else if (ta && !tb) gemm_simt_kernel<true, false, BM, BN><<<grid, kThreads, 0, s>>>(M, N, K, alpha, A, B, beta, C);
  else gemm_simt_kernel<true, true, BM, BN><<<grid, kThreads, 0, s>>>(M, N, K, alpha, A, B, beta, C);
  return cudaGetLastError();
}

}  // namespace

cudaError_t gemm_simt(bool ta, bool tb, int M, int N, int K, float alpha, Operand A, Operand B,
                      float beta, MutOperand C, int batch, cudaStream_t s) {
  if (M <= 0 || N <= 0 || batch <= 0) return cudaSuccess;
  const bool narrow_n = N <= 64;
  if (M <= 32) return narrow_n ? launch_tile<32, 64>(ta, tb, M, N, K, alpha, A, B, beta, C, batch, s)
                               : launch_tile<32, 128>(ta, tb, M, N, K, alpha, A, B, beta, C, batch, s);
  if (M <= 64) return narrow_n ? launch_tile<64, 64>(ta, tb, M, N, K, alpha, A, B, beta, C, batch, s)
                               : launch_tile<64, 128>(ta, tb, M, N, K, alpha, A, B, beta, C, batch, s);
  return narrow_n ? launch_tile<128, 64>(ta, tb, M, N, K, alpha, A, B, beta, C, batch, s)
                  : launch_tile<128, 128>(ta, tb, M, N, K, alpha, A, B, beta, C, batch, s);
}

}  // namespace soap
