// Elementwise parts of the Muon step (Alg. Muon; HBM-bound, grid-stride, float4 where aligned):
//
//  * muon_momentum: M <- beta1 M + (1 - beta1) G and the squared Frobenius norm of every M
//    (block partial sums in double, added atomically per matrix).
//  * muon_init_x: X_0 = M / max(||M||_F, eps) rounded to bf16, written in both orientations
//    (X for the A = X X^T products, X^T as the K-major operand of B X), through 32 x 32
//    shared-memory tiles; a tall matrix (rows > cols) is stored as its transpose.
//  * muon_update: W <- (1 - lr wd) W - lr sqrt(max(rows, cols)) X_n.
#include <algorithm>

#include "profile.h"
#include "soap_internal.h"

namespace soap {
namespace {

constexpr int kThreads = 256;

inline int blocks_for(int64_t elems, int batch) {
  int64_t want = (elems / 4 + kThreads - 1) / kThreads;
  if (want < 1) want = 1;
  const int64_t cap = std::max<int64_t>(4, (8 * 152) / std::max(1, batch));
  return (int)(want < cap ? want : cap);
}

__global__ void muon_momentum_kernel(const float* const* grads, float* M, double* norm2, int64_t elems, float beta1,
                                     int* status) {
  const int b = blockIdx.y;
  const float* g = grads[b];
  float* m = M + (int64_t)b * elems;
  const float c1 = 1.f - beta1;
  double acc = 0.0;
  int bad = 0;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const bool vec = ((reinterpret_cast<uintptr_t>(g) | reinterpret_cast<uintptr_t>(m)) & 15) == 0;
  int64_t tail = 0;
  if (vec) {
    const int64_t n4 = elems / 4;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += stride) {
      const float4 x = reinterpret_cast<const float4*>(g)[i];
      float4 v = reinterpret_cast<float4*>(m)[i];
      bad |= !isfinite(x.x) | !isfinite(x.y) | !isfinite(x.z) | !isfinite(x.w);
      v.x = fmaf(beta1, v.x, c1 * x.x);
      v.y = fmaf(beta1, v.y, c1 * x.y);
      v.z = fmaf(beta1, v.z, c1 * x.z);
      v.w = fmaf(beta1, v.w, c1 * x.w);
      reinterpret_cast<float4*>(m)[i] = v;
      acc += (double)v.x * v.x + (double)v.y * v.y + (double)v.z * v.z + (double)v.w * v.w;
    }
    tail = n4 * 4;
  }
  for (int64_t i = tail + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < elems; i += stride) {
    const float x = g[i];
    bad |= !isfinite(x);
    const float v = fmaf(beta1, m[i], c1 * x);
    m[i] = v;
    acc += (double)v * v;
  }
  __shared__ double red[kThreads];
  red[threadIdx.x] = acc;
  __syncthreads();
  for (int o = kThreads / 2; o > 0; o >>= 1) {
    if ((int)threadIdx.x < o) red[threadIdx.x] += red[threadIdx.x + o];
    __syncthreads();
  }
  if (threadIdx.x == 0) atomicAdd(norm2 + b, red[0]);
  if (__syncthreads_or(bad) && threadIdx.x == 0) atomicOr(status, kStatusNonFinite);
}

// One 32 x 32 tile of M (rows x cols) per block: scaled, rounded to bf16, and written to the
// row-major M-orientation buffer and to its transpose. P (rows x cols) and Pt (cols x rows).
__global__ void muon_init_x_kernel(const float* M, const double* norm2, float eps, __nv_bfloat16* P,
                                   __nv_bfloat16* Pt, int rows, int cols) {
  const int b = blockIdx.z;
  const float inv = 1.f / fmaxf((float)sqrt(norm2[b]), eps);
  const int64_t mn = (int64_t)rows * cols;
  const float* m = M + (int64_t)b * mn;
  __nv_bfloat16* p = P + (int64_t)b * mn;
  __nv_bfloat16* pt = Pt + (int64_t)b * mn;
  __shared__ __nv_bfloat16 tile[32][33];
  const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
  for (int rr = threadIdx.y; rr < 32; rr += blockDim.y) {
    const int r = r0 + rr, c = c0 + threadIdx.x;
    if (r < rows && c < cols) {
      const __nv_bfloat16 v = __float2bfloat16_rn(m[(int64_t)r * cols + c] * inv);
      p[(int64_t)r * cols + c] = v;
      tile[rr][threadIdx.x] = v;
    }
  }
  __syncthreads();
  for (int cc = threadIdx.y; cc < 32; cc += blockDim.y) {
    const int c = c0 + cc, r = r0 + threadIdx.x;
    if (r < rows && c < cols) pt[(int64_t)c * rows + r] = tile[threadIdx.x][cc];
  }
}

__global__ void muon_update_kernel(float* const* params, const __nv_bfloat16* O, int64_t elems, float keep,
                                   float step) {
  const int b = blockIdx.y;
  float* w = params[b];
  const __nv_bfloat16* o = O + (int64_t)b * elems;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const bool vec = (reinterpret_cast<uintptr_t>(w) & 15) == 0 && (reinterpret_cast<uintptr_t>(o) & 7) == 0;
  int64_t tail = 0;
  if (vec) {
    const int64_t n4 = elems / 4;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += stride) {
      float4 x = reinterpret_cast<float4*>(w)[i];
      const uint2 raw = reinterpret_cast<const uint2*>(o)[i];
      const float2 lo = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&raw.x));
      const float2 hi = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&raw.y));
      x.x = fmaf(keep, x.x, -step * lo.x);
      x.y = fmaf(keep, x.y, -step * lo.y);
      x.z = fmaf(keep, x.z, -step * hi.x);
      x.w = fmaf(keep, x.w, -step * hi.y);
      reinterpret_cast<float4*>(w)[i] = x;
    }
    tail = n4 * 4;
  }
  for (int64_t i = tail + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < elems; i += stride)
    w[i] = fmaf(keep, w[i], -step * __bfloat162float(o[i]));
}

}  // namespace

cudaError_t muon_momentum(const float* const* grads, float* M, double* norm2, int64_t elems, int batch, float beta1,
                          int* status, cudaStream_t s) {
  if (elems <= 0 || batch <= 0) return cudaSuccess;
  if (batch > 65535) return cudaErrorInvalidValue;
  ProfScope prof(kFamElementwise, 5.0 * elems * batch, 12.0 * elems * batch, s);
  muon_momentum_kernel<<<dim3(blocks_for(elems, batch), batch), kThreads, 0, s>>>(grads, M, norm2, elems, beta1,
                                                                                  status);
  return cudaGetLastError();
}

cudaError_t muon_init_x(const float* M, const double* norm2, float eps, __nv_bfloat16* X, __nv_bfloat16* Xt, int rows,
                        int cols, int batch, bool transposed, cudaStream_t s) {
  if (rows <= 0 || cols <= 0 || batch <= 0) return cudaSuccess;
  if (batch > 65535 || (rows + 31) / 32 > 65535) return cudaErrorInvalidValue;
  const double e = (double)rows * cols * batch;
  ProfScope prof(kFamElementwise, e, 8.0 * e, s);
  dim3 grid((cols + 31) / 32, (rows + 31) / 32, batch);
  // in M's orientation the first buffer is M-shaped; a transposed class keeps X = M^T
  muon_init_x_kernel<<<grid, dim3(32, 8), 0, s>>>(M, norm2, eps, transposed ? Xt : X, transposed ? X : Xt, rows, cols);
  return cudaGetLastError();
}

cudaError_t muon_update(float* const* params, const __nv_bfloat16* O, int64_t elems, int batch, float lr, float wd,
                        float scale, cudaStream_t s) {
  if (elems <= 0 || batch <= 0) return cudaSuccess;
  if (batch > 65535) return cudaErrorInvalidValue;
  ProfScope prof(kFamElementwise, 3.0 * elems * batch, 10.0 * elems * batch, s);
  muon_update_kernel<<<dim3(blocks_for(elems, batch), batch), kThreads, 0, s>>>(params, O, elems, 1.f - lr * wd,
                                                                                lr * scale);
  return cudaGetLastError();
}

}  // namespace soap
