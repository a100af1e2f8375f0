// Elementwise parts of the SOAP step (HBM-bound; grid-stride, float4 where aligned).
//
//  * momentum_and_copy: the first moment kept in the ORIGINAL basis,
//      M_hat <- beta1 M_hat + (1 - beta1) G,
//    which is Alg. 1's re-projection m <- Q_new^T (Q_old m Q_old^T) Q_new followed
//    by m <- beta1 m + (1 - beta1) Q_new^T G Q_new, written as M_hat = Q m Q^T
//    (exact for the square orthogonal Q of both sides). It also copies G into the
//    library's contiguous gradient arena and flags non-finite gradients.
//  * adam_in_basis: v <- beta2 v + (1 - beta2) G'^2 and N = m / (sqrt(v) + eps)
//    (Alg. 1 "Calculate Adam update"; v is never re-projected), with the zero-column
//    guard.
//  * weight_update: W <- (1 - lr wd) W - lr N for a matrix with no preconditioned
//    side (Alg. 1 "Weight decay and update" with Q_L = Q_R = I).
//  * diag_dot, scale_cols_split: the KL-Shampoo factor form's approximate eigenvalues
//    lam = diag(Q^T F Q) and the column weights sqrt(coef / (lam + eps)) applied to G Q
//    (Alg. 1 "Accumulate Kronecker Factors (KL-Shampoo)").
#include <algorithm>

#include "profile.h"
#include "soap_internal.h"

namespace soap {
namespace {

constexpr int kThreads = 256;

// The tensor core reads an fp32 word as tf32 by dropping its 13 low mantissa bits, so
// an fp32 array serves directly as the "hi" operand. Its lo part is x - trunc(x) (exact
// in fp32) rounded to the nearest tf32, so that the tensor core's own truncation of it
// is exact and hi + lo is x to within half a tf32 unit of lo, without bias.
__device__ __forceinline__ float tf32_trunc(float x) { return __uint_as_float(__float_as_uint(x) & 0xFFFFE000u); }
__device__ __forceinline__ float lo_part(float x) {
  uint32_t r;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x - tf32_trunc(x)));
  return __uint_as_float(r);
}

inline int blocks_for(int64_t elems, int batch) {
  int64_t want = (elems / 4 + kThreads - 1) / kThreads;
  if (want < 1) want = 1;
  // about 8 blocks of 256 threads per SM over the whole launch (152 SMs)
  const int64_t cap = std::max<int64_t>(4, (8 * 152) / std::max(1, batch));
  return (int)(want < cap ? want : cap);
}

__global__ void momentum_copy_kernel(const float* const* grads, float* Gc, float* Mh,
                                     int64_t elems, float beta1, int* status) {
  const int b = blockIdx.y;
  const float* g = grads[b];
  float* gc = Gc + (int64_t)b * elems;
  float* mh = Mh + (int64_t)b * elems;
  const float c1 = 1.f - beta1;
  int bad = 0;
  const bool vec = ((reinterpret_cast<uintptr_t>(g) | reinterpret_cast<uintptr_t>(gc) |
                     reinterpret_cast<uintptr_t>(mh)) & 15) == 0;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  int64_t start = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  int64_t tail = 0;
  if (vec) {
    const int64_t n4 = elems / 4;
    for (int64_t i = start; i < n4; i += stride) {
      float4 x = reinterpret_cast<const float4*>(g)[i];
      float4 m = reinterpret_cast<float4*>(mh)[i];
      bad |= !isfinite(x.x) | !isfinite(x.y) | !isfinite(x.z) | !isfinite(x.w);
      m.x = fmaf(beta1, m.x, c1 * x.x);
      m.y = fmaf(beta1, m.y, c1 * x.y);
      m.z = fmaf(beta1, m.z, c1 * x.z);
      m.w = fmaf(beta1, m.w, c1 * x.w);
      reinterpret_cast<float4*>(gc)[i] = x;
      reinterpret_cast<float4*>(mh)[i] = m;
    }
    tail = n4 * 4;
  }
  for (int64_t i = tail + start; i < elems; i += stride) {
    const float x = g[i];
    bad |= !isfinite(x);
    mh[i] = fmaf(beta1, mh[i], c1 * x);
    gc[i] = x;
  }
  if (__syncthreads_or(bad) && threadIdx.x == 0) atomicOr(status, kStatusNonFinite);
}

// One Adam step in the basis for one element (v updated, N returned).
__device__ __forceinline__ float adam_one(float g, float m, float& v, float beta2, float c2, float eps, float inv_bc1,
                                          float inv_sqrt_bc2) {
  const float vn = fmaf(beta2, v, c2 * g * g);
  v = vn;
  return (m * inv_bc1) / (sqrtf(vn) * inv_sqrt_bc2 + eps);
}

__global__ void adam_kernel(float* Gp, const float* Mp, float* V, int rows, int cols, float beta2,
                            float eps, float inv_bc1, float inv_sqrt_bc2, const uint8_t* skipL,
                            const uint8_t* skipR, float* N_lo, int* status) {
  const int b = blockIdx.y;
  const int64_t elems = (int64_t)rows * cols;
  float* gp = Gp + (int64_t)b * elems;
  const float* mp = Mp + (int64_t)b * elems;
  float* v = V + (int64_t)b * elems;
  float* nl = N_lo ? N_lo + (int64_t)b * elems : nullptr;
  const uint8_t* sl = skipL ? skipL + (int64_t)b * rows : nullptr;
  const uint8_t* sr = skipR ? skipR + (int64_t)b * cols : nullptr;
  const float c2 = 1.f - beta2;
  int bad = 0;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t start = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if ((cols & 3) == 0) {
    // four elements of one row per thread and step, 16-byte accesses (every matrix of the
    // arena starts on a 16-byte boundary when cols is a multiple of 4)
    for (int64_t i4 = start; i4 < elems / 4; i4 += stride) {
      const float4 g = reinterpret_cast<const float4*>(gp)[i4];
      const float4 m = reinterpret_cast<const float4*>(mp)[i4];
      float4 vv = reinterpret_cast<const float4*>(v)[i4];
      float4 o;
      o.x = adam_one(g.x, m.x, vv.x, beta2, c2, eps, inv_bc1, inv_sqrt_bc2);
      o.y = adam_one(g.y, m.y, vv.y, beta2, c2, eps, inv_bc1, inv_sqrt_bc2);
      o.z = adam_one(g.z, m.z, vv.z, beta2, c2, eps, inv_bc1, inv_sqrt_bc2);
      o.w = adam_one(g.w, m.w, vv.w, beta2, c2, eps, inv_bc1, inv_sqrt_bc2);
      if (sl || sr) {
        const int64_t row = (4 * i4) / cols;
        const int col = (int)(4 * i4 - row * cols);
        if (sl && sl[row]) o = make_float4(0.f, 0.f, 0.f, 0.f);
        if (sr) {
          if (sr[col]) o.x = 0.f;
          if (sr[col + 1]) o.y = 0.f;
          if (sr[col + 2]) o.z = 0.f;
          if (sr[col + 3]) o.w = 0.f;
        }
      }
      bad |= !isfinite(o.x) | !isfinite(o.y) | !isfinite(o.z) | !isfinite(o.w);
      reinterpret_cast<float4*>(v)[i4] = vv;
      reinterpret_cast<float4*>(gp)[i4] = o;
      if (nl) reinterpret_cast<float4*>(nl)[i4] = make_float4(lo_part(o.x), lo_part(o.y), lo_part(o.z), lo_part(o.w));
    }
  } else {
    for (int64_t i = start; i < elems; i += stride) {
      float vi = v[i];
      float nv = adam_one(gp[i], mp[i], vi, beta2, c2, eps, inv_bc1, inv_sqrt_bc2);
      v[i] = vi;
      if ((sl && sl[i / cols]) || (sr && sr[i % cols])) nv = 0.f;
      bad |= !isfinite(nv);
      gp[i] = nv;
      if (nl) nl[i] = lo_part(nv);
    }
  }
  if (__syncthreads_or(bad) && threadIdx.x == 0) atomicOr(status, kStatusNonFinite);
}

__global__ void weight_update_kernel(float* const* params, const float* D, int64_t elems, float lr,
                                     float wd) {
  const int b = blockIdx.y;
  float* w = params[b];
  const float* d = D + (int64_t)b * elems;
  const float keep = 1.f - lr * wd;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < elems; i += stride)
    w[i] = fmaf(keep, w[i], -lr * d[i]);
}

__global__ void identity_kernel(float* Q, int n) {
  const int b = blockIdx.y;
  float* q = Q + (int64_t)b * n * n;
  const int64_t nn = (int64_t)n * n;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nn; i += stride)
    q[i] = (i / n == i % n) ? 1.f : 0.f;
}


// One 32 x 32 tile of one matrix per block (32 x 8 threads). Reads G and writes the
// tensor-core operands into the step's workspace: G and its lo part, G^T and its lo part, and
// the momentum EMA M_hat <- b1 M_hat + (1-b1) G, stored back into the optimizer state (Mh) and
// copied with its lo part beside G (Mc, Mc_lo), so that one batched product rotates both.
// M_hat is kept in G's orientation or, with mh_transposed, as M_hat^T (the working orientation
// of a matrix preconditioned on its left side only).
__global__ void momentum_split_kernel(const float* const* grads, float* Gn, float* Gn_lo, float* Gt, float* Gt_lo,
                                      float* Mh, float* Mc, float* Mc_lo, int rows, int cols, float beta1,
                                      int mh_transposed, int* status) {
  __shared__ float tile[32][33];
  const int b = blockIdx.z;
  const int r0 = blockIdx.y * 32, c0 = blockIdx.x * 32;
  const int64_t mn = (int64_t)rows * cols;
  const float* g = grads[b];
  const float c1 = 1.f - beta1;
  int bad = 0;
  for (int i = threadIdx.y; i < 32; i += 8) {
    const int r = r0 + i, c = c0 + threadIdx.x;
    float x = 0.f;
    if (r < rows && c < cols) {
      const int64_t o = (int64_t)b * mn + (int64_t)r * cols + c;
      x = g[(int64_t)r * cols + c];
      bad |= !isfinite(x);
      Gn[o] = x;
      Gn_lo[o] = lo_part(x);
      if (!mh_transposed) {
        const float m = fmaf(beta1, Mh[o], c1 * x);
        Mh[o] = m;
        Mc[o] = m;
        Mc_lo[o] = lo_part(m);
      }
    }
    tile[i][threadIdx.x] = x;
  }
  __syncthreads();
  for (int i = threadIdx.y; i < 32; i += 8) {
    const int c = c0 + i, r = r0 + threadIdx.x;  // G^T[c][r]
    if (r < rows && c < cols) {
      const float x = tile[threadIdx.x][i];
      const int64_t o = (int64_t)b * mn + (int64_t)c * rows + r;
      Gt[o] = x;
      Gt_lo[o] = lo_part(x);
      if (mh_transposed) {
        const float m = fmaf(beta1, Mh[o], c1 * x);
        Mh[o] = m;
        Mc[o] = m;
        Mc_lo[o] = lo_part(m);
      }
    }
  }
  if (__syncthreads_or(bad) && threadIdx.x == 0 && threadIdx.y == 0) atomicOr(status, kStatusNonFinite);
}

// Packed symmetric storage of an n x n factor: only its lower-triangular 32 x 32 tiles, tile
// (I, J) with I >= J at tile index I (I + 1) / 2 + J, each tile row-major; entries beyond n
// are zero. A diagonal tile is stored whole (its upper half mirrors its lower half).
__device__ __forceinline__ void tri_tile(int t, int& I, int& J) {
  int i = (int)((sqrtf(8.f * (float)t + 1.f) - 1.f) * 0.5f);
  while ((i + 1) * (i + 2) / 2 <= t) ++i;
  while (i * (i + 1) / 2 > t) --i;
  I = i;
  J = t - i * (i + 1) / 2;
}

// Full matrix (and, if F_lo is given, its lo part) from packed tiles: one lower tile per
// block (32 x 8 threads), written in place and, off the diagonal, mirrored through shared
// memory.
__global__ void unpack_sym_kernel(const float* P, float* F, float* F_lo, int n, int64_t packed) {
  __shared__ float tile[32][33];
  const int b = blockIdx.y;
  int I, J;
  tri_tile(blockIdx.x, I, J);
  const float* p = P + (int64_t)b * packed + (int64_t)blockIdx.x * 1024;
  float* f = F + (int64_t)b * n * n;
  float* fl = F_lo ? F_lo + (int64_t)b * n * n : nullptr;
  for (int i = threadIdx.y; i < 32; i += 8) {
    const float x = p[i * 32 + threadIdx.x];
    tile[i][threadIdx.x] = x;
    const int r = I * 32 + i, c = J * 32 + threadIdx.x;
    if (r < n && c < n) {
      f[(int64_t)r * n + c] = x;
      if (fl) fl[(int64_t)r * n + c] = lo_part(x);
    }
  }
  if (I == J) return;  // uniform over the block
  __syncthreads();
  for (int i = threadIdx.y; i < 32; i += 8) {
    const int r = J * 32 + i, c = I * 32 + threadIdx.x;
    if (r < n && c < n) {
      const float x = tile[threadIdx.x][i];
      f[(int64_t)r * n + c] = x;
      if (fl) fl[(int64_t)r * n + c] = lo_part(x);
    }
  }
}

// Packed tiles from the lower triangle of a full matrix (the upper triangle is not read
// except inside diagonal tiles, where the lower half is mirrored over it).
__global__ void pack_sym_kernel(const float* F, float* P, int n, int64_t packed) {
  __shared__ float tile[32][33];
  const int b = blockIdx.y;
  int I, J;
  tri_tile(blockIdx.x, I, J);
  const float* f = F + (int64_t)b * n * n;
  float* p = P + (int64_t)b * packed + (int64_t)blockIdx.x * 1024;
  for (int i = threadIdx.y; i < 32; i += 8) {
    const int r = I * 32 + i, c = J * 32 + threadIdx.x;
    tile[i][threadIdx.x] = (r < n && c < n) ? f[(int64_t)r * n + c] : 0.f;
  }
  if (I == J) __syncthreads();  // uniform over the block
  for (int i = threadIdx.y; i < 32; i += 8) {
    const int j = threadIdx.x;
    p[i * 32 + j] = (I != J || i >= j) ? tile[i][j] : tile[j][i];
  }
}

// Writes n (<= kPtrChunk) device pointers handed over as a kernel parameter (the launch copies
// them, so the host array may be reused as soon as the launch call returns).
__global__ void put_ptrs_kernel(void** dst, PtrChunk c, int n) {
  const int i = threadIdx.x;
  if (i < n) dst[i] = c.p[i];
}

// dst_b = src_b^T for `batch` contiguous rows x cols matrices (32 x 32 tiles, 32 x 8 threads).
__global__ void transpose_kernel(const float* src, float* dst, int rows, int cols) {
  __shared__ float tile[32][33];
  const int b = blockIdx.z;
  const int64_t mn = (int64_t)rows * cols;
  const int r0 = blockIdx.y * 32, c0 = blockIdx.x * 32;
  for (int i = threadIdx.y; i < 32; i += 8) {
    const int r = r0 + i, c = c0 + threadIdx.x;
    tile[i][threadIdx.x] = (r < rows && c < cols) ? src[(int64_t)b * mn + (int64_t)r * cols + c] : 0.f;
  }
  __syncthreads();
  for (int i = threadIdx.y; i < 32; i += 8) {
    const int c = c0 + i, r = r0 + threadIdx.x;
    if (r < rows && c < cols) dst[(int64_t)b * mn + (int64_t)c * rows + r] = tile[threadIdx.x][i];
  }
}

// Q -> Q_lo, Q^T, Q^T_lo for `batch` n x n matrices (32 x 32 tiles, 32 x 8 threads).
__global__ void basis_split_kernel(const float* Q, float* Q_lo, float* Qt, float* Qt_lo, int n) {
  __shared__ float tile[32][33];
  const int b = blockIdx.z;
  const int r0 = blockIdx.y * 32, c0 = blockIdx.x * 32;
  const int64_t nn = (int64_t)n * n;
  for (int i = threadIdx.y; i < 32; i += 8) {
    const int r = r0 + i, c = c0 + threadIdx.x;
    float x = 0.f;
    if (r < n && c < n) {
      const int64_t o = (int64_t)b * nn + (int64_t)r * n + c;
      x = Q[o];
      if (Q_lo) Q_lo[o] = lo_part(x);
    }
    tile[i][threadIdx.x] = x;
  }
  __syncthreads();
  for (int i = threadIdx.y; i < 32; i += 8) {
    const int c = c0 + i, r = r0 + threadIdx.x;
    if (r < n && c < n) {
      const float x = tile[threadIdx.x][i];
      const int64_t o = (int64_t)b * nn + (int64_t)c * n + r;
      Qt[o] = x;
      Qt_lo[o] = lo_part(x);
    }
  }
}

// From Q^T and its lo part (one group slice of `batch` n x n bases): a copy of both, and Q
// with its lo part, 32 x 32 tiles (32 x 8 threads). Any output may be null.
__global__ void basis_from_qt_kernel(const float* Qt, const float* Qt_lo, float* Qt_out, float* Qt_lo_out, float* Q,
                                     float* Q_lo, int n) {
  __shared__ float tile[32][33];
  const int b = blockIdx.z;
  const int64_t nn = (int64_t)n * n;
  const int r0 = blockIdx.y * 32, c0 = blockIdx.x * 32;
  for (int i = threadIdx.y; i < 32; i += 8) {
    const int r = r0 + i, c = c0 + threadIdx.x;
    float x = 0.f;
    if (r < n && c < n) {
      const int64_t o = (int64_t)b * nn + (int64_t)r * n + c;
      x = Qt[o];
      if (Qt_out) Qt_out[o] = x;
      if (Qt_lo_out) Qt_lo_out[o] = lo_part(x);
    }
    tile[i][threadIdx.x] = x;
  }
  __syncthreads();
  if (!Q) return;
  for (int i = threadIdx.y; i < 32; i += 8) {
    const int c = c0 + i, r = r0 + threadIdx.x;
    if (r < n && c < n) {
      const float x = tile[threadIdx.x][i];
      const int64_t o = (int64_t)b * nn + (int64_t)c * n + r;
      Q[o] = x;
      if (Q_lo) Q_lo[o] = lo_part(x);
    }
  }
}

// lam[b][i] = sum_k C[b][i][k] Qt[b][i][k] = (Q^T F Q)_ii for C = Q^T F: one warp per row.
__global__ void diag_dot_kernel(const float* C, const float* Qt, float* lam, int n) {
  const int b = blockIdx.y;
  const int row = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  const int lane = threadIdx.x & 31;
  if (row >= n) return;
  const int64_t off = (int64_t)b * n * n + (int64_t)row * n;
  const float4* c = reinterpret_cast<const float4*>(C + off);
  const float4* q = reinterpret_cast<const float4*>(Qt + off);
  float acc = 0.f;
  for (int k = lane; k < n / 4; k += 32) {
    const float4 x = c[k], y = q[k];
    acc = fmaf(x.x, y.x, acc);
    acc = fmaf(x.y, y.y, acc);
    acc = fmaf(x.z, y.z, acc);
    acc = fmaf(x.w, y.w, acc);
  }
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if (lane == 0) lam[(int64_t)b * n + row] = acc;
}

// X[b][i][j] <- X[b][i][j] * sqrt(coef / (max(lam[b][j], 0) + eps)) and its lo part (cols a
// multiple of 4, rows of 16-byte multiples).
__global__ void scale_cols_split_kernel(float* X, float* X_lo, const float* lam, int rows, int cols, float coef,
                                        float eps) {
  const int b = blockIdx.y;
  const int64_t e4 = (int64_t)rows * cols / 4;
  float4* x = reinterpret_cast<float4*>(X + (int64_t)b * rows * cols);
  float4* xl = reinterpret_cast<float4*>(X_lo + (int64_t)b * rows * cols);
  const float* l = lam + (int64_t)b * cols;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < e4; i += stride) {
    const int j = (int)((i * 4) % cols);
    float4 v = x[i];
    v.x *= sqrtf(coef / (fmaxf(l[j], 0.f) + eps));
    v.y *= sqrtf(coef / (fmaxf(l[j + 1], 0.f) + eps));
    v.z *= sqrtf(coef / (fmaxf(l[j + 2], 0.f) + eps));
    v.w *= sqrtf(coef / (fmaxf(l[j + 3], 0.f) + eps));
    x[i] = v;
    xl[i] = make_float4(lo_part(v.x), lo_part(v.y), lo_part(v.z), lo_part(v.w));
  }
}

__global__ void split_kernel(const float* x, float* hi, float* lo, int64_t n) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
    const float v = x[i];
    if (hi) hi[i] = tf32_trunc(v);
    lo[i] = lo_part(v);
  }
}

}  // namespace

cudaError_t momentum_split(const float* const* grads, float* Gn, float* Gn_lo, float* Gt, float* Gt_lo, float* Mhat,
                           float* Mcopy, float* Mcopy_lo, int rows, int cols, int batch, float beta1,
                           bool mhat_transposed, int* status, cudaStream_t s) {
  if (rows <= 0 || cols <= 0 || batch <= 0) return cudaSuccess;
  if (batch > 65535 || (rows + 31) / 32 > 65535) return cudaErrorInvalidValue;
  const double e = (double)rows * cols * batch;
  ProfScope prof(kFamElementwise, 3.0 * e, 36.0 * e, s);
  dim3 grid((cols + 31) / 32, (rows + 31) / 32, batch);
  momentum_split_kernel<<<grid, dim3(32, 8), 0, s>>>(grads, Gn, Gn_lo, Gt, Gt_lo, Mhat, Mcopy, Mcopy_lo, rows, cols,
                                                     beta1, mhat_transposed ? 1 : 0, status);
  return cudaGetLastError();
}

int64_t packed_floats(int n) {
  const int64_t t = (n + 31) / 32;
  return t * (t + 1) / 2 * 1024;
}

cudaError_t unpack_sym(const float* P, float* F, float* F_lo, int n, int batch, cudaStream_t s) {
  if (n <= 0 || batch <= 0) return cudaSuccess;
  if (batch > 65535) return cudaErrorInvalidValue;
  const int64_t tiles = packed_floats(n) / 1024;
  const double e = (double)n * n * batch;
  ProfScope prof(kFamElementwise, 0.0, (2.0 + (F_lo ? 8.0 : 4.0)) * e, s);
  unpack_sym_kernel<<<dim3((unsigned)tiles, batch), dim3(32, 8), 0, s>>>(P, F, F_lo, n, packed_floats(n));
  return cudaGetLastError();
}

cudaError_t pack_sym(const float* F, float* P, int n, int batch, cudaStream_t s) {
  if (n <= 0 || batch <= 0) return cudaSuccess;
  if (batch > 65535) return cudaErrorInvalidValue;
  const int64_t tiles = packed_floats(n) / 1024;
  const double e = (double)n * n * batch;
  ProfScope prof(kFamElementwise, 0.0, 4.0 * e, s);
  pack_sym_kernel<<<dim3((unsigned)tiles, batch), dim3(32, 8), 0, s>>>(F, P, n, packed_floats(n));
  return cudaGetLastError();
}

cudaError_t put_ptrs(void** dst, void* const* src, int64_t n, cudaStream_t s) {
  for (int64_t i = 0; i < n; i += kPtrChunk) {
    PtrChunk c;
    const int k = (int)std::min<int64_t>(kPtrChunk, n - i);
    for (int j = 0; j < k; ++j) c.p[j] = src[i + j];
    ProfScope prof(kFamOther, 0.0, 8.0 * k, s);
    put_ptrs_kernel<<<1, 512, 0, s>>>(dst + i, c, k);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t transpose(const float* src, float* dst, int rows, int cols, int batch, cudaStream_t s) {
  if (rows <= 0 || cols <= 0 || batch <= 0) return cudaSuccess;
  if (batch > 65535 || (rows + 31) / 32 > 65535) return cudaErrorInvalidValue;
  ProfScope prof(kFamOther, 0.0, 8.0 * rows * (double)cols * batch, s);
  dim3 grid((cols + 31) / 32, (rows + 31) / 32, batch);
  transpose_kernel<<<grid, dim3(32, 8), 0, s>>>(src, dst, rows, cols);
  return cudaGetLastError();
}

cudaError_t basis_split(const float* Q, float* Q_lo, float* Qt, float* Qt_lo, int n, int batch, cudaStream_t s) {
  if (n <= 0 || batch <= 0) return cudaSuccess;
  const double e = (double)n * n * batch;
  ProfScope prof(kFamElementwise, 2.0 * e, (Q_lo ? 16.0 : 12.0) * e, s);
  dim3 grid((n + 31) / 32, (n + 31) / 32, batch);
  basis_split_kernel<<<grid, dim3(32, 8), 0, s>>>(Q, Q_lo, Qt, Qt_lo, n);
  return cudaGetLastError();
}

cudaError_t basis_from_qt(const float* Qt, const float* Qt_lo, float* Qt_out, float* Qt_lo_out, float* Q, float* Q_lo,
                          int n, int batch, cudaStream_t s) {
  if (n <= 0 || batch <= 0) return cudaSuccess;
  const double e = (double)n * n * batch;
  ProfScope prof(kFamElementwise, 0.0, (4.0 + (Qt_out ? 4 : 0) + (Qt_lo_out ? 8 : 0) + (Q ? 4 : 0) + (Q_lo ? 4 : 0)) * e, s);
  dim3 grid((n + 31) / 32, (n + 31) / 32, batch);
  basis_from_qt_kernel<<<grid, dim3(32, 8), 0, s>>>(Qt, Qt_lo, Qt_out, Qt_lo_out, Q, Q_lo, n);
  return cudaGetLastError();
}

cudaError_t split_tf32(const float* x, float* hi, float* lo, int64_t n, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  ProfScope prof(kFamElementwise, 2.0 * n, 12.0 * n, s);
  const int64_t want = (n + kThreads - 1) / kThreads;
  split_kernel<<<(int)(want < 4096 ? want : 4096), kThreads, 0, s>>>(x, hi, lo, n);
  return cudaGetLastError();
}

cudaError_t diag_dot(const float* C, const float* Qt, float* lam, int n, int batch, cudaStream_t s) {
  if (n <= 0 || batch <= 0) return cudaSuccess;
  if ((n & 3) || batch > 65535) return cudaErrorInvalidValue;
  const double e = (double)n * n * batch;
  ProfScope prof(kFamElementwise, 2.0 * e, 8.0 * e, s);
  diag_dot_kernel<<<dim3((n + 7) / 8, batch), 256, 0, s>>>(C, Qt, lam, n);
  return cudaGetLastError();
}

cudaError_t scale_cols_split(float* X, float* X_lo, const float* lam, int rows, int cols, int batch, float coef,
                             float eps, cudaStream_t s) {
  const int64_t elems = (int64_t)rows * cols;
  if (elems <= 0 || batch <= 0) return cudaSuccess;
  if ((cols & 3) || batch > 65535) return cudaErrorInvalidValue;
  ProfScope prof(kFamElementwise, 4.0 * elems * batch, 12.0 * elems * batch, s);
  scale_cols_split_kernel<<<dim3(blocks_for(elems, batch), batch), kThreads, 0, s>>>(X, X_lo, lam, rows, cols, coef,
                                                                                     eps);
  return cudaGetLastError();
}

cudaError_t momentum_and_copy(const float* const* grads, float* Gc, float* Mhat, int64_t elems,
                              int batch, float beta1, int* status, cudaStream_t s) {
  if (elems <= 0 || batch <= 0) return cudaSuccess;
  ProfScope prof(kFamElementwise, 3.0 * elems * batch, 16.0 * elems * batch, s);
  momentum_copy_kernel<<<dim3(blocks_for(elems, batch), batch), kThreads, 0, s>>>(grads, Gc, Mhat, elems,
                                                                                   beta1, status);
  return cudaGetLastError();
}

cudaError_t adam_in_basis(float* Gp, const float* Mp, float* V, int rows, int cols, int batch,
                          float beta1, float beta2, float eps, float bc1, float bc2,
                          const uint8_t* skipL, const uint8_t* skipR, float* N_lo, int* status,
                          cudaStream_t s) {
  (void)beta1;
  const int64_t elems = (int64_t)rows * cols;
  if (elems <= 0 || batch <= 0) return cudaSuccess;
  ProfScope prof(kFamElementwise, 8.0 * elems * batch, (N_lo ? 24.0 : 20.0) * elems * batch, s);
  adam_kernel<<<dim3(blocks_for(elems, batch), batch), kThreads, 0, s>>>(
      Gp, Mp, V, rows, cols, beta2, eps, 1.f / bc1, 1.f / sqrtf(bc2), skipL, skipR, N_lo, status);
  return cudaGetLastError();
}

cudaError_t weight_update(float* const* params, const float* D, int64_t elems, int batch, float lr,
                          float wd, cudaStream_t s) {
  if (elems <= 0 || batch <= 0) return cudaSuccess;
  ProfScope prof(kFamElementwise, 3.0 * elems * batch, 12.0 * elems * batch, s);
  weight_update_kernel<<<dim3(blocks_for(elems, batch), batch), kThreads, 0, s>>>(params, D, elems, lr, wd);
  return cudaGetLastError();
}

cudaError_t set_identity(float* Q, int n, int batch, cudaStream_t s) {
  if (n <= 0 || batch <= 0) return cudaSuccess;
  ProfScope prof(kFamOther, 0, 4.0 * n * n * batch, s);
  identity_kernel<<<dim3(blocks_for((int64_t)n * n, batch), batch), kThreads, 0, s>>>(Q, n);
  return cudaGetLastError();
}

}  // namespace soap
