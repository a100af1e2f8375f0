// Batched Householder QR with explicit Q for the eigenbasis refresh
// (Alg. 1, "Eigenbasis Re-computation": Q <- QR(L_t Q).Q, every step as the
// appendix on eigh vs QR settles), with diag(R) >= 0.
//
// Blocked right-looking Householder QR (Golub & Van Loan, 4th ed., section 5.2.3):
//   for each 32-column panel k:
//     1. factor the panel A[k:n, k:k+32] in shared memory          (qr_panel_kernel)
//        -> Householder vectors V (written over the panel) and the
//           compact-WY factor T with H_1...H_32 = I - V T V^T
//     2. trailing update A[k:, k+32:] <- (I - V T^T V^T) A[k:, k+32:] (three GEMMs)
//   then Q = H_1 ... H_n I, accumulated backwards one block at a time (three GEMMs
//   per block).
//
// The panel of an n x n matrix has up to n rows; it is spread over a thread-block
// cluster of ceil((n-k)/1024) CTAs (<= 8 for n <= 8192), 1024 rows each, and the
// column reductions of each Householder step are combined through distributed
// shared memory with one cluster barrier per reduction. No CTA waits on a flag:
// the only waits are hardware cluster barriers that every CTA of the cluster
// reaches unconditionally.
//
// Reflector convention (LAPACK larfg): for x = A[p:n, p] with alpha = x_1 and
// sigma = ||x_2:||^2, beta = -sign(alpha) ||x||, v = x / (alpha - beta) with v_1 = 1,
// tau = (beta - alpha) / beta, so H x = beta e_1 and R_pp = beta; sigma = 0 gives H = I
// and R_pp = alpha. The sign convention diag(R) >= 0 then negates column p of Q
// wherever R_pp < 0; it costs nothing because the backward accumulation of Q starts
// from diag(d_1..d_n), d_p = sign of R_pp, instead of I. A column with
// ||x|| <= tol * ||P||_F is treated as exactly zero: H = I, R_pp = 0, d_p = +1, and the
// column is flagged in skip[]. (The convention matters beyond the sign: the columns of
// Q that complete a rank-deficient P are H_1 ... H_p-1 e_p, which depend on it.)
#include <cooperative_groups.h>

#include <algorithm>

#include "profile.h"
#include "soap_internal.h"

namespace cg = cooperative_groups;

namespace soap {

namespace {

constexpr int NB = 32;            // panel width
constexpr int ROWS = 1024;        // panel rows held by one CTA
constexpr int PT = 512;           // threads per panel CTA
constexpr int LDS = ROWS + 1;     // column stride of the shared panel (bank-conflict padding)
constexpr int MAXC = 8;           // largest cluster (portable limit) -> n <= 8192
constexpr int NWARP = PT / 32;

struct PanelArgs {
  float* A;            // [batch][n][n] working matrices
  float* T;            // [batch][npanel][NB][NB]
  uint8_t* skip;       // [batch][n]
  float* dsign;        // [batch][n] sign of R_pp (+1 for zero columns)
  const float* thresh; // [batch]
  int* status;
  int n, k, kb, panel, npanel;
};

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__global__ void __launch_bounds__(PT, 1) qr_panel_kernel(PanelArgs p) {
  cg::cluster_group cluster = cg::this_cluster();
  const int c = (int)cluster.block_rank();
  const int C = (int)cluster.num_blocks();
  const int b = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

  extern __shared__ float sA[];  // [NB][LDS], column-major panel slice
  __shared__ float s_sig[2][MAXC];
  __shared__ float s_alpha[2];
  __shared__ float s_dot[2][MAXC][NB];
  __shared__ float s_dtot[NB];
  __shared__ float s_red[NWARP];
  __shared__ float s_tau[NB];
  __shared__ int s_skip[NB];
  __shared__ float s_dsign[NB];
  __shared__ float s_gram[MAXC][NB][NB];
  __shared__ float s_T[NB][NB + 1];

  const int n = p.n, k = p.k, kb = p.kb;
  float* A = p.A + (int64_t)b * n * n;
  const int row0 = k + c * ROWS;
  const int nrows = max(0, min(ROWS, n - row0));

  for (int e = tid; e < nrows * kb; e += PT) {
    const int i = e / kb, jj = e % kb;
    sA[jj * LDS + i] = A[(int64_t)(row0 + i) * n + k + jj];
  }
  __syncthreads();
  const float thresh = p.thresh[b];
  int nonfinite = 0;

  for (int j = 0; j < kb; ++j) {
    const int par = j & 1;
    // rows strictly below the pivot (pivot = local row j of rank 0)
    const int ibeg = (c == 0) ? j + 1 : 0;
    float s = 0.f;
    for (int i = ibeg + tid; i < nrows; i += PT) {
      const float x = sA[j * LDS + i];
      s = fmaf(x, x, s);
    }
    s = warp_sum(s);
    if (lane == 0) s_red[warp] = s;
    __syncthreads();
    if (tid == 0) {
      float tot = 0.f;
      for (int w = 0; w < NWARP; ++w) tot += s_red[w];
      const float alpha = (c == 0) ? sA[j * LDS + j] : 0.f;
      for (int q = 0; q < C; ++q) {
        float* rs = cluster.map_shared_rank(&s_sig[par][0], q);
        rs[c] = tot;
        if (c == 0) *cluster.map_shared_rank(&s_alpha[par], q) = alpha;
      }
    }
    cluster.sync();

    // every CTA derives the same reflector from the same reduced values
    float sigma = 0.f;
    for (int q = 0; q < C; ++q) sigma += s_sig[par][q];
    const float alpha = s_alpha[par];
    const float xnorm = sqrtf(fmaf(alpha, alpha, sigma));
    if (!isfinite(xnorm)) nonfinite = 1;
    const bool skip = !(xnorm > thresh);
    float tau = 0.f, v0 = 1.f, rsign = 1.f;
    bool scale = false;
    if (!skip) {
      if (sigma == 0.f) {
        rsign = alpha < 0.f ? -1.f : 1.f;   // H = I, R_pp = alpha
      } else {
        const float beta = alpha >= 0.f ? -xnorm : xnorm;
        v0 = alpha - beta;                   // same sign as alpha: no cancellation
        tau = (beta - alpha) / beta;
        rsign = beta < 0.f ? -1.f : 1.f;
        scale = true;
      }
    }
    // v below the pivot: x / v0, or 0 where H = I or x_2: = 0
    for (int i = ibeg + tid; i < nrows; i += PT) {
      float& x = sA[j * LDS + i];
      x = scale ? x / v0 : 0.f;
    }
    if (tid == 0) {
      s_tau[j] = tau;
      s_skip[j] = skip ? 1 : 0;
      s_dsign[j] = rsign;
    }
    __syncthreads();

    // apply H_j = I - tau v v^T to the panel columns right of j
    if (tau != 0.f && j + 1 < kb) {
      const int pivot_rows = (c == 0) ? j : 0;  // local rows >= this take part
      for (int jj = j + 1 + warp; jj < kb; jj += NWARP) {
        float d = 0.f;
        for (int i = ibeg + lane; i < nrows; i += 32) d = fmaf(sA[j * LDS + i], sA[jj * LDS + i], d);
        d = warp_sum(d);
        if (c == 0) d += sA[jj * LDS + j];  // v_pivot = 1
        if (lane < C) cluster.map_shared_rank(&s_dot[par][0][0], lane)[c * NB + jj] = d;
      }
      cluster.sync();
      if (tid < kb && tid > j) {
        float d = 0.f;
        for (int q = 0; q < C; ++q) d += s_dot[par][q][tid];
        s_dtot[tid] = d;
      }
      __syncthreads();
      for (int i = pivot_rows + tid; i < nrows; i += PT) {
        const float vi = (c == 0 && i == j) ? 1.f : sA[j * LDS + i];
        const float tv = tau * vi;
        for (int jj = j + 1; jj < kb; ++jj) sA[jj * LDS + i] = fmaf(-tv, s_dtot[jj], sA[jj * LDS + i]);
      }
      __syncthreads();
    }
  }

  // V with its unit diagonal and zeros above it (rank 0 holds the top kb rows)
  if (c == 0) {
    for (int e = tid; e < kb * kb; e += PT) {
      const int jj = e / kb, i = e % kb;
      if (i < jj) sA[jj * LDS + i] = 0.f;
      else if (i == jj) sA[jj * LDS + i] = 1.f;
    }
  }
  __syncthreads();
  for (int e = tid; e < nrows * kb; e += PT) {
    const int i = e / kb, jj = e % kb;
    A[(int64_t)(row0 + i) * n + k + jj] = sA[jj * LDS + i];
  }

  // partial Gram V^T V of this CTA's rows, gathered in rank 0
  for (int pr = warp; pr < kb * kb; pr += NWARP) {
    const int a = pr / kb, bb = pr % kb;
    if (bb < a) continue;
    float g = 0.f;
    for (int i = lane; i < nrows; i += 32) g = fmaf(sA[a * LDS + i], sA[bb * LDS + i], g);
    g = warp_sum(g);
    if (lane == 0) cluster.map_shared_rank(&s_gram[0][0][0], 0)[(c * NB + a) * NB + bb] = g;
  }
  if (nonfinite && tid == 0) atomicOr(p.status, kStatusQrBreakdown);
  cluster.sync();
  if (c != 0) return;

  // T: T_jj = tau_j, T(0:j, j) = -tau_j T(0:j, 0:j) (V(:,0:j)^T v_j)   (LAPACK larft, forward)
  for (int j = 0; j < kb; ++j) {
    if (tid < kb) {
      const int i = tid;
      float t = 0.f;
      if (i < j) {
        float acc = 0.f;
        for (int l = i; l < j; ++l) {
          float g = 0.f;
          for (int q = 0; q < C; ++q) g += s_gram[q][l][j];
          acc = fmaf(s_T[i][l], g, acc);
        }
        t = -s_tau[j] * acc;
      } else if (i == j) {
        t = s_tau[j];
      }
      s_T[i][j] = t;
    }
    __syncthreads();
  }
  float* Tout = p.T + ((int64_t)b * p.npanel + p.panel) * NB * NB;
  for (int e = tid; e < NB * NB; e += PT) {
    const int i = e / NB, jj = e % NB;
    Tout[e] = (i < kb && jj < kb) ? s_T[i][jj] : 0.f;
  }
  if (tid < kb) {
    p.skip[(int64_t)b * n + k + tid] = (uint8_t)s_skip[tid];
    p.dsign[(int64_t)b * n + k + tid] = s_dsign[tid];
  }
}

// ||P_b||_F: per-chunk partial sums in double, then tol * sqrt(sum)
constexpr int NORM_CHUNKS = 64;

__global__ void frob_partial_kernel(const float* P, int64_t nn, double* part) {
  const int b = blockIdx.y;
  const float* x = P + (int64_t)b * nn;
  const int64_t per = (nn + NORM_CHUNKS - 1) / NORM_CHUNKS;
  const int64_t beg = blockIdx.x * per, end = min(nn, beg + per);
  double s = 0.0;
  for (int64_t i = beg + threadIdx.x; i < end; i += blockDim.x) s += (double)x[i] * (double)x[i];
  __shared__ double red[256];
  red[threadIdx.x] = s;
  __syncthreads();
  for (int o = 128; o > 0; o >>= 1) {
    if ((int)threadIdx.x < o) red[threadIdx.x] += red[threadIdx.x + o];
    __syncthreads();
  }
  if (threadIdx.x == 0) part[(int64_t)b * NORM_CHUNKS + blockIdx.x] = red[0];
}

__global__ void thresh_kernel(const double* part, float tol, int batch, float* thresh) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= batch) return;
  double s = 0.0;
  for (int i = 0; i < NORM_CHUNKS; ++i) s += part[(int64_t)b * NORM_CHUNKS + i];
  thresh[b] = (float)((double)tol * sqrt(s));
}

__global__ void signed_identity_kernel(float* Q, const float* d, int n) {
  const int b = blockIdx.y;
  float* q = Q + (int64_t)b * n * n;
  const float* db = d + (int64_t)b * n;
  const int64_t nn = (int64_t)n * n;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nn; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = i / n, c = i % n;
    q[i] = r == c ? db[r] : 0.f;
  }
}

struct Workspace {
  float* A;
  float* T;
  float* W1;
  float* W2;
  float* thresh;
  float* dsign;
  double* part;
};

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

Workspace carve(void* base, int n, int batch, size_t* total) {
  const int npanel = (n + NB - 1) / NB;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    size_t o = off;
    off += align256(bytes);
    return o;
  };
  const size_t oA = take((size_t)batch * n * n * sizeof(float));
  const size_t oT = take((size_t)batch * npanel * NB * NB * sizeof(float));
  const size_t oW1 = take((size_t)batch * NB * n * sizeof(float));
  const size_t oW2 = take((size_t)batch * NB * n * sizeof(float));
  const size_t oth = take((size_t)batch * sizeof(float));
  const size_t osg = take((size_t)batch * n * sizeof(float));
  const size_t opart = take((size_t)batch * NORM_CHUNKS * sizeof(double));
  if (total) *total = off;
  char* c = (char*)base;
  return Workspace{(float*)(c + oA), (float*)(c + oT), (float*)(c + oW1), (float*)(c + oW2),
                   (float*)(c + oth), (float*)(c + osg), (double*)(c + opart)};
}

}  // namespace

size_t qr_workspace_bytes(int n, int batch) {
  size_t total = 0;
  carve(nullptr, n, batch, &total);
  return total;
}

cudaError_t qr_q(int n, int batch, const float* P, float* Q, uint8_t* skip, float tol,
                 void* workspace, size_t workspace_bytes, int* status, cudaStream_t s) {
  if (n <= 0 || batch <= 0) return cudaSuccess;
  if (n > MAXC * ROWS || batch > 65535) return cudaErrorInvalidValue;
  size_t need = 0;
  Workspace w = carve(workspace, n, batch, &need);
  if (workspace_bytes < need) return cudaErrorInvalidValue;
  const int npanel = (n + NB - 1) / NB;
  const int64_t nn = (int64_t)n * n;
  cudaError_t e;

  if (P != w.A) {
    e = cudaMemcpyAsync(w.A, P, (size_t)batch * nn * sizeof(float), cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return e;
  }
  {
    ProfScope prof(kFamOther, 2.0 * nn * batch, 4.0 * nn * batch, s);
    frob_partial_kernel<<<dim3(NORM_CHUNKS, batch), 256, 0, s>>>(w.A, nn, w.part);
  }
  {
    ProfScope prof(kFamOther, 0, 8.0 * NORM_CHUNKS * batch, s);
    thresh_kernel<<<(batch + 127) / 128, 128, 0, s>>>(w.part, tol, batch, w.thresh);
  }

  const size_t smem = (size_t)NB * LDS * sizeof(float);
  e = cudaFuncSetAttribute(qr_panel_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;

  for (int pi = 0; pi < npanel; ++pi) {
    const int k = pi * NB, kb = min(NB, n - k);
    const int C = (n - k + ROWS - 1) / ROWS;
    PanelArgs a{w.A, w.T, skip, w.dsign, w.thresh, status, n, k, kb, pi, npanel};
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(C, batch, 1);
    cfg.blockDim = dim3(PT, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = C;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    {
      // Householder work on the (n-k) x kb panel: ~4 (n-k) kb^2 flops, panel read + written
      ProfScope prof(kFamQrPanel, 4.0 * (n - k) * kb * kb * batch, 8.0 * (n - k) * kb * batch, s);
      e = cudaLaunchKernelEx(&cfg, qr_panel_kernel, a);
    }
    if (e != cudaSuccess) return e;

    const int nc = n - k - kb;
    if (nc <= 0) continue;
    const int m = n - k;
    Operand V = strided(w.A, n, nn, (int64_t)k * n + k);
    Operand Cin = strided(w.A, n, nn, (int64_t)k * n + k + kb);
    MutOperand Cout = strided_mut(w.A, n, nn, (int64_t)k * n + k + kb);
    Operand Tp = strided(w.T, NB, (int64_t)npanel * NB * NB, (int64_t)pi * NB * NB);
    // W1 = V^T C  (kb x nc)
    e = gemm(true, false, kb, nc, m, 1.f, V, Cin, 0.f, strided_mut(w.W1, n, (int64_t)NB * n), batch, s);
    if (e != cudaSuccess) return e;
    // W2 = T^T W1
    e = gemm(true, false, kb, nc, kb, 1.f, Tp, strided(w.W1, n, (int64_t)NB * n), 0.f,
             strided_mut(w.W2, n, (int64_t)NB * n), batch, s);
    if (e != cudaSuccess) return e;
    // C -= V W2
    e = gemm(false, false, m, nc, kb, -1.f, V, strided(w.W2, n, (int64_t)NB * n), 1.f, Cout, batch, s);
    if (e != cudaSuccess) return e;
  }

  {
    // Q = H_1 ... H_n diag(d): start the backward accumulation from diag(d)
    ProfScope prof(kFamOther, 0, 4.0 * nn * batch, s);
    const int blocks = (int)std::min<int64_t>((nn + 255) / 256, 1024);
    signed_identity_kernel<<<dim3(blocks, batch), 256, 0, s>>>(Q, w.dsign, n);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  for (int pi = npanel - 1; pi >= 0; --pi) {
    const int k = pi * NB, kb = min(NB, n - k), m = n - k;
    Operand V = strided(w.A, n, nn, (int64_t)k * n + k);
    Operand Qs = strided(Q, n, nn, (int64_t)k * n + k);
    MutOperand Qo = strided_mut(Q, n, nn, (int64_t)k * n + k);
    Operand Tp = strided(w.T, NB, (int64_t)npanel * NB * NB, (int64_t)pi * NB * NB);
    // W1 = V^T Q[k:, k:]; W2 = T W1; Q[k:, k:] -= V W2
    e = gemm(true, false, kb, m, m, 1.f, V, Qs, 0.f, strided_mut(w.W1, n, (int64_t)NB * n), batch, s);
    if (e != cudaSuccess) return e;
    e = gemm(false, false, kb, m, kb, 1.f, Tp, strided(w.W1, n, (int64_t)NB * n), 0.f,
             strided_mut(w.W2, n, (int64_t)NB * n), batch, s);
    if (e != cudaSuccess) return e;
    e = gemm(false, false, m, m, kb, -1.f, V, strided(w.W2, n, (int64_t)NB * n), 1.f, Qo, batch, s);
    if (e != cudaSuccess) return e;
  }
  return cudaGetLastError();
}

}  // namespace soap
