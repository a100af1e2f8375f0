// Batched Householder QR with explicit Q for the eigenbasis refresh
// (Alg. 1, "Eigenbasis Re-computation": Q <- QR(L_t Q).Q, every step as the
// appendix on eigh vs QR settles), with diag(R) >= 0, on tensor cores.
//
// The QR works on At = P^T (row j of At is column j of P), so every product of the
// blocked algorithm is a C = A B^T of K-major operands: the long reductions run on the
// tcgen05 engine, the rank-32 updates (HBM-bound) on the CUDA cores:
//
//   for each 32-column panel at k (rows k..k+31 of At):
//     1. qr_panel_kernel factors the panel rows in distributed shared memory and writes
//        the Householder vectors as rows of Vt (row k+a = v_a over positions k..n-1,
//        zeros before its pivot), T with H_1..H_32 = I - V T V^T, and V T^T and V T
//        (positions x 32), each with its tf32 lo part.
//     2. trailing rows r > k+31 (columns of P): a_r <- a_r - (a_r V) T V^T, i.e.
//          W1  = At_trail Vt^T                (tensor cores: M = rows, N = 32, K = positions)
//          At_trail -= W1 (V T^T)^T           (rank-32 update streaming At_trail once)
//   then Q^T is accumulated backwards from diag(d) (d_j = sign of R_jj) one block at a
//   time, Q^T <- Q^T (I - V T^T V^T):
//          W   = Qt_sub Vt^T ;  Qt_sub -= W (V T)^T
//   and Q = (Q^T)^T is written with its lo part.
//
// The panel of an n x n matrix spans up to n positions; it is spread over a thread-block
// cluster of ceil((n-k)/1024) CTAs (<= 8 for n <= 8192), 1024 positions each, and the
// reductions of each Householder step are combined through distributed shared memory
// with one cluster barrier per reduction. No CTA waits on a flag: the only waits are
// hardware cluster barriers that every CTA of the cluster reaches unconditionally.
//
// Reflector convention (LAPACK larfg): for x = A[p:n, p] with alpha = x_1 and
// sigma = ||x_2:||^2, beta = -sign(alpha) ||x||, v = x / (alpha - beta) with v_1 = 1,
// tau = (beta - alpha) / beta, so H x = beta e_1 and R_pp = beta; sigma = 0 gives H = I
// and R_pp = alpha. The sign convention diag(R) >= 0 then negates column p of Q
// wherever R_pp < 0; it costs nothing because the backward accumulation starts from
// diag(d_1..d_n), d_p = sign of R_pp, instead of I. A column with
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
constexpr int COLS = 1024;        // panel positions held by one CTA
constexpr int PT = 512;           // threads per panel CTA
constexpr int LDS = COLS + 1;     // row stride of the shared panel (bank-conflict padding)
constexpr int MAXC = 8;           // largest cluster (portable limit) -> n <= 8192
constexpr int NWARP = PT / 32;

// lo part of x for the tensor-core products: x - trunc_tf32(x) rounded to the nearest tf32
__device__ __forceinline__ float tf32_lo(float x) {
  uint32_t r;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x - __uint_as_float(__float_as_uint(x) & 0xFFFFE000u)));
  return __uint_as_float(r);
}

struct PanelArgs {
  float* At;           // [batch][n][n] working P^T
  float* Vt;           // [batch][n][n] Householder vectors as rows
  float* Vt_lo;
  float* VTr;          // [batch][n][NB]   V T^T of this panel (row = position)
  float* VTr_lo;
  float* VTq;          // [batch][npanel][n][NB]  V T of every panel
  float* VTq_lo;
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

  extern __shared__ float sA[];  // [NB][LDS]: panel row jj (a column of P), position offset i
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
  const int64_t nn = (int64_t)n * n;
  float* At = p.At + (int64_t)b * nn;
  const int pos0 = k + c * COLS;  // first position held by this CTA
  const int npos = max(0, min(COLS, n - pos0));

  for (int e = tid; e < npos * kb; e += PT) {
    const int jj = e / npos, i = e % npos;
    sA[jj * LDS + i] = At[(int64_t)(k + jj) * n + pos0 + i];
  }
  __syncthreads();
  const float thresh = p.thresh[b];
  int nonfinite = 0;

  for (int j = 0; j < kb; ++j) {
    const int par = j & 1;
    // positions strictly after the pivot (pivot = local position j of rank 0)
    const int ibeg = (c == 0) ? j + 1 : 0;
    float s = 0.f;
    for (int i = ibeg + tid; i < npos; i += PT) {
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
    // v after the pivot: x / v0, or 0 where H = I or x_2: = 0
    for (int i = ibeg + tid; i < npos; i += PT) {
      float& x = sA[j * LDS + i];
      x = scale ? x / v0 : 0.f;
    }
    if (tid == 0) {
      s_tau[j] = tau;
      s_skip[j] = skip ? 1 : 0;
      s_dsign[j] = rsign;
    }
    __syncthreads();

    // apply H_j = I - tau v v^T to the panel rows after j
    if (tau != 0.f && j + 1 < kb) {
      const int piv = (c == 0) ? j : 0;  // local positions >= this take part
      for (int jj = j + 1 + warp; jj < kb; jj += NWARP) {
        float d = 0.f;
        for (int i = ibeg + lane; i < npos; i += 32) d = fmaf(sA[j * LDS + i], sA[jj * LDS + i], d);
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
      for (int i = piv + tid; i < npos; i += PT) {
        const float vi = (c == 0 && i == j) ? 1.f : sA[j * LDS + i];
        const float tv = tau * vi;
        for (int jj = j + 1; jj < kb; ++jj) sA[jj * LDS + i] = fmaf(-tv, s_dtot[jj], sA[jj * LDS + i]);
      }
      __syncthreads();
    }
  }

  // V with its unit diagonal and zeros before it (rank 0 holds the first kb positions)
  if (c == 0) {
    for (int e = tid; e < kb * kb; e += PT) {
      const int jj = e / kb, i = e % kb;
      if (i < jj) sA[jj * LDS + i] = 0.f;
      else if (i == jj) sA[jj * LDS + i] = 1.f;
    }
  }
  __syncthreads();
  float* Vt = p.Vt + (int64_t)b * nn;
  float* Vt_lo = p.Vt_lo + (int64_t)b * nn;
  for (int e = tid; e < npos * kb; e += PT) {
    const int jj = e / npos, i = e % npos;
    const float v = sA[jj * LDS + i];
    const int64_t o = (int64_t)(k + jj) * n + pos0 + i;
    Vt[o] = v;
    Vt_lo[o] = tf32_lo(v);
  }

  // partial Gram V^T V over this CTA's positions, gathered in rank 0
  for (int pr = warp; pr < kb * kb; pr += NWARP) {
    const int a = pr / kb, bb = pr % kb;
    if (bb < a) continue;
    float g = 0.f;
    for (int i = lane; i < npos; i += 32) g = fmaf(sA[a * LDS + i], sA[bb * LDS + i], g);
    g = warp_sum(g);
    if (lane == 0) cluster.map_shared_rank(&s_gram[0][0][0], 0)[(c * NB + a) * NB + bb] = g;
  }
  if (nonfinite && tid == 0) atomicOr(p.status, kStatusQrBreakdown);
  cluster.sync();

  if (c == 0) {
    // sum the partial Grams once, then T: T_jj = tau_j, T(0:j, j) = -tau_j T(0:j, 0:j) g(0:j, j)
    for (int e = tid; e < kb * kb; e += PT) {
      const int l = e / kb, jj = e % kb;
      float g = 0.f;
      if (l < jj)
        for (int q = 0; q < C; ++q) g += s_gram[q][l][jj];
      s_gram[0][l][jj] = g;  // only (l < jj) entries are read below
    }
    __syncthreads();
    for (int j = 0; j < kb; ++j) {
      if (tid < kb) {
        const int i = tid;
        float t = 0.f;
        if (i < j) {
          float acc = 0.f;
          for (int l = i; l < j; ++l) acc = fmaf(s_T[i][l], s_gram[0][l][j], acc);
          t = -s_tau[j] * acc;
        } else if (i == j) {
          t = s_tau[j];
        }
        s_T[i][j] = t;
      }
      __syncthreads();
    }
    // hand T to every CTA of the cluster
    for (int q = 1; q < C; ++q) {
      float* dst = cluster.map_shared_rank(&s_T[0][0], q);
      for (int e = tid; e < NB * (NB + 1); e += PT) dst[e] = (&s_T[0][0])[e];
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
  cluster.sync();

  // V T^T (for this panel's trailing update) and V T (for the Q accumulation), position-major:
  // warp w takes 32 positions at a time, lane a computes output column a (coalesced rows of 32)
  float* VTr = p.VTr + (int64_t)b * n * NB;
  float* VTr_lo = p.VTr_lo + (int64_t)b * n * NB;
  float* VTq = p.VTq + ((int64_t)b * p.npanel + p.panel) * n * NB;
  float* VTq_lo = p.VTq_lo + ((int64_t)b * p.npanel + p.panel) * n * NB;
  const int a = lane;
  for (int i0 = warp * 32; i0 < npos; i0 += NWARP * 32) {
    const int iend = min(i0 + 32, npos);
    for (int i = i0; i < iend; ++i) {
      float r = 0.f, q = 0.f;
      for (int bb = 0; bb < kb; ++bb) {
        const float v = sA[bb * LDS + i];
        r = fmaf((a < kb) ? s_T[a][bb] : 0.f, v, r);
        q = fmaf((a < kb) ? s_T[bb][a] : 0.f, v, q);
      }
      const int64_t o = (int64_t)(pos0 + i) * NB + a;
      VTr[o] = r;
      VTr_lo[o] = tf32_lo(r);
      VTq[o] = q;
      VTq_lo[o] = tf32_lo(q);
    }
  }
}

// Rank-32 update C_b <- C_b - A_b B_b^T (A: M x K, B: N x K, K <= 32, all row-major, N a
// multiple of 4) with the lo part of the result, in exact fp32 FMAs. It streams C once
// (read, write, lo write; 32 FMAs per element), so it is bound by HBM, not by a matrix
// unit. A CTA owns one 128-column strip: it loads that strip's B once (k-major in shared
// memory), then walks down the rows in 64 x 128 tiles, with the C and A tiles of the next
// tile copied in by cp.async while the current one is computed (two stages), so ~64 KB per
// CTA is in flight. Warp w computes rows 8w..8w+7, lane l columns 4l..4l+3; every global
// access to C is a 16-byte vector and a warp covers 512 contiguous bytes of a row.
constexpr int RU_BM = 64, RU_BN = 128, RU_STAGES = 2;
constexpr int RU_SMEM = (RU_STAGES * RU_BM * RU_BN + RU_STAGES * RU_BM * NB + NB * RU_BN) * 4;

__device__ __forceinline__ void cp_async16(void* smem_dst, const void* gmem_src, bool valid) {
  const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(smem_dst));
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(d), "l"(gmem_src), "r"(valid ? 16 : 0)
               : "memory");
}

__global__ void __launch_bounds__(256, 2)
    rank_update_kernel(int M, int N, int K, const float* __restrict__ A, int64_t lda, int64_t sa,
                       const float* __restrict__ B, int64_t ldb, int64_t sb, float* C, float* C_lo, int64_t ldc,
                       int64_t sc) {
  extern __shared__ float4 ru_smem[];
  float* Cs = reinterpret_cast<float*>(ru_smem);     // [stage][RU_BM][RU_BN]
  float* As = Cs + RU_STAGES * RU_BM * RU_BN;        // [stage][RU_BM][NB]
  float* Bs = As + RU_STAGES * RU_BM * NB;           // [NB][RU_BN]
  const int b = blockIdx.z;
  const int c0 = blockIdx.x * RU_BN;
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  const float* Ab = A + (int64_t)b * sa;
  const float* Bb = B + (int64_t)b * sb;
  float* Cb = C + (int64_t)b * sc;
  float* Lb = C_lo + (int64_t)b * sc;
  const int ntiles = (M + RU_BM - 1) / RU_BM;
  const int col = c0 + 4 * lane;

  // one 64 x 128 tile of C and its 64 x 32 slice of A into stage st (zero-filled past the edges)
  auto issue = [&](int tile, int st) {
    const int r0 = tile * RU_BM;
    float* cs = Cs + st * RU_BM * RU_BN;
    float* as = As + st * RU_BM * NB;
    for (int e = tid; e < RU_BM * (RU_BN / 4); e += 256) {
      const int r = e / (RU_BN / 4), q = e % (RU_BN / 4);
      const bool ok = (r0 + r < M) && (c0 + 4 * q < N);
      cp_async16(cs + r * RU_BN + 4 * q, ok ? Cb + (int64_t)(r0 + r) * ldc + c0 + 4 * q : Cb, ok);
    }
    for (int e = tid; e < RU_BM * (NB / 4); e += 256) {
      const int r = e / (NB / 4), q = e % (NB / 4);
      const bool ok = (r0 + r < M) && (4 * q < K);
      cp_async16(as + r * NB + 4 * q, ok ? Ab + (int64_t)(r0 + r) * lda + 4 * q : Ab, ok);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };

  int tile = blockIdx.y;
  if (tile < ntiles) issue(tile, 0);
  for (int e = tid; e < RU_BN * NB; e += 256) {
    const int cc = e / NB, kk = e % NB;
    Bs[kk * RU_BN + cc] = (c0 + cc < N && kk < K) ? Bb[(int64_t)(c0 + cc) * ldb + kk] : 0.f;
  }
  for (int it = 0; tile < ntiles; ++it, tile += gridDim.y) {
    const int st = it & 1;
    const int next = tile + gridDim.y;
    if (next < ntiles) {
      issue(next, st ^ 1);
      asm volatile("cp.async.wait_group 1;" ::: "memory");
    } else {
      asm volatile("cp.async.wait_group 0;" ::: "memory");
    }
    __syncthreads();
    const float* cs = Cs + st * RU_BM * RU_BN;
    const float* as = As + st * RU_BM * NB;
    float acc[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
#pragma unroll 4
    for (int kk = 0; kk < NB; ++kk) {
      const float4 bv = *reinterpret_cast<const float4*>(&Bs[kk * RU_BN + 4 * lane]);
      const float bb[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float a = as[(8 * w + i) * NB + kk];
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a, bb[j], acc[i][j]);
      }
    }
    const int r0 = tile * RU_BM;
    if (col < N) {
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int r = r0 + 8 * w + i;
        if (r >= M) break;
        const float4 c = *reinterpret_cast<const float4*>(&cs[(8 * w + i) * RU_BN + 4 * lane]);
        float4 o;
        o.x = c.x - acc[i][0];
        o.y = c.y - acc[i][1];
        o.z = c.z - acc[i][2];
        o.w = c.w - acc[i][3];
        *reinterpret_cast<float4*>(Cb + (int64_t)r * ldc + col) = o;
        *reinterpret_cast<float4*>(Lb + (int64_t)r * ldc + col) =
            make_float4(tf32_lo(o.x), tf32_lo(o.y), tf32_lo(o.z), tf32_lo(o.w));
      }
    }
    __syncthreads();  // this stage is refilled by the next iteration's prefetch
  }
}

cudaError_t rank_update(int M, int N, int K, int batch, const float* A, int64_t lda, int64_t sa, const float* B,
                        int64_t ldb, int64_t sb, float* C, float* C_lo, int64_t ldc, int64_t sc, cudaStream_t s) {
  if (M <= 0 || N <= 0) return cudaSuccess;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(rank_update_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, RU_SMEM);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  ProfScope prof(kFamQrUpdate, 2.0 * M * N * (double)K * batch, 12.0 * M * (double)N * batch, s);
  const int strips = (N + RU_BN - 1) / RU_BN, ntiles = (M + RU_BM - 1) / RU_BM;
  // about two waves of 2 CTAs per SM; each CTA walks ntiles / gridDim.y row tiles
  const int want = std::max(1, (2 * 2 * 152) / std::max(1, strips * batch));
  dim3 grid(strips, std::min(ntiles, want), batch);
  rank_update_kernel<<<grid, 256, RU_SMEM, s>>>(M, N, K, A, lda, sa, B, ldb, sb, C, C_lo, ldc, sc);
  return cudaGetLastError();
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

// Q^T <- diag(d) (its lo part is zero: +-1 are tf32 values)
__global__ void signed_identity_kernel(float* Qt, float* Qt_lo, const float* d, int n) {
  const int b = blockIdx.y;
  const int64_t nn = (int64_t)n * n;
  float* q = Qt + (int64_t)b * nn;
  float* ql = Qt_lo + (int64_t)b * nn;
  const float* db = d + (int64_t)b * n;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nn; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = i / n, cc = i % n;
    q[i] = r == cc ? db[r] : 0.f;
    ql[i] = 0.f;
  }
}

// Q = (Q^T)^T and its lo part, 32 x 32 tiles through shared memory
__global__ void transpose_out_kernel(const float* Qt, float* Q, float* Q_lo, int n) {
  __shared__ float tile[32][33];
  const int b = blockIdx.z;
  const int64_t nn = (int64_t)n * n;
  const int r0 = blockIdx.y * 32, c0 = blockIdx.x * 32;
  for (int i = threadIdx.y; i < 32; i += 8) {
    const int r = r0 + i, cc = c0 + threadIdx.x;
    tile[i][threadIdx.x] = (r < n && cc < n) ? Qt[(int64_t)b * nn + (int64_t)r * n + cc] : 0.f;
  }
  __syncthreads();
  for (int i = threadIdx.y; i < 32; i += 8) {
    const int r = c0 + i, cc = r0 + threadIdx.x;
    if (r < n && cc < n) {
      const float x = tile[threadIdx.x][i];
      const int64_t o = (int64_t)b * nn + (int64_t)r * n + cc;
      Q[o] = x;
      if (Q_lo) Q_lo[o] = tf32_lo(x);
    }
  }
}

struct Workspace {
  float* At;
  float* At_lo;
  float* Vt;
  float* Vt_lo;
  float* VTq;
  float* VTq_lo;
  float* VTr;
  float* VTr_lo;
  float* W;
  float* W_lo;
  float* T;
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
  const size_t mat = (size_t)batch * n * n * sizeof(float);
  const size_t pan = (size_t)batch * npanel * n * NB * sizeof(float);
  const size_t thin = (size_t)batch * n * NB * sizeof(float);
  const size_t oAt = take(mat), oAtl = take(mat), oVt = take(mat), oVtl = take(mat);
  const size_t oVq = take(pan), oVql = take(pan), oVr = take(thin), oVrl = take(thin);
  const size_t oW = take(thin), oWl = take(thin);
  const size_t oT = take((size_t)batch * npanel * NB * NB * sizeof(float));
  const size_t oth = take((size_t)batch * sizeof(float));
  const size_t osg = take((size_t)batch * n * sizeof(float));
  const size_t opart = take((size_t)batch * NORM_CHUNKS * sizeof(double));
  if (total) *total = off;
  char* c = (char*)base;
  auto f = [&](size_t o) { return (float*)(c + o); };
  return Workspace{f(oAt), f(oAtl), f(oVt), f(oVtl), f(oVq), f(oVql), f(oVr), f(oVrl),
                   f(oW),  f(oWl),  f(oT),  f(oth),  f(osg), (double*)(c + opart)};
}

TcOperand op(const float* hi, const float* lo, int64_t ld, int64_t stride, int batch) {
  return TcOperand{hi, lo, ld, stride, batch};
}

TcEpilogue out(float* C, float* C_lo, int64_t ldc, int64_t stride, float alpha, float beta, int* status) {
  return TcEpilogue{C, nullptr, ldc, stride, C_lo, ldc, stride, 0, alpha, beta, status};
}

}  // namespace

size_t qr_workspace_bytes(int n, int batch) {
  size_t total = 0;
  carve(nullptr, n, batch, &total);
  return total;
}

void qr_input_buffers(void* workspace, int n, int batch, float** At, float** At_lo) {
  Workspace w = carve(workspace, n, batch, nullptr);
  *At = w.At;
  *At_lo = w.At_lo;
}

cudaError_t qr_q_t(int n, int batch, float* Qt, float* Qt_lo, float* Q, float* Q_lo, uint8_t* skip, float tol,
                   void* workspace, size_t workspace_bytes, int* status, cudaStream_t s) {
  if (n <= 0 || batch <= 0) return cudaSuccess;
  if (n > MAXC * COLS || batch > 65535 || (n & 3)) return cudaErrorInvalidValue;
  size_t need = 0;
  Workspace w = carve(workspace, n, batch, &need);
  if (workspace_bytes < need) return cudaErrorInvalidValue;
  if (!Qt) {  // the Q accumulation may reuse the factored matrix's buffers
    Qt = w.At;
    Qt_lo = w.At_lo;
  }
  const int npanel = (n + NB - 1) / NB;
  const int64_t nn = (int64_t)n * n;
  cudaError_t e;

  {
    ProfScope prof(kFamOther, 2.0 * nn * batch, 4.0 * nn * batch, s);
    frob_partial_kernel<<<dim3(NORM_CHUNKS, batch), 256, 0, s>>>(w.At, nn, w.part);
  }
  {
    ProfScope prof(kFamOther, 0, 8.0 * NORM_CHUNKS * batch, s);
    thresh_kernel<<<(batch + 127) / 128, 128, 0, s>>>(w.part, tol, batch, w.thresh);
  }
  const size_t smem = (size_t)NB * LDS * sizeof(float);
  e = cudaFuncSetAttribute(qr_panel_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;

  const int64_t pan_stride = (int64_t)npanel * n * NB;
  for (int pi = 0; pi < npanel; ++pi) {
    const int k = pi * NB, kb = std::min(NB, n - k);
    const int C = (n - k + COLS - 1) / COLS;
    PanelArgs a{w.At, w.Vt, w.Vt_lo, w.VTr, w.VTr_lo, w.VTq, w.VTq_lo, w.T, skip, w.dsign, w.thresh, status,
                n, k, kb, pi, npanel};
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
      // Householder work on the kb x (n-k) panel plus V T^T and V T: ~(4 kb^2 + 4 kb^2) (n-k)
      ProfScope prof(kFamQrPanel, 8.0 * (n - k) * kb * kb * batch, 24.0 * (n - k) * kb * batch, s);
      e = cudaLaunchKernelEx(&cfg, qr_panel_kernel, a);
    }
    if (e != cudaSuccess) return e;

    const int nc = n - k - kb;  // trailing rows of At (columns of P)
    if (nc <= 0) continue;
    const int m = n - k;        // positions from the panel's first pivot on
    const int64_t tr = (int64_t)(k + kb) * n + k;
    // W1 = At_trail Vt^T   (nc x kb)
    e = gemm_tc_nt(nc, kb, m, batch, op(w.At + tr, w.At_lo + tr, n, nn, batch),
                   op(w.Vt + (int64_t)k * n + k, w.Vt_lo + (int64_t)k * n + k, n, nn, batch),
                   out(w.W, w.W_lo, NB, (int64_t)n * NB, 1.f, 0.f, status), s);
    if (e != cudaSuccess) return e;
    // At_trail -= W1 (V T^T)^T
    e = rank_update(nc, m, kb, batch, w.W, NB, (int64_t)n * NB, w.VTr + (int64_t)k * NB, NB, (int64_t)n * NB,
                    w.At + tr, w.At_lo + tr, n, nn, s);
    if (e != cudaSuccess) return e;
  }

  {
    // Q^T = diag(d) H_n ... H_1 accumulated backwards: start from diag(d)
    ProfScope prof(kFamOther, 0, 8.0 * nn * batch, s);
    const int blocks = (int)std::min<int64_t>((nn + 255) / 256, 1024);
    signed_identity_kernel<<<dim3(blocks, batch), 256, 0, s>>>(Qt, Qt_lo, w.dsign, n);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  for (int pi = npanel - 1; pi >= 0; --pi) {
    const int k = pi * NB, kb = std::min(NB, n - k), m = n - k;
    const int64_t sub = (int64_t)k * n + k;
    // W = Qt_sub Vt^T  (m x kb)
    e = gemm_tc_nt(m, kb, m, batch, op(Qt + sub, Qt_lo + sub, n, nn, batch),
                   op(w.Vt + sub, w.Vt_lo + sub, n, nn, batch), out(w.W, w.W_lo, NB, (int64_t)n * NB, 1.f, 0.f, status),
                   s);
    if (e != cudaSuccess) return e;
    // Qt_sub -= W (V T)^T
    const int64_t vq = (int64_t)pi * n * NB + (int64_t)k * NB;
    e = rank_update(m, m, kb, batch, w.W, NB, (int64_t)n * NB, w.VTq + vq, NB, pan_stride, Qt + sub, Qt_lo + sub, n,
                    nn, s);
    if (e != cudaSuccess) return e;
  }
  if (Q) {
    ProfScope prof(kFamOther, 0, 12.0 * nn * batch, s);
    dim3 grid((n + 31) / 32, (n + 31) / 32, batch);
    transpose_out_kernel<<<grid, dim3(32, 8), 0, s>>>(Qt, Q, Q_lo, n);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaGetLastError();
}

cudaError_t qr_q(int n, int batch, const float* P, float* Q, uint8_t* skip, float tol, void* workspace,
                 size_t workspace_bytes, int* status, cudaStream_t s) {
  if (n <= 0 || batch <= 0) return cudaSuccess;
  size_t need = 0;
  Workspace w = carve(workspace, n, batch, &need);
  if (workspace_bytes < need || (n & 3)) return cudaErrorInvalidValue;
  // At = P^T and its lo part
  cudaError_t e = basis_split(P, nullptr, w.At, w.At_lo, n, batch, s);
  if (e != cudaSuccess) return e;
  return qr_q_t(n, batch, nullptr, nullptr, Q, nullptr, skip, tol, workspace, workspace_bytes, status, s);
}

}  // namespace soap
