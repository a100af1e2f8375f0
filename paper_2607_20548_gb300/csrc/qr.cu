// Batched Householder QR with explicit Q for the eigenbasis refresh
// (Alg. 1, "Eigenbasis Re-computation": Q <- QR(L_t Q).Q, every step as the
// appendix on eigh vs QR settles), with diag(R) >= 0, on tensor cores.
//
// The QR works on At = P^T (row j of At is column j of P), so every product of the
// blocked algorithm is a C = A B^T of K-major operands for the tcgen05 engine. It is
// blocked on two levels: 32-column panels are factored in distributed shared memory,
// and the trailing matrix -- the HBM-bound part -- is updated once per 128-column block
// of four panels:
//
//   for each block of 128 rows of At at k0 (columns k0..k0+127 of P):
//     for each 32-row panel at k in the block:
//       qr_panel_kernel (or qr_cols_kernel, then qr_panel_kernel) factors the panel rows,
//       writes the Householder vectors as rows of
//       Vt (row k+a = v_a over positions k0..n-1, zeros before its pivot) and as columns
//       of Vpos (position-major), extends the block's T (H_k0 ... H_k+31 = I - V T V^T)
//       by this panel's columns, and applies the panel's reflectors to the block's rows
//       after the panel;
//     VTr = V T^T and VTq = V T                     (tensor cores, K = 128)
//     trailing rows r >= k0+128: a_r <- a_r - (a_r V) T V^T, i.e.
//       W  = At_trail Vt^T                          (tensor cores: N = 128, K = positions)
//       At_trail -= W VTr^T                         (tensor cores: K = 128, C read in place)
//   then Q^T is accumulated backwards from diag(d) (d_j = sign of R_jj) one block at a
//   time, Q^T <- Q^T (I - V T^T V^T):
//       W = Qt_sub Vt^T ;  Qt_sub -= W VTq^T
//   and Q = (Q^T)^T is written with its lo part.
//
// The panel of an n x n matrix spans up to n positions; it is spread over a thread-block
// cluster of ceil((n-k)/512) CTAs (<= 16 for n <= 8192), 512 positions each, or, on a
// device that cannot run 16-CTA clusters of it, 1024 positions in clusters of <= 8 (a
// factor of at most 1024 rows takes one CTA of 1024 positions). Each Householder step needs
// one cluster-wide reduction: the squared norm of the column below the pivot and its dot
// products with the later panel columns are reduced together (the dot products with v
// follow from them once the reflector is known), and the partial sums are combined through
// distributed shared memory at one cluster barrier. No CTA waits on a flag: the only waits
// are hardware cluster barriers that every CTA of the cluster reaches unconditionally, and
// the tensor-core block product's mbarrier waits, which give up after a bounded time.
// For a batch of at least kSplitBatch factors the panel's 32 Householder steps run as a
// kernel of their own (qr_cols_kernel: two positions per thread, small enough for two CTAs
// per SM), and qr_panel_kernel<512, true> does the rest from the vectors it wrote.
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
#include <atomic>

#include "profile.h"
#include "soap_internal.h"
#include "tc_ptx.h"

namespace cg = cooperative_groups;

namespace soap {

namespace {

constexpr int NB = 32;            // panel width
constexpr int NBO = 128;          // block width: the trailing matrix is updated once per block
constexpr int PT = 512;           // threads per panel CTA
constexpr int MAXC = 16;          // largest cluster (16 needs the non-portable cluster size)
constexpr int NWARP = PT / 32;
constexpr int NREST = NBO - NB;   // most block rows after a panel
constexpr int KSPLIT = 8;         // split-K workspace: 8 partial n x NBO products (shorter ones split up to 16 ways)
constexpr uint64_t kWaitNs = 2000000000ull;  // bound of every mbarrier wait in the panel kernel

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
  float* Vpos;         // [batch][n][NBO] the block's Householder vectors, position-major
  float* Vpos_lo;
  float* T;            // [batch][NBO][NBO] the block's T (upper triangular)
  float* T_lo;
  float* Tt;           // [batch][NBO][NBO] T^T
  float* Tt_lo;
  float* Ypart;        // [batch][MAXC][NBO][NB] per-CTA partial products S V_panel
  uint8_t* skip;       // [batch][n]
  float* dsign;        // [batch][n] sign of R_pp (+1 for zero columns)
  float* tau;          // [batch][n] the reflectors' tau (handed from the column kernel)
  const float* thresh; // [batch]
  int* status;
  int n, k0, kbo, k, kb;  // block start and width, panel start and width
};

// x = hi + lo with hi = tf32(x) rounded to nearest and lo = tf32(x - hi): both as tf32 bits
__device__ __forceinline__ void tf32_split(float x, uint32_t& hi, uint32_t& lo) {
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(hi) : "f"(x));
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(lo) : "f"(x - __uint_as_float(hi)));
}

// d += a b for a 16 x 8 (rows) tf32 A fragment and an 8 x 8 (columns) B fragment, fp32 d
__device__ __forceinline__ void mma_tf32_16x8x8(float (&d)[4], const uint32_t (&a)[4], const uint32_t (&b)[2]) {
  asm volatile(
      "mma.sync.aligned.m16n8k8.row.col.f32.tf32.tf32.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}

// One 32-column panel, spread over a cluster: CTA c holds positions k + c*COLS .. of the
// panel rows in shared memory (row stride LDS, 16-byte aligned rows).
template <int COLS, bool SPLIT = false>
__global__ void __launch_bounds__(PT, 1) qr_panel_kernel(PanelArgs p) {
  static_assert(!SPLIT || COLS == PT, "the column loop runs on its own only for 512 positions per CTA");
  constexpr int LDS = COLS + 4;
  cg::cluster_group cluster = cg::this_cluster();
  const int c = (int)cluster.block_rank();
  const int C = (int)cluster.num_blocks();
  const int b = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

  extern __shared__ float4 smem_dyn[];
  float* sA = reinterpret_cast<float*>(smem_dyn);  // [NB][LDS]: panel row jj, position offset i
  __shared__ float s_part[2][NB];        // this CTA's partial [sigma | x . a_c]
  __shared__ float s_pv[2][NB];          // rank 0: pivot-row values [alpha | a_c,pivot]
  __shared__ float s_scal[2];            // tau and 1 / v0 of the current reflector
  __shared__ float s_w[NB];              // v^T a_c
  __shared__ __align__(16) float s_wl[NB];  // v^T a_(j+l) by offset l from the current row j
  __shared__ float s_red[NWARP][NB];     // per-warp partial sums of the register path
  __shared__ float s_tau[NB];
  __shared__ int s_skip[NB];
  __shared__ float s_dsign[NB];
  __shared__ float s_T[NB][NB + 1];
  __shared__ float s_Y[NBO][NB + 1];     // rank 0: S V_panel summed over the cluster
  __shared__ __align__(16) float s_Z[NREST][NB];  // (S_rest V_panel) T_panel, the in-block update
  // S V_panel: with 512 positions per CTA on the tensor cores (tcgen05): SV_STG chunks of S
  // (128 rows x 32 positions, 128-byte-swizzled) in flight, and two sets of S's lo part and
  // V's hi and lo parts; with 1024 positions as warp-level MMAs over STG staged chunks of
  // 128 x 36
  constexpr int STG = 2;
  constexpr int SV_STG = 4;
  constexpr int A_BYTES = NBO * 32 * 4;
  constexpr int B_BYTES = NB * 32 * 4;
  constexpr int SV_BYTES = COLS == PT ? SV_STG * A_BYTES + 2 * (A_BYTES + 2 * B_BYTES) + 1024 : STG * NBO * 36 * 4;
  __shared__ __align__(1024) uint8_t s_sv[SV_BYTES];
  __shared__ __align__(8) uint64_t s_mma_bar[2];
  __shared__ uint32_t s_tmem;

  const int n = p.n, k = p.k, kb = p.kb, k0 = p.k0, kbo = p.kbo;
  const int jb = k - k0;                // panel offset inside its block
  const int nrest = kbo - jb - kb;      // block rows after the panel
  const int64_t nn = (int64_t)n * n;
  float* At = p.At + (int64_t)b * nn;
  const int pos0 = k + c * COLS;  // first position held by this CTA
  const int npos = max(0, min(COLS, n - pos0));  // a multiple of 4

  const int npad = (npos + 31) & ~31;  // positions read by the chunked S V product
  {
    const int q4n = npad / 4;
    for (int e = tid; e < NB * q4n; e += PT) {
      const int jj = e / q4n, i = 4 * (e % q4n);
      const bool ok = jj < kb && i < npos;
      // after the column kernel: the panel's Householder vectors, as rows of Vt
      const float* rows = SPLIT ? p.Vt + (int64_t)b * nn : At;
      const float* src = ok ? rows + (int64_t)(k + jj) * n + pos0 + i : rows;
      const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(&sA[jj * LDS + i]));
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(d), "l"(src), "r"(ok ? 16 : 0) : "memory");
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
    asm volatile("cp.async.wait_group 0;" ::: "memory");
  }
  if constexpr (SPLIT) {
    if (tid < NB) s_tau[tid] = tid < kb ? p.tau[(int64_t)b * n + k + tid] : 0.f;
  }
  __syncthreads();
  const float thresh = p.thresh[b];
  int nonfinite = 0;

  if constexpr (SPLIT) {
    // the column loop ran in qr_cols_kernel
  } else if constexpr (COLS == PT) {
    // One position per thread: thread tid holds the panel rows' values at position tid in
    // registers, the current row first (a[l] = row j + l; rows past the panel are zero), so
    // that the per-column dot products and the reflector's update never touch shared memory;
    // only v (row j) is written back, for the phases after the loop.
    const int i = tid;
    const bool have = i < npos;
    float a[NB];
#pragma unroll
    for (int l = 0; l < NB; ++l) a[l] = (have && l < kb) ? sA[l * LDS + i] : 0.f;
    for (int j = 0; j < kb; ++j) {
      const int par = j & 1;
      // this position's share of sigma (l = 0) and of x . a_(j+l) (l > 0), for positions
      // strictly after the pivot (pivot = local position j of rank 0)
      const float x = (have && (c != 0 || i > j)) ? a[0] : 0.f;
      float v[NB];
      // transposing butterfly over the warp: lane l ends with the warp's sum for row j + l
#define SOAP_BFLY(o, nh)                                                   \
  {                                                                        \
    const bool up = (lane & (o)) != 0;                                     \
    _Pragma("unroll") for (int q = 0; q < (nh); ++q) {                     \
      const float keep = up ? v[q + (nh)] : v[q];                          \
      const float send = up ? v[q] : v[q + (nh)];                          \
      v[q] = keep + __shfl_xor_sync(0xffffffffu, send, (o));               \
    }                                                                      \
  }
      if (kb - j > NB / 2) {
#pragma unroll
        for (int l = 0; l < NB; ++l) v[l] = x * a[l];
        SOAP_BFLY(16, 16)
        SOAP_BFLY(8, 8)
        SOAP_BFLY(4, 4)
        SOAP_BFLY(2, 2)
        SOAP_BFLY(1, 1)
      } else {
        // at most 16 rows left (the rest of a[] is zero): the butterfly over the 16 live values
        // within each half-warp (lane l ends with row j + (l mod 16)), then across the halves
#pragma unroll
        for (int l = 0; l < NB / 2; ++l) v[l] = x * a[l];
        SOAP_BFLY(8, 8)
        SOAP_BFLY(4, 4)
        SOAP_BFLY(2, 2)
        SOAP_BFLY(1, 1)
        v[0] += __shfl_xor_sync(0xffffffffu, v[0], 16);
      }
#undef SOAP_BFLY
      s_red[warp][lane] = v[0];
      // rank 0's pivot position: alpha and the later rows' values there
      if (c == 0 && i == j) {
#pragma unroll
        for (int l = 0; l < NB; ++l)
          if (j + l < kb) s_pv[par][j + l] = a[l];
      }
      __syncthreads();
      if (warp == 0) {
        float sum = 0.f;
#pragma unroll
        for (int w = 0; w < NWARP; ++w) sum += s_red[w][lane];
        if (j + lane < kb) s_part[par][j + lane] = sum;
      }
      cluster.sync();
      // threads j..kb-1 reduce sigma and their own column's sum (in the same fixed order, so
      // they all derive the same reflector) and form v^T a_tid
      if (warp == 0) {
        s_wl[lane] = 0.f;
        __syncwarp();
      }
      if (tid >= j && tid < kb) {
        float ps[MAXC], pd[MAXC];
#pragma unroll
        for (int q = 0; q < MAXC; ++q) {
          if (q < C) {
            const float* rp = cluster.map_shared_rank(&s_part[par][0], q);
            ps[q] = rp[j];
            pd[q] = rp[tid];
          }
        }
        const float* pv0 = cluster.map_shared_rank(&s_pv[par][0], 0);
        const float alpha = pv0[j], apiv = pv0[tid];
        float d = 0.f, sigma = 0.f;
#pragma unroll
        for (int q = 0; q < MAXC; ++q) {
          if (q < C) {
            sigma += ps[q];
            d += pd[q];
          }
        }
        const float xnorm = sqrtf(fmaf(alpha, alpha, sigma));
        const bool skip = !(xnorm > thresh);
        float tau = 0.f, v0 = 1.f, rsign = 1.f;
        if (!skip) {
          if (sigma == 0.f) {
            rsign = alpha < 0.f ? -1.f : 1.f;   // H = I, R_pp = alpha
          } else {
            const float beta = alpha >= 0.f ? -xnorm : xnorm;
            v0 = alpha - beta;                   // same sign as alpha: no cancellation
            tau = (beta - alpha) / beta;
            rsign = beta < 0.f ? -1.f : 1.f;
          }
        }
        if (tid == j) {
          if (!isfinite(xnorm)) nonfinite = 1;
          s_tau[j] = tau;
          s_skip[j] = skip ? 1 : 0;
          s_dsign[j] = rsign;
          s_scal[0] = tau;
          s_scal[1] = tau != 0.f ? 1.f / v0 : 0.f;
        } else {
          s_wl[tid - j] = tau != 0.f ? apiv + d / v0 : 0.f;  // v^T a_tid, with v = x / v0 after the pivot
        }
      }
      __syncthreads();
      const float tau = s_scal[0], rv0 = s_scal[1];
      // v at this position (x / v0 after the pivot, 1 at it) and H_j = I - tau v v^T on the
      // later rows, shifting them down one register; positions before the pivot only shift
      if (have && (c != 0 || i >= j)) {
        const bool at_pivot = (c == 0 && i == j);
        const float vi = at_pivot ? 1.f : a[0] * rv0;
        if (!at_pivot) sA[j * LDS + i] = vi;
        if (tau != 0.f) {
          const float tv = tau * vi;
#pragma unroll
          for (int l4 = 0; l4 < NB / 4; ++l4) {
            const float4 w4 = reinterpret_cast<const float4*>(s_wl)[l4];
            if (l4 > 0) a[4 * l4 - 1] = fmaf(-tv, w4.x, a[4 * l4]);
            a[4 * l4] = fmaf(-tv, w4.y, a[4 * l4 + 1]);
            a[4 * l4 + 1] = fmaf(-tv, w4.z, a[4 * l4 + 2]);
            a[4 * l4 + 2] = fmaf(-tv, w4.w, a[4 * l4 + 3]);
          }
          a[NB - 1] = 0.f;
        } else {
#pragma unroll
          for (int l = 0; l < NB - 1; ++l) a[l] = a[l + 1];
          a[NB - 1] = 0.f;
        }
      } else {
#pragma unroll
        for (int l = 0; l < NB - 1; ++l) a[l] = a[l + 1];
        a[NB - 1] = 0.f;
      }
      __syncthreads();  // s_wl, s_red and s_scal are rewritten by the next column
    }
  } else {
    for (int j = 0; j < kb; ++j) {
      const int par = j & 1;
      // positions strictly after the pivot (pivot = local position j of rank 0)
      const int ibeg = (c == 0) ? j + 1 : 0;
      // partial sums over this CTA: sigma (cc = j) and x . a_cc (cc > j), kept locally; after
      // the cluster barrier the threads that need them read every CTA's copy. Warp w takes
      // columns j + w and j + w + 16 in one pass over x (kb - j <= 32 columns).
      {
        const int c1 = j + warp, c2 = c1 + NWARP;
        if (c1 < kb) {
          const bool h2 = c2 < kb;
          float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f, b0 = 0.f, b1 = 0.f, b2 = 0.f, b3 = 0.f;
          const float* xr = sA + j * LDS;
          const float* r1 = sA + c1 * LDS;
          const float* r2 = sA + (h2 ? c2 : c1) * LDS;
          int i = ibeg + lane;
          for (; i + 96 < npos; i += 128) {
            const float x0 = xr[i], x1 = xr[i + 32], x2 = xr[i + 64], x3 = xr[i + 96];
            a0 = fmaf(x0, r1[i], a0);
            a1 = fmaf(x1, r1[i + 32], a1);
            a2 = fmaf(x2, r1[i + 64], a2);
            a3 = fmaf(x3, r1[i + 96], a3);
            b0 = fmaf(x0, r2[i], b0);
            b1 = fmaf(x1, r2[i + 32], b1);
            b2 = fmaf(x2, r2[i + 64], b2);
            b3 = fmaf(x3, r2[i + 96], b3);
          }
          for (; i < npos; i += 32) {
            const float x0 = xr[i];
            a0 = fmaf(x0, r1[i], a0);
            b0 = fmaf(x0, r2[i], b0);
          }
          float da = (a0 + a1) + (a2 + a3), db = (b0 + b1) + (b2 + b3);
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) {
            da += __shfl_xor_sync(0xffffffffu, da, o);
            db += __shfl_xor_sync(0xffffffffu, db, o);
          }
          if (lane == 0) {
            s_part[par][c1] = da;
            if (h2) s_part[par][c2] = db;
          }
        }
      }
      if (c == 0 && tid >= j && tid < kb) s_pv[par][tid] = sA[tid * LDS + j];  // alpha (tid == j), a_tid at the pivot
      cluster.sync();
      // threads j..kb-1 reduce sigma and their own column's sum (in the same fixed order, so
      // they all derive the same reflector) and form v^T a_tid
      if (tid >= j && tid < kb) {
        float ps[MAXC], pd[MAXC];
#pragma unroll
        for (int q = 0; q < MAXC; ++q) {
          if (q < C) {
            const float* rp = cluster.map_shared_rank(&s_part[par][0], q);
            ps[q] = rp[j];
            pd[q] = rp[tid];
          }
        }
        const float* pv0 = cluster.map_shared_rank(&s_pv[par][0], 0);
        const float alpha = pv0[j], apiv = pv0[tid];
        float d = 0.f, sigma = 0.f;
#pragma unroll
        for (int q = 0; q < MAXC; ++q) {
          if (q < C) {
            sigma += ps[q];
            d += pd[q];
          }
        }
        const float xnorm = sqrtf(fmaf(alpha, alpha, sigma));
        const bool skip = !(xnorm > thresh);
        float tau = 0.f, v0 = 1.f, rsign = 1.f;
        if (!skip) {
          if (sigma == 0.f) {
            rsign = alpha < 0.f ? -1.f : 1.f;   // H = I, R_pp = alpha
          } else {
            const float beta = alpha >= 0.f ? -xnorm : xnorm;
            v0 = alpha - beta;                   // same sign as alpha: no cancellation
            tau = (beta - alpha) / beta;
            rsign = beta < 0.f ? -1.f : 1.f;
          }
        }
        if (tid == j) {
          if (!isfinite(xnorm)) nonfinite = 1;
          s_tau[j] = tau;
          s_skip[j] = skip ? 1 : 0;
          s_dsign[j] = rsign;
          s_scal[0] = tau;
          s_scal[1] = tau != 0.f ? 1.f / v0 : 0.f;
        } else if (tau != 0.f) {
          s_w[tid] = apiv + d / v0;  // v^T a_tid, with v = x / v0 after the pivot
        }
      }
      __syncthreads();
      const float tau = s_scal[0], rv0 = s_scal[1];

      // v after the pivot (x / v0, or 0 where H = I), and H_j = I - tau v v^T on the later
      // panel rows; every thread owns its positions
      const int piv = (c == 0) ? j : 0;  // local positions >= this take part
      for (int i = piv + tid; i < npos; i += PT) {
        const bool at_pivot = (c == 0 && i == j);
        const float vi = at_pivot ? 1.f : sA[j * LDS + i] * rv0;
        if (!at_pivot) sA[j * LDS + i] = vi;
        if (tau != 0.f) {
          const float tv = tau * vi;
          for (int cc = j + 1; cc < kb; ++cc) sA[cc * LDS + i] = fmaf(-tv, s_w[cc], sA[cc * LDS + i]);
        }
      }
      __syncthreads();
    }
  }
  if (nonfinite) atomicOr(p.status, kStatusQrBreakdown);

  // V with its unit diagonal and zeros before it (rank 0 holds the first kb positions; the
  // column kernel wrote them so)
  if (!SPLIT && c == 0) {
    for (int e = tid; e < kb * kb; e += PT) {
      const int jj = e / kb, i = e % kb;
      if (i < jj) sA[jj * LDS + i] = 0.f;
      else if (i == jj) sA[jj * LDS + i] = 1.f;
    }
  }
  __syncthreads();

  // V as rows of Vt (zeros at the block's positions before the panel) and as columns jb..
  // of the block's position-major Vpos
  float* Vt = p.Vt + (int64_t)b * nn;
  float* Vt_lo = p.Vt_lo + (int64_t)b * nn;
  float* Vpos = p.Vpos + (int64_t)b * n * NBO;
  float* Vpos_lo = p.Vpos_lo + (int64_t)b * n * NBO;
  if constexpr (!SPLIT) {  // (the column kernel wrote Vt)
    const int q4n = npos / 4;
    for (int e = tid; e < kb * q4n; e += PT) {
      const int jj = e / q4n, q = e - jj * q4n;
      const int64_t o = (int64_t)(k + jj) * n + pos0 + 4 * q;
      const float4 v = *reinterpret_cast<const float4*>(&sA[jj * LDS + 4 * q]);
      *reinterpret_cast<float4*>(Vt + o) = v;
      *reinterpret_cast<float4*>(Vt_lo + o) = make_float4(tf32_lo(v.x), tf32_lo(v.y), tf32_lo(v.z), tf32_lo(v.w));
    }
  }
  for (int e = tid; e < npos * (NB / 4); e += PT) {
    const int i = e >> 3, g4 = 4 * (e & 7);  // rows kb.. of sA are zero
    const float4 v = make_float4(sA[g4 * LDS + i], sA[(g4 + 1) * LDS + i], sA[(g4 + 2) * LDS + i], sA[(g4 + 3) * LDS + i]);
    const int64_t o = (int64_t)(pos0 + i) * NBO + jb + g4;
    *reinterpret_cast<float4*>(Vpos + o) = v;
    *reinterpret_cast<float4*>(Vpos_lo + o) = make_float4(tf32_lo(v.x), tf32_lo(v.y), tf32_lo(v.z), tf32_lo(v.w));
  }
  if (c == 0) {
    if (!SPLIT)
      for (int jj = 0; jj < kb; ++jj)
        for (int i = tid; i < jb; i += PT) {
          const int64_t o = (int64_t)(k + jj) * n + k0 + i;
          Vt[o] = 0.f;
          Vt_lo[o] = 0.f;
        }
    for (int e = tid; e < jb * NB; e += PT) {
      const int64_t o = (int64_t)(k0 + e / NB) * NBO + jb + e % NB;
      Vpos[o] = 0.f;
      Vpos_lo[o] = 0.f;
    }
  }
  __syncthreads();  // this CTA's Vt rows are read back below

  // Y = S V_panel over this CTA's positions, S = the block's rows k0 .. k0+kbo-1: the block's
  // Householder vectors so far (rows before the panel's end, from Vt) and the block rows still
  // to be factored (from At), with both operands split into tf32 hi and lo parts (four
  // products: fp32 accuracy), each 32-position chunk summed afresh and added to fp32 registers,
  // so that the tensor core's own accumulation never runs longer than 32 positions.
  if constexpr (COLS == PT) {
    // On the tcgen05 tensor cores: D[128 x 32] (tensor memory) = S chunk (A: 128 rows x 32
    // positions) x V chunk^T (B: 32 rows x 32 positions), both K-major in the 128-byte-swizzled
    // layout. S's rows other than the panel's are copied with cp.async straight into that
    // layout, SV_STG - 1 chunks ahead, and each thread forms the lo part of the units it copied;
    // the panel's rows of S and the V chunk (hi and lo) come from sA. Two accumulators and two
    // lo sets alternate: while the MMAs of chunk ch run, warps 0-3 drain chunk ch-1 (warp w
    // reads lanes 32w..) and its S stage is refilled.
    uint8_t* sv = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(s_sv) + 1023) & ~uintptr_t(1023));
    uint8_t* st_a = sv;                          // [SV_STG] S chunks (fp32, read by the MMA as its hi part)
    uint8_t* st_lo = sv + SV_STG * A_BYTES;      // [2] S lo | V hi | V lo
    constexpr int LO_SET = A_BYTES + 2 * B_BYTES;
    const int nchunk = (npos + 31) / 32;
    if (tid == 0) {
      tc::mbar_init(&s_mma_bar[0], 1);
      tc::mbar_init(&s_mma_bar[1], 1);
      asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 0) {
      asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(tc::smem_u32(&s_tmem)),
                   "r"(64));
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = s_tmem;
    // byte offset of 16-byte unit q of row r in a tile of 128-byte rows, swizzled within
    // 1024-byte groups of 8 rows
    auto swz16 = [](int r, int q) { return (r >> 3) * 1024 + (r & 7) * 128 + ((q ^ (r & 7)) << 4); };
    auto issue = [&](int ch) {
      uint8_t* dst = st_a + (ch % SV_STG) * A_BYTES;
      for (int u = tid; u < NBO * 8; u += PT) {
        const int r = u >> 3, q = u & 7;
        if (r >= jb && r < jb + NB) continue;  // the panel's own rows: V, from sA
        const int row = k0 + r, i = ch * 32 + 4 * q;
        const bool ok = r < kbo && i < npos;  // zero-filled outside the block and past the positions
        const float* src = ok ? (r < jb ? Vt : At) + (int64_t)row * n + pos0 + i : At;
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(tc::smem_u32(dst + swz16(r, q))),
                     "l"(src), "r"(ok ? 16 : 0)
                     : "memory");
      }
    };
    auto lo4 = [](float4 x) { return make_float4(tf32_lo(x.x), tf32_lo(x.y), tf32_lo(x.z), tf32_lo(x.w)); };
    float y[NB];
#pragma unroll
    for (int l = 0; l < NB; ++l) y[l] = 0.f;
    for (int st0 = 0; st0 < SV_STG - 1; ++st0) {
      if (st0 < nchunk) issue(st0);
      asm volatile("cp.async.commit_group;" ::: "memory");
    }
    int issued = 0;  // chunks whose MMAs were issued
    bool aborted = false, bad = false;
    for (int ch = 0; ch < nchunk; ++ch) {
      const int set = ch & 1;
      // this thread's copies of chunk ch have landed: their lo parts; the panel's rows of S and
      // the V chunk (hi and lo) from sA
      asm volatile("cp.async.wait_group %0;" ::"n"(SV_STG - 2) : "memory");
      {
        uint8_t* a = st_a + (ch % SV_STG) * A_BYTES;
        uint8_t* lo = st_lo + set * LO_SET;
        for (int u = tid; u < NBO * 8; u += PT) {
          const int r = u >> 3;
          if (r >= jb && r < jb + NB) continue;
          const int off = swz16(r, u & 7);
          *reinterpret_cast<float4*>(lo + off) = lo4(*reinterpret_cast<const float4*>(a + off));
        }
        uint8_t* bh = lo + A_BYTES;
        uint8_t* bl = bh + B_BYTES;
        for (int u = tid; u < NB * 8; u += PT) {
          const int jj = u >> 3, q = u & 7;
          const float4 x = *reinterpret_cast<const float4*>(&sA[jj * LDS + ch * 32 + 4 * q]);
          const float4 xl = lo4(x);
          const int off = swz16(jj, q), offa = swz16(jb + jj, q);
          *reinterpret_cast<float4*>(bh + off) = x;
          *reinterpret_cast<float4*>(bl + off) = xl;
          *reinterpret_cast<float4*>(a + offa) = x;
          *reinterpret_cast<float4*>(lo + offa) = xl;
        }
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      if (__syncthreads_or(bad)) {
        aborted = true;
        break;
      }
      // the MMAs of chunk ch (its lo set and accumulator were released in the previous pass)
      if (tid == 0) {
        tc::tc_fence_after();
        constexpr uint32_t idesc = tc::idesc_tf32(NBO, NB);
        const uint32_t d = tmem + (uint32_t)(set * 32);
        const uint32_t a_hi = tc::smem_u32(st_a + (ch % SV_STG) * A_BYTES);
        const uint32_t a_lo = tc::smem_u32(st_lo + set * LO_SET);
        const uint32_t b_hi = a_lo + A_BYTES;
        const uint32_t b_lo = b_hi + B_BYTES;
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
          const uint32_t off = kk * 32;  // 8 tf32 = 32 bytes along the positions
          tc::umma_tf32(d, tc::desc_sw128(a_lo + off), tc::desc_sw128(b_lo + off), idesc, kk != 0);
          tc::umma_tf32(d, tc::desc_sw128(a_lo + off), tc::desc_sw128(b_hi + off), idesc, 1u);
          tc::umma_tf32(d, tc::desc_sw128(a_hi + off), tc::desc_sw128(b_lo + off), idesc, 1u);
          tc::umma_tf32(d, tc::desc_sw128(a_hi + off), tc::desc_sw128(b_hi + off), idesc, 1u);
        }
        tc::umma_commit(&s_mma_bar[set]);
      }
      issued = ch + 1;
      // while they run: chunk ch-1's MMAs have completed, so its accumulator is drained and its
      // S stage refilled with chunk ch + SV_STG - 1
      if (ch >= 1) {
        bool ok = tc::mbar_wait(&s_mma_bar[(ch - 1) & 1], ((ch - 1) >> 1) & 1, kWaitNs);
        ok = __all_sync(0xffffffffu, ok);
        if (!ok) {
          bad = true;
        } else if (warp < 4) {
          float v[32];
          tc::tmem_ld32(tmem + (uint32_t)(((ch - 1) & 1) * 32) + ((uint32_t)(32 * warp) << 16), v);
#pragma unroll
          for (int l = 0; l < NB; ++l) y[l] += v[l];
        }
      }
      if (!bad && ch + SV_STG - 1 < nchunk) issue(ch + SV_STG - 1);
      asm volatile("cp.async.commit_group;" ::: "memory");
      tc::tc_fence_before();
    }
    // the last chunk's sum; after a wait that gave up, only the wait for every issued MMA (with
    // the full bound), so that the tensor memory is not freed under one
    bool ok_last = true;
    if (issued > 0)
      ok_last = __all_sync(0xffffffffu, tc::mbar_wait(&s_mma_bar[(issued - 1) & 1], ((issued - 1) >> 1) & 1, kWaitNs));
    if (!aborted && !bad && ok_last && issued > 0 && warp < 4) {
      float v[32];
      tc::tmem_ld32(tmem + (uint32_t)(((issued - 1) & 1) * 32) + ((uint32_t)(32 * warp) << 16), v);
#pragma unroll
      for (int l = 0; l < NB; ++l) y[l] += v[l];
    }
    if (aborted || bad || !ok_last) atomicOr(p.status, kStatusTimeout);
    asm volatile("cp.async.wait_all;" ::: "memory");
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 0) {
      tc::tc_fence_after();
      asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(64));
    }
    // this CTA's partial product, kept in shared memory (the S stages are free) for the cluster
    if (warp < 4) {
      float* yp = reinterpret_cast<float*>(sv) + (32 * warp + lane) * NB;
#pragma unroll
      for (int l4 = 0; l4 < NB / 4; ++l4)
        *reinterpret_cast<float4*>(yp + 4 * l4) = make_float4(y[4 * l4], y[4 * l4 + 1], y[4 * l4 + 2], y[4 * l4 + 3]);
    }
  } else
  // With 1024 positions per CTA (factors of at most 1024 rows): S is streamed through shared
  // memory in 32-position chunks (cp.async, STG buffers, rows padded to 36 floats), and the
  // product runs as warp-level m16n8k8 TF32 MMAs. Warp w owns rows 16 (w mod 8) .. +15 and
  // columns 16 (w / 8) .. +15.
  {
    static_assert(NBO == 128 && NB == 32 && NWARP == 16, "8 x 2 warp tiles of 16 x 16");
    constexpr int CH = 32;       // positions per chunk
    constexpr int CHP = CH + 4;  // padded row stride of a staged chunk
    const int gq = lane >> 2, tg = lane & 3;
    const int m0 = 16 * (warp & 7), nb = 16 * (warp >> 3);
    float y[2][4];
#pragma unroll
    for (int e = 0; e < 4; ++e) y[0][e] = y[1][e] = 0.f;
    const int nchunk = (npos + CH - 1) / CH;
    auto issue = [&](int ch, int buf) {
      float* dst = reinterpret_cast<float*>(s_sv) + buf * NBO * CHP;
      for (int e = tid; e < NBO * (CH / 4); e += PT) {
        const int r = e / (CH / 4), q4 = e % (CH / 4);
        const int row = k0 + r, i = ch * CH + 4 * q4;
        const bool ok = r < kbo && i < npos;
        const float* src = ok ? ((row < k + kb) ? Vt : At) + (int64_t)row * n + pos0 + i : At;
        const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(dst + r * CHP + 4 * q4));
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(d), "l"(src), "r"(ok ? 16 : 0) : "memory");
      }
      asm volatile("cp.async.commit_group;" ::: "memory");
    };
    for (int st0 = 0; st0 < STG - 1; ++st0) {
      if (st0 < nchunk) issue(st0, st0);
      else asm volatile("cp.async.commit_group;" ::: "memory");
    }
    for (int ch = 0; ch < nchunk; ++ch) {
      if (ch + STG - 1 < nchunk) issue(ch + STG - 1, (ch + STG - 1) % STG);
      else asm volatile("cp.async.commit_group;" ::: "memory");  // keeps the group count uniform
      asm volatile("cp.async.wait_group %0;" ::"n"(STG - 1) : "memory");
      __syncthreads();
      const float* st = reinterpret_cast<const float*>(s_sv) + (ch % STG) * NBO * CHP;
      const int i0 = ch * CH;
      float d[2][4];
#pragma unroll
      for (int e = 0; e < 4; ++e) d[0][e] = d[1][e] = 0.f;
#pragma unroll
      for (int ks = 0; ks < CH / 8; ++ks) {
        // positions past npos are zero in the staged chunk and in V (zero-filled copies)
        const int kk = 8 * ks;
        const float av[4] = {st[(m0 + gq) * CHP + kk + tg], st[(m0 + gq + 8) * CHP + kk + tg],
                             st[(m0 + gq) * CHP + kk + tg + 4], st[(m0 + gq + 8) * CHP + kk + tg + 4]};
        uint32_t ah[4], al[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) tf32_split(av[e], ah[e], al[e]);
#pragma unroll
        for (int nt = 0; nt < 2; ++nt) {
          const float* vr = sA + (nb + 8 * nt + gq) * LDS + i0 + kk + tg;
          uint32_t bh[2], bl[2];
          tf32_split(vr[0], bh[0], bl[0]);
          tf32_split(vr[4], bh[1], bl[1]);
          mma_tf32_16x8x8(d[nt], al, bl);
          mma_tf32_16x8x8(d[nt], al, bh);
          mma_tf32_16x8x8(d[nt], ah, bl);
          mma_tf32_16x8x8(d[nt], ah, bh);
        }
      }
#pragma unroll
      for (int nt = 0; nt < 2; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) y[nt][e] += d[nt][e];
      __syncthreads();  // this buffer is refilled STG - 1 chunks later
    }
    float* yp = p.Ypart + ((int64_t)b * MAXC + c) * NBO * NB;
#pragma unroll
    for (int nt = 0; nt < 2; ++nt) {
      const int col = nb + 8 * nt + 2 * tg;
      *reinterpret_cast<float2*>(yp + (m0 + gq) * NB + col) = make_float2(y[nt][0], y[nt][1]);
      *reinterpret_cast<float2*>(yp + (m0 + gq + 8) * NB + col) = make_float2(y[nt][2], y[nt][3]);
    }
  }
  // T_panel from the Gram rows of Y, then U = X T_panel (in place) and Z (rows after the panel);
  // every thread of the CTA takes part (the barriers inside)
  auto form_tuz = [&]() {
    // T of the panel from its Gram matrix g (rows jb.. of Y): T^-1 = diag(1/tau) + striu(g)
    // (H_1 ... H_kb = I - V T V^T); a reflector with tau = 0 (v = 0) gets a zero row and column.
    // Warp w solves columns w and w + 16 by back substitution, lane i holding x_i:
    //   x_i = tau_i (delta_{i,cc} - sum_{i < l <= cc} g_il x_l)   (tau_i read as 1 where it is 0)
    // Each solved x_l is broadcast once and every lane i < l adds g_il x_l to its running sum,
    // so a step costs one shuffle instead of a warp-wide reduction.
    for (int cc = warp; cc < NB; cc += NWARP) {
      float x = 0.f, acc = 0.f;
      for (int l = cc; l >= 0; --l) {
        const float g = s_Y[jb + lane][l];
        if (lane == l) {
          const float tl = l < kb ? s_tau[l] : 0.f;
          x = ((l == cc ? 1.f : 0.f) - acc) * (tl != 0.f ? tl : 1.f);
        }
        const float xl = __shfl_sync(0xffffffffu, x, l);
        if (lane < l) acc = fmaf(g, xl, acc);
      }
      const bool live = cc < kb && s_tau[cc] != 0.f;
      s_T[lane][cc] = (live && lane <= cc && lane < kb && s_tau[lane] != 0.f) ? x : 0.f;
    }
    __syncthreads();
    // U = X T_panel with X = V_before^T V_panel (rows 0..jb-1 of Y), in place, and
    // Z = (S_rest V_panel) T_panel for the block rows after the panel: thread (r, g) forms
    // columns 8g .. 8g+7 of row r
    {
      const int r = tid >> 2, g8 = (tid & 3) * 8;
      const bool act = r < kbo && (r < jb || r >= jb + kb);
      float x[NB];
#pragma unroll
      for (int l = 0; l < NB; ++l) x[l] = act ? s_Y[r][l] : 0.f;
      __syncthreads();  // every row is read before U overwrites it
      if (act) {
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int cc = g8 + u;
          float acc = 0.f;
#pragma unroll
          for (int l = 0; l < NB; ++l)
            if (l <= cc) acc = fmaf(x[l], s_T[l][cc], acc);
          if (r < jb) s_Y[r][cc] = acc;
          else s_Z[r - jb - kb][cc] = acc;
        }
      }
    }
    __syncthreads();
  };
  if constexpr (COLS == PT) {
    // The partial products reduced through distributed shared memory: CTA c sums rows
    // r = c mod C of every CTA's partial, in a fixed order, and every CTA then gathers the summed
    // rows and forms T_panel, U and Z itself (the same values on every CTA).
    uint8_t* sv = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(s_sv) + 1023) & ~uintptr_t(1023));
    float* P_own = reinterpret_cast<float*>(sv);
    float* Ysum = P_own + NBO * NB;
    cluster.sync();  // every CTA's partial is in place
    for (int r = c + C * warp; r < kbo; r += C * NWARP) {
      float part[MAXC];
#pragma unroll
      for (int q = 0; q < MAXC; ++q) part[q] = q < C ? cluster.map_shared_rank(P_own, q)[r * NB + lane] : 0.f;
      float sum = 0.f;
#pragma unroll
      for (int q = 0; q < MAXC; ++q) sum += part[q];
      Ysum[r * NB + lane] = sum;
    }
    cluster.sync();  // every summed row is in place
    for (int e = tid; e < kbo * NB; e += PT) s_Y[e / NB][e % NB] = cluster.map_shared_rank(Ysum, (e / NB) % C)[e];
    // the peers may read this CTA's summed rows until they have gathered theirs: arrive now and
    // wait at the end of the kernel
    asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
    __syncthreads();
    form_tuz();
    __syncthreads();
    if (!SPLIT && c == 0 && tid < kb) {
      p.skip[(int64_t)b * n + k + tid] = (uint8_t)s_skip[tid];
      p.dsign[(int64_t)b * n + k + tid] = s_dsign[tid];
    }
  } else {
    cluster.sync();  // orders the partials in global memory before rank 0 reads them
    // rank 0 sums the partials, forms T_panel, U = X T_panel and Z, and hands Z, U and T_panel
    // to the cluster through global memory (rank 0's slots of Ypart, free once it has summed
    // them): Z at 0, U at 3072 (jb <= 96 rows), T_panel at 6144 floats
    float* xg = p.Ypart + (int64_t)b * MAXC * NBO * NB;
    float* Ug = xg + NREST * NB;
    float* Tpg = xg + 2 * NREST * NB;
    if (c == 0) {
      // sum the partials in a fixed order
      const float* yp = p.Ypart + (int64_t)b * MAXC * NBO * NB;
      for (int e = tid; e < kbo * NB; e += PT) {
        float part[MAXC];
#pragma unroll
        for (int q = 0; q < MAXC; ++q) part[q] = q < C ? yp[(int64_t)q * NBO * NB + e] : 0.f;
        float sum = 0.f;
#pragma unroll
        for (int q = 0; q < MAXC; ++q) sum += part[q];
        s_Y[e / NB][e % NB] = sum;
      }
      __syncthreads();
      form_tuz();
      __syncthreads();
      for (int e = tid; e < nrest * NB; e += PT) xg[e] = s_Z[e / NB][e % NB];
      for (int e = tid; e < jb * NB; e += PT) Ug[e] = s_Y[e / NB][e % NB];
      for (int e = tid; e < NB * NB; e += PT) Tpg[e] = s_T[e / NB][e % NB];
      if (tid < kb) {
        p.skip[(int64_t)b * n + k + tid] = (uint8_t)s_skip[tid];
        p.dsign[(int64_t)b * n + k + tid] = s_dsign[tid];
      }
    }
    cluster.sync();  // Z, U and T_panel in global memory are visible to the cluster
    if (c != 0) {
      for (int e = tid; e < nrest * NB; e += PT) s_Z[e / NB][e % NB] = xg[e];
      for (int e = tid; e < jb * NB; e += PT) s_Y[e / NB][e % NB] = Ug[e];
      for (int e = tid; e < NB * NB; e += PT) s_T[e / NB][e % NB] = Tpg[e];
    }
    __syncthreads();
  }
  // the block's T, rows spread over the cluster (row r by CTA r mod C): column block jb =
  // [-T_before U ; T_panel ; 0] and the row block jb left of it = 0
  {
    float* T = p.T + (int64_t)b * NBO * NBO;
    float* T_lo = p.T_lo + (int64_t)b * NBO * NBO;
    float* Tt = p.Tt + (int64_t)b * NBO * NBO;
    float* Tt_lo = p.Tt_lo + (int64_t)b * NBO * NBO;
    // the rows of T_before (written by the block's earlier panels) that this CTA's rows need,
    // staged in shared memory with independent loads: the S V area is free (on the cluster path
    // past its first 32 KB, the summed rows that peers may still read)
    constexpr int TBS = NBO - NB;  // jb <= 96
    float* Tb = reinterpret_cast<float*>(
        COLS == PT ? ((reinterpret_cast<uintptr_t>(s_sv) + 1023) & ~uintptr_t(1023)) + 2 * NBO * NB * sizeof(float)
                   : reinterpret_cast<uintptr_t>(s_sv));
    static_assert(TBS * TBS * sizeof(float) <= (COLS == PT ? SV_BYTES - 1024 - 2 * NBO * NB * sizeof(float) : SV_BYTES),
                  "T_before staging");
    const int nrl = jb > c ? (jb - c + C - 1) / C : 0;  // this CTA's rows r = c + C rl below jb
    for (int e = tid; e < nrl * jb; e += PT) {
      const int rl = e / jb, l = e - rl * jb, rr = c + C * rl;
      Tb[rl * TBS + l] = l >= rr ? T[rr * NBO + l] : 0.f;
    }
    __syncthreads();
    // one entry (row r = c + C rl, column jb + cc) per work unit, the 32 units of a row on
    // consecutive threads: the triangular product's long rows are spread over all threads in
    // turn. On the cluster path the column block is also staged transposed, so that Tt's rows
    // are written with consecutive stores.
    const int nr = (NBO - c + C - 1) / C;  // this CTA's rows
    float* stt = COLS == PT ? Tb + TBS * TBS : nullptr;  // [NB][NBO]: entry (cc, rl)
    static_assert(COLS != PT || (TBS * TBS + NB * NBO) * sizeof(float) <= SV_BYTES - 1024 - 2 * NBO * NB * sizeof(float),
                  "T column block staging");
    for (int u = tid; u < nr * NB; u += PT) {
      const int rl = u >> 5, cc = u & 31, r = c + C * rl;
      float t = 0.f;
      if (r < jb) {
        const float* tb_row = Tb + rl * TBS;
#pragma unroll 4
        for (int l = r; l < jb; ++l) t = fmaf(-tb_row[l], s_Y[l][cc], t);
      } else if (r < jb + NB) {
        t = s_T[r - jb][cc];
      }
      const int col = jb + cc;
      T[r * NBO + col] = t;
      T_lo[r * NBO + col] = tf32_lo(t);
      if (COLS == PT) {
        stt[cc * NBO + rl] = t;
      } else {
        Tt[col * NBO + r] = t;
        Tt_lo[col * NBO + r] = tf32_lo(t);
      }
    }
    if (COLS == PT) {
      __syncthreads();
      for (int e = tid; e < NB * nr; e += PT) {
        const int cc = e / nr, rl = e - cc * nr;
        const float t = stt[cc * NBO + rl];
        Tt[(jb + cc) * NBO + c + C * rl] = t;
        Tt_lo[(jb + cc) * NBO + c + C * rl] = tf32_lo(t);
      }
    }
    // the row block jb left of the panel is zero: T's rows jb.. and Tt's columns jb.. there
    for (int e = tid; e < NB * jb; e += PT) {
      const int rr = jb + e / jb, col = e % jb;
      if (rr % C != c) continue;
      T[rr * NBO + col] = 0.f;
      T_lo[rr * NBO + col] = 0.f;
    }
    for (int e = tid; e < NB * jb; e += PT) {
      const int col = e / NB, rr = jb + e % NB;
      if (rr % C != c) continue;
      Tt[col * NBO + rr] = 0.f;
      Tt_lo[col * NBO + rr] = 0.f;
    }
  }

  // the panel's reflectors on the block rows after it: a_r -= Z_r V^T at this CTA's
  // positions, eight rows at a time (eight independent loads in flight), then four, then one
  for (int i = tid; i < npos; i += PT) {
    float v[NB];
#pragma unroll
    for (int jj = 0; jj < NB; ++jj) v[jj] = sA[jj * LDS + i];
    float* a = At + (int64_t)(k + kb) * n + pos0 + i;
    int r = 0;
    for (; r + 8 <= nrest; r += 8) {
      float x[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) x[u] = a[(int64_t)(r + u) * n];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        float acc = 0.f;
#pragma unroll
        for (int j4 = 0; j4 < NB / 4; ++j4) {
          const float4 z = *reinterpret_cast<const float4*>(&s_Z[r + u][4 * j4]);
          acc = fmaf(z.x, v[4 * j4], fmaf(z.y, v[4 * j4 + 1], fmaf(z.z, v[4 * j4 + 2], fmaf(z.w, v[4 * j4 + 3], acc))));
        }
        a[(int64_t)(r + u) * n] = x[u] - acc;
      }
    }
    for (; r + 4 <= nrest; r += 4) {
      float x[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) x[u] = a[(int64_t)(r + u) * n];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        float acc = 0.f;
#pragma unroll
        for (int j4 = 0; j4 < NB / 4; ++j4) {
          const float4 z = *reinterpret_cast<const float4*>(&s_Z[r + u][4 * j4]);
          acc = fmaf(z.x, v[4 * j4], fmaf(z.y, v[4 * j4 + 1], fmaf(z.z, v[4 * j4 + 2], fmaf(z.w, v[4 * j4 + 3], acc))));
        }
        a[(int64_t)(r + u) * n] = x[u] - acc;
      }
    }
    for (; r < nrest; ++r) {
      float acc = 0.f;
#pragma unroll
      for (int jj = 0; jj < NB; ++jj) acc = fmaf(s_Z[r][jj], v[jj], acc);
      a[(int64_t)r * n] -= acc;
    }
  }
  if constexpr (COLS == PT) asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// The column loop of a 32-column panel on its own, for factors of more than 1024 rows (the
// Householder steps of qr_panel_kernel's register path): CTA c of the cluster holds positions
// k + 512 c .. of the panel rows, two per thread, in registers. It writes V as rows of Vt with
// their lo parts (zeros before each pivot and at the block's positions before the panel, one at
// the pivot), and tau, skip and dsign; qr_panel_kernel<512, true> then forms the block product,
// T and the in-block update from them. With 256 threads of at most 128 registers and a few KB of
// shared memory, two of these CTAs fit on one SM, so the latency-bound loop holds half an SM
// instead of a whole one.
constexpr int PTA = 256;
constexpr int NWA = PTA / 32;

__global__ void __launch_bounds__(PTA, 2) qr_cols_kernel(PanelArgs p) {
  constexpr int COLS = 2 * PTA;
  cg::cluster_group cluster = cg::this_cluster();
  const int c = (int)cluster.block_rank();
  const int C = (int)cluster.num_blocks();
  const int b = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  __shared__ float s_part[2][NB];
  __shared__ float s_pv[2][NB];
  __shared__ float s_scal[2];
  __shared__ __align__(16) float s_wl[NB];
  __shared__ float s_red[NWA][NB];

  const int n = p.n, k = p.k, kb = p.kb, k0 = p.k0;
  const int jb = k - k0;
  const int64_t nn = (int64_t)n * n;
  const float* At = p.At + (int64_t)b * nn;
  float* Vt = p.Vt + (int64_t)b * nn;
  float* Vt_lo = p.Vt_lo + (int64_t)b * nn;
  const int pos0 = k + c * COLS;
  const int npos = max(0, min(COLS, n - pos0));
  const int i0 = tid, i1 = tid + PTA;  // this thread's positions; i1 is past every pivot
  const bool have0 = i0 < npos, have1 = i1 < npos;
  float a0[NB], a1[NB];
#pragma unroll
  for (int l = 0; l < NB; ++l) {
    a0[l] = (have0 && l < kb) ? At[(int64_t)(k + l) * n + pos0 + i0] : 0.f;
    a1[l] = (have1 && l < kb) ? At[(int64_t)(k + l) * n + pos0 + i1] : 0.f;
  }
  const float thresh = p.thresh[b];
  int nonfinite = 0;
  for (int j = 0; j < kb; ++j) {
    const int par = j & 1;
    // this thread's shares of sigma and of x . a_(j+l), positions strictly after the pivot
    const float x0 = (have0 && (c != 0 || i0 > j)) ? a0[0] : 0.f;
    const float x1 = have1 ? a1[0] : 0.f;
    float v[NB];
#define SOAP_BFLY(o, nh)                                                   \
  {                                                                        \
    const bool up = (lane & (o)) != 0;                                     \
    _Pragma("unroll") for (int q = 0; q < (nh); ++q) {                     \
      const float keep = up ? v[q + (nh)] : v[q];                          \
      const float send = up ? v[q] : v[q + (nh)];                          \
      v[q] = keep + __shfl_xor_sync(0xffffffffu, send, (o));               \
    }                                                                      \
  }
    if (kb - j > NB / 2) {
#pragma unroll
      for (int l = 0; l < NB; ++l) v[l] = fmaf(x1, a1[l], x0 * a0[l]);
      SOAP_BFLY(16, 16)
      SOAP_BFLY(8, 8)
      SOAP_BFLY(4, 4)
      SOAP_BFLY(2, 2)
      SOAP_BFLY(1, 1)
    } else {
#pragma unroll
      for (int l = 0; l < NB / 2; ++l) v[l] = fmaf(x1, a1[l], x0 * a0[l]);
      SOAP_BFLY(8, 8)
      SOAP_BFLY(4, 4)
      SOAP_BFLY(2, 2)
      SOAP_BFLY(1, 1)
      v[0] += __shfl_xor_sync(0xffffffffu, v[0], 16);
    }
#undef SOAP_BFLY
    s_red[warp][lane] = v[0];
    if (c == 0 && i0 == j) {
#pragma unroll
      for (int l = 0; l < NB; ++l)
        if (j + l < kb) s_pv[par][j + l] = a0[l];
    }
    __syncthreads();
    if (warp == 0) {
      float sum = 0.f;
#pragma unroll
      for (int w = 0; w < NWA; ++w) sum += s_red[w][lane];
      if (j + lane < kb) s_part[par][j + lane] = sum;
    }
    cluster.sync();
    if (warp == 0) {
      s_wl[lane] = 0.f;
      __syncwarp();
    }
    if (tid >= j && tid < kb) {
      // the cluster's partial sums in rank order (the same order on every CTA), four peers'
      // loads in flight at a time
      const float* pv0 = cluster.map_shared_rank(&s_pv[par][0], 0);
      const float alpha = pv0[j], apiv = pv0[tid];
      float d = 0.f, sigma = 0.f;
#pragma unroll
      for (int q0 = 0; q0 < MAXC; q0 += 4) {
        if (q0 < C) {
          float ps[4], pd[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const float* rp = cluster.map_shared_rank(&s_part[par][0], q0 + u < C ? q0 + u : 0);
            ps[u] = rp[j];
            pd[u] = rp[tid];
          }
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            if (q0 + u < C) {
              sigma += ps[u];
              d += pd[u];
            }
          }
        }
      }
      const float xnorm = sqrtf(fmaf(alpha, alpha, sigma));
      const bool skip = !(xnorm > thresh);
      float tau = 0.f, v0 = 1.f, rsign = 1.f;
      if (!skip) {
        if (sigma == 0.f) {
          rsign = alpha < 0.f ? -1.f : 1.f;  // H = I, R_pp = alpha
        } else {
          const float beta = alpha >= 0.f ? -xnorm : xnorm;
          v0 = alpha - beta;  // same sign as alpha: no cancellation
          tau = (beta - alpha) / beta;
          rsign = beta < 0.f ? -1.f : 1.f;
        }
      }
      if (tid == j) {
        if (!isfinite(xnorm)) nonfinite = 1;
        s_scal[0] = tau;
        s_scal[1] = tau != 0.f ? 1.f / v0 : 0.f;
        if (c == 0) {
          p.tau[(int64_t)b * n + k + j] = tau;
          p.skip[(int64_t)b * n + k + j] = skip ? 1 : 0;
          p.dsign[(int64_t)b * n + k + j] = rsign;
        }
      } else {
        s_wl[tid - j] = tau != 0.f ? apiv + d / v0 : 0.f;  // v^T a_tid, with v = x / v0 after the pivot
      }
    }
    __syncthreads();
    const float tau = s_scal[0], rv0 = s_scal[1];
    // v at this thread's positions (x / v0 after the pivot, 1 at it, 0 before it on rank 0) into
    // row j of Vt, and H_j = I - tau v v^T on the later rows, shifting them down one register
    {
      const int64_t o = (int64_t)(k + j) * n + pos0 + i0;
      if (have0 && (c != 0 || i0 >= j)) {
        const bool at_pivot = (c == 0 && i0 == j);
        const float vi = at_pivot ? 1.f : a0[0] * rv0;
        Vt[o] = vi;
        Vt_lo[o] = tf32_lo(vi);
        if (tau != 0.f) {
          const float tv = tau * vi;
#pragma unroll
          for (int l4 = 0; l4 < NB / 4; ++l4) {
            const float4 w4 = reinterpret_cast<const float4*>(s_wl)[l4];
            if (l4 > 0) a0[4 * l4 - 1] = fmaf(-tv, w4.x, a0[4 * l4]);
            a0[4 * l4] = fmaf(-tv, w4.y, a0[4 * l4 + 1]);
            a0[4 * l4 + 1] = fmaf(-tv, w4.z, a0[4 * l4 + 2]);
            a0[4 * l4 + 2] = fmaf(-tv, w4.w, a0[4 * l4 + 3]);
          }
          a0[NB - 1] = 0.f;
        } else {
#pragma unroll
          for (int l = 0; l < NB - 1; ++l) a0[l] = a0[l + 1];
          a0[NB - 1] = 0.f;
        }
      } else {
        if (have0) {  // rank 0, before the pivot
          Vt[o] = 0.f;
          Vt_lo[o] = 0.f;
        }
#pragma unroll
        for (int l = 0; l < NB - 1; ++l) a0[l] = a0[l + 1];
        a0[NB - 1] = 0.f;
      }
    }
    if (have1) {
      const int64_t o = (int64_t)(k + j) * n + pos0 + i1;
      const float vi = a1[0] * rv0;
      Vt[o] = vi;
      Vt_lo[o] = tf32_lo(vi);
      if (tau != 0.f) {
        const float tv = tau * vi;
#pragma unroll
        for (int l4 = 0; l4 < NB / 4; ++l4) {
          const float4 w4 = reinterpret_cast<const float4*>(s_wl)[l4];
          if (l4 > 0) a1[4 * l4 - 1] = fmaf(-tv, w4.x, a1[4 * l4]);
          a1[4 * l4] = fmaf(-tv, w4.y, a1[4 * l4 + 1]);
          a1[4 * l4 + 1] = fmaf(-tv, w4.z, a1[4 * l4 + 2]);
          a1[4 * l4 + 2] = fmaf(-tv, w4.w, a1[4 * l4 + 3]);
        }
        a1[NB - 1] = 0.f;
      } else {
#pragma unroll
        for (int l = 0; l < NB - 1; ++l) a1[l] = a1[l + 1];
        a1[NB - 1] = 0.f;
      }
    }
    __syncthreads();  // s_wl, s_red and s_scal are rewritten by the next column
  }
  if (nonfinite) atomicOr(p.status, kStatusQrBreakdown);
  // the block's positions before the panel are zero in the panel's rows of Vt
  if (c == 0)
    for (int e = tid; e < kb * jb; e += PTA) {
      const int64_t o = (int64_t)(k + e / jb) * n + k0 + e % jb;
      Vt[o] = 0.f;
      Vt_lo[o] = 0.f;
    }
  cluster.sync();  // the peers have read this CTA's partial sums
}

// ||P_b||_F: per-chunk partial sums in double (chunks of whole 16-byte units: nn is a
// multiple of 16), then tol * sqrt(sum)
constexpr int NORM_CHUNKS = 64;

// Partial sums of squares of P_b over NORM_CHUNKS chunks. The threshold needs ||P||_F to a few
// digits only, so each thread sums in fp32 (at most a few hundred terms) and the warps' sums are
// added in fp32 too; the chunks' partial sums are added in double by thresh_kernel.
__global__ void frob_partial_kernel(const float* P, int64_t nn, double* part) {
  const int b = blockIdx.y;
  const float4* x = reinterpret_cast<const float4*>(P + (int64_t)b * nn);
  const int64_t n4 = nn / 4;
  const int64_t per = (n4 + NORM_CHUNKS - 1) / NORM_CHUNKS;
  const int64_t beg = blockIdx.x * per, end = min(n4, beg + per);
  float s = 0.f;
  for (int64_t i = beg + threadIdx.x; i < end; i += blockDim.x) {
    const float4 v = x[i];
    s = fmaf(v.x, v.x, s);
    s = fmaf(v.y, v.y, s);
    s = fmaf(v.z, v.z, s);
    s = fmaf(v.w, v.w, s);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  __shared__ float red[8];
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += red[w];
    part[(int64_t)b * NORM_CHUNKS + blockIdx.x] = t;
  }
}

// The zero-column threshold tol * ||P_b||_F; a non-finite norm (a NaN or Inf anywhere in P_b,
// wherever the Householder steps would meet it) is a breakdown of that QR.
__global__ void thresh_kernel(const double* part, float tol, int batch, float* thresh, int* status) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= batch) return;
  double s = 0.0;
  for (int i = 0; i < NORM_CHUNKS; ++i) s += part[(int64_t)b * NORM_CHUNKS + i];
  if (!isfinite(s) && status) atomicOr(status, kStatusQrBreakdown);
  thresh[b] = (float)((double)tol * sqrt(s));
}

// Q^T <- diag(d)
__global__ void signed_identity_kernel(float* Qt, const float* d, int n) {
  const int b = blockIdx.y;
  const int64_t nn = (int64_t)n * n;
  float* q = Qt + (int64_t)b * nn;
  const float* db = d + (int64_t)b * n;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nn; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = i / n, cc = i % n;
    q[i] = r == cc ? db[r] : 0.f;
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

// The panel kernel variant for this device: 512 positions per CTA in clusters of up to 16
// where the device runs 16-CTA clusters of it, else 1024 positions in clusters of up to 8.
struct PanelKernel {
  void (*fn)(PanelArgs);
  void (*cols_fn)(PanelArgs);  // the column loop on its own (then fn forms the rest), or null
  int cols;
  size_t smem;
};

template <int COLS, bool SPLIT = false>
cudaError_t prepare_panel(PanelKernel* pk, bool wide) {
  pk->fn = qr_panel_kernel<COLS, SPLIT>;
  pk->cols_fn = SPLIT ? qr_cols_kernel : nullptr;
  pk->cols = COLS;
  pk->smem = (size_t)NB * (COLS + 4) * sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(pk->fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)pk->smem);
  if (e == cudaSuccess && wide) e = cudaFuncSetAttribute(pk->fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e == cudaSuccess && wide && pk->cols_fn)
    e = cudaFuncSetAttribute(pk->cols_fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  return e;
}

// The cluster shape is chosen once per device (with that device current): 1 = clusters of
// 16 x 512 positions where the device can place them, 2 = clusters of 8 x 1024.
std::atomic<int> g_panel_choice[64];

// Batches of at least this many factors take the column loop as its own kernel: on a GPU
// shared with the other QR groups and the next wave's products, two column-loop CTAs fit on one
// SM and the rest of the panel's work holds the SM for half as long. A smaller batch leaves SMs
// idle anyway, and there the second launch per panel only lengthens the chain.
constexpr int kSplitBatch = 16;

cudaError_t panel_kernel(PanelKernel* pk, int n, int batch) {
  // a factor of at most 1024 rows fits one CTA's 1024 positions: no cluster barrier per column
  if (n <= 1024) return prepare_panel<1024>(pk, false);
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) dev = 0;
  std::atomic<int>* slot = dev < 64 ? &g_panel_choice[dev] : nullptr;
  int choice = slot ? slot->load(std::memory_order_relaxed) : 0;
  if (choice == 0) {
    int ok = 0;
    if (prepare_panel<512, true>(pk, true) == cudaSuccess) {
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(16, 1, 1);
      cfg.blockDim = dim3(PT, 1, 1);
      cfg.dynamicSmemBytes = pk->smem;
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = 16;
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      int clusters = 0;
      if (cudaOccupancyMaxActiveClusters(&clusters, pk->fn, &cfg) == cudaSuccess && clusters > 0) ok = 1;
    }
    cudaGetLastError();
    choice = ok ? 1 : 2;
    if (slot) slot->store(choice, std::memory_order_relaxed);
  }
  if (choice != 1) return prepare_panel<1024>(pk, false);
  return batch >= kSplitBatch ? prepare_panel<512, true>(pk, true) : prepare_panel<512, false>(pk, true);
}

struct Workspace {
  float* At;
  float* At_lo;   // unused (null): the products form A's lo part themselves
  float* Vt;
  float* Vt_lo;
  float* VTq;     // [batch][nblock][n][NBO] V T of every block (kept for the Q accumulation)
  float* VTq_lo;
  float* VTr;     // [batch][n][NBO] V T^T of the current block
  float* VTr_lo;
  float* Vpos;    // [batch][n][NBO]
  float* Vpos_lo;
  float* W;       // [batch][n][NBO]
  float* W_lo;
  float* T;       // [batch][NBO][NBO], and T^T, each with its lo part
  float* T_lo;
  float* Tt;
  float* Tt_lo;
  float* Ypart;   // [batch][MAXC][NBO][NB]
  float* Wsplit;  // [KSPLIT][batch][n][NBO] partial sums of split-K products
  // for the look-ahead schedule only (null otherwise): the far update's own W and split-K
  // buffers, and second V T^T, Vpos and T buffers (blocks alternate: a block's V T^T is read
  // by its far update and its Vpos and T by its V T while the next block is factored)
  float* W2;
  float* W2_lo;
  float* Wsplit2;
  float* VTr2;
  float* VTr2_lo;
  float* Vpos2;
  float* Vpos2_lo;
  float* T2;
  float* T2_lo;
  float* Tt2;
  float* Tt2_lo;
  float* thresh;
  float* dsign;
  float* tau;     // [batch][n] the reflectors' tau, from the column kernel to the panel kernel
  double* part;
};

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

Workspace carve(void* base, int n, int batch, size_t* total, bool lookahead) {
  const int nblock = (n + NBO - 1) / NBO;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    size_t o = off;
    off += align256(bytes);
    return o;
  };
  const size_t mat = (size_t)batch * n * n * sizeof(float);
  const size_t blocks = (size_t)batch * nblock * n * NBO * sizeof(float);
  const size_t thin = (size_t)batch * n * NBO * sizeof(float);
  const size_t tsq = (size_t)batch * NBO * NBO * sizeof(float);
  const size_t oAt = take(mat), oVt = take(mat), oVtl = take(mat);
  const size_t oVq = take(blocks), oVql = take(blocks), oVr = take(thin), oVrl = take(thin);
  const size_t oVp = take(thin), oVpl = take(thin), oW = take(thin), oWl = take(thin);
  const size_t oT = take(tsq), oTl = take(tsq), oTt = take(tsq), oTtl = take(tsq);
  const size_t oY = take((size_t)batch * MAXC * NBO * NB * sizeof(float));
  const size_t oWs = take((size_t)KSPLIT * thin);
  const size_t oW2 = lookahead ? take(thin) : 0, oW2l = lookahead ? take(thin) : 0;
  const size_t oWs2 = lookahead ? take((size_t)KSPLIT * thin) : 0;
  const size_t oVr2 = lookahead ? take(thin) : 0, oVr2l = lookahead ? take(thin) : 0;
  const size_t oVp2 = lookahead ? take(thin) : 0, oVp2l = lookahead ? take(thin) : 0;
  const size_t oT2 = lookahead ? take(tsq) : 0, oT2l = lookahead ? take(tsq) : 0;
  const size_t oTt2 = lookahead ? take(tsq) : 0, oTt2l = lookahead ? take(tsq) : 0;
  const size_t oth = take((size_t)batch * sizeof(float));
  const size_t osg = take((size_t)batch * n * sizeof(float));
  const size_t otau = take((size_t)batch * n * sizeof(float));
  const size_t opart = take((size_t)batch * NORM_CHUNKS * sizeof(double));
  if (total) *total = off;
  char* c = (char*)base;
  auto f = [&](size_t o) { return (float*)(c + o); };
  auto g = [&](size_t o) { return lookahead ? (float*)(c + o) : nullptr; };
  return Workspace{f(oAt), nullptr, f(oVt), f(oVtl), f(oVq), f(oVql), f(oVr), f(oVrl), f(oVp),  f(oVpl),
                   f(oW),  f(oWl),  f(oT),  f(oTl),  f(oTt), f(oTtl), f(oY),  f(oWs), g(oW2),  g(oW2l),
                   g(oWs2), g(oVr2), g(oVr2l), g(oVp2), g(oVp2l), g(oT2),  g(oT2l),  g(oTt2), g(oTt2l),
                   f(oth), f(osg), f(otau), (double*)(c + opart)};
}

TcOperand op(const float* hi, const float* lo, int64_t ld, int64_t stride, int batch) {
  return TcOperand{hi, lo, ld, stride, batch};
}

TcEpilogue out(float* C, float* C_lo, int64_t ldc, int64_t stride, float alpha, float beta, int* status) {
  return TcEpilogue{C, nullptr, ldc, stride, C_lo, ldc, stride, 0, alpha, beta, status};
}

}  // namespace

size_t qr_workspace_bytes(int n, int batch, bool lookahead) {
  size_t total = 0;
  carve(nullptr, n, batch, &total, lookahead);
  return total;
}

void qr_input_buffers(void* workspace, int n, int batch, float** At) {
  Workspace w = carve(workspace, n, batch, nullptr, false);  // the input buffer comes first either way
  *At = w.At;
}

cudaError_t qr_q_t(int n, int batch, float* Qt, float* Qt_lo, float* Q, float* Q_lo, uint8_t* skip, float tol,
                   void* workspace, size_t workspace_bytes, int* status, cudaStream_t s, const QrLookahead* lah) {
  if (n <= 0 || batch <= 0) return cudaSuccess;
  if (n > 8192 || batch > 65535 || (n & 3)) return cudaErrorInvalidValue;
  // look-ahead: a second stream and its events given, and a workspace sized for it
  const bool la = lah && lah->far && lah->vt && lah->far_done && lah->vq[0] && lah->vq[1] &&
                  workspace_bytes >= qr_workspace_bytes(n, batch, true);
  cudaStream_t far = la ? lah->far : nullptr;
  cudaEvent_t ev_vt = la ? lah->vt : nullptr, ev_far = la ? lah->far_done : nullptr;
  size_t need = 0;
  Workspace w = carve(workspace, n, batch, &need, la);
  if (workspace_bytes < need) return cudaErrorInvalidValue;
  if (!Qt) Qt = w.At;  // the Q accumulation may reuse the factored matrix's buffer
  const int nblock = (n + NBO - 1) / NBO;
  const int64_t nn = (int64_t)n * n, thin = (int64_t)n * NBO, vq_stride = (int64_t)nblock * thin;
  cudaError_t e;

  {
    ProfScope prof(kFamOther, 2.0 * nn * batch, 4.0 * nn * batch, s);
    frob_partial_kernel<<<dim3(NORM_CHUNKS, batch), 256, 0, s>>>(w.At, nn, w.part);
  }
  {
    ProfScope prof(kFamOther, 0, 8.0 * NORM_CHUNKS * batch, s);
    thresh_kernel<<<(batch + 127) / 128, 128, 0, s>>>(w.part, tol, batch, w.thresh, status);
  }
  PanelKernel pk;
  e = panel_kernel(&pk, n, batch);
  if (e != cudaSuccess) return e;

  if (la) {
    // the far stream starts after everything enqueued on s so far; ev_far stands for "the
    // previous far update is done" and starts out recorded
    e = cudaEventRecord(ev_far, s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(far, ev_far, 0);
    if (e != cudaSuccess) return e;
  }
  for (int blk = 0; blk < nblock; ++blk) {
    const int k0 = blk * NBO, kbo = std::min(NBO, n - k0), m = n - k0;
    const int par = blk & 1;
    const bool alt = la && par;
    float* vp = alt ? w.Vpos2 : w.Vpos;
    float* vp_lo = alt ? w.Vpos2_lo : w.Vpos_lo;
    float* Tb = alt ? w.T2 : w.T;
    float* Tb_lo = alt ? w.T2_lo : w.T_lo;
    float* Ttb = alt ? w.Tt2 : w.Tt;
    float* Ttb_lo = alt ? w.Tt2_lo : w.Tt_lo;
    // with the look-ahead, this block's Vpos and T buffers were last read by the V T of the
    // block two before, on the far stream
    if (la && blk >= 2) {
      e = cudaStreamWaitEvent(s, lah->vq[par], 0);
      if (e != cudaSuccess) return e;
    }
    for (int k = k0; k < k0 + kbo; k += NB) {
      const int kb = std::min(NB, n - k);
      const int C = (n - k + pk.cols - 1) / pk.cols;
      PanelArgs a{w.At, w.Vt, w.Vt_lo, vp, vp_lo, Tb, Tb_lo, Ttb, Ttb_lo, w.Ypart, skip, w.dsign, w.tau,
                  w.thresh, status, n, k0, kbo, k, kb};
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(C, batch, 1);
      cfg.blockDim = dim3(PT, 1, 1);
      cfg.dynamicSmemBytes = pk.smem;
      cfg.stream = s;
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = C;
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      // Householder steps on the kb x (n-k) panel (~4 kb^2 (n-k)), S V over kbo rows
      // (2 kbo kb (n-k)) and the in-block update (2 kb (kbo-kb) (n-k))
      const double mk = (double)(n - k) * batch;
      if (pk.cols_fn) {
        // the column loop first, on its own (the panel read, V written with its lo part)
        cudaLaunchConfig_t cc = cfg;
        cc.blockDim = dim3(PTA, 1, 1);
        cc.dynamicSmemBytes = 0;
        ProfScope prof(kFamQrPanel, 4.0 * kb * kb * mk, 4.0 * 3.0 * kb * mk, s);
        e = cudaLaunchKernelEx(&cc, pk.cols_fn, a);
        if (e != cudaSuccess) return e;
      }
      {
        const double f = pk.cols_fn ? 4.0 * kbo * kb * mk : (4.0 * kb * kb + 4.0 * kbo * kb) * mk;
        const double by = pk.cols_fn ? 4.0 * 2.0 * kbo * mk : 4.0 * (3.0 * kb + 2.0 * kbo) * mk;
        ProfScope prof(kFamQrPanel, f, by, s);
        e = cudaLaunchKernelEx(&cfg, pk.fn, a);
      }
      if (e != cudaSuccess) return e;
    }
    // VTq = V T (the Q accumulation) and VTr = V T^T (this block's trailing update); with the
    // look-ahead the V T^T buffers alternate between blocks, since the far update of block b
    // still reads its V T^T while block b+1 forms its own
    float* vtr = alt ? w.VTr2 : w.VTr;
    float* vtr_lo = alt ? w.VTr2_lo : w.VTr_lo;
    float* vq = w.VTq + (int64_t)blk * thin + (int64_t)k0 * NBO;
    float* vq_lo = w.VTq_lo + (int64_t)blk * thin + (int64_t)k0 * NBO;
    const TcOperand vpos = op(vp + (int64_t)k0 * NBO, vp_lo + (int64_t)k0 * NBO, NBO, thin, batch);
    auto form_vtq = [&](cudaStream_t st) {
      return gemm_tc_nt(m, kbo, kbo, batch, vpos, op(Ttb, Ttb_lo, NBO, NBO * NBO, batch),
                        out(vq, vq_lo, NBO, vq_stride, 1.f, 0.f, status), st, kFamQrUpdate);
    };
    if (!la) {
      e = form_vtq(s);
      if (e != cudaSuccess) return e;
    }
    const int nc = n - k0 - kbo;  // trailing rows of At (columns of P)
    if (nc > 0) {
      e = gemm_tc_nt(m, kbo, kbo, batch, vpos, op(Tb, Tb_lo, NBO, NBO * NBO, batch),
                     out(vtr + (int64_t)k0 * NBO, vtr_lo + (int64_t)k0 * NBO, NBO, thin, 1.f, 0.f, status), s,
                     kFamQrUpdate);
      if (e != cudaSuccess) return e;
    }
    if (nc <= 0 && !la) continue;
    const TcOperand vtr_trail =
        op(vtr + (int64_t)(k0 + kbo) * NBO, vtr_lo + (int64_t)(k0 + kbo) * NBO, NBO, thin, batch);
    const TcOperand vt_blk = op(w.Vt + (int64_t)k0 * n + k0, w.Vt_lo + (int64_t)k0 * n + k0, n, nn, batch);
    // rows [r0, r0 + rows) of the trailing matrix: a_r -= (a_r V) T V^T, i.e.
    //   W = At_rows Vt^T over positions k0.. ; At_rows -= W VTr^T at positions k0+kbo.. (the
    //   earlier positions of these rows are R's entries, never read again)
    auto update_rows = [&](int r0, int rows, float* Wb, float* Wb_lo, float* ws, cudaStream_t st) -> cudaError_t {
      const int64_t tr = (int64_t)r0 * n;
      cudaError_t e2 = gemm_tc_nt(rows, kbo, m, batch, op(w.At + tr + k0, nullptr, n, nn, batch), vt_blk,
                                  out(Wb, Wb_lo, NBO, thin, 1.f, 0.f, status), st, kFamQrUpdate, ws,
                                  (size_t)KSPLIT * batch * n * NBO);
      if (e2 != cudaSuccess) return e2;
      return gemm_tc_nt(rows, nc, kbo, batch, op(Wb, Wb_lo, NBO, thin, batch), vtr_trail,
                        out(w.At + tr + k0 + kbo, nullptr, n, nn, -1.f, 1.f, status), st,
                        kFamQrUpdate);
    };
    if (!la) {
      e = update_rows(k0 + kbo, nc, w.W, w.W_lo, w.Wsplit, s);
      if (e != cudaSuccess) return e;
      continue;
    }
    // look-ahead: the next block's rows now (they gate its panels), the rest on the far stream,
    // where it overlaps the next block's panels; the next block's rows wait for the previous
    // far update, which covered them. The block's V T follows its far update on the far stream.
    const int knext = std::min(NBO, std::max(nc, 0));
    // (the far update starts once the next block's rows are done, so that those small products
    // do not wait for SMs behind it)
    e = cudaSuccess;
    if (nc > 0) e = cudaStreamWaitEvent(s, ev_far, 0);
    if (e == cudaSuccess && nc > 0) e = update_rows(k0 + kbo, knext, w.W, w.W_lo, w.Wsplit, s);
    if (e == cudaSuccess) e = cudaEventRecord(ev_vt, s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(far, ev_vt, 0);
    if (e == cudaSuccess && nc > knext) e = update_rows(k0 + kbo + knext, nc - knext, w.W2, w.W2_lo, w.Wsplit2, far);
    if (e == cudaSuccess) e = cudaEventRecord(ev_far, far);
    if (e == cudaSuccess) e = form_vtq(far);
    if (e == cudaSuccess) e = cudaEventRecord(lah->vq[par], far);
    if (e != cudaSuccess) return e;
  }
  if (la) {
    // the last far update and the last V T before the Q accumulation
    e = cudaEventRecord(ev_far, far);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(s, ev_far, 0);
    if (e != cudaSuccess) return e;
  }

  {
    // Q^T = diag(d) H_n ... H_1 accumulated backwards: start from diag(d)
    ProfScope prof(kFamOther, 0, 4.0 * nn * batch, s);
    const int blocks = (int)std::min<int64_t>((nn + 255) / 256, 1024);
    signed_identity_kernel<<<dim3(blocks, batch), 256, 0, s>>>(Qt, w.dsign, n);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  for (int blk = nblock - 1; blk >= 0; --blk) {
    const int k0 = blk * NBO, kbo = std::min(NBO, n - k0), m = n - k0;
    const int64_t sub = (int64_t)k0 * n + k0;
    // W = Qt_sub Vt^T  (m x kbo)
    e = gemm_tc_nt(m, kbo, m, batch, op(Qt + sub, nullptr, n, nn, batch),
                   op(w.Vt + sub, w.Vt_lo + sub, n, nn, batch), out(w.W, w.W_lo, NBO, thin, 1.f, 0.f, status), s,
                   kFamQrUpdate, w.Wsplit, (size_t)KSPLIT * batch * n * NBO);
    if (e != cudaSuccess) return e;
    // Qt_sub -= W VTq^T
    const int64_t vq = (int64_t)blk * thin + (int64_t)k0 * NBO;
    e = gemm_tc_nt(m, m, kbo, batch, op(w.W, w.W_lo, NBO, thin, batch),
                   op(w.VTq + vq, w.VTq_lo + vq, NBO, vq_stride, batch),
                   out(Qt + sub, nullptr, n, nn, -1.f, 1.f, status), s, kFamQrUpdate);
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
  Workspace w = carve(workspace, n, batch, &need, false);
  if (workspace_bytes < need || (n & 3)) return cudaErrorInvalidValue;
  // At = P^T and its lo part
  cudaError_t e = transpose(P, w.At, n, n, batch, s);
  if (e != cudaSuccess) return e;
  return qr_q_t(n, batch, nullptr, nullptr, Q, nullptr, skip, tol, workspace, workspace_bytes, status, s, nullptr);
}

}  // namespace soap
