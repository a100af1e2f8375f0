// fp32-accurate batched GEMM on the 5th-generation tensor cores (tcgen05, sm_103a).
//
//   C_b = alpha * A_b * B_{b mod bmod}^T + beta * C_b
//
// A_b is M x K and B is N x K, both row-major ("K-major"), so TMA copies their tiles
// straight into the canonical 128-byte-swizzled K-major shared-memory layout that
// tcgen05.mma reads. Every operand comes as a pair (hi, lo): the tensor core reads an
// fp32 word as tf32 by dropping its 13 low mantissa bits, so hi may be the fp32 array
// itself, and lo = x - trunc_tf32(x) rounded to the nearest tf32 (read exactly). The
// accumulator (fp32, in TMEM) receives
//   a_lo b_lo + a_lo b_hi + a_hi b_lo + a_hi b_hi
// = (hi + lo)(hi + lo), each operand within 2^-22 of x and without the bias that
// truncation would leave: products with fp32 accuracy at tensor-core rate, as the
// optimizer step's fp32 arithmetic requires.
//
// The tensor core's own accumulation rounds toward zero at every MMA, so a long chain
// of MMAs into one accumulator drifts (relative error growing ~linearly in K: 6e-5 at
// K = 8192). Each 32-wide K block is therefore accumulated afresh in one of four TMEM
// accumulators, used in turn, while the epilogue warps drain finished ones into fp32
// registers with round-to-nearest adds; the drain of block k overlaps the MMAs of the
// next blocks, and the error stays at the level of an fp32 dot product.
//
// CTA: warp 0 issues the TMA loads (one elected lane), warp 1 allocates tensor memory and
// issues the MMAs (one elected lane), and 8 epilogue warps (4 for BN = 32) drain the
// accumulators: tensor memory -> registers (a warp reads the 32 accumulator lanes of its
// quadrant, two warps split a quadrant's columns) -> alpha/beta -> a swizzled 32 x 32
// block in shared memory -> 16-byte global stores, optionally transposed and optionally
// also writing the lo part of the result for a later product. When the epilogue reads C
// (beta != 0), the epilogue warps copy their part of the C tile into shared memory with
// cp.async while the MMAs run. For short K a CTA runs several consecutive tiles, so that
// the next tile's loads and MMAs proceed while the epilogue stores the current one.
// Stages are handed over with mbarriers; every wait gives up after a bounded time (2 s of
// %globaltimer time unless soap_wait_limit set another), records kStatusTimeout and lets the
// CTA drain -- TMA copies already issued land, issued MMAs complete -- and free its tensor
// memory instead of hanging. The drains themselves always keep the full 2 s bound.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <atomic>
#include <mutex>

#include "profile.h"
#include "soap_internal.h"
#include "tc_ptx.h"

namespace soap {
namespace tc {

constexpr int BM = 128;
constexpr int BK = 32;  // fp32 elements per K block = one 128-byte swizzle row
constexpr uint64_t kWaitNs = 2000000000ull;

template <int BN, int STAGES, bool PRE>
struct Cfg {
  static constexpr int EPI = BN >= 64 ? 8 : 4;      // epilogue warps (two per TMEM lane quadrant if 8)
  static constexpr int THREADS = 64 + 32 * EPI;
  static constexpr int CPW = BN * 4 / EPI;          // accumulator columns drained by one epilogue warp
  static constexpr int NCH = CPW / 32;              // 32-column chunks per epilogue warp
  static constexpr int TILE_A = BM * BK * 4;
  static constexpr int TILE_B = BN * BK * 4;
  static constexpr int STAGE = 2 * TILE_A + 2 * TILE_B;
  // per epilogue warp: its whole 32 x CPW block of C when C is prefetched, else one 32 x 32
  // staging block (both swizzled in 16-byte units)
  static constexpr int OBUF = PRE ? 32 * CPW : 32 * 32;
  static constexpr int SMEM = STAGES * STAGE + EPI * OBUF * 4 + 1024 + 256;
  // four accumulators used in turn: a K block's partial sum may wait three K blocks of MMAs
  // for the epilogue warps to drain it
  static constexpr int NACC = 4;
  static constexpr uint32_t TMEM_COLS = NACC * BN;
  static_assert(CPW % 32 == 0, "epilogue chunking");
  static_assert(SMEM <= 232448, "shared memory budget");
};

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}

// Bounded wait until *flag != 0 (a flag set from outside the kernel): false after `limit_ns`.
__device__ __forceinline__ bool flag_wait(const int* flag, uint64_t limit_ns) {
  const volatile int* f = flag;
  if (*f != 0) return true;
  const uint64_t t0 = globaltimer();
  while (*f == 0)
    if (globaltimer() - t0 > limit_ns) return false;
  return true;
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, uint64_t* bar, int c0, int c1,
                                            int c2) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(
          dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(c0), "r"(c1), "r"(c2)
      : "memory");
}

__device__ __forceinline__ void cp_async16(float* smem_dst, const float* gmem_src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(smem_dst)), "l"(gmem_src),
               "r"(valid ? 16 : 0)
               : "memory");
}

// Word offset of element (r, j) of a 32 x 32 block stored row-major with its 16-byte units
// XOR-swizzled by r mod 8: a warp touching one 16-byte unit per row, or one row, is
// conflict-free.
__device__ __forceinline__ int swz(int r, int j) { return r * 32 + ((((j >> 2) ^ (r & 7))) << 2) + (j & 3); }

// Tile t of a launch -> (m0, n0, batch index). Within a matrix the tiles go in groups of GM
// row tiles: m fastest inside a group, then n, then the next group. The ~152 tiles in flight
// at a time then read about GM A row panels and 152/GM B column panels, whose current K
// slices stay in L2, instead of all of B once per row of tiles.
constexpr int GM = 8;
__device__ __forceinline__ void tile_coords(int t, int ntm, int ntn, int BN_, int& m0, int& n0, int& b) {
  const int per = ntm * ntn;
  b = t / per;
  const int r = t - b * per;
  const int g = r / (GM * ntn);
  const int first = g * GM;
  const int gsz = min(GM, ntm - first);
  const int w = r - g * GM * ntn;
  m0 = (first + w % gsz) * BM;
  n0 = (w / gsz) * BN_;
}

// Symmetric products (C = alpha A A^T + beta C, M = N): tile t -> (m0, n0, batch index) over the
// tiles on or below the diagonal only, row by row (tile (i, j), j <= i, at i (i + 1) / 2 + j).
__device__ __forceinline__ void tile_coords_sym(int t, int ntm, int& m0, int& n0, int& b) {
  const int per = ntm * (ntm + 1) / 2;
  b = t / per;
  const int r = t - b * per;
  int i = (int)((sqrtf(8.f * (float)r + 1.f) - 1.f) * 0.5f);
  while ((i + 1) * (i + 2) / 2 <= r) ++i;
  while (i * (i + 1) / 2 > r) --i;
  m0 = i * BM;
  n0 = (r - i * (i + 1) / 2) * BM;
}

// A CTA takes `tpc` consecutive tiles, so that the loads and MMAs of its next tile overlap
// the epilogue of the current one. With ksplit > 1 the K blocks are split into ksplit
// consecutive ranges; split s of matrix b is written as output matrix s * batch + b (partial
// sums that the caller adds up).
// With CVTA the A operand comes as fp32 only: the epilogue warps form its lo part in shared
// memory, beside the tile TMA brought in (for HBM-bound products whose A is read once; the
// extra shared-memory traffic would slow a compute-bound product).
// With SYM (A = B, M = N, BN = BM) only the tiles on or below the diagonal are computed, and each
// one below it is also stored transposed in the mirror position, so C stays exactly symmetric
// with about half of the MMAs.
template <int BN, int STAGES, bool PRE, bool CVTA, bool TR, bool LO, bool VEC, bool SYM>
__global__ void __launch_bounds__(Cfg<BN, STAGES, PRE>::THREADS, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap ta_hi, const __grid_constant__ CUtensorMap ta_lo,
                   const __grid_constant__ CUtensorMap tb_hi, const __grid_constant__ CUtensorMap tb_lo, int M,
                   int N, int K, int batch, int a_mod, int b_mod, int tpc, int ksplit, TcEpilogue ep) {
  using C = Cfg<BN, STAGES, PRE>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  float* obuf_all = reinterpret_cast<float*>(smem + STAGES * C::STAGE);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * C::STAGE + C::EPI * C::OBUF * 4);
  uint64_t* empty = full + STAGES;
  uint64_t* conv = empty + STAGES;          // [STAGES] CVTA: the stage's A lo part is in place
  uint64_t* acc_full = conv + STAGES;       // [NACC] accumulator a holds a finished K block
  uint64_t* acc_empty = acc_full + C::NACC;  // [NACC] accumulator a has been drained
  uint64_t* mma_done = acc_empty + C::NACC;  // every MMA this CTA issued has completed
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(mma_done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);
  volatile int* consumed = abort_flag + 1;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint64_t lim = ep.wait_ns ? ep.wait_ns : kWaitNs;  // bound of every wait but the drains
  const int kblocks = (K + BK - 1) / BK;
  const int kper = (kblocks + ksplit - 1) / ksplit;  // K blocks of one split
  const int ntn = (N + BN - 1) / BN, ntm = (M + BM - 1) / BM;
  const int ntiles = (SYM ? ntm * (ntm + 1) / 2 : ntn * ntm) * batch * ksplit;
  // the K blocks [kb0, kb1) of tile t, and its operand and output matrix indices
  auto krange = [&](int bo, int& kb0, int& kb1) {
    kb0 = (bo / batch) * kper;
    kb1 = min(kblocks, kb0 + kper);
  };
  const int t_begin = blockIdx.x * tpc;
  const int t_end = min(ntiles, t_begin + tpc);

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
      mbar_init(&conv[s], C::EPI);  // one arrival per epilogue warp
    }
    for (int a = 0; a < C::NACC; ++a) {
      mbar_init(&acc_full[a], 1);
      mbar_init(&acc_empty[a], C::EPI);  // one arrival per epilogue warp
    }
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    *consumed = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0 && lane == 0) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&ta_hi)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&ta_lo)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tb_hi)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tb_lo)) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_holder)),
                 "r"(C::TMEM_COLS));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;

  if (warp == 0) {
    if (lane == 0) {
      int g = 0, issued = 0;  // k blocks over all of this CTA's tiles
      for (int t = t_begin; t < t_end && !*abort_flag; ++t) {
        int m0, n0, bo, kb0, kb1;
        if (SYM) tile_coords_sym(t, ntm, m0, n0, bo);
        else tile_coords(t, ntm, ntn, BN, m0, n0, bo);
        krange(bo, kb0, kb1);
        const int b = bo % batch;
        for (int kb = kb0; kb < kb1; ++kb, ++g) {
          const int s = g % STAGES;
          const uint32_t ph = (g / STAGES) & 1;
          if (!mbar_wait(&empty[s], ph ^ 1, lim) || *abort_flag) {
            *abort_flag = 1;
            if (ep.status) atomicOr(ep.status, kStatusTimeout);
            break;
          }
          mbar_expect_tx(&full[s], CVTA ? C::STAGE - C::TILE_A : C::STAGE);
          const uint32_t st = smem_u32(smem + s * C::STAGE);
          const int kc = kb * BK;
          tma_load_3d(st, &ta_hi, &full[s], kc, m0, b % a_mod);
          if (!CVTA) tma_load_3d(st + C::TILE_A, &ta_lo, &full[s], kc, m0, b % a_mod);
          tma_load_3d(st + 2 * C::TILE_A, &tb_hi, &full[s], kc, n0, b % b_mod);
          tma_load_3d(st + 2 * C::TILE_A + C::TILE_B, &tb_lo, &full[s], kc, n0, b % b_mod);
          issued = g + 1;
        }
      }
      if (*abort_flag) {
        // let copies already in flight land before the CTA's shared memory goes away
        for (int gg = *consumed; gg < issued; ++gg) mbar_wait(&full[gg % STAGES], (gg / STAGES) & 1, kWaitNs);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_tf32(BM, BN);
      int g = 0;
      bool ok = true;
      for (int t = t_begin; t < t_end && ok && !*abort_flag; ++t) {
        int m0, n0, bo, kb0, kb1;
        if (SYM) tile_coords_sym(t, ntm, m0, n0, bo);
        else tile_coords(t, ntm, ntn, BN, m0, n0, bo);
        krange(bo, kb0, kb1);
        for (int kb = kb0; kb < kb1; ++kb, ++g) {
          const int s = g % STAGES;
          const uint32_t ph = (g / STAGES) & 1;
          const int a = g % C::NACC;
          if (!mbar_wait(CVTA ? &conv[s] : &full[s], ph, lim) ||
              (g >= C::NACC && !mbar_wait(&acc_empty[a], ((g / C::NACC) & 1) ^ 1, lim)) || *abort_flag) {
            ok = false;
            break;
          }
          *consumed = g + 1;
          tc_fence_after();
          const uint32_t d = tmem + static_cast<uint32_t>(a * BN);
          const uint32_t a_hi = smem_u32(smem + s * C::STAGE);
          const uint32_t a_lo = a_hi + C::TILE_A;
          const uint32_t b_hi = a_hi + 2 * C::TILE_A;
          const uint32_t b_lo = b_hi + C::TILE_B;
#pragma unroll
          for (int kk = 0; kk < BK / 8; ++kk) {
            const uint32_t off = kk * 32;  // 8 tf32 = 32 bytes along K inside the swizzle row
            umma_tf32(d, desc_sw128(a_lo + off), desc_sw128(b_lo + off), idesc, kk != 0);
            umma_tf32(d, desc_sw128(a_lo + off), desc_sw128(b_hi + off), idesc, 1u);
            umma_tf32(d, desc_sw128(a_hi + off), desc_sw128(b_lo + off), idesc, 1u);
            umma_tf32(d, desc_sw128(a_hi + off), desc_sw128(b_hi + off), idesc, 1u);
          }
          umma_commit(&empty[s]);     // frees the stage once these MMAs have read it
          umma_commit(&acc_full[a]);  // hands the K block's sum to the epilogue warps
        }
      }
      if (!ok) {
        *abort_flag = 1;
        if (ep.status) atomicOr(ep.status, kStatusTimeout);
      }
      // the tensor memory is freed below: every MMA issued must have completed first (this
      // matters only when a wait gave up; otherwise the epilogue has drained them all)
      if (g > 0) {
        umma_commit(mma_done);
        mbar_wait(mma_done, 0, kWaitNs);
      }
    }
  } else {
    const int q = warp & 3;  // this warp may read accumulator lanes 32q .. 32q+31
    const int colbase = ((warp - 2) / 4) * C::CPW;
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(32 * q) << 16);
    float* obuf = obuf_all + (warp - 2) * C::OBUF;
    // CVTA: the lo part of k block gc's A tile, x - trunc_tf32(x) rounded to the nearest tf32,
    // written beside it for the tensor core (which reads it through the async proxy)
    auto convert = [&](int gc) -> bool {
      const int s = gc % STAGES;
      if (!mbar_wait(&full[s], (gc / STAGES) & 1, lim) || *abort_flag) return false;
      const float4* src = reinterpret_cast<const float4*>(smem + s * C::STAGE);
      float4* dst = reinterpret_cast<float4*>(smem + s * C::STAGE + C::TILE_A);
      for (int u = (warp - 2) * 32 + lane; u < C::TILE_A / 16; u += C::EPI * 32) {
        const float4 v = src[u];
        dst[u] = make_float4(tf32_lo(v.x), tf32_lo(v.y), tf32_lo(v.z), tf32_lo(v.w));
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      __syncwarp();
      if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(&conv[s])) : "memory");
      return true;
    };
    int gtotal = 0;  // K blocks over this CTA's tiles
    if (CVTA)
      for (int t = t_begin; t < t_end; ++t) {
        int m0, n0, bo, kb0, kb1;
        if (SYM) tile_coords_sym(t, ntm, m0, n0, bo);
        else tile_coords(t, ntm, ntn, BN, m0, n0, bo);
        krange(bo, kb0, kb1);
        gtotal += kb1 - kb0;
      }
    int gconv = 0;  // next K block to convert, kept STAGES - 1 ahead of the drains
    int g = 0;
    bool valid = true;
    if (ep.hold && !flag_wait(ep.hold, lim)) {
      // the timeout path under test: no tile is drained, the other warps' waits run out too
      valid = false;
      *abort_flag = 1;
      if (lane == 0 && ep.status) atomicOr(ep.status, kStatusTimeout);
    }
    for (int t = t_begin; t < t_end && valid; ++t) {
      int m0, n0, b, kb0, kb1;  // b: output matrix (split * batch + operand matrix)
      if (SYM) tile_coords_sym(t, ntm, m0, n0, b);
      else tile_coords(t, ntm, ntn, BN, m0, n0, b);
      krange(b, kb0, kb1);
      float* Cb = ep.C_ptrs ? ep.C_ptrs[b] : (ep.C ? ep.C + (int64_t)b * ep.c_stride : nullptr);
      float* Lb = LO && ep.C_lo ? ep.C_lo + (int64_t)b * ep.lo_stride : nullptr;
      const int row0 = m0 + 32 * q;   // first of this warp's 32 rows
      const int col0 = n0 + colbase;  // first of its CPW columns
      // 16-byte vector access to C (and C_lo) needs 16-byte aligned rows
      // (a kernel that prefetches C is only launched on 16-byte aligned C, lo part and rows)
      const bool vec = PRE || VEC || Cb && (ep.ldc & 3) == 0 && (reinterpret_cast<uintptr_t>(Cb) & 15) == 0 &&
                       (!Lb || ((ep.ld_lo & 3) == 0 && (reinterpret_cast<uintptr_t>(Lb) & 15) == 0));
      // the prefetch copies whole 16-byte units: the dimension they run along must be a multiple of 4
      const bool pre = PRE;
      if (pre) {
        // this warp's C block, copied in while the MMAs run; only 16-byte units wholly inside C
        for (int c = 0; c < C::NCH; ++c) {
          float* cb = obuf + 1024 * c;
          for (int u = lane; u < 256; u += 32) {
            const int x = u >> 3, y4 = u & 7;  // x: row (or column if transposed), y4: 16-byte unit
            int r, col;
            if (!TR) {
              r = row0 + x;
              col = col0 + 32 * c + 4 * y4;
            } else {
              col = col0 + 32 * c + x;
              r = row0 + 4 * y4;
            }
            const bool ok = TR ? (col < N && r + 3 < M) : (r < M && col + 3 < N);
            const float* src = !ok ? Cb : TR ? Cb + (int64_t)col * ep.ldc + r : Cb + (int64_t)r * ep.ldc + col;
            cp_async16(cb + x * 32 + ((y4 ^ (x & 7)) << 2), src, ok);
          }
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
      }
      float acc[C::NCH][32];
#pragma unroll
      for (int c = 0; c < C::NCH; ++c)
#pragma unroll
        for (int j = 0; j < 32; ++j) acc[c][j] = 0.f;
      for (int kb = kb0; kb < kb1; ++kb, ++g) {
        if (CVTA)
          while (valid && gconv < gtotal && gconv <= g + STAGES - 1) valid = convert(gconv++);
        const int a = g % C::NACC;
        if (!valid || !mbar_wait(&acc_full[a], (g / C::NACC) & 1, lim) || *abort_flag) {
          valid = false;
          break;
        }
        tc_fence_after();
#pragma unroll
        for (int c = 0; c < C::NCH; ++c) {
          float v[32];
          tmem_ld32(lane_base + static_cast<uint32_t>(a * BN + colbase + 32 * c), v);
#pragma unroll
          for (int j = 0; j < 32; ++j) acc[c][j] += v[j];
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0)
          asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(&acc_empty[a])) : "memory");
      }
      if (pre) {
        asm volatile("cp.async.wait_all;" ::: "memory");
        __syncwarp();
      }
      if (!valid) {
        if (lane == 0 && ep.status) atomicOr(ep.status, kStatusTimeout);
        break;
      }
      // out = alpha acc + beta C through the warp's shared block, then 16-byte stores
#pragma unroll
      for (int c = 0; c < C::NCH; ++c) {
        float* cb = obuf + (PRE ? 1024 * c : 0);
        const int cc0 = col0 + 32 * c;
        if (!TR) {
          const int r = row0 + lane;  // this lane's row
#pragma unroll
          for (int j4 = 0; j4 < 8; ++j4) {
            float4 o;
            o.x = ep.alpha * acc[c][4 * j4];
            o.y = ep.alpha * acc[c][4 * j4 + 1];
            o.z = ep.alpha * acc[c][4 * j4 + 2];
            o.w = ep.alpha * acc[c][4 * j4 + 3];
            float4* slot = reinterpret_cast<float4*>(cb + swz(lane, 4 * j4));
            if (ep.beta != 0.f) {
              float4 cv;
              if (pre) {
                cv = *slot;
              } else {
                const int col = cc0 + 4 * j4;
                const float* src = Cb + (int64_t)r * ep.ldc + col;
                const bool in = Cb && r < M;
                cv.x = (in && col < N) ? src[0] : 0.f;
                cv.y = (in && col + 1 < N) ? src[1] : 0.f;
                cv.z = (in && col + 2 < N) ? src[2] : 0.f;
                cv.w = (in && col + 3 < N) ? src[3] : 0.f;
              }
              o.x = fmaf(ep.beta, cv.x, o.x);
              o.y = fmaf(ep.beta, cv.y, o.y);
              o.z = fmaf(ep.beta, cv.z, o.z);
              o.w = fmaf(ep.beta, cv.w, o.w);
            }
            *slot = o;
          }
          __syncwarp();
#pragma unroll
          for (int it = 0; it < 8; ++it) {
            const int rr = 4 * it + (lane >> 3), j4 = lane & 7;
            const int r2 = row0 + rr, col = cc0 + 4 * j4;
            if (r2 >= M || col >= N) continue;
            const float4 o = *reinterpret_cast<const float4*>(cb + swz(rr, 4 * j4));
            const float ov[4] = {o.x, o.y, o.z, o.w};
            if (vec && col + 3 < N) {
              if (Cb) *reinterpret_cast<float4*>(Cb + (int64_t)r2 * ep.ldc + col) = o;
              if (Lb)
                *reinterpret_cast<float4*>(Lb + (int64_t)r2 * ep.ld_lo + col) =
                    make_float4(tf32_lo(o.x), tf32_lo(o.y), tf32_lo(o.z), tf32_lo(o.w));
            } else {
              for (int e = 0; e < 4 && col + e < N; ++e) {
                if (Cb) Cb[(int64_t)r2 * ep.ldc + col + e] = ov[e];
                if (Lb) Lb[(int64_t)r2 * ep.ld_lo + col + e] = tf32_lo(ov[e]);
              }
            }
          }
          if (SYM && m0 != n0) {
            // the mirror tile: element (r, j) of this block also goes to C[j][r]
#pragma unroll 1
            for (int it = 0; it < 8; ++it) {
              const int jj = 4 * it + (lane >> 3), r4 = 4 * (lane & 7);
              const int mrow = cc0 + jj, mcol = row0 + r4;  // row and column in C
              if (mrow >= N || mcol + 3 >= M) continue;    // M = N, a multiple of 4
              const float4 o = make_float4(cb[swz(r4, jj)], cb[swz(r4 + 1, jj)], cb[swz(r4 + 2, jj)],
                                           cb[swz(r4 + 3, jj)]);
              *reinterpret_cast<float4*>(Cb + (int64_t)mrow * ep.ldc + mcol) = o;
              if (Lb)
                *reinterpret_cast<float4*>(Lb + (int64_t)mrow * ep.ld_lo + mcol) =
                    make_float4(tf32_lo(o.x), tf32_lo(o.y), tf32_lo(o.z), tf32_lo(o.w));
            }
          }
          __syncwarp();
        } else {
          // C^T: element (row r = this lane, column j) is stored at column-major block position (j, r)
          const int r = row0 + lane;
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            float o = ep.alpha * acc[c][j];
            float* slot = cb + swz(j, lane);
            if (ep.beta != 0.f) {
              const int col = cc0 + j;
              const float cv = pre ? *slot : ((Cb && r < M && col < N) ? Cb[(int64_t)col * ep.ldc + r] : 0.f);
              o = fmaf(ep.beta, cv, o);
            }
            *slot = o;
          }
          __syncwarp();
#pragma unroll
          for (int it = 0; it < 8; ++it) {
            const int jj = 4 * it + (lane >> 3), r4 = lane & 7;
            const int col = cc0 + jj, r2 = row0 + 4 * r4;
            if (col >= N || r2 >= M) continue;
            const float4 o = *reinterpret_cast<const float4*>(cb + swz(jj, 4 * r4));
            const float ov[4] = {o.x, o.y, o.z, o.w};
            if (vec && r2 + 3 < M) {
              if (Cb) *reinterpret_cast<float4*>(Cb + (int64_t)col * ep.ldc + r2) = o;
              if (Lb)
                *reinterpret_cast<float4*>(Lb + (int64_t)col * ep.ld_lo + r2) =
                    make_float4(tf32_lo(o.x), tf32_lo(o.y), tf32_lo(o.z), tf32_lo(o.w));
            } else {
              for (int e = 0; e < 4 && r2 + e < M; ++e) {
                if (Cb) Cb[(int64_t)col * ep.ldc + r2 + e] = ov[e];
                if (Lb) Lb[(int64_t)col * ep.ld_lo + r2 + e] = tf32_lo(ov[e]);
              }
            }
          }
          __syncwarp();
        }
      }
    }
    // copies of a tile abandoned after a timeout still land before shared memory goes away
    if (PRE) asm volatile("cp.async.wait_all;" ::: "memory");
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(C::TMEM_COLS));
  }
}

// ---- host side ---------------------------------------------------------------------

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// Tensor map of `batch` row-major rows x K fp32 matrices, tiles of box_rows x 32.
bool make_map(CUtensorMap* map, const float* base, int rows, int K, int64_t ld, int64_t batch_stride, int batch,
              int box_rows) {
  auto fn = encode_fn();
  if (!fn || !base) return false;
  if ((reinterpret_cast<uintptr_t>(base) & 15) || (ld & 3) || ld < K) return false;
  if (batch <= 1) batch_stride = ld * rows;
  if ((batch_stride & 3) || batch_stride < ld * rows) return false;
  cuuint64_t dims[3] = {(cuuint64_t)K, (cuuint64_t)rows, (cuuint64_t)(batch < 1 ? 1 : batch)};
  cuuint64_t strides[2] = {(cuuint64_t)ld * 4, (cuuint64_t)batch_stride * 4};
  cuuint32_t box[3] = {(cuuint32_t)BK, (cuuint32_t)box_rows, 1};
  cuuint32_t es[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<float*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int BN, int STAGES, bool PRE, bool CVTA = false, bool TR = false, bool LO = false, bool VEC = false,
          bool SYM = false>
cudaError_t launch(const TcOperand& A, const TcOperand& B, int M, int N, int K, int batch, const TcEpilogue& ep,
                   cudaStream_t s, int ksplit = 1) {
  using C = Cfg<BN, STAGES, PRE>;
  CUtensorMap m[4];
  const int amod = A.batch > 0 ? A.batch : batch;
  const int bmod = B.batch > 0 ? B.batch : batch;
  if (!make_map(&m[0], A.hi, M, K, A.ld, A.stride, amod, BM) ||
      !make_map(&m[1], CVTA ? A.hi : A.lo, M, K, A.ld, A.stride, amod, BM) ||
      !make_map(&m[2], B.hi, N, K, B.ld, B.stride, bmod, BN) || !make_map(&m[3], B.lo, N, K, B.ld, B.stride, bmod, BN))
    return cudaErrorInvalidValue;
  // the shared-memory attribute belongs to each device's context: one bit per device that has it
  static std::atomic<uint64_t> attr_set{0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) dev = 0;
  const uint64_t bit = (dev >= 0 && dev < 64) ? uint64_t(1) << dev : 0;
  if (bit == 0 || !(attr_set.load(std::memory_order_relaxed) & bit)) {
    cudaError_t e =
        cudaFuncSetAttribute(gemm_tc_kernel<BN, STAGES, PRE, CVTA, TR, LO, VEC, SYM>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             C::SMEM);
    if (e != cudaSuccess) return e;
    attr_set.fetch_or(bit, std::memory_order_relaxed);
  }
  const int64_t ntm = (M + BM - 1) / BM;
  const int64_t ntiles = (SYM ? ntm * (ntm + 1) / 2 : (int64_t)((N + BN - 1) / BN) * ntm) * batch * ksplit;
  if (ntiles > (int64_t)1 << 30) return cudaErrorInvalidValue;
  // K up to 2048: a CTA runs several tiles so that the next tile's loads and MMAs overlap the
  // current epilogue, keeping about four waves of CTAs over the 152 SMs (for longer K the
  // epilogue is a small part of a tile's time)
  const int kblocks = (K + BK - 1) / BK;
  const int tpc = kblocks > 64 ? 1 : (int)std::max<int64_t>(1, std::min<int64_t>(8, ntiles / (4 * 152)));
  const int grid = (int)((ntiles + tpc - 1) / tpc);
  gemm_tc_kernel<BN, STAGES, PRE, CVTA, TR, LO, VEC, SYM><<<grid, C::THREADS, C::SMEM, s>>>(m[0], m[1], m[2], m[3], M, N, K, batch, amod,
                                                                     bmod, tpc, ksplit, ep);
  return cudaGetLastError();
}

// C_b = alpha * sum_s P_(s*batch+b) (M x N partial sums, contiguous) and its lo part,
// 16-byte units along N (N a multiple of 4).
__global__ void split_reduce_kernel(const float* P, int ksplit, int batch, int M, int N, float alpha, float* C,
                                    int64_t ldc, int64_t c_stride, float* C_lo) {
  const int b = blockIdx.y;
  const int64_t mn = (int64_t)M * N, n4 = mn / 4;
  for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < n4; u += (int64_t)gridDim.x * blockDim.x) {
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int sp = 0; sp < ksplit; ++sp) {
      const float4 v = reinterpret_cast<const float4*>(P + ((int64_t)sp * batch + b) * mn)[u];
      acc.x += v.x;
      acc.y += v.y;
      acc.z += v.z;
      acc.w += v.w;
    }
    const float4 o = make_float4(alpha * acc.x, alpha * acc.y, alpha * acc.z, alpha * acc.w);
    const int64_t e = 4 * u, i = e / N, j = e - i * N;
    *reinterpret_cast<float4*>(C + (int64_t)b * c_stride + i * ldc + j) = o;
    if (C_lo)
      *reinterpret_cast<float4*>(C_lo + (int64_t)b * c_stride + i * ldc + j) =
          make_float4(tf32_lo(o.x), tf32_lo(o.y), tf32_lo(o.z), tf32_lo(o.w));
  }
}

// One instantiation per (transposed output, lo output): each kernel's epilogue then carries
// only the store path it uses.
// With `vec` (C and its lo part 16-byte aligned, rows of 16-byte multiples) the kernel has no
// element-wise store path either.
template <int BN, int STAGES, bool PRE, bool CVTA, bool VEC>
cudaError_t launch_tlv(bool tr, bool lo, const TcOperand& A, const TcOperand& B, int M, int N, int K, int batch,
                       const TcEpilogue& ep, cudaStream_t s) {
  if (tr) return lo ? launch<BN, STAGES, PRE, CVTA, true, true, VEC>(A, B, M, N, K, batch, ep, s)
                    : launch<BN, STAGES, PRE, CVTA, true, false, VEC>(A, B, M, N, K, batch, ep, s);
  return lo ? launch<BN, STAGES, PRE, CVTA, false, true, VEC>(A, B, M, N, K, batch, ep, s)
            : launch<BN, STAGES, PRE, CVTA, false, false, VEC>(A, B, M, N, K, batch, ep, s);
}
template <int BN, int STAGES, bool PRE, bool CVTA>
cudaError_t launch_tl(bool tr, bool lo, bool vec, const TcOperand& A, const TcOperand& B, int M, int N, int K,
                      int batch, const TcEpilogue& ep, cudaStream_t s) {
  if constexpr (PRE) {
    return launch_tlv<BN, STAGES, PRE, CVTA, true>(tr, lo, A, B, M, N, K, batch, ep, s);
  } else {
    if (vec) return launch_tlv<BN, STAGES, PRE, CVTA, true>(tr, lo, A, B, M, N, K, batch, ep, s);
    return launch_tlv<BN, STAGES, PRE, CVTA, false>(tr, lo, A, B, M, N, K, batch, ep, s);
  }
}

// How many K splits give the fewest idle SMs in the last wave, for a launch of `tiles` tiles
// with kblocks K blocks (each split keeps at least 16 K blocks, at most 16 splits), within `cap`
// partial matrices.
int choose_ksplit(int64_t tiles, int kblocks, int64_t cap) {
  if (kblocks < 32 || tiles >= 2 * 152) return 1;
  int best = 1;
  double best_eff = 0.0;
  for (int sp = 1; sp <= 16 && kblocks / sp >= 16 && sp <= cap; ++sp) {
    const int64_t ctas = tiles * sp;
    const double eff = (double)ctas / (double)(((ctas + 151) / 152) * 152);
    if (eff > best_eff + 0.02) {
      best_eff = eff;
      best = sp;
    }
  }
  const int kper = (kblocks + best - 1) / best;
  return (kblocks + kper - 1) / kper;  // no empty split
}

}  // namespace tc

namespace {
// soap_wait_limit's settings, read by every launch
std::atomic<uint64_t> g_wait_ns{0};
std::atomic<const int*> g_hold{nullptr};
}  // namespace

void set_wait_limit(uint64_t ns, const int* hold) {
  g_wait_ns.store(ns, std::memory_order_relaxed);
  g_hold.store(hold, std::memory_order_relaxed);
}

cudaError_t gemm_tc_nt(int M, int N, int K, int batch, const TcOperand& A, const TcOperand& B,
                       const TcEpilogue& ep_in, cudaStream_t s, int family, float* split_ws, size_t split_ws_floats) {
  if (M <= 0 || N <= 0 || batch <= 0) return cudaSuccess;
  TcEpilogue ep = ep_in;
  ep.wait_ns = g_wait_ns.load(std::memory_order_relaxed);
  ep.hold = g_hold.load(std::memory_order_relaxed);
  if (batch > 65535) return cudaErrorInvalidValue;
  const double flops = 2.0 * M * N * (double)K * batch;  // algorithmic (4 tf32 products each on the pipe)
  const double bytes = 4.0 * ((A.lo ? 2.0 : 1.0) * (double)M * K * (A.batch > 0 ? A.batch : batch) +
                              2.0 * (double)N * K * (B.batch > 0 ? B.batch : batch) +
                              (double)M * N * batch * ((ep.beta != 0.f ? 2 : 1) + (ep.C_lo ? 1 : 0)));
  ProfScope prof(family, flops, bytes, s);
  // an epilogue that reads C gives one pipeline stage's shared memory to the C tile, which it
  // prefetches in 16-byte units: C (and its lo part) 16-byte aligned with rows of 16-byte
  // multiples; otherwise the kernel without the prefetch reads C element by element
  auto al16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; };
  const bool pre = ep.beta != 0.f && (ep.C || ep.C_ptrs) && (ep.ldc & 3) == 0 && (ep.c_stride & 3) == 0 &&
                   (!ep.C || al16(ep.C)) && ((ep.transpose ? M : N) & 3) == 0 &&
                   (!ep.C_lo || ((ep.ld_lo & 3) == 0 && (ep.lo_stride & 3) == 0 && al16(ep.C_lo)));
  // few tiles and a long K: split K over more CTAs (plain row-major outputs only)
  int ksplit = 1;
  const bool splittable = split_ws && ep.C && !ep.C_ptrs && !ep.transpose && ep.beta == 0.f && (N & 3) == 0 &&
                          (ep.ldc & 3) == 0 && (ep.c_stride & 3) == 0 && (!ep.C_lo || (ep.ld_lo == ep.ldc && ep.lo_stride == ep.c_stride)) &&
                          (reinterpret_cast<uintptr_t>(ep.C) & 15) == 0;
  if (splittable) {
    const int bn = N <= 32 ? 32 : 128;
    const int64_t tiles = (int64_t)((N + bn - 1) / bn) * ((M + tc::BM - 1) / tc::BM) * batch;
    ksplit = tc::choose_ksplit(tiles, (K + tc::BK - 1) / tc::BK, (int64_t)(split_ws_floats / ((size_t)M * N * batch)));
  }
  // an A given without its lo part gets it formed in the kernel (products whose C is not read)
  const bool cvt = A.lo == nullptr;
  if (cvt && (pre || ep.transpose)) return cudaErrorInvalidValue;
  if (B.lo == nullptr) return cudaErrorInvalidValue;
  if (ksplit > 1) {
    TcEpilogue pe{split_ws, nullptr, N, (int64_t)M * N, nullptr, N, (int64_t)M * N, 0, 1.f, 0.f, ep.status};
    pe.wait_ns = ep.wait_ns;
    pe.hold = ep.hold;
    cudaError_t e = N <= 32 ? (cvt ? tc::launch<32, 5, false, true>(A, B, M, N, K, batch, pe, s, ksplit)
                                   : tc::launch<32, 5, false>(A, B, M, N, K, batch, pe, s, ksplit))
                            : (cvt ? tc::launch<128, 3, false, true>(A, B, M, N, K, batch, pe, s, ksplit)
                                   : tc::launch<128, 3, false>(A, B, M, N, K, batch, pe, s, ksplit));
    if (e != cudaSuccess) return e;
    const int64_t n4 = (int64_t)M * N / 4;
    const int blocks = (int)std::min<int64_t>((n4 + 255) / 256, std::max(1, 1216 / batch));
    tc::split_reduce_kernel<<<dim3(blocks, batch), 256, 0, s>>>(split_ws, ksplit, batch, M, N, ep.alpha, ep.C, ep.ldc,
                                                                ep.c_stride, ep.C_lo);
    return cudaGetLastError();
  }
  const bool tr = ep.transpose != 0, lo = ep.C_lo != nullptr;
  const bool vec = !ep.C_ptrs && ep.C && al16(ep.C) && (ep.ldc & 3) == 0 && (ep.c_stride & 3) == 0 &&
                   ((tr ? M : N) & 3) == 0 &&
                   (!ep.C_lo || ((ep.ld_lo & 3) == 0 && (ep.lo_stride & 3) == 0 && al16(ep.C_lo)));
  if (cvt)
    return N <= 32 ? tc::launch_tl<32, 5, false, true>(false, lo, vec, A, B, M, N, K, batch, ep, s)
                   : tc::launch_tl<128, 3, false, true>(false, lo, vec, A, B, M, N, K, batch, ep, s);
  if (N <= 32)
    return pre ? tc::launch_tl<32, 4, true, false>(tr, lo, vec, A, B, M, N, K, batch, ep, s)
               : tc::launch_tl<32, 5, false, false>(tr, lo, vec, A, B, M, N, K, batch, ep, s);
  return pre ? tc::launch_tl<128, 2, true, false>(tr, lo, vec, A, B, M, N, K, batch, ep, s)
             : tc::launch_tl<128, 3, false, false>(tr, lo, vec, A, B, M, N, K, batch, ep, s);
}

cudaError_t gemm_tc_syrk(int M, int K, int batch, const TcOperand& A, const TcEpilogue& ep_in, cudaStream_t s,
                         int family) {
  if (M <= 0 || batch <= 0) return cudaSuccess;
  if (batch > 65535) return cudaErrorInvalidValue;
  auto al16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; };
  // the symmetric kernel stores row-major C and its lo part with 16-byte stores, both halves
  const bool ok = ep_in.C && !ep_in.C_ptrs && !ep_in.transpose && ep_in.C_lo && A.lo && al16(ep_in.C) &&
                  al16(ep_in.C_lo) && (M & 3) == 0 && (ep_in.ldc & 3) == 0 && (ep_in.c_stride & 3) == 0 &&
                  (ep_in.ld_lo & 3) == 0 && (ep_in.lo_stride & 3) == 0;
  if (!ok) return gemm_tc_nt(M, M, K, batch, A, A, ep_in, s, family);
  TcEpilogue ep = ep_in;
  ep.wait_ns = g_wait_ns.load(std::memory_order_relaxed);
  ep.hold = g_hold.load(std::memory_order_relaxed);
  const double ntm = (double)((M + tc::BM - 1) / tc::BM);
  const double tiles = ntm * (ntm + 1) / 2 * batch;
  const double flops = 2.0 * tc::BM * tc::BM * (double)K * tiles;  // the lower tiles' products
  const double bytes = 4.0 * (2.0 * (double)M * K * (A.batch > 0 ? A.batch : batch) +
                              (double)M * M * batch * ((ep.beta != 0.f ? 1.5 : 1.0) + 1.0));
  ProfScope prof(family, flops, bytes, s);
  return ep.beta != 0.f ? tc::launch<128, 2, true, false, false, true, true, true>(A, A, M, M, K, batch, ep, s)
                        : tc::launch<128, 3, false, false, false, true, true, true>(A, A, M, M, K, batch, ep, s);
}

}  // namespace soap
