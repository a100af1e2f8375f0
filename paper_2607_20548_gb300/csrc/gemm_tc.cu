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
// K = 8192). Each 32-wide K block is therefore accumulated afresh in one of two TMEM
// accumulators while the epilogue warps drain the other into fp32 registers with
// round-to-nearest adds; the drain of block k overlaps the MMAs of block k+1, and the
// error stays at the level of an fp32 dot product.
//
// CTA: 192 threads. Warp 0 issues the TMA loads (one elected lane), warp 1 allocates
// tensor memory and issues the MMAs (one elected lane), warps 2-5 drain the
// accumulators and run the epilogue: tensor memory -> registers (each warp owns 32 of
// the 128 accumulator lanes) -> alpha/beta -> global, optionally transposed and optionally also writing the lo part
// of the result for a later product. When the epilogue reads C (beta != 0), the
// epilogue warps copy their part of the C tile into shared memory with cp.async while
// the MMAs run, so the epilogue does not wait on one global load per output row.
// Stages are handed over with mbarriers; every
// wait gives up after ~2 s of %globaltimer time, records kStatusTimeout and lets the
// CTA drain and free its tensor memory instead of hanging.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "profile.h"
#include "soap_internal.h"

namespace soap {
namespace tc {

constexpr int BM = 128;
constexpr int BK = 32;  // fp32 elements per K block = one 128-byte swizzle row
constexpr int THREADS = 192;
constexpr uint64_t kWaitNs = 2000000000ull;

template <int BN, int STAGES, bool PRE>
struct Cfg {
  static constexpr int TILE_A = BM * BK * 4;
  static constexpr int TILE_B = BN * BK * 4;
  static constexpr int STAGE = 2 * TILE_A + 2 * TILE_B;
  static constexpr int STAGING = 4 * 32 * 33 * 4;  // per epilogue warp: one 32 x 32 block (+pad)
  static constexpr int CPRE = PRE ? 4 * 32 * BN * 4 : 0;  // prefetched C tile (32 rows per warp)
  static constexpr int SMEM = STAGES * STAGE + STAGING + CPRE + 1024 + 256;
  static constexpr uint32_t TMEM_COLS = 2 * BN;  // two accumulators, used alternately
  static_assert(SMEM <= 232448, "shared memory budget");
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait on an mbarrier phase: false after kWaitNs without completion.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
  if (mbar_try(bar, parity)) return true;
  const uint64_t t0 = globaltimer();
  for (;;) {
    for (int i = 0; i < 256; ++i)
      if (mbar_try(bar, parity)) return true;
    if (globaltimer() - t0 > kWaitNs) return false;
  }
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, uint64_t* bar, int c0, int c1,
                                            int c2) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(
          dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(c0), "r"(c1), "r"(c2)
      : "memory");
}

// Shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row atoms 1024 B apart.
__device__ __forceinline__ uint64_t desc_sw128(uint32_t addr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((addr & 0x3FFFF) >> 4);  // start address
  d |= static_cast<uint64_t>(1) << 16;                 // leading byte offset (unused for this layout)
  d |= static_cast<uint64_t>(1024 >> 4) << 32;         // stride byte offset: next 8-row atom
  d |= static_cast<uint64_t>(1) << 46;                 // descriptor version (sm_100 family)
  d |= static_cast<uint64_t>(2) << 61;                 // 128-byte swizzle
  return d;
}

// Instruction descriptor for kind::tf32: D = f32, A = B = tf32, both K-major.
__host__ __device__ constexpr uint32_t idesc_tf32(int M, int N) {
  return (1u << 4) | (2u << 7) | (2u << 10) | (static_cast<uint32_t>(N >> 3) << 17) |
         (static_cast<uint32_t>(M >> 4) << 24);
}

__device__ __forceinline__ void umma_tf32(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate));
}

__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// tf32 value the tensor core reads from an fp32 word (13 low mantissa bits dropped), and
// the lo part x - trunc(x) rounded to the nearest tf32 (so the tensor core reads it exactly).
__device__ __forceinline__ float tf32_trunc(float x) { return __uint_as_float(__float_as_uint(x) & 0xFFFFE000u); }
__device__ __forceinline__ float tf32_lo(float x) {
  uint32_t r;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x - tf32_trunc(x)));
  return __uint_as_float(r);
}

__device__ __forceinline__ void cp_async16(float* smem_dst, const float* gmem_src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(smem_dst)), "l"(gmem_src),
               "r"(valid ? 16 : 0)
               : "memory");
}

template <int BN, int STAGES, bool PRE>
__global__ void __launch_bounds__(THREADS, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap ta_hi, const __grid_constant__ CUtensorMap ta_lo,
                   const __grid_constant__ CUtensorMap tb_hi, const __grid_constant__ CUtensorMap tb_lo, int M,
                   int N, int K, int a_mod, int b_mod, TcEpilogue ep) {
  using C = Cfg<BN, STAGES, PRE>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  float* staging = reinterpret_cast<float*>(smem + STAGES * C::STAGE);
  float* cpre_all = reinterpret_cast<float*>(smem + STAGES * C::STAGE + C::STAGING);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * C::STAGE + C::STAGING + C::CPRE);
  uint64_t* empty = full + STAGES;
  uint64_t* acc_full = empty + STAGES;  // [2] accumulator a holds a finished K block
  uint64_t* acc_empty = acc_full + 2;   // [2] accumulator a has been drained
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(acc_empty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);
  volatile int* consumed = abort_flag + 1;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n0 = blockIdx.x * BN, m0 = blockIdx.y * BM, b = blockIdx.z;
  const int kblocks = (K + BK - 1) / BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&acc_full[a], 1);
      mbar_init(&acc_empty[a], 4);  // one arrival per epilogue warp
    }
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
      int issued = 0;
      for (int kb = 0; kb < kblocks; ++kb) {
        const int s = kb % STAGES;
        const uint32_t ph = (kb / STAGES) & 1;
        if (!mbar_wait(&empty[s], ph ^ 1) || *abort_flag) {
          *abort_flag = 1;
          break;
        }
        mbar_expect_tx(&full[s], C::STAGE);
        const uint32_t st = smem_u32(smem + s * C::STAGE);
        const int kc = kb * BK;
        tma_load_3d(st, &ta_hi, &full[s], kc, m0, b % a_mod);
        tma_load_3d(st + C::TILE_A, &ta_lo, &full[s], kc, m0, b % a_mod);
        tma_load_3d(st + 2 * C::TILE_A, &tb_hi, &full[s], kc, n0, b % b_mod);
        tma_load_3d(st + 2 * C::TILE_A + C::TILE_B, &tb_lo, &full[s], kc, n0, b % b_mod);
        issued = kb + 1;
      }
      if (*abort_flag) {
        // let copies already in flight land before the CTA's shared memory goes away
        for (int kb = *consumed; kb < issued; ++kb) mbar_wait(&full[kb % STAGES], (kb / STAGES) & 1);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_tf32(BM, BN);
      for (int kb = 0; kb < kblocks; ++kb) {
        const int s = kb % STAGES;
        const uint32_t ph = (kb / STAGES) & 1;
        const int a = kb & 1;
        if (!mbar_wait(&full[s], ph) || (kb >= 2 && !mbar_wait(&acc_empty[a], ((kb >> 1) & 1) ^ 1)) ||
            *abort_flag) {
          *abort_flag = 1;
          break;
        }
        *consumed = kb + 1;
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
  } else {
    const int q = warp & 3;  // this warp may read accumulator lanes 32q .. 32q+31
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(32 * q) << 16);
    float* Cb = ep.C_ptrs ? ep.C_ptrs[b] : (ep.C ? ep.C + (int64_t)b * ep.c_stride : nullptr);
    const int row0 = m0 + 32 * q;  // first of this warp's 32 rows
    // this warp's part of the C tile, copied in while the MMAs run: rows row0.. x BN columns
    // ([row][col]), or for a transposed C the BN columns' 32 entries each ([col][row]);
    // only 16-byte chunks wholly inside C are copied, so partial chunks disable it
    float* cpre = cpre_all + q * 32 * BN;
    const bool pre = PRE && Cb && ep.beta != 0.f && (ep.ldc & 3) == 0 &&
                     (reinterpret_cast<uintptr_t>(Cb) & 15) == 0 && ((ep.transpose ? M : N) & 3) == 0;
    if (pre) {
      if (!ep.transpose) {
        for (int i = lane; i < 32 * (BN / 4); i += 32) {
          const int rr = i / (BN / 4), ch = i % (BN / 4);
          const int r = row0 + rr, col = n0 + 4 * ch;
          const bool ok = r < M && col < N;
          cp_async16(cpre + rr * BN + 4 * ch, ok ? Cb + (int64_t)r * ep.ldc + col : Cb, ok);
        }
      } else {
        for (int i = lane; i < BN * 8; i += 32) {
          const int cc = i / 8, ch = i % 8;
          const int col = n0 + cc, r = row0 + 4 * ch;
          const bool ok = r < M && col < N;
          cp_async16(cpre + cc * 32 + 4 * ch, ok ? Cb + (int64_t)col * ep.ldc + r : Cb, ok);
        }
      }
      asm volatile("cp.async.commit_group;" ::: "memory");
    }
    float acc[BN / 32][32];
#pragma unroll
    for (int c = 0; c < BN / 32; ++c)
#pragma unroll
      for (int j = 0; j < 32; ++j) acc[c][j] = 0.f;
    bool valid = true;
    for (int kb = 0; kb < kblocks; ++kb) {
      const int a = kb & 1;
      if (!mbar_wait(&acc_full[a], (kb >> 1) & 1) || *abort_flag) {
        valid = false;
        break;
      }
      tc_fence_after();
#pragma unroll
      for (int c = 0; c < BN / 32; ++c) {
        float v[32];
        tmem_ld32(lane_base + static_cast<uint32_t>(a * BN + 32 * c), v);
#pragma unroll
        for (int j = 0; j < 32; ++j) acc[c][j] += v[j];
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0)
        asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(&acc_empty[a])) : "memory");
    }
    if (!valid && lane == 0 && ep.status) atomicOr(ep.status, kStatusTimeout);
    if (pre) {
      // the copies complete even when a wait gave up, before the CTA's shared memory goes away
      asm volatile("cp.async.wait_all;" ::: "memory");
      __syncwarp();
    }
    float* Lb = ep.C_lo ? ep.C_lo + (int64_t)b * ep.lo_stride : nullptr;
    if (valid && ep.transpose) {
      // C^T: for a fixed column the 32 lanes (32 consecutive rows) write 128 contiguous bytes
      const int r = row0 + lane;
#pragma unroll
      for (int c = 0; c < BN / 32; ++c) {
        const int col0 = n0 + 32 * c;
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const int col = col0 + j;
          if (col >= N || r >= M) continue;
          const int64_t off = (int64_t)col * ep.ldc + r;
          float out = ep.alpha * acc[c][j];
          if (Cb) {
            if (ep.beta != 0.f) out = fmaf(ep.beta, pre ? cpre[(32 * c + j) * 32 + lane] : Cb[off], out);
            Cb[off] = out;
          }
          if (Lb) Lb[(int64_t)col * ep.ld_lo + r] = tf32_lo(out);
        }
      }
    } else if (valid) {
      // C: each lane holds one row; stage the warp's 32 x 32 block in shared memory so that
      // every global access instruction covers 32 consecutive columns of one row
      float* st = staging + q * (32 * 33);
#pragma unroll
      for (int c = 0; c < BN / 32; ++c) {
        const int col0 = n0 + 32 * c;
        if (col0 >= N) break;  // warp-uniform
#pragma unroll
        for (int j = 0; j < 32; ++j) st[lane * 33 + j] = acc[c][j];
        __syncwarp();
        const int col = col0 + lane;
        for (int rr = 0; rr < 32; ++rr) {
          const int r = row0 + rr;
          if (r >= M) break;  // warp-uniform
          if (col < N) {
            float out = ep.alpha * st[rr * 33 + lane];
            if (Cb) {
              const int64_t off = (int64_t)r * ep.ldc + col;
              if (ep.beta != 0.f) out = fmaf(ep.beta, pre ? cpre[rr * BN + 32 * c + lane] : Cb[off], out);
              Cb[off] = out;
            }
            if (Lb) Lb[(int64_t)r * ep.ld_lo + col] = tf32_lo(out);
          }
        }
        __syncwarp();
      }
    }
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

template <int BN, int STAGES, bool PRE>
cudaError_t launch(const TcOperand& A, const TcOperand& B, int M, int N, int K, int batch, const TcEpilogue& ep,
                   cudaStream_t s) {
  using C = Cfg<BN, STAGES, PRE>;
  CUtensorMap m[4];
  const int amod = A.batch > 0 ? A.batch : batch;
  const int bmod = B.batch > 0 ? B.batch : batch;
  if (!make_map(&m[0], A.hi, M, K, A.ld, A.stride, amod, BM) || !make_map(&m[1], A.lo, M, K, A.ld, A.stride, amod, BM) ||
      !make_map(&m[2], B.hi, N, K, B.ld, B.stride, bmod, BN) || !make_map(&m[3], B.lo, N, K, B.ld, B.stride, bmod, BN))
    return cudaErrorInvalidValue;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e =
        cudaFuncSetAttribute(gemm_tc_kernel<BN, STAGES, PRE>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  dim3 grid((N + BN - 1) / BN, (M + BM - 1) / BM, batch);
  gemm_tc_kernel<BN, STAGES, PRE><<<grid, THREADS, C::SMEM, s>>>(m[0], m[1], m[2], m[3], M, N, K, amod, bmod, ep);
  return cudaGetLastError();
}

}  // namespace tc

cudaError_t gemm_tc_nt(int M, int N, int K, int batch, const TcOperand& A, const TcOperand& B, const TcEpilogue& ep,
                       cudaStream_t s, int family) {
  if (M <= 0 || N <= 0 || batch <= 0) return cudaSuccess;
  if (batch > 65535 || (M + tc::BM - 1) / tc::BM > 65535) return cudaErrorInvalidValue;
  const double flops = 2.0 * M * N * (double)K * batch;  // algorithmic (4 tf32 products each on the pipe)
  const double bytes = 4.0 * (2.0 * (double)M * K * (A.batch > 0 ? A.batch : batch) +
                              2.0 * (double)N * K * (B.batch > 0 ? B.batch : batch) +
                              (double)M * N * batch * ((ep.beta != 0.f ? 2 : 1) + (ep.C_lo ? 1 : 0)));
  ProfScope prof(family, flops, bytes, s);
  // an epilogue that reads C gives one pipeline stage's shared memory to the C tile
  const bool pre = ep.beta != 0.f && (ep.C || ep.C_ptrs);
  if (N <= 32) return pre ? tc::launch<32, 4, true>(A, B, M, N, K, batch, ep, s)
                          : tc::launch<32, 5, false>(A, B, M, N, K, batch, ep, s);
  return pre ? tc::launch<128, 2, true>(A, B, M, N, K, batch, ep, s)
             : tc::launch<128, 3, false>(A, B, M, N, K, batch, ep, s);
}

}  // namespace soap
