// Batched bf16 GEMM on the 5th-generation tensor cores (tcgen05, kind::f16), fp32 accumulation:
//
//   out_b = alpha * A_b * B_b^T + beta * Cin_b       (A_b M x K, B_b N x K, both row-major)
//
// written as bf16 (row-major, and optionally transposed as well) and/or fp32. It serves the
// Newton-Schulz iterations of Muon, which run in bf16 (products of bf16 operands accumulated
// in fp32, results stored in bf16).
//
// Persistent CTAs (one per SM) walk the output tiles (128 x 128) in groups of 8 row tiles.
// Warp 0 issues the TMA loads of 64-element K slices (one 128-byte swizzle row per matrix
// row) into a 4-stage ring, warp 1 issues the MMAs (M = 128, N = 128, K = 16 per instruction)
// into one of two TMEM accumulators, used in turn by consecutive tiles so that a tile's
// epilogue overlaps the next tile's MMAs, and 8 epilogue warps drain the accumulator
// (tensor memory -> registers -> alpha/beta -> bf16/fp32 stores). Every mbarrier wait gives
// up after ~2 s of %globaltimer time, records kStatusTimeout and lets the CTA drain and free
// its tensor memory instead of hanging.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <atomic>
#include <mutex>

#include "profile.h"
#include "soap_internal.h"

namespace soap {
namespace bf16g {
namespace {

constexpr int BM = 128;
constexpr int BN = 128;
constexpr int BK = 64;  // bf16 elements per K slice = one 128-byte swizzle row
constexpr int STAGES = 4;
constexpr int NACC = 2;
constexpr int EPI = 8;
constexpr int THREADS = 64 + 32 * EPI;
constexpr int TILE_A = BM * BK * 2;
constexpr int TILE_B = BN * BK * 2;
constexpr int STAGE = TILE_A + TILE_B;
constexpr int SMEM = STAGES * STAGE + 1024 + 256;
constexpr uint32_t TMEM_COLS = NACC * BN;
constexpr int GM = 8;
constexpr uint64_t kWaitNs = 2000000000ull;

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

// Instruction descriptor for kind::f16: D = f32, A = B = bf16, both K-major.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(N >> 3) << 17) |
         (static_cast<uint32_t>(M >> 4) << 24);
}

__device__ __forceinline__ void umma_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(tmem_d),
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

// Tile t -> (m0, n0, batch index), in groups of GM row tiles (m fastest inside a group).
__device__ __forceinline__ void tile_coords(int t, int ntm, int ntn, int& m0, int& n0, int& b) {
  const int per = ntm * ntn;
  b = t / per;
  const int r = t - b * per;
  const int g = r / (GM * ntn);
  const int first = g * GM;
  const int gsz = min(GM, ntm - first);
  const int w = r - g * GM * ntn;
  m0 = (first + w % gsz) * BM;
  n0 = (w / gsz) * BN;
}

__global__ void __launch_bounds__(THREADS, 1)
    gemm_bf16_kernel(const __grid_constant__ CUtensorMap ta, const __grid_constant__ CUtensorMap tb, int M, int N,
                     int K, int batch, Bf16Epilogue ep) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE);
  uint64_t* empty = full + STAGES;
  uint64_t* acc_full = empty + STAGES;
  uint64_t* acc_empty = acc_full + NACC;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(acc_empty + NACC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);
  volatile int* consumed = abort_flag + 1;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int kblocks = (K + BK - 1) / BK;
  const int ntn = (N + BN - 1) / BN, ntm = (M + BM - 1) / BM;
  const int ntiles = ntn * ntm * batch;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < NACC; ++a) {
      mbar_init(&acc_full[a], 1);
      mbar_init(&acc_empty[a], EPI);
    }
    *abort_flag = 0;
    *consumed = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0 && lane == 0) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&ta)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tb)) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_holder)),
                 "r"(TMEM_COLS));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;

  if (warp == 0) {
    if (lane == 0) {
      int g = 0, issued = 0;
      for (int t = blockIdx.x; t < ntiles && !*abort_flag; t += gridDim.x) {
        int m0, n0, b;
        tile_coords(t, ntm, ntn, m0, n0, b);
        for (int kb = 0; kb < kblocks; ++kb, ++g) {
          const int s = g % STAGES;
          if (!mbar_wait(&empty[s], ((g / STAGES) & 1) ^ 1) || *abort_flag) {
            *abort_flag = 1;
            break;
          }
          mbar_expect_tx(&full[s], STAGE);
          const uint32_t st = smem_u32(smem + s * STAGE);
          tma_load_3d(st, &ta, &full[s], kb * BK, m0, b);
          tma_load_3d(st + TILE_A, &tb, &full[s], kb * BK, n0, b);
          issued = g + 1;
        }
      }
      if (*abort_flag) {
        // let copies already in flight land before the CTA's shared memory goes away
        for (int gg = *consumed; gg < issued; ++gg) mbar_wait(&full[gg % STAGES], (gg / STAGES) & 1);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16(BM, BN);
      int g = 0, tl = 0;
      for (int t = blockIdx.x; t < ntiles && !*abort_flag; t += gridDim.x, ++tl) {
        const int a = tl % NACC;
        if (tl >= NACC && !mbar_wait(&acc_empty[a], ((tl / NACC) & 1) ^ 1)) {
          *abort_flag = 1;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + static_cast<uint32_t>(a * BN);
        bool ok = true;
        for (int kb = 0; kb < kblocks; ++kb, ++g) {
          const int s = g % STAGES;
          if (!mbar_wait(&full[s], (g / STAGES) & 1) || *abort_flag) {
            ok = false;
            break;
          }
          *consumed = g + 1;
          tc_fence_after();
          const uint32_t a_s = smem_u32(smem + s * STAGE);
          const uint32_t b_s = a_s + TILE_A;
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk) {
            const uint32_t off = kk * 32;  // 16 bf16 = 32 bytes along K inside the swizzle row
            umma_bf16(d, desc_sw128(a_s + off), desc_sw128(b_s + off), idesc, (kb | kk) != 0);
          }
          umma_commit(&empty[s]);  // frees the stage once these MMAs have read it
        }
        if (!ok) {
          *abort_flag = 1;
          break;
        }
        umma_commit(&acc_full[a]);  // hands the tile's sum to the epilogue warps
      }
    }
  } else {
    const int q = warp & 3;                  // accumulator lanes 32q .. 32q+31
    const int colbase = ((warp - 2) / 4) * 64;  // columns colbase .. colbase+63
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(32 * q) << 16);
    int tl = 0;
    for (int t = blockIdx.x; t < ntiles; t += gridDim.x, ++tl) {
      int m0, n0, b;
      tile_coords(t, ntm, ntn, m0, n0, b);
      const int a = tl % NACC;
      if (!mbar_wait(&acc_full[a], (tl / NACC) & 1) || *abort_flag) {
        if (lane == 0 && ep.status) atomicOr(ep.status, kStatusTimeout);
        *abort_flag = 1;
        break;
      }
      tc_fence_after();
      float v[2][32];
      tmem_ld32(lane_base + static_cast<uint32_t>(a * BN + colbase), v[0]);
      tmem_ld32(lane_base + static_cast<uint32_t>(a * BN + colbase + 32), v[1]);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(&acc_empty[a])) : "memory");
      const int r = m0 + 32 * q + lane;  // this lane's output row
      if (r >= M) continue;
      const int64_t ob = (int64_t)b * ep.stride;
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        const int c0 = n0 + colbase + 32 * c;
        if (c0 >= N) continue;
        float o[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) o[j] = ep.alpha * v[c][j];
        if (ep.beta != 0.f && ep.cin) {
          const __nv_bfloat16* src = ep.cin + ob + (int64_t)r * ep.ld + c0;
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            if (c0 + 8 * u >= N) break;
            const uint4 w = *reinterpret_cast<const uint4*>(src + 8 * u);
            const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&w);
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const float2 f = __bfloat1622float2(h2[e]);
              o[8 * u + 2 * e] = fmaf(ep.beta, f.x, o[8 * u + 2 * e]);
              o[8 * u + 2 * e + 1] = fmaf(ep.beta, f.y, o[8 * u + 2 * e + 1]);
            }
          }
        }
        if (ep.out) {
          __nv_bfloat16* dst = ep.out + ob + (int64_t)r * ep.ld + c0;
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            if (c0 + 8 * u >= N) break;
            uint4 w;
            __nv_bfloat162* h2 = reinterpret_cast<__nv_bfloat162*>(&w);
#pragma unroll
            for (int e = 0; e < 4; ++e) h2[e] = __floats2bfloat162_rn(o[8 * u + 2 * e], o[8 * u + 2 * e + 1]);
            *reinterpret_cast<uint4*>(dst + 8 * u) = w;
          }
        }
        if (ep.out_t) {
          // transposed copy: for each column the warp's 32 rows are 32 consecutive elements
          __nv_bfloat16* dst = ep.out_t + (int64_t)b * ep.stride_t + r;
#pragma unroll
          for (int j = 0; j < 32; ++j)
            if (c0 + j < N) dst[(int64_t)(c0 + j) * ep.ld_t] = __float2bfloat16_rn(o[j]);
        }
        if (ep.out_f32) {
          float* dst = ep.out_f32 + (int64_t)b * ep.stride_f32 + (int64_t)r * ep.ld_f32 + c0;
#pragma unroll
          for (int u = 0; u < 8; ++u)
            if (c0 + 4 * u < N)
              *reinterpret_cast<float4*>(dst + 4 * u) = make_float4(o[4 * u], o[4 * u + 1], o[4 * u + 2], o[4 * u + 3]);
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TMEM_COLS));
  }
}

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

// Tensor map of `batch` row-major rows x K bf16 matrices, tiles of box_rows x 64.
bool make_map(CUtensorMap* map, const __nv_bfloat16* base, int rows, int K, int64_t ld, int64_t stride, int batch,
              int box_rows) {
  auto fn = encode_fn();
  if (!fn || !base) return false;
  if ((reinterpret_cast<uintptr_t>(base) & 15) || (ld & 7) || ld < K) return false;
  if (batch <= 1) stride = ld * rows;
  if ((stride & 7) || stride < ld * rows) return false;
  cuuint64_t dims[3] = {(cuuint64_t)K, (cuuint64_t)rows, (cuuint64_t)(batch < 1 ? 1 : batch)};
  cuuint64_t strides[2] = {(cuuint64_t)ld * 2, (cuuint64_t)stride * 2};
  cuuint32_t box[3] = {(cuuint32_t)BK, (cuuint32_t)box_rows, 1};
  cuuint32_t es[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<__nv_bfloat16*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace
}  // namespace bf16g

cudaError_t gemm_bf16_nt(int M, int N, int K, int batch, const __nv_bfloat16* A, int64_t lda, int64_t a_stride,
                         const __nv_bfloat16* B, int64_t ldb, int64_t b_stride, const Bf16Epilogue& ep,
                         cudaStream_t s) {
  using namespace bf16g;
  if (M <= 0 || N <= 0 || batch <= 0) return cudaSuccess;
  if (K <= 0 || batch > 65535 || (N & 7) || (K & 7)) return cudaErrorInvalidValue;
  if ((ep.out || ep.cin) && ((ep.ld & 7) || (ep.stride & 7))) return cudaErrorInvalidValue;
  if (ep.out_f32 && ((ep.ld_f32 & 3) || (ep.stride_f32 & 3))) return cudaErrorInvalidValue;
  ProfScope prof(kFamGemmTc, 2.0 * M * N * (double)K * batch,
                 2.0 * ((double)M * K + (double)N * K) * batch +
                     (double)M * N * batch * ((ep.out ? 2 : 0) + (ep.out_t ? 2 : 0) + (ep.out_f32 ? 4 : 0) +
                                              (ep.beta != 0.f && ep.cin ? 2 : 0)),
                 s);
  CUtensorMap ta, tb;
  if (!make_map(&ta, A, M, K, lda, a_stride, batch, BM) || !make_map(&tb, B, N, K, ldb, b_stride, batch, BN))
    return cudaErrorInvalidValue;
  // the shared-memory attribute belongs to each device's context: one bit per device that has it
  static std::atomic<uint64_t> attr_set{0};
  int dev = 0, sms = 152;
  if (cudaGetDevice(&dev) != cudaSuccess) dev = 0;
  const uint64_t bit = (dev >= 0 && dev < 64) ? uint64_t(1) << dev : 0;
  if (bit == 0 || !(attr_set.load(std::memory_order_relaxed) & bit)) {
    cudaError_t e = cudaFuncSetAttribute(gemm_bf16_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM);
    if (e != cudaSuccess) return e;
    attr_set.fetch_or(bit, std::memory_order_relaxed);
  }
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t ntiles = (int64_t)((N + BN - 1) / BN) * ((M + BM - 1) / BM) * batch;
  if (ntiles > (int64_t)1 << 30) return cudaErrorInvalidValue;
  const int grid = (int)std::min<int64_t>(ntiles, sms);
  gemm_bf16_kernel<<<grid, THREADS, SMEM, s>>>(ta, tb, M, N, K, batch, ep);
  return cudaGetLastError();
}

}  // namespace soap
