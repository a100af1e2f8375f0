// soap_qr_static: the batched QR refresh of soap_qr, with its workspace taken from a
// fixed array compiled into the library instead of from the caller.
//
// Who needs it: a caller that cannot hand out device memory at the moment it wants a QR.
// Some run where a cudaMalloc/cudaFree is not acceptable because either call may wait
// for the whole device to go idle; others do not own their process's device memory at
// all (a framework's caching pool or a fixed budget handed out at start-up owns it) and
// have no way to give this library a buffer. This entry point asks them for nothing but
// the inputs and outputs.
#include <cstdint>
#include <mutex>

#include "soap_internal.h"

namespace {

// 32 MiB: room for the workspace of one 1024 x 1024 matrix (about 29 MB) or of several
// smaller ones (e.g. 3 of 512 x 512). Every GPU that loads the library keeps this array
// until the process exits.
constexpr size_t kScratchBytes = size_t(32) << 20;
__device__ __align__(256) unsigned char g_qr_scratch[kScratchBytes];

// Device address of g_qr_scratch per device, looked up once with that device current.
constexpr int kMaxDevices = 64;
std::mutex g_scratch_mutex;
void* g_scratch_addr[kMaxDevices] = {};

}  // namespace

extern "C" soap_status_t soap_qr_static(int32_t n, int32_t batch, const float* P, float* Q, uint8_t* skip,
                                        float tol, int32_t* status, soap_stream_t stream) {
  if (n <= 0 || n > 8192 || (n & 3) || batch <= 0 || batch > 65535 || !P || !Q || !skip || !(tol >= 0.f))
    return SOAP_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(P) | reinterpret_cast<uintptr_t>(Q)) & 15) return SOAP_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(status) & 3) return SOAP_ERR_INVALID_ARG;
  const size_t qb = soap::qr_workspace_bytes(n, batch);
  if (qb + 256 > kScratchBytes) return SOAP_ERR_INVALID_ARG;  // more than the fixed array holds
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return SOAP_ERR_CUDA;
  void* base = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_scratch_mutex);
    if (!g_scratch_addr[dev]) {
      // host code only has a stand-in for the array's name: ask the runtime where it lives
      void* p = nullptr;
      if (cudaGetSymbolAddress(&p, g_qr_scratch) != cudaSuccess || !p) return SOAP_ERR_CUDA;
      g_scratch_addr[dev] = p;
    }
    base = g_scratch_addr[dev];
  }
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  // the array keeps the previous call's contents; only the status word must start at zero
  // (every other region is written before it is read). The word is the caller's if given, so
  // that a breakdown or a wait that gave up can be read back; else it sits in the array.
  int* word = status ? reinterpret_cast<int*>(status) : reinterpret_cast<int*>(static_cast<char*>(base) + qb);
  if (cudaMemsetAsync(word, 0, sizeof(int), s) != cudaSuccess) return SOAP_ERR_CUDA;
  return soap::qr_q(n, batch, P, Q, skip, tol, base, qb, word, s) == cudaSuccess ? SOAP_OK : SOAP_ERR_CUDA;
}
