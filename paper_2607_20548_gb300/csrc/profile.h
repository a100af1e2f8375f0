// Per-launch CUDA-event timing of the library's kernels (enabled by soap_profile_begin).
//
// While a Profiler is installed for the calling thread, every kernel launch the library
// makes is bracketed by two events recorded on the launch stream, and tagged with its
// kernel family and its algorithmic FLOPs and bytes. soap_profile_end() synchronises and
// sums the durations per family.
#pragma once

#include <cuda_runtime.h>

#include <vector>

namespace soap {

enum KernelFamily : int {
  kFamGemmSimt = 0,   // CUDA-core fp32 GEMM
  kFamGemmTc = 1,     // tcgen05 GEMM: fp32 as four TF32 products, or bf16 (Muon)
  kFamQrPanel = 2,    // cluster panel factorisation of the QR
  kFamElementwise = 3,// momentum / Adam / weight update
  kFamOther = 4,      // norms, identity fills
  kFamQrUpdate = 5,   // tensor-core products of the QR's block updates (at the roofline ridge)
  kNumFamilies = 6,
};

struct Profiler {
  std::vector<cudaEvent_t> events;
  struct Rec {
    int family;
    double flops;
    double bytes;
  };
  std::vector<Rec> recs;
  size_t capacity = 0;  // records
  bool overflow = false;
  bool serial = false;  // each timed launch starts on an idle device
};

extern thread_local Profiler* t_profiler;

// RAII bracket around one launch; a no-op unless a profiler is installed.
class ProfScope {
 public:
  ProfScope(int family, double flops, double bytes, cudaStream_t s);
  ~ProfScope();

 private:
  int idx_ = -1;
  cudaStream_t s_;
};

}  // namespace soap
