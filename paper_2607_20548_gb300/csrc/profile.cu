#include "profile.h"

namespace soap {

thread_local Profiler* t_profiler = nullptr;

ProfScope::ProfScope(int family, double flops, double bytes, cudaStream_t s) : s_(s) {
  Profiler* p = t_profiler;
  if (!p) return;
  if (p->recs.size() >= p->capacity) {
    p->overflow = true;
    return;
  }
  if (p->serial) cudaDeviceSynchronize();
  idx_ = (int)p->recs.size();
  p->recs.push_back({family, flops, bytes});
  cudaEventRecord(p->events[2 * idx_], s_);
}

ProfScope::~ProfScope() {
  if (idx_ >= 0 && t_profiler) cudaEventRecord(t_profiler->events[2 * idx_ + 1], s_);
}

}  // namespace soap
