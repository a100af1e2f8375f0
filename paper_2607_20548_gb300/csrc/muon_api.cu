// libsoap's Muon ABI (include/muon.h): Alg. Muon batched by shape class.
//
// Per class (same rows x cols), with (r, c) = (rows, cols), or (cols, rows) for a tall class
// that is orthogonalized as its transpose:
//   M <- b1 M + (1-b1) G, ||M||_F^2                     muon_momentum
//   X = M / max(||M||_F, eps) in bf16, and X^T          muon_init_x
//   per Newton-Schulz step i (bf16 tensor-core products, fp32 accumulation):
//     A = X X^T                  A-op X, B-op X                      (r x r, K = c)
//     B = c_i A A^T + b_i A      A-op A, B-op A (A symmetric)        (r x r, K = r)
//     X' = B X + a_i X, X'^T     A-op B, B-op X^T                    (r x c, K = r)
//   (a step with c_i = 0 folds B into the last product: X' = b_i A X + a_i X)
//   W <- (1 - lr wd) W - lr sqrt(max(rows, cols)) X_n     muon_update
#include <algorithm>
#include <cmath>
#include <cstring>
#include <map>
#include <string>
#include <utility>
#include <vector>

#include "../../include/muon.h"
#include "profile.h"
#include "soap_internal.h"

namespace {

struct MuonClass {
  int rows = 0, cols = 0;
  bool tr = false;  // orthogonalized as the transpose (rows > cols)
  int count = 0;
  std::vector<int> members;
  size_t ptr_offset = 0;
  float* M = nullptr;  // [count][rows][cols]
};

}  // namespace

struct muon_s {
  int device = 0;
  muon_hparams hp{};
  std::vector<float> coeffs;  // 3 per Newton-Schulz step
  float lr = 0.f, wd = 0.f;
  std::vector<soap_shape> shapes;
  std::vector<std::pair<int, int>> loc;
  std::vector<MuonClass> classes;
  __nv_bfloat16 *X = nullptr, *X2 = nullptr, *Xt = nullptr, *Xt2 = nullptr, *A = nullptr, *B = nullptr;
  double* norm2 = nullptr;
  int* d_status = nullptr;
  int* h_status = nullptr;
  cudaEvent_t status_ev = nullptr;
  bool status_pending = false;
  void** h_ptrs = nullptr;
  void** d_ptrs = nullptr;
  size_t nptrs = 0;
  cudaEvent_t stage_ev = nullptr;
  bool stage_pending = false;
  std::vector<void*> last_ptrs;
  std::vector<void*> allocs;
  soap::Profiler prof;
  std::string err;
};

namespace {

soap_status_t fail(muon_handle h, soap_status_t code, const std::string& msg) {
  if (h) h->err = msg;
  return code;
}

#define MUON_CUDA(h, expr)                                                                                 \
  do {                                                                                                     \
    cudaError_t e_ = (expr);                                                                               \
    if (e_ != cudaSuccess)                                                                                 \
      return fail(h, e_ == cudaErrorMemoryAllocation ? SOAP_ERR_OOM : SOAP_ERR_CUDA,                      \
                  std::string(#expr) + ": " + cudaGetErrorString(e_));                                    \
  } while (0)

struct DeviceGuard {
  int prev = -1;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
    if (prev != dev) cudaSetDevice(dev);
  }
  ~DeviceGuard() {
    int cur = -1;
    if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
  }
};

cudaError_t dalloc(muon_handle h, void** p, size_t bytes) {
  *p = nullptr;
  if (bytes == 0) return cudaSuccess;
  cudaError_t e = cudaMalloc(p, bytes);
  if (e == cudaSuccess) h->allocs.push_back(*p);
  return e;
}

void free_all(muon_handle h) {
  if (soap::t_profiler == &h->prof) soap::t_profiler = nullptr;
  for (cudaEvent_t ev : h->prof.events) cudaEventDestroy(ev);
  h->prof.events.clear();
  for (void* p : h->allocs) cudaFree(p);
  h->allocs.clear();
  if (h->h_status) cudaFreeHost(h->h_status);
  if (h->h_ptrs) cudaFreeHost(h->h_ptrs);
  if (h->status_ev) cudaEventDestroy(h->status_ev);
  if (h->stage_ev) cudaEventDestroy(h->stage_ev);
  h->h_status = nullptr;
  h->h_ptrs = nullptr;
  h->status_ev = h->stage_ev = nullptr;
}

soap::Bf16Epilogue bepi(muon_handle h, __nv_bfloat16* out, int64_t ld, int64_t stride, const __nv_bfloat16* cin,
                        float alpha, float beta) {
  soap::Bf16Epilogue e{};
  e.out = out;
  e.ld = ld;
  e.stride = stride;
  e.cin = cin;
  e.alpha = alpha;
  e.beta = beta;
  e.status = h->d_status;
  return e;
}

soap_status_t step_class(muon_handle h, MuonClass& c, float* const* params, const float* const* grads,
                         cudaStream_t s) {
  const int B = c.count;
  const int r = c.tr ? c.cols : c.rows, k = c.tr ? c.rows : c.cols;
  const int64_t rk = (int64_t)r * k, rr = (int64_t)r * r, mn = (int64_t)c.rows * c.cols;
  MUON_CUDA(h, cudaMemsetAsync(h->norm2, 0, sizeof(double) * B, s));
  MUON_CUDA(h, soap::muon_momentum(grads, c.M, h->norm2, mn, B, h->hp.beta1, h->d_status, s));
  MUON_CUDA(h, soap::muon_init_x(c.M, h->norm2, h->hp.eps, h->X, h->Xt, c.rows, c.cols, B, c.tr, s));
  __nv_bfloat16 *X = h->X, *Xt = h->Xt, *Xn = h->X2, *Xtn = h->Xt2;
  for (int i = 0; i < h->hp.ns_steps; ++i) {
    const float a = h->coeffs[3 * i], b = h->coeffs[3 * i + 1], cc = h->coeffs[3 * i + 2];
    // A = X X^T
    MUON_CUDA(h, soap::gemm_bf16_nt(r, r, k, B, X, k, rk, X, k, rk, bepi(h, h->A, r, rr, nullptr, 1.f, 0.f), s));
    const __nv_bfloat16* P = h->A;
    float alpha = b;
    if (cc != 0.f) {
      // B = c A A^T + b A
      MUON_CUDA(h, soap::gemm_bf16_nt(r, r, r, B, h->A, r, rr, h->A, r, rr, bepi(h, h->B, r, rr, h->A, cc, b), s));
      P = h->B;
      alpha = 1.f;
    }
    // X' = P X + a X, and X'^T
    soap::Bf16Epilogue e = bepi(h, Xn, k, rk, X, alpha, a);
    e.out_t = Xtn;
    e.ld_t = r;
    e.stride_t = rk;
    MUON_CUDA(h, soap::gemm_bf16_nt(r, k, r, B, P, r, rr, Xt, r, rk, e, s));
    std::swap(X, Xn);
    std::swap(Xt, Xtn);
  }
  // X_n in W's orientation: X (r x k) for a wide class, X^T for a tall one
  const float scale = std::sqrt((float)std::max(c.rows, c.cols));
  MUON_CUDA(h, soap::muon_update(params, c.tr ? Xt : X, mn, B, h->lr, h->wd, scale, s));
  return SOAP_OK;
}

}  // namespace

extern "C" {

void muon_default_hparams(muon_hparams* hp) {
  if (!hp) return;
  hp->lr = 3e-3f;
  hp->beta1 = 0.9f;
  hp->weight_decay = 0.1f;
  hp->eps = 1e-7f;
  hp->ns_steps = 16;
  hp->coeffs = nullptr;
}

soap_status_t muon_create(const soap_shape* shapes, int32_t n, const muon_hparams* hp, int32_t device,
                          muon_handle* out) {
  if (!out) return SOAP_ERR_INVALID_ARG;
  *out = nullptr;
  if (!shapes || n <= 0 || !hp) return SOAP_ERR_INVALID_ARG;
  if (hp->ns_steps < 1 || hp->ns_steps > 64 || !(hp->eps > 0.f)) return SOAP_ERR_INVALID_ARG;
  for (int i = 0; i < n; ++i) {
    const soap_shape& s = shapes[i];
    if (s.rows < 8 || s.cols < 8 || (s.rows & 7) || (s.cols & 7) || s.rows > 65536 || s.cols > 65536)
      return SOAP_ERR_INVALID_ARG;
    if (s.rows * s.cols > (int64_t(1) << 31) - 1) return SOAP_ERR_INVALID_ARG;
  }
  int ndev = 0;
  if (cudaGetDeviceCount(&ndev) != cudaSuccess || device < 0 || device >= ndev) return SOAP_ERR_CUDA;
  DeviceGuard g(device);
  muon_handle h = new muon_s();
  h->device = device;
  h->hp = *hp;
  h->hp.coeffs = nullptr;
  h->lr = hp->lr;
  h->wd = hp->weight_decay;
  for (int i = 0; i < hp->ns_steps; ++i) {
    if (hp->coeffs) {
      h->coeffs.insert(h->coeffs.end(), hp->coeffs + 3 * i, hp->coeffs + 3 * i + 3);
    } else {
      // X p(X^T X) with p(x) = (15 - 10 x + 3 x^2) / 8: the second-order expansion of
      // (1 - e)^(-1/2) at e = 1 - x, whose fixed point is the polar factor
      h->coeffs.insert(h->coeffs.end(), {15.f / 8.f, -10.f / 8.f, 3.f / 8.f});
    }
  }
  h->shapes.assign(shapes, shapes + n);
  h->loc.resize(n);
  std::map<std::pair<int64_t, int64_t>, int> index;
  for (int i = 0; i < n; ++i) {
    auto key = std::make_pair(shapes[i].rows, shapes[i].cols);
    auto it = index.find(key);
    int ci;
    if (it == index.end()) {
      ci = (int)h->classes.size();
      index[key] = ci;
      MuonClass c;
      c.rows = (int)shapes[i].rows;
      c.cols = (int)shapes[i].cols;
      c.tr = c.rows > c.cols;
      h->classes.push_back(c);
    } else {
      ci = it->second;
    }
    h->loc[i] = {ci, h->classes[ci].count};
    h->classes[ci].members.push_back(i);
    h->classes[ci].count++;
  }
  cudaError_t e = cudaSuccess;
  size_t off = 0, ws_rk = 0, ws_rr = 0;
  int max_batch = 0;
  for (auto& c : h->classes) {
    if (c.count > 65535) e = cudaErrorInvalidValue;
    const size_t mn = (size_t)c.count * c.rows * c.cols;
    const size_t r = std::min(c.rows, c.cols);
    c.ptr_offset = off;
    off += 2 * (size_t)c.count;
    if (e == cudaSuccess) e = dalloc(h, (void**)&c.M, mn * 4);
    if (e == cudaSuccess) e = cudaMemset(c.M, 0, mn * 4);
    ws_rk = std::max(ws_rk, mn);
    ws_rr = std::max(ws_rr, (size_t)c.count * r * r);
    max_batch = std::max(max_batch, c.count);
  }
  h->nptrs = off;
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->X, ws_rk * 2);
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->X2, ws_rk * 2);
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->Xt, ws_rk * 2);
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->Xt2, ws_rk * 2);
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->A, ws_rr * 2);
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->B, ws_rr * 2);
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->norm2, (size_t)max_batch * sizeof(double));
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->d_status, sizeof(int));
  if (e == cudaSuccess) e = dalloc(h, (void**)&h->d_ptrs, h->nptrs * sizeof(void*));
  if (e == cudaSuccess) e = cudaMemset(h->d_status, 0, sizeof(int));
  if (e == cudaSuccess) e = cudaMallocHost((void**)&h->h_status, sizeof(int));
  if (e == cudaSuccess) e = cudaMallocHost((void**)&h->h_ptrs, h->nptrs * sizeof(void*));
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->status_ev, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->stage_ev, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    const soap_status_t code = e == cudaErrorMemoryAllocation ? SOAP_ERR_OOM
                               : e == cudaErrorInvalidValue   ? SOAP_ERR_INVALID_ARG
                                                              : SOAP_ERR_CUDA;
    free_all(h);
    delete h;
    cudaGetLastError();
    return code;
  }
  *h->h_status = 0;
  h->last_ptrs.assign(h->nptrs, nullptr);
  *out = h;
  return SOAP_OK;
}

soap_status_t muon_step(muon_handle h, float* const* params, const float* const* grads, soap_stream_t stream_) {
  if (!h) return SOAP_ERR_INVALID_ARG;
  if (!params || !grads) return fail(h, SOAP_ERR_INVALID_ARG, "muon_step: null pointer array");
  const int n = (int)h->shapes.size();
  for (int i = 0; i < n; ++i)
    if (!params[i] || !grads[i] || (reinterpret_cast<uintptr_t>(params[i]) & 15) ||
        (reinterpret_cast<uintptr_t>(grads[i]) & 15))
      return fail(h, SOAP_ERR_INVALID_ARG,
                  "muon_step: matrix " + std::to_string(i) + " has a null or non-16-byte-aligned pointer");
  DeviceGuard g(h->device);
  cudaStream_t s = (cudaStream_t)stream_;
  if (h->status_pending && cudaEventQuery(h->status_ev) == cudaSuccess) {
    h->status_pending = false;
    const int bits = *h->h_status;
    if (bits & soap::kStatusTimeout) return fail(h, SOAP_ERR_TIMEOUT, "muon_step: a device wait timed out earlier");
    if (bits & soap::kStatusNonFinite) return fail(h, SOAP_ERR_NONFINITE, "muon_step: non-finite gradient earlier");
  }
  bool changed = false;
  for (auto& c : h->classes)
    for (int j = 0; j < c.count; ++j) {
      void* pp = params[c.members[j]];
      void* gp = const_cast<float*>(grads[c.members[j]]);
      if (h->last_ptrs[c.ptr_offset + j] != pp || h->last_ptrs[c.ptr_offset + c.count + j] != gp) changed = true;
      h->last_ptrs[c.ptr_offset + j] = pp;
      h->last_ptrs[c.ptr_offset + c.count + j] = gp;
    }
  if (changed) {
    if (h->stage_pending) MUON_CUDA(h, cudaEventSynchronize(h->stage_ev));
    std::memcpy(h->h_ptrs, h->last_ptrs.data(), h->nptrs * sizeof(void*));
    MUON_CUDA(h, cudaMemcpyAsync(h->d_ptrs, h->h_ptrs, h->nptrs * sizeof(void*), cudaMemcpyHostToDevice, s));
    MUON_CUDA(h, cudaEventRecord(h->stage_ev, s));
    h->stage_pending = true;
  }
  for (auto& c : h->classes) {
    const soap_status_t st = step_class(h, c, reinterpret_cast<float* const*>(h->d_ptrs + c.ptr_offset),
                                        reinterpret_cast<const float* const*>(h->d_ptrs + c.ptr_offset + c.count), s);
    if (st != SOAP_OK) return st;
  }
  MUON_CUDA(h, cudaMemcpyAsync(h->h_status, h->d_status, sizeof(int), cudaMemcpyDeviceToHost, s));
  MUON_CUDA(h, cudaEventRecord(h->status_ev, s));
  h->status_pending = true;
  return SOAP_OK;
}

soap_status_t muon_set_lr(muon_handle h, float lr, float weight_decay) {
  if (!h || !(lr >= 0.f) || !(weight_decay >= 0.f)) return SOAP_ERR_INVALID_ARG;
  h->lr = lr;
  h->wd = weight_decay;
  return SOAP_OK;
}

soap_status_t muon_state_get(muon_handle h, int32_t idx, void* dst, soap_stream_t stream) {
  if (!h || idx < 0 || idx >= (int)h->shapes.size() || !dst) return SOAP_ERR_INVALID_ARG;
  DeviceGuard g(h->device);
  const auto [ci, slot] = h->loc[idx];
  const MuonClass& c = h->classes[ci];
  const size_t mn = (size_t)c.rows * c.cols;
  MUON_CUDA(h, cudaMemcpyAsync(dst, c.M + slot * mn, mn * 4, cudaMemcpyDefault, (cudaStream_t)stream));
  return SOAP_OK;
}

soap_status_t muon_state_set(muon_handle h, int32_t idx, const void* src, soap_stream_t stream) {
  if (!h || idx < 0 || idx >= (int)h->shapes.size() || !src) return SOAP_ERR_INVALID_ARG;
  DeviceGuard g(h->device);
  const auto [ci, slot] = h->loc[idx];
  const MuonClass& c = h->classes[ci];
  const size_t mn = (size_t)c.rows * c.cols;
  MUON_CUDA(h, cudaMemcpyAsync(c.M + slot * mn, src, mn * 4, cudaMemcpyDefault, (cudaStream_t)stream));
  return SOAP_OK;
}

soap_status_t muon_status(muon_handle h, soap_stream_t stream) {
  if (!h) return SOAP_ERR_INVALID_ARG;
  DeviceGuard g(h->device);
  MUON_CUDA(h, cudaMemcpyAsync(h->h_status, h->d_status, sizeof(int), cudaMemcpyDeviceToHost, (cudaStream_t)stream));
  MUON_CUDA(h, cudaStreamSynchronize((cudaStream_t)stream));
  const int bits = *h->h_status;
  if (bits & soap::kStatusTimeout) return SOAP_ERR_TIMEOUT;
  if (bits & soap::kStatusNonFinite) return SOAP_ERR_NONFINITE;
  return SOAP_OK;
}

soap_status_t muon_profile_begin(muon_handle h, int64_t max_launches) {
  if (!h || max_launches < 1 || max_launches > (int64_t(1) << 22)) return SOAP_ERR_INVALID_ARG;
  DeviceGuard g(h->device);
  soap::Profiler& p = h->prof;
  while ((int64_t)p.events.size() < 2 * max_launches) {
    cudaEvent_t ev;
    MUON_CUDA(h, cudaEventCreate(&ev));
    p.events.push_back(ev);
  }
  p.capacity = (size_t)max_launches;
  p.recs.clear();
  p.overflow = false;
  soap::t_profiler = &p;
  return SOAP_OK;
}

soap_status_t muon_profile_end(muon_handle h, soap_stream_t stream, soap_kernel_stats* out, int32_t* overflow) {
  if (!h || !out) return SOAP_ERR_INVALID_ARG;
  DeviceGuard g(h->device);
  if (soap::t_profiler == &h->prof) soap::t_profiler = nullptr;
  MUON_CUDA(h, cudaStreamSynchronize((cudaStream_t)stream));
  MUON_CUDA(h, cudaDeviceSynchronize());
  for (int f = 0; f < soap::kNumFamilies; ++f) out[f] = soap_kernel_stats{f, 0, 0.0, 0.0, 0.0};
  const soap::Profiler& p = h->prof;
  for (size_t i = 0; i < p.recs.size(); ++i) {
    float ms = 0.f;
    MUON_CUDA(h, cudaEventElapsedTime(&ms, p.events[2 * i], p.events[2 * i + 1]));
    soap_kernel_stats& o = out[p.recs[i].family];
    o.launches += 1;
    o.ms += ms;
    o.flops += p.recs[i].flops;
    o.bytes += p.recs[i].bytes;
  }
  if (overflow) *overflow = p.overflow ? 1 : 0;
  h->prof.recs.clear();
  return SOAP_OK;
}

const char* muon_last_error(muon_handle h) { return h ? h->err.c_str() : "null handle"; }

void muon_destroy(muon_handle h) {
  if (!h) return;
  DeviceGuard g(h->device);
  cudaDeviceSynchronize();
  free_all(h);
  delete h;
}

}  // extern "C"
