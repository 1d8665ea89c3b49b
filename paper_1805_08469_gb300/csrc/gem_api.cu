// Host side of the GEM commit ABI (include/gem.h): handle life cycle, argument checks,
// stream plumbing and the staging of host-resident gradients.
#include <cmath>
#include <cstdint>
#include <cstdlib>
#include <new>
#include <vector>

#include "gem_internal.h"

namespace {

// Makes the handle's device current for the duration of a call, then restores the
// caller's device.
class DeviceScope {
 public:
  explicit DeviceScope(int device) {
    if (cudaGetDevice(&prev_) != cudaSuccess) prev_ = -1;
    if (prev_ != device) ok_ = cudaSetDevice(device) == cudaSuccess;
    target_ = device;
  }
  ~DeviceScope() {
    if (prev_ >= 0 && prev_ != target_) cudaSetDevice(prev_);
  }
  bool ok() const { return ok_; }

 private:
  int prev_ = -1;
  int target_ = 0;
  bool ok_ = true;
};

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int cuda_status(gem_t* h, cudaError_t e) {
  if (e == cudaSuccess) return GEM_OK;
  if (h) h->broken = true;
  return GEM_ECUDA;
}

int check_handle(const gem_t* h) {
  if (!h) return GEM_EINVAL;
  if (h->broken) return GEM_ESTATE;
  return GEM_OK;
}

// Launch the commits [0, K) in order; GEM_ECUDA marks the handle broken.
int launch_commits(gem_t* h, const int* order, const float* const* grads, int K) {
  return cuda_status(h, gem::commit_ordered(h, order, grads, K));
}

int check_batch(const gem_t* h, const int* order, const float* const* grads, int K) {
  if (K < 0) return GEM_EINVAL;
  if (K > 0 && (!order || !grads)) return GEM_EINVAL;
  for (int k = 0; k < K; ++k) {
    if (order[k] < 0 || order[k] >= h->n) return GEM_EINVAL;
    if (!grads[k] || !aligned16(grads[k])) return GEM_EINVAL;
  }
  return GEM_OK;
}

int ensure_staging(gem_t* h) {
  if (h->stage) return GEM_OK;
  const size_t bytes = size_t(2 * gem::kStageChunk) * h->stride * sizeof(float);
  if (cudaMalloc(&h->stage, bytes) != cudaSuccess) {
    cudaGetLastError();
    h->stage = nullptr;
    return GEM_ENOMEM;
  }
  cudaError_t e = cudaStreamCreateWithFlags(&h->copy_stream, cudaStreamNonBlocking);
  for (int i = 0; i < 2 && e == cudaSuccess; ++i) {
    e = cudaEventCreateWithFlags(&h->stage_filled[i], cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->stage_free[i], cudaEventDisableTiming);
  }
  return cuda_status(h, e);
}

}  // namespace

namespace gem {

cudaError_t commit_ordered(gem_ctx* h, const int* order, const float* const* grads, int K,
                           float* const* pi_out, unsigned* pi_counts, const long long* pi_seg,
                           int pi_nseg) {
  if (pi_counts && (K > kMaxBatchPerLaunch || K * pi_nseg * 2 > kMaxCountWords || !pi_out))
    return cudaErrorInvalidValue;   // counts are kept by one launch
  BatchArgs a;
  a.pi_counts = pi_counts;
  a.pi_seg = pi_seg;
  a.pi_nseg = pi_nseg;
  a.count_smem_at = 0;
  a.theta = h->theta;
  a.m = h->m;
  a.s = h->s;
  a.P = h->P;
  a.stride = h->stride;
  a.eta = h->eta;
  a.mu = h->mu;
  a.eps = h->eps;
  a.energy_scale = 1.f;
  switch (h->mode) {
    case GEM_MODE_KAPPA_SQRT:
      a.rule = kRuleScaled;
      a.energy_scale = sqrtf(h->kappa);  // correctly rounded fp32 square root
      break;
    case GEM_MODE_KAPPA_LINEAR:
      a.rule = kRuleScaled;
      a.energy_scale = h->kappa;
      break;
    case GEM_MODE_DOWNPOUR:
    case GEM_MODE_ADAPTIVE:
      a.rule = kRuleFixed;
      break;
    case GEM_MODE_MOMENTUM:
      a.rule = kRuleMomentum;
      break;
    default:
      a.rule = kRuleGem;
      break;
  }
  for (int k0 = 0; k0 < K; k0 += kMaxBatchPerLaunch) {
    const int kc = (K - k0) < kMaxBatchPerLaunch ? (K - k0) : kMaxBatchPerLaunch;
    a.K = kc;
    a.record_pi = 0;
    for (int k = 0; k < kc; ++k) {
      a.pi_out[k] = pi_out ? pi_out[k0 + k] : nullptr;
      if (a.pi_out[k]) a.record_pi = 1;
    }
    for (int k = 0; k < kc; ++k) {
      const int w = order[k0 + k];
      a.worker[k] = w;
      a.grad[k] = grads[k0 + k];
      // staleness: commits by the other workers since w's last commit (and pull)
      const int64_t tau = h->clock - h->last[size_t(w)] - 1;
      h->last[size_t(w)] = h->clock;
      h->clock += 1;
      // adaptive staleness: pi = 1 / (tau + 1) in fp32 (IEEE division); DOWNPOUR: pi = 1
      a.pi[k] = h->mode == GEM_MODE_ADAPTIVE ? 1.0f / (static_cast<float>(tau) + 1.0f) : 1.0f;
    }
    plan_slots(a);
    const cudaError_t e = launch_commit_batch(a, h->sm_count, h->stream);
    if (e != cudaSuccess) return e;
    h->launches += 1;
  }
  return cudaSuccess;
}

}  // namespace gem

extern "C" {

const char* gem_status_string(int status) {
  switch (status) {
    case GEM_OK: return "GEM_OK";
    case GEM_EINVAL: return "GEM_EINVAL: invalid argument";
    case GEM_ENOMEM: return "GEM_ENOMEM: allocation failed";
    case GEM_ECUDA: return "GEM_ECUDA: CUDA error";
    case GEM_ESTATE: return "GEM_ESTATE: handle unusable after an earlier CUDA error";
    default: return "unknown gem_status";
  }
}

int gem_create(size_t P, int n, float eta, float mu, float eps, gem_t** out) {
  if (!out) return GEM_EINVAL;
  *out = nullptr;
  if (P == 0 || n < 1) return GEM_EINVAL;
  if (!(eta > 0.0f) || !(mu >= 0.0f) || !(mu < 1.0f) || !(eps > 0.0f)) return GEM_EINVAL;
  const size_t stride = (P + gem::kStrideAlign - 1) / gem::kStrideAlign * gem::kStrideAlign;
  if (stride > (SIZE_MAX / sizeof(float)) / (size_t(n) + 1)) return GEM_EINVAL;
  gem_t* h = new (std::nothrow) gem_t();
  if (!h) return GEM_ENOMEM;
  h->P = P;
  h->stride = stride;
  h->n = n;
  h->eta = eta;
  h->mu = mu;
  h->eps = eps;
  try {
    h->last.assign(size_t(n), -1);
  } catch (...) {
    delete h;
    return GEM_ENOMEM;
  }
  if (cudaGetDevice(&h->device) != cudaSuccess ||
      cudaDeviceGetAttribute(&h->sm_count, cudaDevAttrMultiProcessorCount, h->device) !=
          cudaSuccess) {
    cudaGetLastError();
    delete h;
    return GEM_ECUDA;
  }
  const size_t row = stride * sizeof(float);
  const size_t rows = size_t(n) * row;
  if (cudaMalloc(&h->theta, row) != cudaSuccess || cudaMalloc(&h->m, rows) != cudaSuccess ||
      cudaMalloc(&h->s, rows) != cudaSuccess) {
    cudaGetLastError();
    cudaFree(h->theta);
    cudaFree(h->m);
    cudaFree(h->s);
    delete h;
    return GEM_ENOMEM;
  }
  cudaError_t e = cudaMemset(h->theta, 0, row);
  if (e == cudaSuccess) e = cudaMemset(h->m, 0, rows);
  if (e == cudaSuccess) e = cudaMemset(h->s, 0, rows);
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    cudaFree(h->theta);
    cudaFree(h->m);
    cudaFree(h->s);
    delete h;
    return GEM_ECUDA;
  }
  *out = h;
  return GEM_OK;
}

void gem_destroy(gem_t* h) {
  if (!h) return;
  DeviceScope scope(h->device);
  cudaStreamSynchronize(h->stream);
  if (h->copy_stream) cudaStreamSynchronize(h->copy_stream);
  for (int i = 0; i < 2; ++i) {
    if (h->stage_filled[i]) cudaEventDestroy(h->stage_filled[i]);
    if (h->stage_free[i]) cudaEventDestroy(h->stage_free[i]);
  }
  if (h->copy_stream) cudaStreamDestroy(h->copy_stream);
  cudaFree(h->stage);
  cudaFree(h->select_scratch);
  cudaFree(h->theta);
  cudaFree(h->m);
  cudaFree(h->s);
  cudaGetLastError();
  delete h;
}

int gem_set_stream(gem_t* h, void* stream) {
  if (!h) return GEM_EINVAL;
  h->stream = static_cast<cudaStream_t>(stream);
  return GEM_OK;
}

int gem_set_theta(gem_t* h, const float* theta0) {
  int rc = check_handle(h);
  if (rc) return rc;
  if (!theta0) return GEM_EINVAL;
  DeviceScope scope(h->device);
  if (!scope.ok()) return GEM_ECUDA;
  const size_t row = h->stride * sizeof(float);
  cudaError_t e = cudaMemcpyAsync(h->theta, theta0, h->P * sizeof(float), cudaMemcpyDefault,
                                  h->stream);
  for (int w = 0; w < h->n && e == cudaSuccess; ++w)
    e = cudaMemcpyAsync(h->s + size_t(w) * h->stride, h->theta, row, cudaMemcpyDeviceToDevice,
                        h->stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(h->m, 0, size_t(h->n) * row, h->stream);
  h->clock = 0;
  for (auto& t : h->last) t = -1;
  return cuda_status(h, e);
}

int gem_set_mode(gem_t* h, int mode, float kappa) {
  int rc = check_handle(h);
  if (rc) return rc;
  if (mode < GEM_MODE_GEM || mode > GEM_MODE_MOMENTUM) return GEM_EINVAL;
  if ((mode == GEM_MODE_KAPPA_SQRT || mode == GEM_MODE_KAPPA_LINEAR) &&
      !(kappa > 0.0f && kappa <= 3.0e38f))
    return GEM_EINVAL;
  h->mode = mode;
  h->kappa = (mode == GEM_MODE_KAPPA_SQRT || mode == GEM_MODE_KAPPA_LINEAR) ? kappa : 1.0f;
  return GEM_OK;
}

int gem_get_mode(const gem_t* h, int* mode, float* kappa) {
  if (!h) return GEM_EINVAL;
  if (mode) *mode = h->mode;
  if (kappa) *kappa = h->kappa;
  return GEM_OK;
}

int gem_get_clock(const gem_t* h, int64_t* clock, int64_t* last) {
  if (!h) return GEM_EINVAL;
  if (clock) *clock = h->clock;
  if (last)
    for (int w = 0; w < h->n; ++w) last[w] = h->last[size_t(w)];
  return GEM_OK;
}

int gem_set_clock(gem_t* h, int64_t clock, const int64_t* last) {
  int rc = check_handle(h);
  if (rc) return rc;
  if (clock < 0) return GEM_EINVAL;
  if (last)
    for (int w = 0; w < h->n; ++w)
      if (last[w] < -1 || last[w] >= clock) return GEM_EINVAL;
  h->clock = clock;
  for (int w = 0; w < h->n; ++w) h->last[size_t(w)] = last ? last[w] : -1;
  return GEM_OK;
}

int gem_staleness(const gem_t* h, int worker, int64_t* tau) {
  if (!h || !tau || worker < 0 || worker >= h->n) return GEM_EINVAL;
  *tau = h->clock - h->last[size_t(worker)] - 1;
  return GEM_OK;
}

int gem_pull(gem_t* h, int worker, const float** snapshot) {
  int rc = check_handle(h);
  if (rc) return rc;
  if (!snapshot || worker < 0 || worker >= h->n) return GEM_EINVAL;
  *snapshot = h->s + size_t(worker) * h->stride;
  return GEM_OK;
}

int gem_moment(gem_t* h, int worker, const float** moment) {
  int rc = check_handle(h);
  if (rc) return rc;
  if (!moment || worker < 0 || worker >= h->n) return GEM_EINVAL;
  *moment = h->m + size_t(worker) * h->stride;
  return GEM_OK;
}

int gem_theta(gem_t* h, const float** theta) {
  int rc = check_handle(h);
  if (rc) return rc;
  if (!theta) return GEM_EINVAL;
  *theta = h->theta;
  return GEM_OK;
}

int gem_shape(const gem_t* h, size_t* P, int* n, size_t* stride) {
  if (!h) return GEM_EINVAL;
  if (P) *P = h->P;
  if (n) *n = h->n;
  if (stride) *stride = h->stride;
  return GEM_OK;
}

uint64_t gem_launch_count(const gem_t* h) { return h ? h->launches : 0; }

int gem_shard_range(size_t P, int world, int rank, size_t* begin, size_t* end) {
  if (P < 1 || world < 1 || rank < 0 || rank >= world || !begin || !end) return GEM_EINVAL;
  const size_t units = (P + gem::kStrideAlign - 1) / gem::kStrideAlign;   // 128-byte units
  const size_t w = size_t(world), r = size_t(rank);
  const size_t per = units / w, extra = units % w;
  const size_t u0 = r * per + (r < extra ? r : extra);
  const size_t u1 = u0 + per + (r < extra ? 1 : 0);
  *begin = u0 * gem::kStrideAlign < P ? u0 * gem::kStrideAlign : P;
  *end = u1 * gem::kStrideAlign < P ? u1 * gem::kStrideAlign : P;
  return GEM_OK;
}

int gem_commit(gem_t* h, int worker, const float* grad) {
  int rc = check_handle(h);
  if (rc) return rc;
  rc = check_batch(h, &worker, &grad, 1);
  if (rc) return rc;
  DeviceScope scope(h->device);
  if (!scope.ok()) return GEM_ECUDA;
  return launch_commits(h, &worker, &grad, 1);
}

int gem_commit_batch(gem_t* h, const int* order, const float* const* grads, int K) {
  int rc = check_handle(h);
  if (rc) return rc;
  rc = check_batch(h, order, grads, K);
  if (rc || K == 0) return rc;
  DeviceScope scope(h->device);
  if (!scope.ok()) return GEM_ECUDA;
  return launch_commits(h, order, grads, K);
}

int gem_commit_batch_pi(gem_t* h, const int* order, const float* const* grads, int K,
                        float* const* pi) {
  int rc = check_handle(h);
  if (rc) return rc;
  rc = check_batch(h, order, grads, K);
  if (rc) return rc;
  if (pi)
    for (int k = 0; k < K; ++k)
      if (pi[k] && !aligned16(pi[k])) return GEM_EINVAL;
  if (K == 0) return GEM_OK;
  DeviceScope scope(h->device);
  if (!scope.ok()) return GEM_ECUDA;
  return cuda_status(h, gem::commit_ordered(h, order, grads, K, pi));
}

int gem_pi_median(gem_t* h, const float* const* pi, int K, const int64_t* seg, int nseg,
                  float* lo, float* hi) {
  int rc = check_handle(h);
  if (rc) return rc;
  if (K < 0 || nseg < 1 || nseg > gem::kMaxPiSegments || !seg) return GEM_EINVAL;
  if (seg[0] < 0 || seg[nseg] > int64_t(h->P)) return GEM_EINVAL;
  for (int i = 0; i < nseg; ++i)
    if (seg[i + 1] < seg[i] || seg[i + 1] - seg[i] > int64_t(UINT32_MAX)) return GEM_EINVAL;
  if (K == 0) return GEM_OK;
  if (!pi || !lo || !hi) return GEM_EINVAL;
  const uintptr_t align4 = 3u;
  if ((reinterpret_cast<uintptr_t>(lo) & align4) || (reinterpret_cast<uintptr_t>(hi) & align4))
    return GEM_EINVAL;
  for (int k = 0; k < K; ++k)
    if (!pi[k] || (reinterpret_cast<uintptr_t>(pi[k]) & align4)) return GEM_EINVAL;
  DeviceScope scope(h->device);
  if (!scope.ok()) return GEM_ECUDA;
  const cudaError_t e = gem::pi_median_ordered(h, pi, K, seg, nseg, lo, hi);
  if (e == cudaErrorMemoryAllocation) {
    cudaGetLastError();
    return GEM_ENOMEM;
  }
  return cuda_status(h, e);
}

int gem_commit_batch_pi_median(gem_t* h, const int* order, const float* const* grads, int K,
                               float* const* pi, const int64_t* seg, int nseg, float* lo,
                               float* hi) {
  int rc = check_handle(h);
  if (rc) return rc;
  rc = check_batch(h, order, grads, K);
  if (rc) return rc;
  if (nseg < 1 || nseg > gem::kMaxPiSegments || !seg) return GEM_EINVAL;
  if (seg[0] < 0 || seg[nseg] > int64_t(h->P)) return GEM_EINVAL;
  for (int i = 0; i < nseg; ++i)
    if (seg[i + 1] < seg[i] || seg[i + 1] - seg[i] > int64_t(UINT32_MAX)) return GEM_EINVAL;
  if (K == 0) return GEM_OK;
  if (!pi || !lo || !hi) return GEM_EINVAL;
  const uintptr_t align4 = 3u;
  if ((reinterpret_cast<uintptr_t>(lo) & align4) || (reinterpret_cast<uintptr_t>(hi) & align4))
    return GEM_EINVAL;
  for (int k = 0; k < K; ++k)
    if (!pi[k] || !aligned16(pi[k])) return GEM_EINVAL;
  DeviceScope scope(h->device);
  if (!scope.ok()) return GEM_ECUDA;
  const cudaError_t e = gem::commit_pi_median_ordered(h, order, grads, K, pi, seg, nseg, lo, hi);
  if (e == cudaErrorMemoryAllocation) {
    cudaGetLastError();
    return GEM_ENOMEM;
  }
  return cuda_status(h, e);
}

int gem_commit_batch_host(gem_t* h, const int* order, const float* const* grads, int K) {
  int rc = check_handle(h);
  if (rc) return rc;
  if (K < 0 || (K > 0 && (!order || !grads))) return GEM_EINVAL;
  for (int k = 0; k < K; ++k)
    if (order[k] < 0 || order[k] >= h->n || !grads[k]) return GEM_EINVAL;
  if (K == 0) return GEM_OK;
  DeviceScope scope(h->device);
  if (!scope.ok()) return GEM_ECUDA;
  // Page-locked host memory is readable by the device in place (over the host link): when
  // every gradient is, the commit kernel reads them there and nothing is staged.
  {
    std::vector<const float*> dev(static_cast<size_t>(K));
    bool in_place = true;
    for (int k = 0; k < K && in_place; ++k) {
      cudaPointerAttributes attr;
      if (cudaPointerGetAttributes(&attr, grads[k]) != cudaSuccess) {
        cudaGetLastError();
        in_place = false;
        break;
      }
      in_place = attr.type == cudaMemoryTypeHost && attr.devicePointer != nullptr &&
                 aligned16(attr.devicePointer);
      dev[size_t(k)] = static_cast<const float*>(attr.devicePointer);
    }
    if (in_place) return launch_commits(h, order, dev.data(), K);
  }
  rc = ensure_staging(h);
  if (rc) return rc;
  // Chunk j uses staging half j % 2: the copy stream fills it once the commits that last
  // read it have finished, and the commit stream starts on it once it is filled, so the
  // copy of chunk j + 1 overlaps the commits of chunk j.
  const float* slot[gem::kStageChunk];
  for (int k0 = 0, j = 0; k0 < K; k0 += gem::kStageChunk, ++j) {
    const int half = j & 1;
    const int kc = (K - k0) < gem::kStageChunk ? (K - k0) : gem::kStageChunk;
    cudaError_t e = cudaStreamWaitEvent(h->copy_stream, h->stage_free[half], 0);
    for (int i = 0; i < kc && e == cudaSuccess; ++i) {
      float* dst = h->stage + size_t(half * gem::kStageChunk + i) * h->stride;
      e = cudaMemcpyAsync(dst, grads[k0 + i], h->P * sizeof(float), cudaMemcpyDefault,
                          h->copy_stream);
      slot[i] = dst;
    }
    if (e == cudaSuccess) e = cudaEventRecord(h->stage_filled[half], h->copy_stream);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(h->stream, h->stage_filled[half], 0);
    rc = cuda_status(h, e);
    if (rc) return rc;
    rc = launch_commits(h, order + k0, slot, kc);
    if (rc) return rc;
    rc = cuda_status(h, cudaEventRecord(h->stage_free[half], h->stream));
    if (rc) return rc;
  }
  return GEM_OK;
}

namespace {

// Copies between the strided state rows [n][stride] and dense rows [n][P].
cudaError_t copy_rows(void* dst, size_t dpitch, const void* src, size_t spitch, size_t width,
                      size_t rows, cudaStream_t st) {
  return cudaMemcpy2DAsync(dst, dpitch, src, spitch, width, rows, cudaMemcpyDefault, st);
}

}  // namespace

int gem_save_state(gem_t* h, float* theta, float* m, float* s) {
  int rc = check_handle(h);
  if (rc) return rc;
  DeviceScope scope(h->device);
  if (!scope.ok()) return GEM_ECUDA;
  const size_t row = h->P * sizeof(float), pitch = h->stride * sizeof(float);
  cudaError_t e = cudaSuccess;
  if (theta) e = cudaMemcpyAsync(theta, h->theta, row, cudaMemcpyDefault, h->stream);
  if (m && e == cudaSuccess) e = copy_rows(m, row, h->m, pitch, row, size_t(h->n), h->stream);
  if (s && e == cudaSuccess) e = copy_rows(s, row, h->s, pitch, row, size_t(h->n), h->stream);
  return cuda_status(h, e);
}

int gem_load_state(gem_t* h, const float* theta, const float* m, const float* s) {
  int rc = check_handle(h);
  if (rc) return rc;
  DeviceScope scope(h->device);
  if (!scope.ok()) return GEM_ECUDA;
  const size_t row = h->P * sizeof(float), pitch = h->stride * sizeof(float);
  cudaError_t e = cudaSuccess;
  if (theta) e = cudaMemcpyAsync(h->theta, theta, row, cudaMemcpyDefault, h->stream);
  if (m && e == cudaSuccess) e = copy_rows(h->m, pitch, m, row, row, size_t(h->n), h->stream);
  if (s && e == cudaSuccess) e = copy_rows(h->s, pitch, s, row, row, size_t(h->n), h->stream);
  return cuda_status(h, e);
}

int gem_read_theta(gem_t* h, float* out) {
  int rc = check_handle(h);
  if (rc) return rc;
  if (!out) return GEM_EINVAL;
  DeviceScope scope(h->device);
  if (!scope.ok()) return GEM_ECUDA;
  return cuda_status(h, cudaMemcpyAsync(out, h->theta, h->P * sizeof(float), cudaMemcpyDefault,
                                        h->stream));
}

int gem_sync(gem_t* h) {
  if (!h) return GEM_EINVAL;
  if (h->broken) return GEM_ESTATE;
  DeviceScope scope(h->device);
  if (!scope.ok()) return GEM_ECUDA;
  cudaError_t e = cudaStreamSynchronize(h->stream);
  if (e == cudaSuccess && h->copy_stream) e = cudaStreamSynchronize(h->copy_stream);
  if (e == cudaSuccess) e = cudaGetLastError();
  return cuda_status(h, e);
}

}  // extern "C"
