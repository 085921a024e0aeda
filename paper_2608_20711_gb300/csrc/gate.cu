// gate.cu -- GatedEval timing and the commit gate of AsmEvo (Sec. 3.4,
// Algorithm 1; Eq. 2).  Host code: the statistics of event-timed launches
// and the variance-aware commit threshold; plus the event-timing loop
// itself, which only records CUDA events around the caller's launches.
#include <algorithm>
#include <cmath>
#include <vector>

#include <cuda_runtime.h>

#include "asmv.h"
#include "nvtx_range.h"

namespace {

bool finite_nonneg(double x) { return std::isfinite(x) && x >= 0.0; }

}  // namespace

extern "C" {

int asmv_timing_summary(const double *samples_ms, size_t r, asmv_timing *out) {
  if (samples_ms == nullptr || out == nullptr || r == 0) return ASMV_EINVAL;
  for (size_t i = 0; i < r; ++i)
    if (!std::isfinite(samples_ms[i]) || samples_ms[i] <= 0.0) return ASMV_EINVAL;
  std::vector<double> v(samples_ms, samples_ms + r);
  std::sort(v.begin(), v.end());
  const double median = (r % 2) ? v[r / 2] : (v[r / 2 - 1] + v[r / 2]) / 2.0;
  double sum = 0.0;
  for (size_t i = 0; i < r; ++i) sum += samples_ms[i];
  const double mean = sum / (double)r;
  double cv = 0.0;
  if (r > 1) {
    double ss = 0.0;
    for (size_t i = 0; i < r; ++i) {
      const double d = samples_ms[i] - mean;
      ss += d * d;
    }
    cv = std::sqrt(ss / (double)(r - 1)) / mean;
  }
  out->median_ms = median;
  out->mean_ms = mean;
  out->cv = cv;
  out->r = r;
  return ASMV_OK;
}

int asmv_commit_gate(int all_eq, double s_cand, double s_best, double cv,
                     const asmv_gate_params *params, double *m_star, int *commit) {
  if (params == nullptr || m_star == nullptr || commit == nullptr) return ASMV_EINVAL;
  if (!finite_nonneg(s_cand) || !finite_nonneg(s_best) || s_best == 0.0 || !finite_nonneg(cv) ||
      !finite_nonneg(params->eps) || !finite_nonneg(params->k) || !finite_nonneg(params->s_floor))
    return ASMV_EINVAL;
  const double kcv = params->k * cv;
  const double margin = std::max(params->eps, kcv);
  const double m = (1.0 + margin) * s_best;
  *m_star = m;
  *commit = (all_eq != 0) && s_cand >= std::max(m, params->s_floor);
  return ASMV_OK;
}

int asmv_time_launches(asmv_launch_fn fn, void *user, int warmup, size_t r,
                       double *samples_ms, asmv_stream_t stream, int *cuda_error) {
  ASMV_NVTX_RANGE("asmv_time_launches");
  if (fn == nullptr || samples_ms == nullptr || r == 0 || warmup < 0) return ASMV_EINVAL;
  const cudaStream_t s = (cudaStream_t)stream;
  std::vector<cudaEvent_t> ev(2 * r, nullptr);
  cudaError_t e = cudaSuccess;
  size_t made = 0;
  for (; made < ev.size(); ++made)
    if ((e = cudaEventCreate(&ev[made])) != cudaSuccess) break;
  if (e == cudaSuccess) {
    for (int i = 0; i < warmup; ++i) fn(user, stream);
    for (size_t i = 0; i < r && e == cudaSuccess; ++i) {
      if ((e = cudaEventRecord(ev[2 * i], s)) != cudaSuccess) break;
      fn(user, stream);
      e = cudaEventRecord(ev[2 * i + 1], s);
    }
    if (e == cudaSuccess) e = cudaEventSynchronize(ev[2 * r - 1]);
    for (size_t i = 0; i < r && e == cudaSuccess; ++i) {
      float ms = 0.0f;
      if ((e = cudaEventElapsedTime(&ms, ev[2 * i], ev[2 * i + 1])) == cudaSuccess)
        samples_ms[i] = (double)ms;
    }
  }
  for (size_t i = 0; i < made; ++i) cudaEventDestroy(ev[i]);
  if (e != cudaSuccess) {
    if (cuda_error) *cuda_error = (int)e;
    return ASMV_ECUDA;
  }
  if (cuda_error) *cuda_error = 0;
  return ASMV_OK;
}

}  // extern "C"
