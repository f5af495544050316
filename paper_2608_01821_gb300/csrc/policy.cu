// policy.cu -- the denoising-aware allocation policy on the device (Sec. 4.2,
// Eq. 6-8; Sec. 4.3, Eq. 9), so that a captured step loop chooses each
// step's evidence view without a host round trip.
//
// Envelope (once per request): phase profile p_t (early: 1 - (t-0.5)/T, late:
// (t-0.5)/T), normalizer N(p; target) = clip(s p, 0, 1) with the mean equal
// to the target, lower = N(p; (1-rho) B), upper = N(p; (1-rho+rho d) B).
// The scale s is found exactly: p is monotone in t, so the steps clipped at 1
// are the m largest entries, and for the right m,
//     s = (T * target - m) / (sum of the other entries),
// checked against the clip condition of the m-th and (m+1)-th largest.
//
// Step (once per denoising step): r_1 = 1, r_t = 1 - alpha c_{t-1} (1 - chi_{t-1})
// from the previous unmasking call's statistics, b_t = lower_t + r_t
// (upper_t - lower_t), view = coarse / mixed / high by thirds, mapped to a
// pyramid level through a caller table.  All arithmetic is fp64: these
// kernels are tiny, and the quantization then decides at the oracle's
// precision.
#include "common.cuh"

namespace davet {
namespace pol {

constexpr int kMaxT = 4096;

// Entry k of the profile sorted in decreasing order (k = 0 is the largest).
__device__ __forceinline__ double profile_desc(int k, int T, int orientation) {
  // early grounding: p_t decreases with t, so the k-th largest is t = k + 1;
  // late verification: p_t increases, so the k-th largest is t = T - k
  const int t = orientation == 0 ? k + 1 : T - k;
  const double u = (t - 0.5) / T;
  return orientation == 0 ? 1.0 - u : u;
}

// clip(s p_t, 0, 1) for every t, with mean equal to `target`
__device__ void normalize(int T, int orientation, double target, double* out) {
  if (target <= 0.0) {
    for (int t = 0; t < T; ++t) out[t] = 0.0;
    return;
  }
  if (target >= 1.0) {
    for (int t = 0; t < T; ++t) out[t] = 1.0;
    return;
  }
  double total = 0.0;
  for (int k = 0; k < T; ++k) total += profile_desc(k, T, orientation);
  double top = 0.0;  // sum of the m largest entries
  double s = 0.0;
  for (int m = 0; m < T; ++m) {
    const double rest = total - top;
    const double cand = (T * target - m) / rest;
    const double p_next = profile_desc(m, T, orientation);          // largest unclipped entry
    const bool rest_ok = cand * p_next <= 1.0;
    const bool top_ok = m == 0 || cand * profile_desc(m - 1, T, orientation) >= 1.0;
    if (cand >= 0.0 && rest_ok && top_ok) {
      s = cand;
      break;
    }
    top += p_next;
    s = cand;
  }
  for (int t = 1; t <= T; ++t) {
    const double u = (t - 0.5) / T;
    const double p = orientation == 0 ? 1.0 - u : u;
    out[t - 1] = fmin(fmax(s * p, 0.0), 1.0);
  }
}

__global__ void envelope_kernel(int T, int orientation, double B, double rho, const double* __restrict__ demand,
                                int batch, double* __restrict__ lower, double* __restrict__ upper) {
  pdl_launch_dependents();
  pdl_wait();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= batch) return;
  const double d = demand ? demand[b] : 1.0;
  normalize(T, orientation, (1.0 - rho) * B, lower + static_cast<long long>(b) * T);
  normalize(T, orientation, (1.0 - rho + rho * d) * B, upper + static_cast<long long>(b) * T);
}

struct StepArgs {
  int t, T, batch;
  double alpha;
  int view_level[3];
  const double* lower;
  const double* upper;
  const float* stats_prev;
  int32_t* level_out;
  double* budget_out;
};

__global__ void step_kernel(StepArgs a) {
  pdl_launch_dependents();
  pdl_wait();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= a.batch) return;
  double r = 1.0;  // no prediction state before the first update
  if (a.t > 0 && a.stats_prev) {
    const double cbar = a.stats_prev[2 * b + 0];
    const double chi = a.stats_prev[2 * b + 1];
    r = 1.0 - a.alpha * cbar * (1.0 - chi);
  }
  const long long i = static_cast<long long>(b) * a.T + a.t;
  const double lo = a.lower[i], up = a.upper[i];
  const double bt = lo + r * (up - lo);
  const int view = bt < 1.0 / 3.0 ? 0 : (bt < 2.0 / 3.0 ? 1 : 2);
  a.level_out[b] = a.view_level[view];
  if (a.budget_out) a.budget_out[b] = bt;
}

}  // namespace pol
}  // namespace davet

extern "C" davet_status davet_policy_envelope(int T, int orientation, double B, double rho, const double* demand_dev,
                                              int batch, double* lower_dev, double* upper_dev, void* stream) {
  using namespace davet;
  if (T < 1 || T > pol::kMaxT || (orientation != 0 && orientation != 1) || batch < 0) return DAVET_ERR_INVALID_ARG;
  if (!(B >= 0.0 && B <= 1.0) || !(rho >= 0.0 && rho <= 1.0)) return DAVET_ERR_INVALID_ARG;
  if (batch == 0) return DAVET_OK;
  if (!lower_dev || !upper_dev) return DAVET_ERR_INVALID_ARG;
  const int threads = 64;
  const cudaError_t e = launch(pol::envelope_kernel, dim3((batch + threads - 1) / threads), dim3(threads), 0,
                               static_cast<cudaStream_t>(stream), T, orientation, B, rho, demand_dev, batch,
                               lower_dev, upper_dev);
  return e == cudaSuccess ? DAVET_OK : cuda_fail(e);
}

extern "C" davet_status davet_policy_step(int t, int T, const double* lower_dev, const double* upper_dev,
                                          const float* stats_prev_dev, int batch, double alpha,
                                          const int32_t* view_level, int32_t* level_out_dev, double* budget_out_dev,
                                          void* stream) {
  using namespace davet;
  if (T < 1 || t < 0 || t >= T || batch < 0 || !(alpha >= 0.0 && alpha <= 1.0) || !view_level)
    return DAVET_ERR_INVALID_ARG;
  if (batch == 0) return DAVET_OK;
  if (!lower_dev || !upper_dev || !level_out_dev) return DAVET_ERR_INVALID_ARG;
  pol::StepArgs a;
  a.t = t;
  a.T = T;
  a.batch = batch;
  a.alpha = alpha;
  for (int v = 0; v < 3; ++v) a.view_level[v] = view_level[v];
  a.lower = lower_dev;
  a.upper = upper_dev;
  a.stats_prev = stats_prev_dev;
  a.level_out = level_out_dev;
  a.budget_out = budget_out_dev;
  const int threads = 64;
  const cudaError_t e = launch(pol::step_kernel, dim3((batch + threads - 1) / threads), dim3(threads), 0,
                               static_cast<cudaStream_t>(stream), a);
  return e == cudaSuccess ? DAVET_OK : cuda_fail(e);
}
