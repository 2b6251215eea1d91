// K3: revised PPO-EWMA update of the proximal parameters (Eq. 5, App. B, Sec. 5.2).
//
// A one-thread prologue turns the device state (w, streak) and the latest loss
// statistics (rho = n_active / n_valid) into the step's coefficients:
//   reset  (rho < tau for min_streak steps, or forced): theta_prox <- theta, w <- 1
//   update: w' = 1 + beta w, a = beta w / w', b = 1 / w'  (a + b = 1)
// and the streaming body applies theta_prox <- theta_prox + b (theta - theta_prox),
// which is a theta_prox + b theta written so that a constant theta is a fixed
// point exactly.  b = 1 (first step of an empty history, or a reset) copies
// theta bit for bit.  HBM traffic: 12 bytes per parameter (two reads, one write).
#include "occ_common.cuh"

namespace occ {

constexpr int kK3Threads = 256;
constexpr int kK3Unroll = 4;

__global__ void k3_ewma_prologue(occ_ewma_state* st, const occ_loss_stats* stats, double beta,
                                 double tau, int min_streak, int force_reset) {
  const double w = st->w;
  int streak = st->streak;
  bool evidence = false;
  if (stats) {
    const long long nv = stats->n_valid;
    if (nv > 0) {
      evidence = true;
      const double rho = (double)stats->n_active / (double)nv;
      streak = rho < tau ? streak + 1 : 0;
    }
  }
  const bool reset = force_reset || (evidence && streak >= min_streak);
  if (reset) {
    st->w = 1.0;
    st->coef_a = 0.0;
    st->coef_b = 1.0;
    st->streak = 0;
    st->n_resets += 1;
    st->last_reset = 1;
  } else {
    const double wn = 1.0 + beta * w;
    st->coef_a = beta * w / wn;
    st->coef_b = 1.0 / wn;
    st->w = wn;
    st->streak = streak;
    st->last_reset = 0;
  }
}

__device__ __forceinline__ float4 ld_f4(const float4* p) {
  const uint4 r = ld_stream_v4(p);
  return make_float4(__uint_as_float(r.x), __uint_as_float(r.y), __uint_as_float(r.z),
                     __uint_as_float(r.w));
}

__device__ __forceinline__ float lerp_b(float tp, float th, float b) { return fmaf(b, th - tp, tp); }

template <int NT, int U>
__global__ void __launch_bounds__(NT) k3_ewma_vec(float4* __restrict__ tp,
                                                  const float4* __restrict__ th, int64_t n4,
                                                  const occ_ewma_state* __restrict__ st) {
  const double bd = st->coef_b;
  const bool copy = (bd == 1.0);
  const float b = (float)bd;
  const int64_t stride = (int64_t)gridDim.x * NT;
  int64_t i = (int64_t)blockIdx.x * NT + threadIdx.x;
  for (; i + (int64_t)(U - 1) * stride < n4; i += (int64_t)U * stride) {
    float4 x[U], y[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      y[u] = ld_f4(th + i + u * stride);
      if (!copy) x[u] = ld_f4(tp + i + u * stride);
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      float4 o = y[u];
      if (!copy)
        o = make_float4(lerp_b(x[u].x, y[u].x, b), lerp_b(x[u].y, y[u].y, b),
                        lerp_b(x[u].z, y[u].z, b), lerp_b(x[u].w, y[u].w, b));
      st_stream_v4(tp + i + u * stride, make_uint4(__float_as_uint(o.x), __float_as_uint(o.y),
                                                   __float_as_uint(o.z), __float_as_uint(o.w)));
    }
  }
  for (; i < n4; i += stride) {
    const float4 y = ld_f4(th + i);
    float4 o = y;
    if (!copy) {
      const float4 x = ld_f4(tp + i);
      o = make_float4(lerp_b(x.x, y.x, b), lerp_b(x.y, y.y, b), lerp_b(x.z, y.z, b),
                      lerp_b(x.w, y.w, b));
    }
    st_stream_v4(tp + i, make_uint4(__float_as_uint(o.x), __float_as_uint(o.y),
                                    __float_as_uint(o.z), __float_as_uint(o.w)));
  }
}

// Scalar elements [i0, n): the ragged tail of the vector kernel, or every
// element when the arrays are not 16-byte aligned.
template <int NT>
__global__ void __launch_bounds__(NT) k3_ewma_scalar(float* __restrict__ tp,
                                                     const float* __restrict__ th, int64_t i0,
                                                     int64_t n,
                                                     const occ_ewma_state* __restrict__ st) {
  const double bd = st->coef_b;
  const bool copy = (bd == 1.0);
  const float b = (float)bd;
  for (int64_t i = i0 + (int64_t)blockIdx.x * NT + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * NT)
    tp[i] = copy ? th[i] : lerp_b(tp[i], th[i], b);
}

__global__ void k3_state_init(occ_ewma_state* st, double w0) {
  st->w = w0;
  st->coef_a = 0.0;
  st->coef_b = 0.0;
  st->streak = 0;
  st->n_resets = 0;
  st->last_reset = 0;
  st->reserved = 0;
}

}  // namespace occ

using namespace occ;

extern "C" occ_status occ_ewma_update(float* theta_prox, const float* theta, int64_t n,
                                      double beta, occ_ewma_state* st,
                                      const occ_loss_stats* stats, double tau, int32_t min_streak,
                                      int32_t force_reset, void* stream) {
  clear_error();
  if (n < 0) return fail(OCC_ERR_INVALID_ARG, "n < 0");
  if (!st || !aligned(st, 8)) return fail(OCC_ERR_INVALID_ARG, "state null or misaligned");
  if (stats && !aligned(stats, 8)) return fail(OCC_ERR_MISALIGNED, "stats misaligned");
  if (!(beta >= 0.0 && beta < 1.0)) return fail(OCC_ERR_INVALID_ARG, "beta must be in [0, 1)");
  if (min_streak < 1) return fail(OCC_ERR_INVALID_ARG, "min_streak must be >= 1");
  if (isnan(tau)) return fail(OCC_ERR_INVALID_ARG, "tau is NaN");
  if (n > 0) {
    if (!theta_prox || !theta) return fail(OCC_ERR_INVALID_ARG, "null theta_prox/theta");
    if (!aligned(theta_prox, 4) || !aligned(theta, 4))
      return fail(OCC_ERR_MISALIGNED, "parameter arrays must be 4-byte aligned");
    if (overlaps(theta_prox, (size_t)n * 4, theta, (size_t)n * 4))
      return fail(OCC_ERR_INVALID_ARG, "theta_prox overlaps theta");
  }
  cudaStream_t s = (cudaStream_t)stream;
  k3_ewma_prologue<<<1, 1, 0, s>>>(st, stats, beta, tau, min_streak, force_reset ? 1 : 0);
  occ_status rc = check_launch("k3_ewma_prologue");
  if (rc != OCC_OK || n == 0) return rc;
  const int64_t blocks_cap = (int64_t)sm_count() * 8;
  if (aligned(theta_prox, 16) && aligned(theta, 16)) {
    const int64_t n4 = n / 4;
    if (n4 > 0) {
      const int64_t need = (n4 + kK3Threads * kK3Unroll - 1) / (kK3Threads * kK3Unroll);
      const unsigned grid = (unsigned)std::max<int64_t>(1, std::min(need, blocks_cap));
      k3_ewma_vec<kK3Threads, kK3Unroll><<<grid, kK3Threads, 0, s>>>(
          (float4*)theta_prox, (const float4*)theta, n4, st);
    }
    if (n - n4 * 4 > 0)
      k3_ewma_scalar<kK3Threads><<<1, kK3Threads, 0, s>>>(theta_prox, theta, n4 * 4, n, st);
  } else {
    const int64_t need = (n + kK3Threads - 1) / kK3Threads;
    const unsigned grid = (unsigned)std::max<int64_t>(1, std::min(need, blocks_cap));
    k3_ewma_scalar<kK3Threads><<<grid, kK3Threads, 0, s>>>(theta_prox, theta, 0, n, st);
  }
  return check_launch("occ_ewma_update");
}

extern "C" occ_status occ_ewma_state_init(occ_ewma_state* st, double w0, void* stream) {
  clear_error();
  if (!st || !aligned(st, 8)) return fail(OCC_ERR_INVALID_ARG, "state null or misaligned");
  if (!(w0 >= 0.0) || isinf(w0)) return fail(OCC_ERR_INVALID_ARG, "w0 must be finite and >= 0");
  k3_state_init<<<1, 1, 0, (cudaStream_t)stream>>>(st, w0);
  return check_launch("occ_ewma_state_init");
}
