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

#include <algorithm>

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


// ------------------------------------------------------------------ bf16 buffers
//
// The proximal parameters may be kept in bf16 (2 bytes per parameter, the
// footprint the paper reports for its host-side EWMA copy, Table 3a).  The
// update is computed in float32 from the bf16 value and rounded back either
// to nearest-even or stochastically (seed != 0), which keeps small EWMA steps
// (b (theta - theta_prox) below half a bf16 ulp) from being lost in
// expectation.

// The i-th output of SplitMix64 (Steele, Lea and Flood, 2014) started at
// `seed`, used as a counter-based generator: state_i = seed + (i + 1) gamma.
__device__ __forceinline__ uint64_t splitmix64_at(uint64_t seed, uint64_t i) {
  uint64_t z = seed + (i + 1) * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// float32 -> bf16 bits: nearest-even (seed == 0) or stochastic with the 16
// random bits r: they are added below the bf16 unit in the last place and the
// result truncated, so the magnitude rounds up with probability equal to the
// dropped fraction.  Parameter i takes 16-bit lane (i mod 4) of the (i / 4)-th
// SplitMix64 output (lane 0 = the least significant bits).
__device__ __forceinline__ uint16_t round_bf16_bits(float x, bool sr, uint32_t r) {
  const uint32_t u = __float_as_uint(x);
  if (!sr || (u & 0x7f800000u) == 0x7f800000u) {
    unsigned short h;
    asm("cvt.rn.bf16.f32 %0, %1;" : "=h"(h) : "f"(x));
    return h;
  }
  return (uint16_t)((u + r) >> 16);
}
__device__ __forceinline__ uint16_t round_bf16(float x, uint64_t seed, uint64_t idx) {
  const uint32_t r =
      seed ? (uint32_t)(splitmix64_at(seed, idx >> 2) >> (16 * (idx & 3))) & 0xffffu : 0u;
  return round_bf16_bits(x, seed != 0, r);
}

// Eight theta values as loaded (raw 16-byte words) and unpacked to float.
template <typename ThT>
struct Raw8;
template <>
struct Raw8<float> {
  uint4 a, b;
  __device__ __forceinline__ void load(const float* p) {
    a = ld_stream_v4(p);
    b = ld_stream_v4(p + 4);
  }
  __device__ __forceinline__ void unpack(float (&x)[8]) const {
    x[0] = __uint_as_float(a.x); x[1] = __uint_as_float(a.y);
    x[2] = __uint_as_float(a.z); x[3] = __uint_as_float(a.w);
    x[4] = __uint_as_float(b.x); x[5] = __uint_as_float(b.y);
    x[6] = __uint_as_float(b.z); x[7] = __uint_as_float(b.w);
  }
};
template <>
struct Raw8<bf16_t> {
  uint4 a;
  __device__ __forceinline__ void load(const bf16_t* p) { a = ld_stream_v4(p); }
  __device__ __forceinline__ void unpack(float (&x)[8]) const { Elem<bf16_t>::unpack(a, x); }
};
__device__ __forceinline__ float load1(const float* p) { return *p; }
__device__ __forceinline__ float load1(const bf16_t* p) {
  return __uint_as_float(((uint32_t)p->bits) << 16);
}

// theta_prox (bf16, 16-byte aligned) <- theta_prox + b (theta - theta_prox),
// eight parameters per vector, U vectors of each operand in flight per thread;
// elements [8 n8, n) in a scalar tail.  On a copy step (b = 1) theta_prox is
// not read.
// Launch shape of the bf16 update (measured on GB300 over 4e9 parameters,
// fraction of the measured copy bandwidth, float32 theta nearest / stochastic
// and bf16 theta stochastic): 2 vectors of each operand in flight per thread
// and grids of 6 / 8 CTAs of 256 threads per SM reach 1.05 / 1.03 and 0.97;
// 4 vectors in flight with one resident wave of 3 / 4 CTAs per SM reached
// 0.95 / 0.93 and 0.94, 1 vector 0.98 / 0.97 and 0.84, 512-thread CTAs 0.89 /
// 0.86 and 0.90.  The register bound keeps 3 / 4 CTAs resident at least.
constexpr int kK3Bf16Unroll = 2;
template <typename ThT>
constexpr int k3_bf16_min_ctas() {
  return sizeof(ThT) == 4 ? 3 : 4;
}
template <typename ThT>
constexpr int k3_bf16_grid_per_sm() {
  return sizeof(ThT) == 4 ? 6 : 8;
}

template <typename ThT, int NT, int U>
__global__ void __launch_bounds__(NT, k3_bf16_min_ctas<ThT>())
    k3_ewma_bf16(bf16_t* __restrict__ tp, const ThT* __restrict__ th, int64_t n, bool vec,
                 const occ_ewma_state* __restrict__ st, uint64_t seed, uint64_t idx0) {
  const double bd = st->coef_b;
  const bool copy = (bd == 1.0);
  const float b = (float)bd;
  const int64_t stride = (int64_t)gridDim.x * NT;
  const int64_t gtid = (int64_t)blockIdx.x * NT + threadIdx.x;
  int64_t done = 0;
  if (vec) {
    const int64_t n8 = n / 8;
    // The rounding is written to keep the integer (ALU) pipe light, which
    // otherwise co-limits the bf16-theta update: nearest-even rounds a pair per
    // conversion; the stochastic path checks the eight values for inf / NaN
    // once, with multiplies (0 * v is NaN only for them), takes each 16-bit
    // lane of the generator outputs in one operation, and packs two rounded
    // values with one byte permutation.  The bits are those of
    // round_bf16_bits, which the rare vector holding inf or NaN still takes.
    auto emit = [&](int64_t iv, const uint4& xr, const Raw8<ThT>& yr) {
      float x[8], y[8], v[8];
      Elem<bf16_t>::unpack(xr, x);
      yr.unpack(y);
#pragma unroll
      for (int k = 0; k < 8; ++k) v[k] = copy ? y[k] : fmaf(b, y[k] - x[k], x[k]);
      uint32_t w[4];
      if (!seed) {
#pragma unroll
        for (int j = 0; j < 4; ++j) w[j] = pack_bf16x2(v[2 * j], v[2 * j + 1]);
      } else {
        const uint64_t g0 = idx0 + 8 * iv;  // idx0 is a multiple of 8: two whole generator outputs
        const uint64_t r0 = splitmix64_at(seed, g0 >> 2);
        const uint64_t r1 = splitmix64_at(seed, (g0 >> 2) + 1);
        const uint32_t q[4] = {(uint32_t)r0, (uint32_t)(r0 >> 32), (uint32_t)r1,
                               (uint32_t)(r1 >> 32)};
        float s = 0.f;
#pragma unroll
        for (int k = 0; k < 8; ++k) s = fmaf(v[k], 0.f, s);
        if (s == 0.f) {
#pragma unroll
          for (int j = 0; j < 4; ++j)  // lanes 2j, 2j + 1 = low and high half of q[j]
            w[j] = __byte_perm(__float_as_uint(v[2 * j]) + (q[j] & 0xffffu),
                               __float_as_uint(v[2 * j + 1]) + (q[j] >> 16), 0x7632);
        } else {
#pragma unroll
          for (int j = 0; j < 4; ++j)
            w[j] = (uint32_t)round_bf16_bits(v[2 * j], true, q[j] & 0xffffu) |
                   ((uint32_t)round_bf16_bits(v[2 * j + 1], true, q[j] >> 16) << 16);
        }
      }
      st_stream_v4(tp + 8 * iv, make_uint4(w[0], w[1], w[2], w[3]));
    };
    int64_t i = gtid;
    for (; i + (int64_t)(U - 1) * stride < n8; i += (int64_t)U * stride) {
      uint4 xr[U];
      Raw8<ThT> yr[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        yr[u].load(th + 8 * (i + u * stride));
        xr[u] = copy ? make_uint4(0, 0, 0, 0) : ld_stream_v4(tp + 8 * (i + u * stride));
      }
#pragma unroll
      for (int u = 0; u < U; ++u) emit(i + u * stride, xr[u], yr[u]);
    }
    for (; i < n8; i += stride) {
      Raw8<ThT> yr;
      yr.load(th + 8 * i);
      emit(i, copy ? make_uint4(0, 0, 0, 0) : ld_stream_v4(tp + 8 * i), yr);
    }
    done = n8 * 8;
  }
  for (int64_t i = done + gtid; i < n; i += stride) {
    const float y = load1(th + i);
    const float v = copy ? y : fmaf(b, y - load1(tp + i), load1(tp + i));
    tp[i].bits = round_bf16(v, seed, idx0 + i);
  }
}

}  // namespace occ

using namespace occ;

namespace {
// Launches the float32 update of n parameters (vector body + scalar tail).
occ_status launch_f32_body(float* tp, const float* th, int64_t n, const occ_ewma_state* st,
                           cudaStream_t s);
}  // namespace

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
  return launch_f32_body(theta_prox, theta, n, st, s);
}

extern "C" occ_status occ_ewma_state_init(occ_ewma_state* st, double w0, void* stream) {
  clear_error();
  if (!st || !aligned(st, 8)) return fail(OCC_ERR_INVALID_ARG, "state null or misaligned");
  if (!(w0 >= 0.0) || isinf(w0)) return fail(OCC_ERR_INVALID_ARG, "w0 must be finite and >= 0");
  k3_state_init<<<1, 1, 0, (cudaStream_t)stream>>>(st, w0);
  return check_launch("occ_ewma_state_init");
}


// ------------------------------------------------------------------ F4 entry points

namespace {

occ_status validate_ewma(int64_t n, double beta, occ_ewma_state* st, const occ_loss_stats* stats,
                         double tau, int32_t min_streak) {
  if (n < 0) return fail(OCC_ERR_INVALID_ARG, "n < 0");
  if (!st || !aligned(st, 8)) return fail(OCC_ERR_INVALID_ARG, "state null or misaligned");
  if (stats && !aligned(stats, 8)) return fail(OCC_ERR_MISALIGNED, "stats misaligned");
  if (!(beta >= 0.0 && beta < 1.0)) return fail(OCC_ERR_INVALID_ARG, "beta must be in [0, 1)");
  if (min_streak < 1) return fail(OCC_ERR_INVALID_ARG, "min_streak must be >= 1");
  if (isnan(tau)) return fail(OCC_ERR_INVALID_ARG, "tau is NaN");
  return OCC_OK;
}

// Launches the bf16 update of n parameters whose global index starts at idx0.
occ_status launch_bf16_body(bf16_t* tp, const void* th, occ_dtype theta_dt, int64_t n,
                            const occ_ewma_state* st, uint64_t seed, uint64_t idx0,
                            cudaStream_t s) {
  if (n == 0) return OCC_OK;
  const bool vec = aligned(tp, 16) && aligned(th, 16);
  const int64_t work = vec ? (n + 7) / 8 : n;
  const int64_t need = (work + kK3Threads * kK3Bf16Unroll - 1) / (kK3Threads * kK3Bf16Unroll);
  auto grid_for = [&](int per_sm) {
    return (unsigned)std::max<int64_t>(1, std::min<int64_t>(need, (int64_t)sm_count() * per_sm));
  };
  note_kernel("k3_ewma_bf16");
  if (theta_dt == OCC_BF16)
    k3_ewma_bf16<bf16_t, kK3Threads, kK3Bf16Unroll>
        <<<grid_for(k3_bf16_grid_per_sm<bf16_t>()), kK3Threads, 0, s>>>(tp, (const bf16_t*)th, n,
                                                                         vec, st, seed, idx0);
  else
    k3_ewma_bf16<float, kK3Threads, kK3Bf16Unroll>
        <<<grid_for(k3_bf16_grid_per_sm<float>()), kK3Threads, 0, s>>>(tp, (const float*)th, n,
                                                                        vec, st, seed, idx0);
  return check_launch("k3_ewma_bf16");
}

// Launches the float32 update of n parameters (vector body + scalar tail).
occ_status launch_f32_body(float* tp, const float* th, int64_t n, const occ_ewma_state* st,
                           cudaStream_t s) {
  if (n == 0) return OCC_OK;
  const int64_t blocks_cap = (int64_t)sm_count() * 8;
  if (aligned(tp, 16) && aligned(th, 16)) {
    const int64_t n4 = n / 4;
    note_kernel(n4 > 0 ? "k3_ewma_vec" : "k3_ewma_scalar");
    if (n4 > 0) {
      const int64_t need = (n4 + kK3Threads * kK3Unroll - 1) / (kK3Threads * kK3Unroll);
      const unsigned grid = (unsigned)std::max<int64_t>(1, std::min(need, blocks_cap));
      k3_ewma_vec<kK3Threads, kK3Unroll><<<grid, kK3Threads, 0, s>>>((float4*)tp,
                                                                     (const float4*)th, n4, st);
    }
    if (n - n4 * 4 > 0) k3_ewma_scalar<kK3Threads><<<1, kK3Threads, 0, s>>>(tp, th, n4 * 4, n, st);
  } else {
    note_kernel("k3_ewma_scalar");
    const int64_t need = (n + kK3Threads - 1) / kK3Threads;
    const unsigned grid = (unsigned)std::max<int64_t>(1, std::min(need, blocks_cap));
    k3_ewma_scalar<kK3Threads><<<grid, kK3Threads, 0, s>>>(tp, th, 0, n, st);
  }
  return check_launch("k3_ewma body");
}

}  // namespace

extern "C" occ_status occ_ewma_update_bf16(void* theta_prox, const void* theta, occ_dtype theta_dt,
                                           int64_t n, double beta, occ_ewma_state* st,
                                           const occ_loss_stats* stats, double tau,
                                           int32_t min_streak, int32_t force_reset,
                                           uint64_t sr_seed, void* stream) {
  clear_error();
  occ_status rc = validate_ewma(n, beta, st, stats, tau, min_streak);
  if (rc != OCC_OK) return rc;
  if (theta_dt != OCC_F32 && theta_dt != OCC_BF16)
    return fail(OCC_ERR_UNSUPPORTED, "theta dtype %d", (int)theta_dt);
  const size_t es = dtype_size(theta_dt);
  if (n > 0) {
    if (!theta_prox || !theta) return fail(OCC_ERR_INVALID_ARG, "null theta_prox/theta");
    if (!aligned(theta_prox, 2) || !aligned(theta, es))
      return fail(OCC_ERR_MISALIGNED, "arrays must be aligned to their element size");
    if (overlaps(theta_prox, (size_t)n * 2, theta, (size_t)n * es))
      return fail(OCC_ERR_INVALID_ARG, "theta_prox overlaps theta");
  }
  cudaStream_t s = (cudaStream_t)stream;
  k3_ewma_prologue<<<1, 1, 0, s>>>(st, stats, beta, tau, min_streak, force_reset ? 1 : 0);
  rc = check_launch("k3_ewma_prologue");
  if (rc != OCC_OK) return rc;
  return launch_bf16_body((bf16_t*)theta_prox, theta, theta_dt, n, st, sr_seed, 0, s);
}

extern "C" occ_status occ_ewma_update_host(void* theta_prox_host, occ_dtype prox_dt,
                                           const void* theta, occ_dtype theta_dt, int64_t n,
                                           double beta, occ_ewma_state* st,
                                           const occ_loss_stats* stats, double tau,
                                           int32_t min_streak, int32_t force_reset,
                                           uint64_t sr_seed, void* staging, size_t staging_bytes,
                                           void* stream0, void* stream1) {
  clear_error();
  occ_status rc = validate_ewma(n, beta, st, stats, tau, min_streak);
  if (rc != OCC_OK) return rc;
  if ((prox_dt != OCC_F32 && prox_dt != OCC_BF16) || (theta_dt != OCC_F32 && theta_dt != OCC_BF16))
    return fail(OCC_ERR_UNSUPPORTED, "dtypes %d/%d", (int)prox_dt, (int)theta_dt);
  if (prox_dt == OCC_F32 && theta_dt != OCC_F32)
    return fail(OCC_ERR_UNSUPPORTED, "a float32 proximal buffer needs float32 theta");
  const size_t pes = dtype_size(prox_dt), tes = dtype_size(theta_dt);
  if (n > 0) {
    if (!theta_prox_host || !theta || !staging)
      return fail(OCC_ERR_INVALID_ARG, "null theta_prox_host/theta/staging");
    if (!aligned(theta_prox_host, 16) || !aligned(staging, 16) || !aligned(theta, tes))
      return fail(OCC_ERR_MISALIGNED, "host buffer and staging must be 16-byte aligned");
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, theta_prox_host) != cudaSuccess ||
        at.type != cudaMemoryTypeHost) {
      cudaGetLastError();
      return fail(OCC_ERR_INVALID_ARG, "theta_prox_host must be pinned (page-locked) host memory");
    }
  }
  // two staging slots, each a whole number of 16-byte groups
  const int64_t chunk = (int64_t)(staging_bytes / 2 / pes) / 8 * 8;
  if (n > 0 && chunk <= 0)
    return fail(OCC_ERR_WORKSPACE, "staging needs at least %zu bytes", 2 * 8 * pes);
  cudaStream_t s[2] = {(cudaStream_t)stream0, (cudaStream_t)stream1};
  k3_ewma_prologue<<<1, 1, 0, s[0]>>>(st, stats, beta, tau, min_streak, force_reset ? 1 : 0);
  rc = check_launch("k3_ewma_prologue");
  if (rc != OCC_OK || n == 0) return rc;
  cudaEvent_t ev;
  if (cudaEventCreateWithFlags(&ev, cudaEventDisableTiming) != cudaSuccess)
    return check_launch("cudaEventCreate");
  if (s[1] != s[0]) {  // stream 1 starts after the coefficients exist
    cudaEventRecord(ev, s[0]);
    cudaStreamWaitEvent(s[1], ev, 0);
  }
  char* host = (char*)theta_prox_host;
  char* stage[2] = {(char*)staging, (char*)staging + (size_t)chunk * pes};
  for (int64_t k = 0, off = 0; off < n; ++k, off += chunk) {
    const int64_t m = std::min(chunk, n - off);
    cudaStream_t q = s[k & 1];
    char* buf = stage[k & 1];
    cudaMemcpyAsync(buf, host + (size_t)off * pes, (size_t)m * pes, cudaMemcpyHostToDevice, q);
    const void* th = (const char*)theta + (size_t)off * tes;
    rc = prox_dt == OCC_F32
             ? launch_f32_body((float*)buf, (const float*)th, m, st, q)
             : launch_bf16_body((bf16_t*)buf, th, theta_dt, m, st, sr_seed, (uint64_t)off, q);
    if (rc != OCC_OK) break;
    cudaMemcpyAsync(host + (size_t)off * pes, buf, (size_t)m * pes, cudaMemcpyDeviceToHost, q);
  }
  if (s[1] != s[0]) {  // the call completes on stream 0
    cudaEventRecord(ev, s[1]);
    cudaStreamWaitEvent(s[0], ev, 0);
  }
  cudaEventDestroy(ev);
  if (rc != OCC_OK) return rc;
  return check_launch("occ_ewma_update_host");
}
