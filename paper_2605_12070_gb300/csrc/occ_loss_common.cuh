// Pieces shared by the decoupled-loss kernels (K0, K2 variants, the fused
// old+current kernel): the per-token scalar math of Eqs. 1-4, gradient
// stores, the token-count and finalize kernels, and the workspace layout.
#pragma once

#include <math.h>

#include <cmath>

#include "occ_common.cuh"

namespace occ {

constexpr int kK2Threads = 512;  // streaming kernel
constexpr int kK0Threads = 1024;
constexpr int kFinThreads = 1024;
constexpr uint8_t kWsBadId = 0x80;           // workspace flag: dropped for a bad id

struct LossKParams {
  ff log_rd_lo, log_rd_hi;        // log of the r_d band (may be -inf / +inf), float-float
  ff log_clip_lo, log_clip_hi;    // log(1 - eps_low), log(1 + eps_high), float-float
  float clip_lo, clip_hi;         // 1 - eps_low, 1 + eps_high
  float grad_scale;
  int rd_weight;
  long long denom;                // > 0: caller's N; else read from the workspace
  int proxy;                      // OCC_PROXY_*: how log pi_old is obtained
  double alpha;                   // behaviour-policy weight of the proxy
};

// log pi_prox of a token from log mu_old and log pi_theta (Table 1 proxies,
// App. A), in float64:
//   log-linear:  alpha log mu + (1 - alpha) log pi_theta
//   arithmetic:  log(alpha mu + (1 - alpha) pi_theta), written around the larger
//                term as log1p of an expm1 so that it keeps relative precision.
__device__ __forceinline__ double proxy_logprob(int proxy, double alpha, double lmu, double lth) {
  if (proxy == OCC_PROXY_LOGLINEAR) return alpha * lmu + (1.0 - alpha) * lth;
  const double d = lth - lmu;
  if (d <= 0.0)  // mu >= pi_theta: alpha mu + (1-alpha) pi = mu (1 + (1-alpha) (e^d - 1))
    return lmu + log1p((1.0 - alpha) * expm1(d));
  return lth + log1p(alpha * expm1(-d));
}

struct K2Args {
  const void* logits;
  int64_t T, V, ld, S, row0;
  int64_t stage_bytes;  // bytes of the shared-memory head of the row (two-pass kernels)
  int* ws_err;          // device-detected error bits, OR-ed into stats.err
  unsigned* ws_rows;    // row counter of the persistent fused kernel (K0 clears it)
  const int32_t* ids;
  const float* lp_old;
  const float* lp_mu;
  const float* adv;
  const uint8_t* mask;
  const long long* ws_N;
  float* ws_loss;
  uint8_t* ws_flags;
  float* logp_out;
  uint8_t* flags_out;
  void* dlogits;
  int64_t ld_grad;
  LossKParams kp;
};

// Per-token scalar part (R2..R8): threshold decisions in float-float log space
// (the proxies of Table 1 are formed in float64: log1p / expm1).
__device__ __forceinline__ void token_math(const LossKParams& kp, ff lse, float zy, ff lpo,
                                           float lpm, float A, long long N, float& g,
                                           float& loss_t, uint32_t& flags, float& logp_f) {
  const ff logp = ff_add(ff_neg(lse), zy);
  if (kp.proxy != OCC_PROXY_NONE) {
    const double d = proxy_logprob(kp.proxy, kp.alpha, (double)lpm, (double)logp.hi + (double)logp.lo);
    const float h = (float)d;
    lpo = ff{h, isfinite(h) ? (float)(d - (double)h) : 0.f};
  }
  const ff log_rd = ff_add(lpo, -lpm);
  const bool in_band = ff_le(kp.log_rd_lo, log_rd) && ff_le(log_rd, kp.log_rd_hi);
  const ff log_rs = ff_sub(logp, lpo);
  const bool mis = (A >= 0.f) ? ff_le(log_rs, kp.log_clip_hi) : ff_le(kp.log_clip_lo, log_rs);
  const float r_s = expf(ff_round(log_rs));
  const float r_d = expf(ff_round(log_rd));
  const float w = kp.rd_weight ? r_d : 1.f;
  const float rc = fminf(fmaxf(r_s, kp.clip_lo), kp.clip_hi);
  const float s = fminf(r_s * A, rc * A);
  const bool active = in_band && mis;
  loss_t = in_band ? -w * s : 0.f;
  g = (active && N > 0) ? __fdividef(-kp.grad_scale * w * r_s * A, (float)N) : 0.f;
  flags = (in_band ? OCC_FLAG_IN_BAND : 0) | (mis ? 0 : OCC_FLAG_CLIPPED) |
          (active ? OCC_FLAG_ACTIVE : 0) | OCC_FLAG_VALID;
  logp_f = ff_round(logp);
}

// Exponent offset of the backward pass, g folded in: dlogits_v = -sign(g)
// 2^(z_v L - cb) (+ g at the sampled token) with cb = lse L - log2|g|, from the
// base-2 lse l2; 0 when g = 0.
__device__ __forceinline__ float backward_offset(ff l2, float g) {
  if (g == 0.f) return 0.f;
  int e;
  const float fm = frexpf(fabsf(g), &e);  // |g| = fm 2^e
  return ff_round(ff_add(ff_add(l2, -(float)e), -log2f(fm)));
}

// Writes VEC gradient values starting at a 16-byte aligned output address.
template <typename Tout, int VEC>
struct OutVec;
template <>
struct OutVec<bf16_t, 8> {
  __device__ __forceinline__ static void store(bf16_t* p, const float (&d)[8]) {
    uint4 v;
    v.x = pack_bf16x2(d[0], d[1]);
    v.y = pack_bf16x2(d[2], d[3]);
    v.z = pack_bf16x2(d[4], d[5]);
    v.w = pack_bf16x2(d[6], d[7]);
    st_stream_v4(p, v);
  }
  __device__ __forceinline__ static void zero(bf16_t* p) { st_stream_v4(p, make_uint4(0, 0, 0, 0)); }
};
template <>
struct OutVec<float, 8> {
  __device__ __forceinline__ static void store(float* p, const float (&d)[8]) {
    st_stream_v4(p, make_uint4(__float_as_uint(d[0]), __float_as_uint(d[1]),
                               __float_as_uint(d[2]), __float_as_uint(d[3])));
    st_stream_v4(p + 4, make_uint4(__float_as_uint(d[4]), __float_as_uint(d[5]),
                                   __float_as_uint(d[6]), __float_as_uint(d[7])));
  }
  __device__ __forceinline__ static void zero(float* p) {
    st_stream_v4(p, make_uint4(0, 0, 0, 0));
    st_stream_v4(p + 4, make_uint4(0, 0, 0, 0));
  }
};
template <>
struct OutVec<float, 4> {
  __device__ __forceinline__ static void store(float* p, const float (&d)[4]) {
    st_stream_v4(p, make_uint4(__float_as_uint(d[0]), __float_as_uint(d[1]),
                               __float_as_uint(d[2]), __float_as_uint(d[3])));
  }
  __device__ __forceinline__ static void zero(float* p) { st_stream_v4(p, make_uint4(0, 0, 0, 0)); }
};

__device__ __forceinline__ void out_scalar(float* p, float x) { *p = x; }
__device__ __forceinline__ void out_scalar(bf16_t* p, float x) { st_bf16(p, x); }

// Zeroes n gradient entries of a row slice (vector body + scalar tail).
template <typename Tout, int VEC, int NT>
__device__ __forceinline__ void zero_slice_vec(Tout* d, int64_t n) {
  const int64_t nvec = n / VEC;
  for (int64_t i = threadIdx.x; i < nvec; i += NT) OutVec<Tout, VEC>::zero(d + i * VEC);
  const int64_t t0 = nvec * VEC;
  if ((int64_t)threadIdx.x < n - t0) out_scalar(d + t0 + threadIdx.x, 0.f);
}

// Outputs of a dropped token (mask 0 or id out of range).
__device__ __forceinline__ void dropped_token_outputs(const K2Args& a, int64_t row, bool m,
                                                      bool id_ok) {
  a.ws_loss[row] = 0.f;
  a.ws_flags[row] = (m && !id_ok) ? kWsBadId : 0;
  if (a.logp_out) a.logp_out[row] = id_ok ? 0.f : __int_as_float(0x7fc00000);
  if (a.flags_out) a.flags_out[row] = 0;
}

// Writes VEC gradient values with an L2 policy (16 bytes per 8 bf16 / 4 f32).
template <typename Tout, int VEC>
struct OutVecHint;
template <>
struct OutVecHint<bf16_t, 8> {
  __device__ __forceinline__ static void store(bf16_t* p, const float (&d)[8], uint64_t pol) {
    st_hint_v4(p, make_uint4(pack_bf16x2(d[0], d[1]), pack_bf16x2(d[2], d[3]),
                             pack_bf16x2(d[4], d[5]), pack_bf16x2(d[6], d[7])), pol);
  }
  __device__ __forceinline__ static void zero(bf16_t* p, uint64_t pol) {
    st_hint_v4(p, make_uint4(0, 0, 0, 0), pol);
  }
};
template <>
struct OutVecHint<float, 8> {
  __device__ __forceinline__ static void store(float* p, const float (&d)[8], uint64_t pol) {
    st_hint_v4(p, make_uint4(__float_as_uint(d[0]), __float_as_uint(d[1]), __float_as_uint(d[2]),
                             __float_as_uint(d[3])), pol);
    st_hint_v4(p + 4, make_uint4(__float_as_uint(d[4]), __float_as_uint(d[5]),
                                 __float_as_uint(d[6]), __float_as_uint(d[7])), pol);
  }
  __device__ __forceinline__ static void zero(float* p, uint64_t pol) {
    st_hint_v4(p, make_uint4(0, 0, 0, 0), pol);
    st_hint_v4(p + 4, make_uint4(0, 0, 0, 0), pol);
  }
};
template <>
struct OutVecHint<float, 4> {
  __device__ __forceinline__ static void store(float* p, const float (&d)[4], uint64_t pol) {
    st_hint_v4(p, make_uint4(__float_as_uint(d[0]), __float_as_uint(d[1]), __float_as_uint(d[2]),
                             __float_as_uint(d[3])), pol);
  }
  __device__ __forceinline__ static void zero(float* p, uint64_t pol) {
    st_hint_v4(p, make_uint4(0, 0, 0, 0), pol);
  }
};

// K0: N = number of tokens with mask set and id in range.
template <int NT>
__global__ void __launch_bounds__(NT) k0_count_valid(const uint8_t* __restrict__ mask,
                                                     const int32_t* __restrict__ ids, int64_t T,
                                                     int64_t V, long long* __restrict__ ws_N,
                                                     int* __restrict__ ws_err,
                                                     unsigned* __restrict__ ws_rows) {
  __shared__ long long part[NT / 32];
  if (threadIdx.x == 0) {
    *ws_err = 0;
    *ws_rows = 0;
  }
  long long c = 0;
  for (int64_t t0 = threadIdx.x; t0 < T; t0 += 8 * (int64_t)NT) {
    int idv[8];
    uint8_t mv[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int64_t t = t0 + (int64_t)j * NT;
      idv[j] = t < T ? ids[t] : -1;
      mv[j] = (t < T && mask) ? mask[t] : (uint8_t)1;
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) c += (mv[j] != 0 && idv[j] >= 0 && (int64_t)idv[j] < V) ? 1 : 0;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = c;
  __syncthreads();
  if (threadIdx.x == 0) {
    long long s = 0;
    for (int w = 0; w < NT / 32; ++w) s += part[w];
    *ws_N = s;
  }
}

// Fixed-order reduction of the per-token losses and flags into the stats.
template <int NT>
__global__ void __launch_bounds__(NT) k2_finalize(int64_t T, const float* __restrict__ ws_loss,
                                                  const uint8_t* __restrict__ ws_flags,
                                                  const long long* __restrict__ ws_N,
                                                  const int* __restrict__ ws_err,
                                                  long long denom_fixed, occ_loss_stats* st) {
  __shared__ float2 ps[NT / 32];
  __shared__ long long pc[4][NT / 32];
  __shared__ int pb[NT / 32];
  float2 s = make_float2(0.f, 0.f);
  long long nv = 0, nout = 0, nclip = 0, nact = 0;
  int bad = 0;
  for (int64_t t = threadIdx.x; t < T; t += NT) {
    const float l = ws_loss[t];
    const uint32_t f = ws_flags[t];
    s = pair_add(s, make_float2(l, 0.f));
    if (f & OCC_FLAG_VALID) {
      ++nv;
      nout += (f & OCC_FLAG_IN_BAND) ? 0 : 1;
      nclip += (f & OCC_FLAG_CLIPPED) ? 1 : 0;
      nact += (f & OCC_FLAG_ACTIVE) ? 1 : 0;
    }
    bad |= (f & kWsBadId) ? 1 : 0;
  }
  s = warp_pair_sum(s);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    nv += __shfl_xor_sync(0xffffffffu, nv, o);
    nout += __shfl_xor_sync(0xffffffffu, nout, o);
    nclip += __shfl_xor_sync(0xffffffffu, nclip, o);
    nact += __shfl_xor_sync(0xffffffffu, nact, o);
    bad |= __shfl_xor_sync(0xffffffffu, bad, o);
  }
  const int w = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) {
    ps[w] = s;
    pc[0][w] = nv;
    pc[1][w] = nout;
    pc[2][w] = nclip;
    pc[3][w] = nact;
    pb[w] = bad;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float2 S = make_float2(0.f, 0.f);
    long long c[4] = {0, 0, 0, 0};
    int b = 0;
    for (int k = 0; k < NT / 32; ++k) {
      S = pair_add(S, ps[k]);
      for (int q = 0; q < 4; ++q) c[q] += pc[q][k];
      b |= pb[k];
    }
    const long long N = denom_fixed > 0 ? denom_fixed : *ws_N;
    const double loss_sum = (double)S.x + (double)S.y;
    st->loss_sum = loss_sum;
    st->loss = N > 0 ? loss_sum / (double)N : 0.0;
    st->n_valid = c[0];
    st->n_rd_out = c[1];
    st->n_clipped = c[2];
    st->n_active = c[3];
    st->denom = N;
    st->err = (b ? OCC_DATA_ERR_BAD_ID : 0) | *ws_err;
    st->reserved = 0;
  }
}

// --------------------------------------------------------------- host side

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

struct WsLayout {
  size_t off_N, off_err, off_rows, off_loss, off_flags, total;
};
inline WsLayout ws_layout(int64_t T) {
  const size_t t = T > 0 ? (size_t)T : 0;
  WsLayout w;
  w.off_N = 0;
  w.off_err = 8;
  w.off_rows = 12;
  w.off_loss = 256;
  w.off_flags = w.off_loss + align_up(4 * t, 256);
  w.total = w.off_flags + align_up(t, 256);
  return w;
}


// Online (c, s, sv): s = sum 2^(x L - c), sv = sum 2^(x L - c) v.
struct LseAccV {
  float c, s, sv;
};

template <int N, bool WV>
__device__ __forceinline__ void accv_add(LseAccV& a, const float (&x)[N], const float (&v)[N]) {
  float t = 0.f, tv = 0.f;
#pragma unroll
  for (int j = 0; j < N; ++j) {
    const float e = ex2_approx(fmaf(x[j], kLog2e, -a.c));
    t += e;
    if (WV) tv = fmaf(e, v[j], tv);
  }
  if (t <= 1.8446744073709552e19f) {  // 2^64; false for inf / NaN and for c = -inf
    a.s += t;
    a.sv += tv;
    return;
  }
  float m = x[0];
#pragma unroll
  for (int j = 1; j < N; ++j) m = fmaxf(m, x[j]);
  const float ms = m * kLog2e;
  if (ms > a.c + kRescale) {
    const float f = exp2f(a.c - ms);
    a.s *= f;
    a.sv *= f;
    a.c = ms;
  }
  if (a.c == -INFINITY) return;
  t = 0.f;
  tv = 0.f;
#pragma unroll
  for (int j = 0; j < N; ++j) {
    const float e = ex2_approx(fmaf(x[j], kLog2e, -a.c));
    t += e;
    if (WV) tv = fmaf(e, v[j], tv);
  }
  a.s += t;
  a.sv += tv;
}

struct FusedRed {
  float c[2][32];
  float2 s[2][32];
  float sv[2][32];
};

// Block merge of two accumulators; the results are valid in thread 0.
template <int NT>
__device__ __forceinline__ void block_lse_v2(const LseAccV (&acc)[2], FusedRed& r, float (&C)[2],
                                             float2 (&S)[2], float (&SV)[2]) {
  constexpr int NW = NT / 32;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
#pragma unroll
  for (int k = 0; k < 2; ++k) {
    const float wm = warp_max(acc[k].c);
    const float f = acc[k].c == -INFINITY ? 0.f : exp2f(acc[k].c - wm);
    float2 v = warp_pair_sum(make_float2(acc[k].s * f, 0.f));
    float sv = acc[k].sv * f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sv += __shfl_xor_sync(0xffffffffu, sv, o);
    if (lane == 0) {
      r.c[k][wid] = wm;
      r.s[k][wid] = v;
      r.sv[k][wid] = sv;
    }
  }
  __syncthreads();
  if (wid == 0) {
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      const float cw = lane < NW ? r.c[k][lane] : -INFINITY;
      const float cm = warp_max(cw);
      float2 w = make_float2(0.f, 0.f);
      float sv = 0.f;
      if (lane < NW && cw != -INFINITY) {
        const float f = exp2f(cw - cm);
        const float2 p = r.s[k][lane];
        const float hi = p.x * f;
        w = make_float2(hi, fmaf(p.x, f, -hi) + p.y * f);
        sv = r.sv[k][lane] * f;
      }
      w = warp_pair_sum(w);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) sv += __shfl_xor_sync(0xffffffffu, sv, o);
      C[k] = cm;
      S[k] = w;
      SV[k] = sv;
    }
  }
}


// Host: a double threshold as a normalised float-float pair.
inline ff ff_of(double x) {
  const float h = (float)x;
  return ff{h, std::isfinite(h) ? (float)(x - (double)h) : 0.f};
}

// Host: validates the arguments every loss entry point shares (all but the
// source of log pi_old), fills the kernel arguments and reports whether the
// rows qualify for the 16-byte vector kernels.
inline occ_status prepare_loss_args(const void* logits, occ_dtype dt, int64_t T, int64_t V,
                                    int64_t ld, const int32_t* ids, const float* logp_mu,
                                    const float* adv, const uint8_t* loss_mask,
                                    const occ_loss_params* p, float* logp_out, uint8_t* flags_out,
                                    void* dlogits, int64_t ld_grad, occ_loss_stats* stats,
                                    void* workspace, size_t ws_bytes, K2Args& a, bool& vec) {
  if (dt != OCC_F32 && dt != OCC_BF16) return fail(OCC_ERR_UNSUPPORTED, "dtype %d", (int)dt);
  if (!p) return fail(OCC_ERR_INVALID_ARG, "params pointer is null");
  if (T < 0 || V < 1 || ld < V)
    return fail(OCC_ERR_INVALID_ARG, "need T >= 0, V >= 1, ld >= V (T=%lld V=%lld ld=%lld)",
                (long long)T, (long long)V, (long long)ld);
  if (V > 0x7fffffffLL)  // token ids are int32; row-local indices are 32-bit
    return fail(OCC_ERR_UNSUPPORTED, "V = %lld exceeds 2^31 - 1", (long long)V);
  if (!(p->rd_lo >= 0.0) || !(p->rd_hi >= p->rd_lo) || !(p->eps_low >= 0.0) ||
      !(p->eps_low <= 1.0) || !(p->eps_high >= 0.0) || !isfinite(p->grad_scale) ||
      (p->rd_weight != 0 && p->rd_weight != 1) || (p->dlogits_f32 != 0 && p->dlogits_f32 != 1) ||
      p->proxy < OCC_PROXY_NONE || p->proxy > OCC_PROXY_ARITHMETIC ||
      (p->proxy != OCC_PROXY_NONE && !(p->alpha >= 0.0 && p->alpha <= 1.0)))
    return fail(OCC_ERR_INVALID_ARG,
                "thresholds must satisfy 0 <= rd_lo <= rd_hi, 0 <= eps_low <= 1, eps_high >= 0; "
                "grad_scale finite; rd_weight and dlogits_f32 in {0,1}; proxy in {0,1,2} with "
                "alpha in [0,1]");
  if (!stats || !aligned(stats, 8)) return fail(OCC_ERR_INVALID_ARG, "stats null or misaligned");
  const WsLayout wl = ws_layout(T);
  if (!workspace || !aligned(workspace, 16) || ws_bytes < wl.total)
    return fail(OCC_ERR_WORKSPACE, "workspace needs %zu bytes, 16-byte aligned (got %zu)",
                wl.total, ws_bytes);
  const size_t es = dtype_size(dt);
  const size_t es_out = p->dlogits_f32 ? 4 : es;
  if (T > 0) {
    if (!logits || !ids || !logp_mu || !adv)
      return fail(OCC_ERR_INVALID_ARG, "null logits/ids/logp_mu/adv");
    if (!aligned(logits, es) || !aligned(ids, 4) || !aligned(logp_mu, 4) || !aligned(adv, 4) ||
        (logp_out && !aligned(logp_out, 4)))
      return fail(OCC_ERR_MISALIGNED, "arrays must be aligned to their element size");
    if (dlogits) {
      if (ld_grad < V) return fail(OCC_ERR_INVALID_ARG, "ld_grad < V");
      if (!aligned(dlogits, es_out)) return fail(OCC_ERR_MISALIGNED, "dlogits misaligned");
      if (dlogits == logits) {
        if (es_out != es || ld_grad != ld)
          return fail(OCC_ERR_INVALID_ARG,
                      "in-place dlogits needs the logits dtype and the same row stride");
      } else {
        const size_t in_bytes = ((size_t)(T - 1) * (size_t)ld + (size_t)V) * es;
        const size_t out_bytes = ((size_t)(T - 1) * (size_t)ld_grad + (size_t)V) * es_out;
        if (overlaps(logits, in_bytes, dlogits, out_bytes))
          return fail(OCC_ERR_INVALID_ARG, "dlogits overlaps logits without being identical");
      }
    }
  }
  char* ws = (char*)workspace;
  a.logits = logits;
  a.T = T;
  a.V = V;
  a.ld = ld;
  a.S = V;
  a.row0 = 0;
  a.stage_bytes = 0;
  a.ids = ids;
  a.lp_old = nullptr;
  a.lp_mu = logp_mu;
  a.adv = adv;
  a.mask = loss_mask;
  a.ws_N = (const long long*)(ws + wl.off_N);
  a.ws_err = (int*)(ws + wl.off_err);
  a.ws_rows = (unsigned*)(ws + wl.off_rows);
  a.ws_loss = (float*)(ws + wl.off_loss);
  a.ws_flags = (uint8_t*)(ws + wl.off_flags);
  a.logp_out = logp_out;
  a.flags_out = flags_out;
  a.dlogits = dlogits;
  a.ld_grad = ld_grad;
  a.kp.log_rd_lo = ff_of(p->rd_lo > 0.0 ? log(p->rd_lo) : -INFINITY);
  a.kp.log_rd_hi = ff_of(isinf(p->rd_hi) ? INFINITY : log(p->rd_hi));
  a.kp.log_clip_lo = ff_of(p->eps_low < 1.0 ? log1p(-p->eps_low) : -INFINITY);
  a.kp.log_clip_hi = ff_of(log1p(p->eps_high));
  a.kp.clip_lo = (float)(1.0 - p->eps_low);
  a.kp.clip_hi = (float)(1.0 + p->eps_high);
  a.kp.grad_scale = (float)p->grad_scale;
  a.kp.rd_weight = p->rd_weight;
  a.kp.denom = p->denom > 0 ? (long long)p->denom : 0;
  a.kp.proxy = p->proxy;
  a.kp.alpha = p->alpha;
  vec = T > 0 && aligned(logits, 16) && ((ld * (int64_t)es) % 16 == 0) &&
        (!dlogits || (aligned(dlogits, 16) && ((ld_grad * (int64_t)es_out) % 16 == 0)));
  return OCC_OK;
}

// Host: K0 (valid-token count and cleared error word; always launched because
// the workspace starts undefined).
inline occ_status launch_k0(const K2Args& a, cudaStream_t s) {
  k0_count_valid<kK0Threads><<<1, kK0Threads, 0, s>>>(a.mask, a.ids, a.T, a.V,
                                                      const_cast<long long*>(a.ws_N), a.ws_err,
                                                      a.ws_rows);
  return check_launch("k0_count_valid");
}

// Host: the fixed-order reduction of the per-token records into the stats.
inline occ_status launch_finalize(const K2Args& a, occ_loss_stats* stats, cudaStream_t s) {
  k2_finalize<kFinThreads><<<1, kFinThreads, 0, s>>>(a.T, a.ws_loss, a.ws_flags, a.ws_N, a.ws_err,
                                                     a.kp.denom, stats);
  return check_launch("k2_finalize");
}

}  // namespace occ
