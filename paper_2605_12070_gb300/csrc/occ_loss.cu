// K0 + K2: the decoupled PPO loss over policy logits, forward and backward in
// one pass over the vocabulary.
//
// Per token t (Sec. 3.2 and Eqs. 1-4; the role of r_d follows Table 5):
//   logp   = z[t, y] - lse(z[t])                       (streamed, as in K1)
//   r_d    = pi_old / mu_old, masked to [rd_lo, rd_hi] (Eq. 4)
//   r_s    = pi_theta / pi_old under the sign-dependent clip (Eqs. 2-3)
//   loss_t = -m M_d w_d min(r_s A, clip(r_s) A), token mean over N valid tokens
//   dz[v]  = g (1[v = y] - softmax(z[t])_v), g = -grad_scale m M_d MIS w_d r_s A / N
//
// Kernel layout (vector path): one thread-block cluster of C CTAs per row.
// Each CTA owns a V/C slice, loads it once from HBM with 16-byte coalesced
// loads, keeps it in shared memory, and folds it into an online log-sum-exp.
// The C partial (c, s) pairs are exchanged through distributed shared memory,
// every CTA of the cluster derives the same lse and per-token scalars, and
// the slice is turned into dlogits straight out of shared memory.  So the
// logits are read from HBM once and dlogits written once: 2 * V * sizeof(T)
// bytes per valid token, V * sizeof(T_out) per dropped token (no read).
// A scalar-load two-pass kernel handles rows that are not 16-byte aligned
// and vocabularies too large for the cluster's shared memory.
//
// K0 counts the valid tokens N before K2 runs (the token-mean denominator is
// needed by every row's gradient).  A final one-CTA kernel reduces the
// per-token losses and flags in a fixed order (deterministic float64 loss).
#include <math.h>

#include "occ_common.cuh"

namespace occ {

constexpr int kK2Threads = 512;
constexpr int kK2Unroll = 8;
constexpr int kK0Threads = 1024;
constexpr int kFinThreads = 1024;
constexpr size_t kSliceTarget = 100 * 1024;  // two CTAs per SM
constexpr size_t kSliceMax = 200 * 1024;     // one CTA per SM
constexpr uint8_t kWsBadId = 0x80;           // workspace flag: dropped for a bad id

struct LossKParams {
  double log_rd_lo, log_rd_hi;    // log of the r_d band (may be -inf / +inf)
  double log_clip_lo, log_clip_hi;  // log(1 - eps_low), log(1 + eps_high)
  float clip_lo, clip_hi;         // 1 - eps_low, 1 + eps_high
  float grad_scale;
  int rd_weight;
  long long denom;                // > 0: caller's N; else read from the workspace
};

struct K2Args {
  const void* logits;
  int64_t T, V, ld, S, row0;
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

// Per-token scalar part (R2..R8): threshold decisions in float64 log space.
__device__ __forceinline__ void token_math(const LossKParams& kp, double lse, float zy, float lpo,
                                           float lpm, float A, long long N, float& g,
                                           float& loss_t, uint32_t& flags, float& logp_f) {
  const double logp = (double)zy - lse;
  const double log_rd = (double)lpo - (double)lpm;
  const bool in_band = (log_rd >= kp.log_rd_lo) && (log_rd <= kp.log_rd_hi);
  const double log_rs = logp - (double)lpo;
  const bool mis = (A >= 0.f) ? (log_rs <= kp.log_clip_hi) : (log_rs >= kp.log_clip_lo);
  const float r_s = expf((float)log_rs);
  const float r_d = expf((float)log_rd);
  const float w = kp.rd_weight ? r_d : 1.f;
  const float rc = fminf(fmaxf(r_s, kp.clip_lo), kp.clip_hi);
  const float s = fminf(r_s * A, rc * A);
  const bool active = in_band && mis;
  loss_t = in_band ? -w * s : 0.f;
  g = (active && N > 0) ? (-kp.grad_scale * w * r_s * A) / (float)N : 0.f;
  flags = (in_band ? OCC_FLAG_IN_BAND : 0) | (mis ? 0 : OCC_FLAG_CLIPPED) |
          (active ? OCC_FLAG_ACTIVE : 0) | OCC_FLAG_VALID;
  logp_f = (float)logp;
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

template <typename Tin, typename Tout, int NT, int U>
__global__ void __launch_bounds__(NT, 2) k2_loss_smem(const K2Args a) {
  constexpr int VEC = Elem<Tin>::kVec;
  extern __shared__ __align__(16) uint4 sm_row[];
  __shared__ RedScratch red;
  __shared__ __align__(16) float4 cta_part;
  __shared__ float bc_g, bc_cb;

  const uint32_t C = cluster_nctarank();
  const uint32_t rank = cluster_ctarank();
  const int64_t row = a.row0 + blockIdx.x / C;
  const int tid = threadIdx.x;
  const int id = a.ids[row];
  const bool m = (a.mask == nullptr) || (a.mask[row] != 0);
  const bool id_ok = (id >= 0) && ((int64_t)id < a.V);
  const int64_t v0 = (int64_t)rank * a.S;
  const int64_t n = max((int64_t)0, min(a.S, a.V - v0));
  Tout* drow = a.dlogits ? (Tout*)a.dlogits + row * a.ld_grad + v0 : nullptr;

  if (!(m && id_ok)) {  // uniform over the cluster: no barrier is entered
    if (drow) zero_slice_vec<Tout, VEC, NT>(drow, n);
    if (rank == 0 && tid == 0) dropped_token_outputs(a, row, m, id_ok);
    return;
  }

  const Tin* zrow = (const Tin*)a.logits + row * a.ld;
  float zy = 0.f, lpo = 0.f, lpm = 0.f, A = 0.f;
  if (tid == 0) {
    zy = Elem<Tin>::load(zrow + id);
    lpo = a.lp_old[row];
    lpm = a.lp_mu[row];
    A = a.adv[row];
  }

  // Forward: HBM -> registers -> (shared memory copy, online log-sum-exp).
  const uint4* zv = reinterpret_cast<const uint4*>(zrow + v0);
  const int64_t nvec = n / VEC;
  LseAcc acc;
  acc_init(acc);
  int64_t i = tid;
  for (; i + (int64_t)(U - 1) * NT < nvec; i += (int64_t)U * NT) {
    uint4 r[U];
#pragma unroll
    for (int u = 0; u < U; ++u) r[u] = ld_stream_v4(zv + i + u * NT);
#pragma unroll
    for (int u = 0; u < U; ++u) {
      sm_row[i + u * NT] = r[u];
      float x[VEC];
      Elem<Tin>::unpack(r[u], x);
      acc_add(acc, x);
    }
  }
  for (; i < nvec; i += NT) {
    const uint4 r = ld_stream_v4(zv + i);
    sm_row[i] = r;
    float x[VEC];
    Elem<Tin>::unpack(r, x);
    acc_add(acc, x);
  }
  const int64_t t0 = nvec * VEC;
  if ((int64_t)tid < n - t0) {
    float x[1] = {Elem<Tin>::load(zrow + v0 + t0 + tid)};
    Elem<Tin>::put(reinterpret_cast<Tin*>(sm_row) + t0 + tid, x[0]);
    acc_add(acc, x);
  }

  float Cr;
  float2 Sr;
  block_lse<NT>(acc, red, Cr, Sr);
  if (C > 1) {
    if (tid == 0) cta_part = make_float4(Cr, Sr.x, Sr.y, 0.f);
    cluster_arrive_release();
    cluster_wait_acquire();
    if (tid == 0) {  // merge the C partials in rank order (same order in every CTA)
      float Cm = -INFINITY;
      for (uint32_t r = 0; r < C; ++r) Cm = fmaxf(Cm, ld_dsmem_f4(&cta_part, r).x);
      float2 s = make_float2(0.f, 0.f);
      for (uint32_t r = 0; r < C; ++r) {
        const float4 P = ld_dsmem_f4(&cta_part, r);
        if (P.x == -INFINITY) continue;
        const float f = exp2f(P.x - Cm);
        const float hi = P.y * f;
        s = pair_add(s, make_float2(hi, fmaf(P.y, f, -hi) + P.z * f));
      }
      Cr = Cm;
      Sr = s;
    }
    cluster_arrive_release();  // this CTA is done reading the others' shared memory
  }

  if (tid == 0) {
    const double lse = lse_from(Cr, Sr);
    const long long N = a.kp.denom > 0 ? a.kp.denom : *a.ws_N;
    float g, loss_t, logp_f;
    uint32_t fl;
    token_math(a.kp, lse, zy, lpo, lpm, A, N, g, loss_t, fl, logp_f);
    bc_g = g;
    bc_cb = (float)(lse * (double)kLog2e);  // p_v = 2^(z_v L - cb)
    if (rank == 0) {
      a.ws_loss[row] = loss_t;
      a.ws_flags[row] = (uint8_t)fl;
      if (a.logp_out) a.logp_out[row] = logp_f;
      if (a.flags_out) a.flags_out[row] = (uint8_t)fl;
    }
  }
  __syncthreads();

  // Backward straight from shared memory.
  if (drow) {
    const float g = bc_g;
    if (g == 0.f) {
      zero_slice_vec<Tout, VEC, NT>(drow, n);
    } else {
      const float cb = bc_cb;
      const int64_t yl = (int64_t)id - v0;  // sampled token, local index (may be outside)
#pragma unroll 4
      for (int64_t j = tid; j < nvec; j += NT) {
        float x[VEC], d[VEC];
        Elem<Tin>::unpack(sm_row[j], x);
#pragma unroll
        for (int k = 0; k < VEC; ++k) {
          d[k] = -g * ex2_approx(fmaf(x[k], kLog2e, -cb));
          if (j * VEC + k == yl) d[k] += g;
        }
        OutVec<Tout, VEC>::store(drow + j * VEC, d);
      }
      if ((int64_t)tid < n - t0) {
        const int64_t k = t0 + tid;
        float xs;
        if (sizeof(Tin) == 2)
          xs = __uint_as_float(((uint32_t)reinterpret_cast<const uint16_t*>(sm_row)[k]) << 16);
        else
          xs = reinterpret_cast<const float*>(sm_row)[k];
        float dv = -g * ex2_approx(fmaf(xs, kLog2e, -cb));
        if (k == yl) dv += g;
        out_scalar(drow + k, dv);
      }
    }
  }
  if (C > 1) cluster_wait_acquire();
}

// Any alignment / any V: element loads, forward pass then backward pass over
// global memory (the second read of the row is served from L2 when it fits).
template <typename Tin, typename Tout, int NT>
__global__ void __launch_bounds__(NT) k2_loss_stream(const K2Args a) {
  __shared__ RedScratch red;
  __shared__ float bc_g, bc_cb;
  const int64_t row = a.row0 + blockIdx.x;
  const int tid = threadIdx.x;
  const int id = a.ids[row];
  const bool m = (a.mask == nullptr) || (a.mask[row] != 0);
  const bool id_ok = (id >= 0) && ((int64_t)id < a.V);
  const int64_t V = a.V;
  Tout* drow = a.dlogits ? (Tout*)a.dlogits + row * a.ld_grad : nullptr;
  if (!(m && id_ok)) {
    if (drow)
      for (int64_t v = tid; v < V; v += NT) out_scalar(drow + v, 0.f);
    if (tid == 0) dropped_token_outputs(a, row, m, id_ok);
    return;
  }
  const Tin* z = (const Tin*)a.logits + row * a.ld;
  float zy = 0.f, lpo = 0.f, lpm = 0.f, A = 0.f;
  if (tid == 0) {
    zy = Elem<Tin>::load(z + id);
    lpo = a.lp_old[row];
    lpm = a.lp_mu[row];
    A = a.adv[row];
  }
  LseAcc acc;
  acc_init(acc);
  for (int64_t v0 = tid; v0 < V; v0 += 8 * (int64_t)NT) {
    float x[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int64_t v = v0 + (int64_t)j * NT;
      x[j] = v < V ? Elem<Tin>::load(z + v) : -INFINITY;
    }
    acc_add(acc, x);
  }
  float Cr;
  float2 Sr;
  block_lse<NT>(acc, red, Cr, Sr);
  if (tid == 0) {
    const double lse = lse_from(Cr, Sr);
    const long long N = a.kp.denom > 0 ? a.kp.denom : *a.ws_N;
    float g, loss_t, logp_f;
    uint32_t fl;
    token_math(a.kp, lse, zy, lpo, lpm, A, N, g, loss_t, fl, logp_f);
    bc_g = g;
    bc_cb = (float)(lse * (double)kLog2e);
    a.ws_loss[row] = loss_t;
    a.ws_flags[row] = (uint8_t)fl;
    if (a.logp_out) a.logp_out[row] = logp_f;
    if (a.flags_out) a.flags_out[row] = (uint8_t)fl;
  }
  __syncthreads();
  if (drow) {
    const float g = bc_g, cb = bc_cb;
    for (int64_t v = tid; v < V; v += NT) {
      float dv = 0.f;
      if (g != 0.f) {
        dv = -g * ex2_approx(fmaf(Elem<Tin>::load(z + v), kLog2e, -cb));
        if (v == id) dv += g;
      }
      out_scalar(drow + v, dv);
    }
  }
}

// K0: N = number of tokens with mask set and id in range.
template <int NT>
__global__ void __launch_bounds__(NT) k0_count_valid(const uint8_t* __restrict__ mask,
                                                     const int32_t* __restrict__ ids, int64_t T,
                                                     int64_t V, long long* __restrict__ ws_N) {
  __shared__ long long part[NT / 32];
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
    st->err = b ? OCC_DATA_ERR_BAD_ID : 0;
    st->reserved = 0;
  }
}

// --------------------------------------------------------------- host side

static inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

struct WsLayout {
  size_t off_N, off_loss, off_flags, total;
};
static WsLayout ws_layout(int64_t T) {
  const size_t t = T > 0 ? (size_t)T : 0;
  WsLayout w;
  w.off_N = 0;
  w.off_loss = 256;
  w.off_flags = w.off_loss + align_up(4 * t, 256);
  w.total = w.off_flags + align_up(t, 256);
  return w;
}

struct ClusterPlan {
  int C;       // CTAs per row (0: use the streaming kernel)
  int64_t S;   // elements per CTA slice (multiple of the vector width)
  size_t smem; // dynamic shared memory per CTA
};

static ClusterPlan plan_cluster(int64_t V, size_t es) {
  const int64_t vec = 16 / (int64_t)es;
  for (size_t cap : {kSliceTarget, kSliceMax}) {
    for (int C : {1, 2, 4, 8}) {
      int64_t S = (V + C - 1) / C;
      S = (S + vec - 1) / vec * vec;
      if ((size_t)S * es <= cap) return ClusterPlan{C, S, (size_t)S * es};
    }
  }
  return ClusterPlan{0, V, 0};
}

template <typename Tin, typename Tout>
static occ_status launch_k2(K2Args a, bool vec, cudaStream_t s) {
  const int64_t T = a.T;
  ClusterPlan pl = vec ? plan_cluster(a.V, sizeof(Tin)) : ClusterPlan{0, a.V, 0};
  if (pl.C == 0) {
    const int64_t step = 0x7fffffffLL;
    for (int64_t r0 = 0; r0 < T; r0 += step) {
      a.row0 = r0;
      const unsigned grid = (unsigned)std::min<int64_t>(step, T - r0);
      k2_loss_stream<Tin, Tout, kK2Threads><<<grid, kK2Threads, 0, s>>>(a);
    }
    return check_launch("occ_decoupled_loss_fwd_bwd (stream kernel)");
  }
  auto kern = k2_loss_smem<Tin, Tout, kK2Threads, kK2Unroll>;
  cudaError_t e =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)pl.smem);
  if (e != cudaSuccess)
    return fail(OCC_ERR_CUDA, "cudaFuncSetAttribute(smem=%zu): %s", pl.smem, cudaGetErrorString(e));
  a.S = pl.S;
  const int64_t step = 0x7fffffffLL / pl.C;
  for (int64_t r0 = 0; r0 < T; r0 += step) {
    a.row0 = r0;
    const int64_t rows = std::min<int64_t>(step, T - r0);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(rows * pl.C), 1, 1);
    cfg.blockDim = dim3(kK2Threads, 1, 1);
    cfg.dynamicSmemBytes = pl.smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = pl.C;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pl.C > 1 ? 1 : 0;
    e = cudaLaunchKernelEx(&cfg, kern, a);
    if (e != cudaSuccess)
      return fail(OCC_ERR_CUDA, "k2 cluster launch (C=%d, smem=%zu): %s", pl.C, pl.smem,
                  cudaGetErrorString(e));
  }
  return check_launch("occ_decoupled_loss_fwd_bwd");
}

}  // namespace occ

using namespace occ;

extern "C" size_t occ_loss_workspace_bytes(int64_t T, int64_t V) {
  (void)V;
  return ws_layout(T).total;
}

extern "C" occ_status occ_decoupled_loss_fwd_bwd(
    const void* logits, occ_dtype dt, int64_t T, int64_t V, int64_t ld, const int32_t* ids,
    const float* logp_old, const float* logp_mu, const float* adv, const uint8_t* loss_mask,
    const occ_loss_params* p, float* logp_out, uint8_t* flags_out, void* dlogits,
    int64_t ld_grad, occ_loss_stats* stats, void* workspace, size_t ws_bytes, void* stream) {
  clear_error();
  if (dt != OCC_F32 && dt != OCC_BF16) return fail(OCC_ERR_UNSUPPORTED, "dtype %d", (int)dt);
  if (!p) return fail(OCC_ERR_INVALID_ARG, "params pointer is null");
  if (T < 0 || V < 1 || ld < V)
    return fail(OCC_ERR_INVALID_ARG, "need T >= 0, V >= 1, ld >= V (T=%lld V=%lld ld=%lld)",
                (long long)T, (long long)V, (long long)ld);
  if (!(p->rd_lo >= 0.0) || !(p->rd_hi >= p->rd_lo) || !(p->eps_low >= 0.0) ||
      !(p->eps_low <= 1.0) || !(p->eps_high >= 0.0) || !isfinite(p->grad_scale) ||
      (p->rd_weight != 0 && p->rd_weight != 1) || (p->dlogits_f32 != 0 && p->dlogits_f32 != 1))
    return fail(OCC_ERR_INVALID_ARG,
                "thresholds must satisfy 0 <= rd_lo <= rd_hi, 0 <= eps_low <= 1, eps_high >= 0; "
                "grad_scale finite; rd_weight and dlogits_f32 in {0,1}");
  if (!stats || !aligned(stats, 8)) return fail(OCC_ERR_INVALID_ARG, "stats null or misaligned");
  const WsLayout wl = ws_layout(T);
  if (!workspace || !aligned(workspace, 16) || ws_bytes < wl.total)
    return fail(OCC_ERR_WORKSPACE, "workspace needs %zu bytes, 16-byte aligned (got %zu)",
                wl.total, ws_bytes);
  const size_t es = dtype_size(dt);
  const size_t es_out = p->dlogits_f32 ? 4 : es;
  if (T > 0) {
    if (!logits || !ids || !logp_old || !logp_mu || !adv)
      return fail(OCC_ERR_INVALID_ARG, "null logits/ids/logp_old/logp_mu/adv");
    if (!aligned(logits, es) || !aligned(ids, 4) || !aligned(logp_old, 4) ||
        !aligned(logp_mu, 4) || !aligned(adv, 4) || (logp_out && !aligned(logp_out, 4)))
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
  K2Args a;
  a.logits = logits;
  a.T = T;
  a.V = V;
  a.ld = ld;
  a.S = V;
  a.row0 = 0;
  a.ids = ids;
  a.lp_old = logp_old;
  a.lp_mu = logp_mu;
  a.adv = adv;
  a.mask = loss_mask;
  a.ws_N = (const long long*)(ws + wl.off_N);
  a.ws_loss = (float*)(ws + wl.off_loss);
  a.ws_flags = (uint8_t*)(ws + wl.off_flags);
  a.logp_out = logp_out;
  a.flags_out = flags_out;
  a.dlogits = dlogits;
  a.ld_grad = ld_grad;
  a.kp.log_rd_lo = p->rd_lo > 0.0 ? log(p->rd_lo) : -INFINITY;
  a.kp.log_rd_hi = isinf(p->rd_hi) ? INFINITY : log(p->rd_hi);
  a.kp.log_clip_lo = p->eps_low < 1.0 ? log1p(-p->eps_low) : -INFINITY;
  a.kp.log_clip_hi = log1p(p->eps_high);
  a.kp.clip_lo = (float)(1.0 - p->eps_low);
  a.kp.clip_hi = (float)(1.0 + p->eps_high);
  a.kp.grad_scale = (float)p->grad_scale;
  a.kp.rd_weight = p->rd_weight;
  a.kp.denom = p->denom > 0 ? (long long)p->denom : 0;

  cudaStream_t s = (cudaStream_t)stream;
  if (a.kp.denom == 0) {
    k0_count_valid<kK0Threads><<<1, kK0Threads, 0, s>>>(loss_mask, ids, T, V,
                                                        (long long*)(ws + wl.off_N));
    occ_status st = check_launch("k0_count_valid");
    if (st != OCC_OK) return st;
  }
  if (T > 0) {
    const bool vec = aligned(logits, 16) && ((ld * (int64_t)es) % 16 == 0) &&
                     (!dlogits || (aligned(dlogits, 16) && ((ld_grad * (int64_t)es_out) % 16 == 0)));
    occ_status st;
    if (dt == OCC_BF16)
      st = p->dlogits_f32 ? launch_k2<bf16_t, float>(a, vec, s) : launch_k2<bf16_t, bf16_t>(a, vec, s);
    else
      st = launch_k2<float, float>(a, vec, s);
    if (st != OCC_OK) return st;
  }
  k2_finalize<kFinThreads><<<1, kFinThreads, 0, s>>>(T, a.ws_loss, a.ws_flags, a.ws_N, a.kp.denom,
                                                     stats);
  return check_launch("k2_finalize");
}
