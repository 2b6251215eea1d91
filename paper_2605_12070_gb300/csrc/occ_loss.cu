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
#include <stdlib.h>
#include <string.h>

#include <mutex>
#include <vector>

#include "occ_loss_common.cuh"

namespace occ {

// Backward over one row slice held in shared memory.  dz = -g p_v (+ g at the
// sampled token), with p_v g folded into one exponential: |dz| =
// 2^(z L - cb) where cb = lse L - log2|g|; NEG is the sign of -g.
template <typename Tin, typename Tout, int NT, bool NEG>
__device__ __forceinline__ void backward_slice(const uint4* sv, int64_t nvec, int tail, float xt,
                                               Tout* drow, float cb, float g, int64_t yl) {
  constexpr int VEC = Elem<Tin>::kVec;
#pragma unroll 4
  for (int64_t j = threadIdx.x; j < nvec; j += NT) {
    float x[VEC], d[VEC];
    Elem<Tin>::unpack(sv[j], x);
#pragma unroll
    for (int q = 0; q < VEC; ++q) {
      const float e = ex2_approx(fmaf(x[q], kLog2e, -cb));
      d[q] = NEG ? -e : e;
    }
    if (yl >= j * VEC && yl < (j + 1) * VEC) {
#pragma unroll
      for (int q = 0; q < VEC; ++q)
        if (j * VEC + q == yl) d[q] += g;
    }
    OutVec<Tout, VEC>::store(drow + j * VEC, d);
  }
  if ((int)threadIdx.x < tail) {
    const int64_t q = nvec * VEC + threadIdx.x;
    const float e = ex2_approx(fmaf(xt, kLog2e, -cb));
    float dv = NEG ? -e : e;
    if (q == yl) dv += g;
    out_scalar(drow + q, dv);
  }
}


// Persistent, TMA-pipelined cluster kernel.  Cluster c of the grid handles rows
// c, c + ncl, c + 2 ncl, ...; CTA `rank` of the cluster owns columns
// [rank S, rank S + S).  Thread 0 prefetches the slice of row k + STAGES - 1
// with one cp.async.bulk into a free shared-memory stage while the CTA works
// on row k, so HBM reads of the next rows overlap this row's reduction,
// cluster exchange and dlogits stores.
template <typename Tin, typename Tout, int NT, int STAGES>
__global__ void __launch_bounds__(NT, 2) k2_loss_tma(const K2Args a) {
  constexpr int VEC = Elem<Tin>::kVec;
  constexpr int NW = NT / 32;
  extern __shared__ __align__(128) unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t bars[STAGES];
  __shared__ __align__(16) float4 part[2];  // this CTA's (c, s_hi, s_lo, z_y), by valid-row parity
  __shared__ float red_c[NW];
  __shared__ float2 red_s[NW];
  __shared__ float bc_g, bc_cb;

  const uint32_t C = cluster_nctarank();
  const uint32_t rank = cluster_ctarank();
  const int64_t cid = blockIdx.x / C;
  const int64_t ncl = gridDim.x / C;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const int64_t T = a.T, V = a.V;
  const int64_t v0 = (int64_t)rank * a.S;
  const int64_t n = max((int64_t)0, min(a.S, V - v0));
  const int64_t nvec = n / VEC;
  const uint32_t bulk = (uint32_t)(nvec * 16);
  const int tail = (int)(n - nvec * VEC);
  const size_t stage_bytes = (size_t)a.stage_bytes;
  const Tin* logits = (const Tin*)a.logits;

  if (tid == 0) {
    for (int st = 0; st < STAGES; ++st) mbar_init(&bars[st], 1);
    fence_mbarrier_init();
  }
  __syncthreads();

  auto row_ok = [&](int64_t r) -> bool {
    const int id = a.ids[r];
    return (a.mask == nullptr || a.mask[r] != 0) && id >= 0 && (int64_t)id < V;
  };
  // Producer state, thread 0 only: stages with a copy whose completion thread 0
  // has not observed (pend), the parity each of them completes (ppar), and the
  // parity the next copy into each stage will complete (ipar).
  uint32_t pend = 0, ppar = 0, ipar = 0;
  bool fault = false;
  auto issue = [&](int64_t r, int st) {
    const uint32_t bit = 1u << st;
    fence_proxy_async_smem();
    mbar_arrive_expect_tx(&bars[st], bulk);
    tma_load_1d(smem_raw + (size_t)st * stage_bytes, logits + r * a.ld + v0, bulk, &bars[st]);
    pend |= bit;
    ppar = (ppar & ~bit) | (ipar & bit);
    ipar ^= bit;
  };
  if (tid == 0 && bulk > 0)
    for (int st = 0; st < STAGES - 1; ++st) {
      const int64_t r = cid + (int64_t)st * ncl;
      if (r < T && r != a.lost_copy_row && row_ok(r)) issue(r, st);
    }

  const long long N = a.kp.denom > 0 ? a.kp.denom : *a.ws_N;
  uint32_t phase = 0;  // consumer side: parity of the next completion of each stage
  int64_t nvalid_done = 0;
  int k = 0;
  for (int64_t row = cid; row < T; row += ncl, ++k) {
    const int st = k % STAGES;
    if (tid == 0 && bulk > 0 && !fault) {
      const int64_t r = row + (int64_t)(STAGES - 1) * ncl;
      const int sn = (k + STAGES - 1) % STAGES;
      if (r < T && r != a.lost_copy_row && row_ok(r)) issue(r, sn);
    }
    const int id = a.ids[row];
    const bool m = (a.mask == nullptr) || (a.mask[row] != 0);
    const bool id_ok = id >= 0 && (int64_t)id < V;
    Tout* drow = a.dlogits ? (Tout*)a.dlogits + row * a.ld_grad + v0 : nullptr;
    if (!(m && id_ok)) {  // uniform over the cluster: no barrier is entered
      if (drow) zero_slice_vec<Tout, VEC, NT>(drow, n);
      if (rank == 0 && tid == 0) dropped_token_outputs(a, row, m, id_ok);
      continue;
    }
    float lpo = 0.f, lpm = 0.f, A = 0.f;
    if (tid == 0) {
      lpo = a.lp_old ? a.lp_old[row] : 0.f;
      lpm = a.lp_mu[row];
      A = a.adv[row];
    }
    unsigned char* sp = smem_raw + (size_t)st * stage_bytes;
    if (bulk > 0) {
      const uint32_t par = (phase >> st) & 1u;
      const bool ok = mbar_wait_bounded(&bars[st], par, fault ? 0 : a.wait_ns);
      phase ^= 1u << st;
      if (!ok) fault = true;
      if (tid == 0 && ok) pend &= ~(1u << st);
    }
    // ragged tail of the last slice: plain loads, kept in registers and smem
    const Tin* zs = logits + row * a.ld + v0;
    float xt = 0.f;
    LseAcc acc;
    acc_init(acc);
    if (tid < tail) {
      xt = Elem<Tin>::load(zs + nvec * VEC + tid);
      Elem<Tin>::put(reinterpret_cast<Tin*>(sp) + nvec * VEC + tid, xt);
      float x1[1] = {xt};
      acc_add(acc, x1);
    }
    // forward: online log-sum-exp over the slice in shared memory
    const uint4* sv = reinterpret_cast<const uint4*>(sp);
#pragma unroll 4
    for (int64_t j = tid; j < nvec; j += NT) {
      float x[VEC];
      Elem<Tin>::unpack(sv[j], x);
      acc_add_fast(acc, x);
    }
    // CTA reduction: warp max, one rescale per lane, compensated warp sums
    const float wmax = warp_max(acc.c);
    float2 v = make_float2(acc.c == -INFINITY ? 0.f : acc.s * exp2f(acc.c - wmax), 0.f);
    v = warp_pair_sum(v);
    if (lane == 0) {
      red_c[wid] = wmax;
      red_s[wid] = v;
    }
    __syncthreads();
    const int slot = (int)(nvalid_done & 1);
    if (wid == 0) {
      const float c = lane < NW ? red_c[lane] : -INFINITY;
      const float cm = warp_max(c);
      float2 w = make_float2(0.f, 0.f);
      if (lane < NW && c != -INFINITY) {
        const float f = exp2f(c - cm);
        const float2 p = red_s[lane];
        const float hi = p.x * f;
        w = make_float2(hi, fmaf(p.x, f, -hi) + p.y * f);
      }
      w = warp_pair_sum(w);
      if (lane == 0) {
        const int64_t yl = (int64_t)id - v0;
        float zy = 0.f;
        if (yl >= 0 && yl < n) {
          if (sizeof(Tin) == 2)
            zy = __uint_as_float(((uint32_t)reinterpret_cast<const uint16_t*>(sp)[yl]) << 16);
          else
            zy = reinterpret_cast<const float*>(sp)[yl];
        }
        part[slot] = make_float4(cm, w.x, w.y, zy);
      }
    }
    // exchange the C partials (cluster barrier; a CTA barrier when C = 1)
    if (C > 1) {
      cluster_arrive_release();
      cluster_wait_acquire();
    } else {
      __syncthreads();
    }
    if (wid == 0) {
      float4 P = make_float4(-INFINITY, 0.f, 0.f, 0.f);
      if (lane < (int)C) P = (C > 1) ? ld_dsmem_f4(&part[slot], (uint32_t)lane) : part[slot];
      const float cm = warp_max(P.x);
      float2 w = make_float2(0.f, 0.f);
      if (lane < (int)C && P.x != -INFINITY) {
        const float f = exp2f(P.x - cm);
        const float hi = P.y * f;
        w = make_float2(hi, fmaf(P.y, f, -hi) + P.z * f);
      }
      w = warp_pair_sum(w);
      const float zy = __shfl_sync(0xffffffffu, P.w, (int)((int64_t)id / a.S));
      if (lane == 0) {
        const double lse = lse_from(cm, w);
        float g, loss_t, logp_f;
        uint32_t fl;
        token_math(a.kp, lse, zy, lpo, lpm, A, N, g, loss_t, fl, logp_f);
        float cb = 0.f;
        if (g != 0.f) {
          int e;
          const float fm = frexpf(fabsf(g), &e);  // |g| = fm 2^e
          cb = (float)(lse * (double)kLog2e - (double)e - (double)log2f(fm));
        }
        bc_g = g;
        bc_cb = cb;
        if (rank == 0) {
          a.ws_loss[row] = loss_t;
          a.ws_flags[row] = (uint8_t)fl;
          if (a.logp_out) a.logp_out[row] = logp_f;
          if (a.flags_out) a.flags_out[row] = (uint8_t)fl;
        }
      }
    }
    __syncthreads();
    if (drow) {
      const float g = bc_g;
      if (g == 0.f) {
        zero_slice_vec<Tout, VEC, NT>(drow, n);
      } else if (g > 0.f) {
        backward_slice<Tin, Tout, NT, true>(sv, nvec, tail, xt, drow, bc_cb, g, (int64_t)id - v0);
      } else {
        backward_slice<Tin, Tout, NT, false>(sv, nvec, tail, xt, drow, bc_cb, g, (int64_t)id - v0);
      }
    }
    __syncthreads();  // stage st and the broadcast slots are free again
    ++nvalid_done;
  }
  if (C > 1) {  // no CTA leaves while a peer may still read its partials
    cluster_arrive_release();
    cluster_wait_acquire();
  }
  if (tid == 0) {
    if (fault) atomicOr(a.ws_err, OCC_DATA_ERR_TIMEOUT);
    // copies still in flight (only after a timeout): wait, bounded, before exiting
    for (int st = 0; st < STAGES; ++st)
      if (pend & (1u << st)) {
        if (!mbar_wait_bounded(&bars[st], (ppar >> st) & 1u, a.wait_ns))
          atomicOr(a.ws_err, OCC_DATA_ERR_TIMEOUT);
      }
  }
}

// Packed bf16 max of the eight values of a 16-byte vector, as a float.
__device__ __forceinline__ uint32_t bf16x2_max(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("max.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}
template <typename Tin>
struct VecMax;
template <>
struct VecMax<bf16_t> {
  __device__ __forceinline__ static float of(const uint4& r) {
    const uint32_t m = bf16x2_max(bf16x2_max(r.x, r.y), bf16x2_max(r.z, r.w));
    return fmaxf(bf16_lo(m), bf16_hi(m));
  }
};
template <>
struct VecMax<float> {
  __device__ __forceinline__ static float of(const uint4& r) {
    return fmaxf(fmaxf(__uint_as_float(r.x), __uint_as_float(r.y)),
                 fmaxf(__uint_as_float(r.z), __uint_as_float(r.w)));
  }
};

// Register-resident persistent kernel for rows whose CTA slice fits EV
// vectors per thread.  The forward pass keeps every term e_v = 2^(z_v L - c)
// of the thread's share of the slice in registers (c = the thread's own
// maximum, so e_v <= 1), which makes the backward a multiplication:
//   dz_v = k e_v (+ g at the sampled token),  k = -g 2^(c - lse L),
// one exponential per element for forward and backward together.  The
// shared-memory stage only lands the TMA copy and is handed back to the
// prefetcher as soon as the forward pass has read it.
template <typename Tin, typename Tout, int NT, int EV, int STAGES>
__global__ void __launch_bounds__(NT, 2) k2_loss_reg(const K2Args a) {
  constexpr int VEC = Elem<Tin>::kVec;
  constexpr int NW = NT / 32;
  extern __shared__ __align__(128) unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t bars[STAGES];
  __shared__ __align__(16) float4 part[2];  // (c, s_hi, s_lo, z_y) by valid-row parity
  __shared__ float red_c[NW];
  __shared__ float2 red_s[NW];
  __shared__ float bc_g, zy_sh;
  __shared__ double bc_lseL;

  const uint32_t C = cluster_nctarank();
  const uint32_t rank = cluster_ctarank();
  const int64_t cid = blockIdx.x / C;
  const int64_t ncl = gridDim.x / C;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const int64_t T = a.T, V = a.V;
  const int64_t v0 = (int64_t)rank * a.S;
  const int64_t n = max((int64_t)0, min(a.S, V - v0));
  const int64_t nvec = n / VEC;
  const uint32_t bulk = (uint32_t)(nvec * 16);
  const int tail = (int)(n - nvec * VEC);
  const size_t stage_bytes = (size_t)a.stage_bytes;
  const Tin* logits = (const Tin*)a.logits;

  if (tid == 0) {
    for (int st = 0; st < STAGES; ++st) mbar_init(&bars[st], 1);
    fence_mbarrier_init();
  }
  __syncthreads();

  auto row_ok = [&](int64_t r) -> bool {
    const int id = a.ids[r];
    return (a.mask == nullptr || a.mask[r] != 0) && id >= 0 && (int64_t)id < V;
  };
  uint32_t pend = 0, ppar = 0, ipar = 0;  // producer bookkeeping (thread 0)
  bool fault = false;
  auto issue = [&](int64_t r, int st) {
    const uint32_t bit = 1u << st;
    fence_proxy_async_smem();
    mbar_arrive_expect_tx(&bars[st], bulk);
    tma_load_1d(smem_raw + (size_t)st * stage_bytes, logits + r * a.ld + v0, bulk, &bars[st]);
    pend |= bit;
    ppar = (ppar & ~bit) | (ipar & bit);
    ipar ^= bit;
  };
  // refill stage st with the row STAGES iterations ahead (thread 0)
  auto refill = [&](int64_t row, int st) {
    if (tid == 0 && bulk > 0 && !fault) {
      const int64_t r = row + (int64_t)STAGES * ncl;
      if (r < T && r != a.lost_copy_row && row_ok(r)) issue(r, st);
    }
  };
  if (tid == 0 && bulk > 0)
    for (int st = 0; st < STAGES; ++st) {
      const int64_t r = cid + (int64_t)st * ncl;
      if (r < T && r != a.lost_copy_row && row_ok(r)) issue(r, st);
    }

  const long long N = a.kp.denom > 0 ? a.kp.denom : *a.ws_N;
  uint32_t phase = 0;
  int64_t nvalid_done = 0;
  int k = 0;
  for (int64_t row = cid; row < T; row += ncl, ++k) {
    const int st = k % STAGES;
    const int id = a.ids[row];
    const bool m = (a.mask == nullptr) || (a.mask[row] != 0);
    const bool id_ok = id >= 0 && (int64_t)id < V;
    Tout* drow = a.dlogits ? (Tout*)a.dlogits + row * a.ld_grad + v0 : nullptr;
    if (!(m && id_ok)) {  // uniform over the cluster: no barrier is entered
      refill(row, st);
      if (drow) zero_slice_vec<Tout, VEC, NT>(drow, n);
      if (rank == 0 && tid == 0) dropped_token_outputs(a, row, m, id_ok);
      continue;
    }
    float lpo = 0.f, lpm = 0.f, A = 0.f;
    if (tid == 0) {
      lpo = a.lp_old ? a.lp_old[row] : 0.f;
      lpm = a.lp_mu[row];
      A = a.adv[row];
    }
    const unsigned char* sp = smem_raw + (size_t)st * stage_bytes;
    if (bulk > 0) {
      const bool ok = mbar_wait_bounded(&bars[st], (phase >> st) & 1u, fault ? 0 : a.wait_ns);
      phase ^= 1u << st;
      if (!ok) fault = true;
      if (tid == 0 && ok) pend &= ~(1u << st);
    }
    const int64_t yl = (int64_t)id - v0;  // sampled token in slice coordinates
    float xt = -INFINITY;
    if (tid < tail) xt = Elem<Tin>::load(logits + row * a.ld + v0 + nvec * VEC + tid);
    // pass 1: the thread's maximum
    const uint4* sv = reinterpret_cast<const uint4*>(sp);
    float mx = xt;
#pragma unroll
    for (int e = 0; e < EV; ++e) {
      const int64_t j = tid + (int64_t)e * NT;
      if (j < nvec) mx = fmaxf(mx, VecMax<Tin>::of(sv[j]));
    }
    const float c = mx * kLog2e;  // -inf when the thread holds nothing finite
    // pass 2: terms e_v = 2^(z_v L - c) kept in registers
    float E[EV][VEC];
    float s = 0.f, et = 0.f;
    if (c != -INFINITY) {
#pragma unroll
      for (int e = 0; e < EV; ++e) {
        const int64_t j = tid + (int64_t)e * NT;
        if (j < nvec) {
          float x[VEC];
          Elem<Tin>::unpack(sv[j], x);
          float t = 0.f;
#pragma unroll
          for (int q = 0; q < VEC; ++q) {
            E[e][q] = ex2_approx(fmaf(x[q], kLog2e, -c));
            t += E[e][q];
          }
          s += t;
          if (yl >= j * VEC && yl < (j + 1) * VEC) {
#pragma unroll
            for (int q = 0; q < VEC; ++q)
              if (j * VEC + q == yl) zy_sh = x[q];
          }
        }
      }
      if (tid < tail) {
        et = ex2_approx(fmaf(xt, kLog2e, -c));
        s += et;
      }
    } else {
#pragma unroll
      for (int e = 0; e < EV; ++e)
#pragma unroll
        for (int q = 0; q < VEC; ++q) E[e][q] = 0.f;
    }
    if (tid < tail && nvec * VEC + tid == yl) zy_sh = xt;
    // CTA reduction: warp max, one rescale per lane, compensated warp sums
    const float wmax = warp_max(c);
    float2 v = make_float2(c == -INFINITY ? 0.f : s * exp2f(c - wmax), 0.f);
    v = warp_pair_sum(v);
    if (lane == 0) {
      red_c[wid] = wmax;
      red_s[wid] = v;
    }
    __syncthreads();   // the stage has been read: hand it to the prefetcher
    refill(row, st);
    const int slot = (int)(nvalid_done & 1);
    if (wid == 0) {
      const float cw = lane < NW ? red_c[lane] : -INFINITY;
      const float cm = warp_max(cw);
      float2 w = make_float2(0.f, 0.f);
      if (lane < NW && cw != -INFINITY) {
        const float f = exp2f(cw - cm);
        const float2 p = red_s[lane];
        const float hi = p.x * f;
        w = make_float2(hi, fmaf(p.x, f, -hi) + p.y * f);
      }
      w = warp_pair_sum(w);
      if (lane == 0) part[slot] = make_float4(cm, w.x, w.y, (yl >= 0 && yl < n) ? zy_sh : 0.f);
    }
    if (C > 1) {
      cluster_arrive_release();
      cluster_wait_acquire();
    } else {
      __syncthreads();
    }
    if (wid == 0) {
      float4 P = make_float4(-INFINITY, 0.f, 0.f, 0.f);
      if (lane < (int)C) P = (C > 1) ? ld_dsmem_f4(&part[slot], (uint32_t)lane) : part[slot];
      const float cm = warp_max(P.x);
      float2 w = make_float2(0.f, 0.f);
      if (lane < (int)C && P.x != -INFINITY) {
        const float f = exp2f(P.x - cm);
        const float hi = P.y * f;
        w = make_float2(hi, fmaf(P.y, f, -hi) + P.z * f);
      }
      w = warp_pair_sum(w);
      const float zy = __shfl_sync(0xffffffffu, P.w, (int)((int64_t)id / a.S));
      if (lane == 0) {
        const double lse = lse_from(cm, w);
        float g, loss_t, logp_f;
        uint32_t fl;
        token_math(a.kp, lse, zy, lpo, lpm, A, N, g, loss_t, fl, logp_f);
        bc_g = g;
        bc_lseL = lse * (double)kLog2e;
        if (rank == 0) {
          a.ws_loss[row] = loss_t;
          a.ws_flags[row] = (uint8_t)fl;
          if (a.logp_out) a.logp_out[row] = logp_f;
          if (a.flags_out) a.flags_out[row] = (uint8_t)fl;
        }
      }
    }
    __syncthreads();
    if (drow) {
      const float g = bc_g;
      if (g == 0.f) {
        zero_slice_vec<Tout, VEC, NT>(drow, n);
      } else {
        const float kf = c == -INFINITY ? 0.f : -g * exp2f((float)((double)c - bc_lseL));
#pragma unroll
        for (int e = 0; e < EV; ++e) {
          const int64_t j = tid + (int64_t)e * NT;
          if (j < nvec) {
            float d[VEC];
#pragma unroll
            for (int q = 0; q < VEC; ++q) d[q] = kf * E[e][q];
            if (yl >= j * VEC && yl < (j + 1) * VEC) {
#pragma unroll
              for (int q = 0; q < VEC; ++q)
                if (j * VEC + q == yl) d[q] += g;
            }
            OutVec<Tout, VEC>::store(drow + j * VEC, d);
          }
        }
        if (tid < tail) {
          const int64_t q = nvec * VEC + tid;
          float dv = kf * et;
          if (q == yl) dv += g;
          out_scalar(drow + q, dv);
        }
      }
    }
    ++nvalid_done;
  }
  if (C > 1) {  // no CTA leaves while a peer may still read its partials
    cluster_arrive_release();
    cluster_wait_acquire();
  }
  if (tid == 0) {
    if (fault) atomicOr(a.ws_err, OCC_DATA_ERR_TIMEOUT);
    for (int st = 0; st < STAGES; ++st)
      if (pend & (1u << st)) {
        if (!mbar_wait_bounded(&bars[st], (ppar >> st) & 1u, a.wait_ns))
          atomicOr(a.ws_err, OCC_DATA_ERR_TIMEOUT);
      }
  }
}

// One CTA per row, two streaming passes (the K1 layout), with the head of the
// row kept in shared memory.  The forward pass reads the row from HBM once:
// its first `head` vectors are also stored in shared memory, the rest is read
// with an L2 evict-last policy.  The backward pass takes the head from shared
// memory and re-reads only the remainder, oldest data first and with an
// evict-first policy (its last use), so the re-read is served by L2 and HBM
// sees the logits once and dlogits once.  Oldest-first bounds the time a line
// waits in L2 by the longer of the two passes (newest-first lets the first
// lines wait through both).  dlogits are written evict-first.
template <typename Tin, typename Tout, int NT, int U, bool PEEL>
__global__ void __launch_bounds__(NT, 1024 / NT) k2_loss_l2(const K2Args a) {
  constexpr int VEC = Elem<Tin>::kVec;
  extern __shared__ __align__(16) uint4 head_sm[];
  __shared__ RedScratch red;
  __shared__ float bc_g, bc_cb;
  const uint64_t keep = l2_policy_evict_last();
  const uint64_t last = l2_policy_evict_first();
  const int tid = threadIdx.x;
  const int64_t V = a.V;
  const long long N = a.kp.denom > 0 ? a.kp.denom : *a.ws_N;
  for (int64_t row = a.row0 + blockIdx.x; row < a.T; row += gridDim.x) {
    const int id = a.ids[row];
    const bool m = (a.mask == nullptr) || (a.mask[row] != 0);
    const bool id_ok = id >= 0 && (int64_t)id < V;
    // PEEL: the row's first `lead` elements (up to its 16-byte boundary) are
    // scalar; the gradient row has the same byte offset (checked on the host)
    const Tin* z0 = (const Tin*)a.logits + row * a.ld;
    const int64_t lead =
        PEEL ? min(V, (int64_t)(((16 - ((uintptr_t)z0 & 15)) & 15) / sizeof(Tin))) : 0;
    const Tin* z = z0 + lead;
    const int64_t nvec = (V - lead) / VEC;
    const int64_t tail0 = nvec * VEC;  // relative to z
    const int64_t ntail = V - lead - tail0;
    const int64_t head = min(nvec, (int64_t)(a.stage_bytes / 16));  // vectors kept on chip
    const int idr = id - (int)lead;  // the sampled token relative to z
    Tout* drow0 = a.dlogits ? (Tout*)a.dlogits + row * a.ld_grad : nullptr;
    Tout* drow = drow0 ? drow0 + lead : nullptr;
    if (!(m && id_ok)) {
      if (drow) {
        for (int64_t i = tid; i < nvec; i += NT) OutVecHint<Tout, VEC>::zero(drow + i * VEC, last);
        if ((int64_t)tid < ntail) out_scalar(drow + tail0 + tid, 0.f);
        if (PEEL && (int64_t)tid < lead) out_scalar(drow0 + tid, 0.f);
      }
      if (tid == 0) dropped_token_outputs(a, row, m, id_ok);
      continue;
    }
    float zy = 0.f, lpo = 0.f, lpm = 0.f, A = 0.f;
    if (tid == 0) {
      zy = Elem<Tin>::load(z0 + id);
      lpo = a.lp_old ? a.lp_old[row] : 0.f;
      lpm = a.lp_mu[row];
      A = a.adv[row];
    }
    const uint4* zv = reinterpret_cast<const uint4*>(z);
    LseAcc acc;
    acc_init(acc);
    // Row walk (GB300, bf16, against one load at a time in the last round):
    // clamped rounds in the 128- and 512-thread tiers (V = 151936: 6.31 -> 5.93
    // ms; 32000: 1.48 -> 1.37 ms; 24000: 1.34 -> 1.18 ms), one load at a time
    // in the 256-thread tier (V = 50000: 1.30 against 1.33 ms) and for peeled
    // rows (V = 50257: 1.32 against 1.35 ms).
    constexpr Walk kW = (PEEL || NT == 256) ? Walk::kSerialTail : Walk::kClampAll;
    const int nh = (int)head;
    walk_row<kW, U, NT>(
        tid, (int)nvec, [&](int j) { return ld_hint_v4(zv + j, keep); },
        [&](int j, const uint4& r) {
          if (j < nh) head_sm[j] = r;
          float x[VEC];
          Elem<Tin>::unpack(r, x);
          acc_add_fast(acc, x);
        });
    float xt = 0.f, xp = 0.f;
    if ((int64_t)tid < ntail) {
      xt = Elem<Tin>::load(z + tail0 + tid);
      float x1[1] = {xt};
      acc_add(acc, x1);
    }
    if (PEEL && (int64_t)tid < lead) {
      xp = Elem<Tin>::load(z0 + tid);
      float x1[1] = {xp};
      acc_add(acc, x1);
    }
    float Cr;
    float2 Sr;
    block_lse<NT>(acc, red, Cr, Sr);
    if (tid == 0) {
      const double lse = lse_from(Cr, Sr);
      float g, loss_t, logp_f;
      uint32_t fl;
      token_math(a.kp, lse, zy, lpo, lpm, A, N, g, loss_t, fl, logp_f);
      float cb = 0.f;
      if (g != 0.f) {
        int e;
        const float fm = frexpf(fabsf(g), &e);
        cb = (float)(lse * (double)kLog2e - (double)e - (double)log2f(fm));
      }
      bc_g = g;
      bc_cb = cb;
      a.ws_loss[row] = loss_t;
      a.ws_flags[row] = (uint8_t)fl;
      if (a.logp_out) a.logp_out[row] = logp_f;
      if (a.flags_out) a.flags_out[row] = (uint8_t)fl;
    }
    __syncthreads();
    if (drow) {
      const float g = bc_g, cb = bc_cb;
      if (g == 0.f) {
        for (int64_t j = tid; j < nvec; j += NT) OutVecHint<Tout, VEC>::zero(drow + j * VEC, last);
        if ((int64_t)tid < ntail) out_scalar(drow + tail0 + tid, 0.f);
        if (PEEL && (int64_t)tid < lead) out_scalar(drow0 + tid, 0.f);
      } else {
        const float sgn = g > 0.f ? -1.f : 1.f;
        auto emit = [&](int64_t jj, const uint4& r) {
          float x[VEC], d[VEC];
          Elem<Tin>::unpack(r, x);
#pragma unroll
          for (int q = 0; q < VEC; ++q) d[q] = sgn * ex2_approx(fmaf(x[q], kLog2e, -cb));
          if (idr >= jj * VEC && idr < (jj + 1) * VEC) {
#pragma unroll
            for (int q = 0; q < VEC; ++q)
              if (jj * VEC + q == idr) d[q] += g;
          }
          OutVecHint<Tout, VEC>::store(drow + jj * VEC, d, last);
        };
        // re-read part, oldest first: vectors head+tid, head+tid+NT, ... < nvec
        const int64_t nre = nvec - head;
        const uint4* zr = zv + head;
        walk_row<kW, U, NT>(
            tid, (int)nre, [&](int j) { return ld_hint_v4(zr + j, last); },
            [&](int j, const uint4& r) { emit(head + j, r); });
        // on-chip head
#pragma unroll 4
        for (int64_t j = tid; j < head; j += NT) emit(j, head_sm[j]);
        if ((int64_t)tid < ntail) {
          float dv = sgn * ex2_approx(fmaf(xt, kLog2e, -cb));
          if (tail0 + tid == idr) dv += g;
          out_scalar(drow + tail0 + tid, dv);
        }
        if (PEEL && (int64_t)tid < lead) {
          float dv = sgn * ex2_approx(fmaf(xp, kLog2e, -cb));
          if (tid == id) dv += g;
          out_scalar(drow0 + tid, dv);
        }
      }
    }
    __syncthreads();
  }
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
    lpo = a.lp_old ? a.lp_old[row] : 0.f;
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

struct ClusterPlan {
  int C;               // CTAs per row (0: use the streaming kernel)
  int64_t S;           // elements per CTA slice (multiple of the vector width)
  size_t stage_bytes;  // one pipeline stage, rounded to 128 bytes
};

constexpr int kK2Stages = 2;
constexpr size_t kSmemTarget = 80 * 1024;   // two CTAs per SM
constexpr size_t kSmemMax = 200 * 1024;     // one CTA per SM

static ClusterPlan plan_cluster(int64_t V, size_t es, int stages) {
  const int64_t vec = 16 / (int64_t)es;
  for (size_t cap : {kSmemTarget, kSmemMax}) {
    for (int C : {1, 2, 4, 8}) {
      int64_t S = (V + C - 1) / C;
      S = (S + vec - 1) / vec * vec;
      const size_t sb = align_up((size_t)S * es, 128);
      if (sb * stages <= cap) return ClusterPlan{C, S, sb};
    }
  }
  return ClusterPlan{0, V, 0};
}

// Co-resident clusters for a kernel configuration (cached per device).
static int max_active_clusters(const void* kern, int C, int NT, size_t smem) {
  struct Key {
    const void* k;
    int C, NT, dev;
    size_t smem;
    int n;
  };
  static std::mutex mu;
  static std::vector<Key> cache;
  int dev = 0;
  cudaGetDevice(&dev);
  std::lock_guard<std::mutex> lk(mu);
  for (const Key& e : cache)
    if (e.k == kern && e.C == C && e.NT == NT && e.dev == dev && e.smem == smem) return e.n;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(C, 1, 1);
  cfg.blockDim = dim3(NT, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) {
    cudaGetLastError();
    n = 0;
  }
  cache.push_back(Key{kern, C, NT, dev, smem, n});
  return n;
}

template <typename Kern>
static occ_status launch_persistent(Kern kern, int NT, K2Args a, const ClusterPlan& pl, int stages,
                                    cudaStream_t s) {
  // Test hooks of the bounded waits: OCC_TEST_LOST_COPY_ROW makes the producer
  // skip one row's copy so that its consumers' wait runs out (after
  // OCC_TEST_WAIT_TIMEOUT_NS); the kernel then reports OCC_DATA_ERR_TIMEOUT.
  if (const char* e = getenv("OCC_TEST_LOST_COPY_ROW")) a.lost_copy_row = atoll(e);
  if (const char* e = getenv("OCC_TEST_WAIT_TIMEOUT_NS")) a.wait_ns = strtoull(e, nullptr, 10);
  const size_t smem = (size_t)stages * pl.stage_bytes;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess)
    return fail(OCC_ERR_CUDA, "cudaFuncSetAttribute(smem=%zu): %s", smem, cudaGetErrorString(e));
  int ncl = max_active_clusters((const void*)kern, pl.C, NT, smem);
  if (ncl <= 0)
    return fail(OCC_ERR_CUDA, "no co-resident cluster of %d CTAs with %zu bytes of shared memory",
                pl.C, smem);
  ncl = (int)std::min<int64_t>(ncl, a.T);
  a.S = pl.S;
  a.stage_bytes = (int64_t)pl.stage_bytes;
  a.row0 = 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(ncl * pl.C), 1, 1);
  cfg.blockDim = dim3(NT, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = pl.C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, kern, a);
  if (e != cudaSuccess)
    return fail(OCC_ERR_CUDA, "k2 launch (clusters=%d x %d CTAs, smem=%zu): %s", ncl, pl.C, smem,
                cudaGetErrorString(e));
  return check_launch("occ_decoupled_loss_fwd_bwd");
}

// Register-resident kernel geometry: 256 threads, 80 float registers of terms
// per thread, so a CTA slice holds at most 20480 elements.
constexpr int kRegThreads = 256;
constexpr int64_t kRegSliceElems = 20480;

static ClusterPlan plan_reg(int64_t V, size_t es, int stages) {
  const int64_t vec = 16 / (int64_t)es;
  for (int C : {1, 2, 4, 8}) {
    int64_t S = (V + C - 1) / C;
    S = (S + vec - 1) / vec * vec;
    const size_t sb = align_up((size_t)S * es, 128);
    if (S <= kRegSliceElems && sb * stages <= kSmemMax) return ClusterPlan{C, S, sb};
  }
  return ClusterPlan{0, V, 0};
}

// Threads per CTA of the TMA kernel (OCC_K2_THREADS=256|512 overrides, for tuning).
static int k2_threads() {
  static int nt = [] {
    const char* v = getenv("OCC_K2_THREADS");
    return (v && atoi(v) == 512) ? 512 : 256;
  }();
  return nt;
}

// Kernel variant for aligned rows: "l2" (default), "l2_1024", "reg" or "tma"
// (OCC_K2_VARIANT overrides, for tuning).
static int k2_variant() {
  static int v = [] {
    const char* e = getenv("OCC_K2_VARIANT");
    if (e && !strcmp(e, "reg")) return 1;
    if (e && !strcmp(e, "tma")) return 2;
    if (e && !strcmp(e, "l2_1024")) return 3;
    return 0;
  }();
  return v;
}

using K2Kern = void (*)(const K2Args);

template <typename Tin, typename Tout, bool PEEL>
static K2Kern l2_kernel(int var, int nt, int unroll) {
  return (var == 3)      ? k2_loss_l2<Tin, Tout, 1024, 8, PEEL>
         : (nt == 128)   ? k2_loss_l2<Tin, Tout, 128, 8, PEEL>
         : (nt == 256)   ? k2_loss_l2<Tin, Tout, 256, 8, PEEL>
         : (unroll == 4) ? k2_loss_l2<Tin, Tout, 512, 4, PEEL>
                         : k2_loss_l2<Tin, Tout, 512, 8, PEEL>;
}

// Rows that are not 16-byte aligned can run the vector kernel peeled when the
// gradient rows sit at the same byte offsets as the logits rows (same element
// size, base addresses and row strides congruent modulo 16 bytes) and a row
// holds at least a few vectors.  Only the same-size instantiations exist.
template <typename Tin, typename Tout>
static bool k2_peel_ok(const K2Args& a) {
  const int64_t es = (int64_t)sizeof(Tin);
  if (sizeof(Tout) != sizeof(Tin)) return false;
  if (a.V < 16 * Elem<Tin>::kVec || ((uintptr_t)a.logits % es) != 0) return false;
  if (!a.dlogits) return true;
  return (((uintptr_t)a.dlogits - (uintptr_t)a.logits) % 16) == 0 &&
         (((a.ld_grad - a.ld) * es) % 16) == 0;
}

template <typename Tin, typename Tout>
static occ_status launch_k2(K2Args a, bool vec, cudaStream_t s) {
  const int64_t T = a.T;
  const bool peel = !vec && k2_peel_ok<Tin, Tout>(a);
  if (vec || peel) {
    const int var = vec ? k2_variant() : 0;  // the cluster variants need aligned rows
    if (var == 1) {
      const ClusterPlan pr = plan_reg(a.V, sizeof(Tin), kK2Stages);
      if (pr.C > 0) {
        note_kernel("k2_loss_reg");
        constexpr int EV = (int)(kRegSliceElems / kRegThreads / Elem<Tin>::kVec);
        return launch_persistent(k2_loss_reg<Tin, Tout, kRegThreads, EV, kK2Stages>, kRegThreads,
                                 a, pr, kK2Stages, s);
      }
    }
    if (var == 2) {
      const ClusterPlan pl = plan_cluster(a.V, sizeof(Tin), kK2Stages);
      if (pl.C > 0) {
        note_kernel("k2_loss_tma");
        if (k2_threads() == 512)
          return launch_persistent(k2_loss_tma<Tin, Tout, 512, kK2Stages>, 512, a, pl, kK2Stages,
                                   s);
        return launch_persistent(k2_loss_tma<Tin, Tout, 256, kK2Stages>, 256, a, pl, kK2Stages, s);
      }
    }
    // Row-size tiers (measured on GB300, V = 32000 to 151936 bf16): 128 threads
    // and a 16 KB head up to 64 KB rows, 256 threads and no head up to 112 KB,
    // 512 threads beyond, with the largest head that keeps two CTAs in the
    // 164 KB shared-memory carveout (80 KB for this kernel).  OCC_K2_L2_THREADS and
    // OCC_K2_HEAD_KB override (0 = pure L2 re-read).
    const size_t row_bytes = (size_t)(a.V / Elem<Tin>::kVec) * 16;
    const int nt_auto = row_bytes <= 64 * 1024 ? 128 : row_bytes <= 112 * 1024 ? 256 : 512;
    static const long head_env = [] {
      const char* e = getenv("OCC_K2_HEAD_KB");
      return e ? atol(e) * 1024 : -1L;
    }();
    static const int unroll = [] {
      const char* e = getenv("OCC_K2_UNROLL");
      return e ? atoi(e) : 8;
    }();
    static const int nt_env = [] {
      const char* e = getenv("OCC_K2_L2_THREADS");
      return e ? atoi(e) : 0;
    }();
    const int nt_small = nt_env ? nt_env : nt_auto;
    K2Kern kern = l2_kernel<Tin, Tout, false>(var, nt_small, unroll);
    if constexpr (sizeof(Tin) == sizeof(Tout))
      if (peel) kern = l2_kernel<Tin, Tout, true>(var, nt_small, unroll);
    const size_t head_auto = nt_auto == 128   ? 16 * 1024
                             : nt_auto == 256 ? 0
                                              : two_cta_smem_budget((const void*)kern);
    const size_t head_bytes =
        std::min(head_env >= 0 ? (size_t)head_env : head_auto, row_bytes);
    a.stage_bytes = (int64_t)head_bytes;
    const int nt = (var == 3) ? 1024 : (nt_small == 128 || nt_small == 256) ? nt_small : 512;
    if (head_bytes > 0) {
      cudaError_t e =
          cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)head_bytes);
      if (e != cudaSuccess)
        return fail(OCC_ERR_CUDA, "cudaFuncSetAttribute(smem=%zu): %s", head_bytes,
                    cudaGetErrorString(e));
    }
    note_kernel(peel ? "k2_loss_l2/peel" : "k2_loss_l2");
    const int64_t step = 0x7fffffffLL;
    for (int64_t r0 = 0; r0 < T; r0 += step) {
      a.row0 = r0;
      const unsigned grid = (unsigned)std::min<int64_t>(step, T - r0);
      kern<<<grid, nt, head_bytes, s>>>(a);
    }
    return check_launch("occ_decoupled_loss_fwd_bwd");
  }
  note_kernel("k2_loss_stream");
  const int64_t step = 0x7fffffffLL;
  for (int64_t r0 = 0; r0 < T; r0 += step) {
    a.row0 = r0;
    const unsigned grid = (unsigned)std::min<int64_t>(step, T - r0);
    k2_loss_stream<Tin, Tout, kK2Threads><<<grid, kK2Threads, 0, s>>>(a);
  }
  return check_launch("occ_decoupled_loss_fwd_bwd (stream kernel)");
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
  K2Args a;
  bool vec = false;
  occ_status st = prepare_loss_args(logits, dt, T, V, ld, ids, logp_mu, adv, loss_mask, p,
                                    logp_out, flags_out, dlogits, ld_grad, stats, workspace,
                                    ws_bytes, a, vec);
  if (st != OCC_OK) return st;
  if (T > 0 && p->proxy == OCC_PROXY_NONE && !logp_old)
    return fail(OCC_ERR_INVALID_ARG, "logp_old is null (and no proxy selected)");
  if (logp_old && !aligned(logp_old, 4)) return fail(OCC_ERR_MISALIGNED, "logp_old misaligned");
  a.lp_old = logp_old;
  cudaStream_t s = (cudaStream_t)stream;
  st = launch_k0(a, s);
  if (st != OCC_OK) return st;
  if (T > 0) {
    if (dt == OCC_BF16)
      st = p->dlogits_f32 ? launch_k2<bf16_t, float>(a, vec, s) : launch_k2<bf16_t, bf16_t>(a, vec, s);
    else
      st = launch_k2<float, float>(a, vec, s);
    if (st != OCC_OK) return st;
  }
  return launch_finalize(a, stats, s);
}
