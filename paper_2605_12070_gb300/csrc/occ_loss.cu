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
// Kernel layout (vector path): one CTA per row and two passes over it.  The
// forward pass streams the row from HBM once with 16-byte loads, keeps its
// first part in shared memory and leaves the rest in L2 (evict-last); after
// the CTA reduction and the token's scalars, the backward pass turns the
// shared-memory part and the L2 re-read of the rest into dlogits.  So HBM
// sees the logits once and dlogits once: V * sizeof(T) read per valid token
// plus V * sizeof(T_out) written per token (a dropped token is not read).
// Rows long enough for it keep another part in tensor memory (the tier of
// occ_common.cuh), which shrinks the re-read that the dirty dlogits lines in
// L2 would otherwise push out.  A scalar-load two-pass kernel handles rows
// that cannot be vectorised.
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

// One CTA per row, two streaming passes (the K1 layout), with the head of the
// row kept in shared memory.  The forward pass reads the row from HBM once:
// its first `head` vectors are also stored in shared memory, the rest is read
// with an L2 evict-last policy.  The backward pass takes the head from shared
// memory and re-reads only the remainder, oldest data first and with an
// evict-first policy (its last use), so the re-read is served by L2 and HBM
// sees the logits once and dlogits once.  Oldest-first bounds the time a line
// waits in L2 by the longer of the two passes (newest-first lets the first
// lines wait through both).  dlogits are written evict-first.
//
// TM: the tensor-memory tier of occ_common.cuh keeps 16 more blocks of NT
// vectors of the row on chip (128 KB at 512 threads, 64 KB at 256, 32 KB at
// 128), and the kernel runs persistent, 1024 / NT CTAs per SM fetching rows
// from the workspace's counter.
template <typename Tin, typename Tout, int NT, int U, bool PEEL, bool TM = false>
__global__ void __launch_bounds__(NT, 1024 / NT) k2_loss_l2(const K2Args a) {
  static_assert(!TM || NT == kTmThreads || NT == 256 || NT == 128, "the tensor-memory tier");
  // head blocks before the tensor-memory part: 72 KB at 512 threads, none at 256 and 16 KB at
  // 128 (as the plain kernel)
  constexpr int kHB = NT == kTmThreads ? kTmHeadBlocks : NT == 256 ? 0 : 8;
  constexpr int VEC = Elem<Tin>::kVec;
  extern __shared__ __align__(16) uint4 head_sm[];
  __shared__ RedScratch red;
  __shared__ float bc_g, bc_cb;
  __shared__ uint32_t tmem_sm;  // TM: the CTA's tensor-memory address
  __shared__ long long row_sm;  // TM: the row fetched for the CTA
  const uint64_t keep = l2_policy_evict_last();
  const uint64_t last = l2_policy_evict_first();
  const int tid = threadIdx.x;
  const int64_t V = a.V;
  const long long N = a.kp.denom > 0 ? a.kp.denom : *a.ws_N;
  if constexpr (TM) {
    if (tid < 32) {
      __syncwarp();
      tmem_alloc(&tmem_sm, tm_cols<NT>());
    }
    tmem_fence_before_sync();
    __syncthreads();
    tmem_fence_after_sync();
  }
  for (int64_t row_i = a.row0 + blockIdx.x;; row_i += gridDim.x) {
    int64_t row = row_i;
    if constexpr (TM) {
      __syncthreads();
      if (tid == 0) row_sm = (long long)atomicAdd(a.ws_rows, 1u) + a.row0;
      __syncthreads();
      row = row_sm;
    }
    if (row >= a.T) break;
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
    // ms; 32000: 1.48 -> 1.37 ms; 24000: 1.34 -> 1.18 ms; peeled 32001: 1.64 ->
    // 1.47 ms), one load at a time in the 256-thread tier (V = 50000: 1.30
    // against 1.33 ms) and for peeled rows of the larger tiers (V = 50257: 1.32
    // against 1.35 ms).
    constexpr Walk kW = (NT == 256 || (PEEL && NT != 128)) ? Walk::kSerialTail : Walk::kClampAll;
    const int nh = (int)head;
    walk_row<kW, U, NT>(
        tid, (int)nvec, [&](int j) { return ld_hint_v4(zv + j, keep); },
        [&](int j, const uint4& r) {
          if (j < nh) head_sm[j] = r;
          if constexpr (TM) {  // block k of the tensor-memory part: the same for the whole CTA
            const int k = j / NT - kHB;
            if (k >= 0 && k < kTmBlocks) {
              __syncwarp();
              tmem_st16(tmem_warp_base(tmem_sm) + 4u * (uint32_t)k, r);
            }
          }
          float x[VEC];
          Elem<Tin>::unpack(r, x);
          acc_add_fast(acc, x);
        });
    if constexpr (TM) {
      __syncwarp();
      tmem_wait_st();
    }
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
      const ff l2 = lse2_from(Cr, Sr);
      float g, loss_t, logp_f;
      uint32_t fl;
      token_math(a.kp, lse_nat(l2), zy, ff{lpo, 0.f}, lpm, A, N, g, loss_t, fl, logp_f);
      bc_g = g;
      bc_cb = backward_offset(l2, g);
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
        // re-read part, oldest first: vectors rb+tid, rb+tid+NT, ... < nvec
        const int64_t rb = TM ? (int64_t)(kHB + kTmBlocks) * NT : head;
        const int64_t nre = nvec - rb;
        const uint4* zr = zv + rb;
        walk_row<kW, U, NT>(
            tid, (int)nre, [&](int j) { return ld_hint_v4(zr + j, last); },
            [&](int j, const uint4& r) { emit(rb + j, r); });
        if constexpr (TM) {
          __syncwarp();
          const uint32_t tw = tmem_warp_base(tmem_sm);
          for (int k = 0; k < kTmBlocks; ++k) {
            const uint4 r = tmem_ld16(tw + 4u * (uint32_t)k);
            tmem_wait_ld();
            emit((int64_t)(kHB + k) * NT + tid, r);
          }
        }
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
  if constexpr (TM) {
    tmem_fence_before_sync();
    __syncthreads();
    tmem_fence_after_sync();
    if (tid < 32) {
      __syncwarp();
      tmem_dealloc(tmem_sm, tm_cols<NT>());
    }
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
    const ff l2 = lse2_from(Cr, Sr);
    const long long N = a.kp.denom > 0 ? a.kp.denom : *a.ws_N;
    float g, loss_t, logp_f;
    uint32_t fl;
    token_math(a.kp, lse_nat(l2), zy, ff{lpo, 0.f}, lpm, A, N, g, loss_t, fl, logp_f);
    bc_g = g;
    bc_cb = ff_round(l2);
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

using K2Kern = void (*)(const K2Args);

// Vectors in flight per thread of the 512-thread tier: 8 for aligned rows
// (V = 151936, GB300: 5.92 ms against 6.08 with 6), 6 for peeled ones
// (V = 151937: 6.20 ms against 6.46 with 8 and 6.50 with 4); `unroll` > 0
// overrides.
template <typename Tin, typename Tout, bool PEEL>
static K2Kern l2_kernel(int nt, int unroll) {
  const int u = unroll > 0 ? unroll : (PEEL ? 6 : 8);
  return (nt == 128)   ? k2_loss_l2<Tin, Tout, 128, 8, PEEL>
         : (nt == 256) ? k2_loss_l2<Tin, Tout, 256, 8, PEEL>
         : (u == 4)    ? k2_loss_l2<Tin, Tout, 512, 4, PEEL>
         : (u == 6)    ? k2_loss_l2<Tin, Tout, 512, 6, PEEL>
                       : k2_loss_l2<Tin, Tout, 512, 8, PEEL>;
}

// The tensor-memory tier's instantiation for a CTA size: the plain kernel's
// vectors in flight (6 for peeled 512-thread rows, else 8).
template <typename Tin, typename Tout, bool PEEL>
static K2Kern tm_kernel(int nt) {
  return nt == kTmThreads ? k2_loss_l2<Tin, Tout, kTmThreads, PEEL ? 6 : 8, PEEL, true>
         : nt == 256      ? k2_loss_l2<Tin, Tout, 256, 8, PEEL, true>
                          : k2_loss_l2<Tin, Tout, 128, 8, PEEL, true>;
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
    // Row-size tiers (measured on GB300, V = 32000 to 151936 bf16): 128 threads
    // and a 16 KB head up to 64 KB rows, 256 threads and no head up to 112 KB,
    // 512 threads beyond, with the largest head that keeps two CTAs in the
    // 164 KB shared-memory carveout (80 KB for this kernel).  The options
    // OCC_OPT_K2_THREADS, OCC_OPT_K2_HEAD_BYTES (0 = pure L2 re-read) and
    // OCC_OPT_K2_UNROLL override the choice.
    const size_t row_bytes = (size_t)(a.V / Elem<Tin>::kVec) * 16;
    const int nt_auto = row_bytes <= 64 * 1024 ? 128 : row_bytes <= 112 * 1024 ? 256 : 512;
    const int64_t nt_opt = option(OCC_OPT_K2_THREADS);
    const int64_t head_opt = option(OCC_OPT_K2_HEAD_BYTES);
    const int unroll = (int)option(OCC_OPT_K2_UNROLL);  // -1: by the row layout
    const int nt = nt_opt > 0 ? (int)nt_opt : nt_auto;
    K2Kern kern = l2_kernel<Tin, Tout, false>(nt, unroll);
    if constexpr (sizeof(Tin) == sizeof(Tout))
      if (peel) kern = l2_kernel<Tin, Tout, true>(nt, unroll);
    const size_t head_auto = nt_auto == 128   ? 16 * 1024
                             : nt_auto == 256 ? 0
                                              : two_cta_smem_budget((const void*)kern);
    size_t head_bytes = std::min(head_opt >= 0 ? (size_t)head_opt : head_auto, row_bytes);
    // Aligned rows in the 512- and 128-thread tiers take the tensor-memory tier when
    // every tensor-memory block lies in whole rounds of the walk (8 blocks per round);
    // OCC_OPT_K2_TMEM = 0 or a shape option keeps the plain kernel.
    bool tm = false;
    const int64_t step = 0x7fffffffLL;
    const int hb = nt == kTmThreads ? kTmHeadBlocks : nt == 256 ? 0 : 8;
    const int tu = (peel && nt == kTmThreads) ? 6 : 8;  // vectors in flight, as the plain kernel's
    // rows of a peeled call lose up to VEC - 1 elements to their scalar lead
    const int64_t nvec_min = (a.V - (peel ? Elem<Tin>::kVec - 1 : 0)) / Elem<Tin>::kVec;
    const int64_t full_blocks = nvec_min / ((int64_t)tu * nt) * tu;
    if ((vec || peel) && (nt == kTmThreads || nt == 256 || nt == 128) &&
        option(OCC_OPT_K2_TMEM) != 0 && nt_opt < 0 && head_opt < 0 && unroll < 0 && T < step &&
        full_blocks >= hb + kTmBlocks) {
      K2Kern kt = tm_kernel<Tin, Tout, false>(nt);
      if constexpr (sizeof(Tin) == sizeof(Tout))
        if (peel) kt = tm_kernel<Tin, Tout, true>(nt);
      const size_t tm_head = (size_t)hb * nt * 16;
      if (nt != kTmThreads || two_cta_smem_budget((const void*)kt) >= tm_head) {
        kern = kt;
        head_bytes = tm_head;
        tm = true;
      }
    }
    a.stage_bytes = (int64_t)head_bytes;
    if (head_bytes > 0) {
      cudaError_t e =
          cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)head_bytes);
      if (e != cudaSuccess)
        return fail(OCC_ERR_CUDA, "cudaFuncSetAttribute(smem=%zu): %s", head_bytes,
                    cudaGetErrorString(e));
    }
    note_kernel(tm ? (peel ? "k2_loss_l2/peel/tmem" : "k2_loss_l2/tmem")
                   : peel ? "k2_loss_l2/peel" : "k2_loss_l2");
    if (tm) {  // persistent: 1024 / nt CTAs per SM (the register limit), rows from the counter
      a.row0 = 0;
      kern<<<(unsigned)std::min<int64_t>(T, (int64_t)sm_count() * (1024 / nt)), nt, head_bytes,
             s>>>(a);
    } else {
      for (int64_t r0 = 0; r0 < T; r0 += step) {
        a.row0 = r0;
        const unsigned grid = (unsigned)std::min<int64_t>(step, T - r0);
        kern<<<grid, nt, head_bytes, s>>>(a);
      }
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
