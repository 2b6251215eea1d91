// K1 + K2 fused: log pi_old, the decoupled loss and dlogits in one launch,
// with optional per-token diagnostics of the proximal reference.
//
// One CTA per row streams the old (or proxy) logits row and the current
// logits row side by side in the forward pass: log pi_old(y_t) and
// log pi_theta(y_t) come out of the same CTA (Eq. 1 factors), log pi_old stays
// in float-float into the ratio decisions (Eqs. 2-4), and the old row of a dropped
// token is never read.  The backward pass is the K2 one (the current row's
// head from shared memory, the rest re-read from L2).
//
// Rows long enough for it keep more of the current row on chip: after the
// shared-memory head, 16 blocks of NT vectors in tensor memory (128 KB at 512
// threads, 64 KB at 256, 32 KB at 128), which no step of this path needs for
// matrix work.  Only the rest of the row is re-read from L2, and the re-reads
// that the gradient writes would push out of L2 are gone.  That kernel is
// persistent (1024 / NT CTAs per SM, rows fetched from a counter), so each CTA
// allocates its tensor memory once.
//
// Diagnostics (optional, no extra HBM bytes): the entropy of pi_theta,
// H = lse - E_p[z], and KL(pi_old || pi_theta) = E_{p_old}[z_old - z] -
// lse_old + lse, which track the reference-policy lag that the revised
// PPO-EWMA is built to limit (Sec. 5.2, Sec. 6.5, App. E).
#include <cstring>

#include "occ_fused_common.cuh"

namespace occ {

// One 16-byte vector of the current row and the old row.
struct RowPair {
  uint4 t, o;
};

// Vector path: 16-byte rows.  U vectors of each row in flight per thread.
// PEEL: rows that start off a 16-byte boundary take their first `lead`
// elements (up to the boundary) as scalars; the old-logits and gradient rows
// have the same byte offset (checked on the host).
template <typename Tin, typename Tout, int NT, int U, bool DIAG, bool PEEL, bool TM = false>
__global__ void __launch_bounds__(NT, 1024 / NT) k2_fused_l2(const FusedArgs f) {
  static_assert(!TM || NT == kTmThreads || NT == 256 || NT == 128, "the tensor-memory tier");
  // head blocks before the tensor-memory part: 72 KB at 512 threads, none at 256 and 128 (the
  // plain kernel has none there either)
  constexpr int kHB = NT == kTmThreads ? kTmHeadBlocks : 0;
  constexpr int VEC = Elem<Tin>::kVec;
  extern __shared__ __align__(16) uint4 head_sm[];
  __shared__ FusedRed red;
  __shared__ float bc_g, bc_cb;
  __shared__ FusedTok tk_sm;  // thread 0's token scalars, kept over the broadcast
  __shared__ uint32_t tmem_sm;  // TM: the CTA's tensor-memory address
  __shared__ long long row_sm;  // TM: the row fetched for the CTA
  const K2Args& a = f.a;
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
    if constexpr (TM) {  // rows from a counter that K0 cleared: no tail of unequal CTAs
      __syncthreads();
      if (tid == 0) row_sm = (long long)atomicAdd(a.ws_rows, 1u) + a.row0;
      __syncthreads();
      row = row_sm;
    }
    if (row >= a.T) break;
    const int id = a.ids[row];
    const bool m = (a.mask == nullptr) || (a.mask[row] != 0);
    const bool id_ok = id >= 0 && (int64_t)id < V;
    const Tin* z0 = (const Tin*)a.logits + row * a.ld;
    const Tin* zo0 = (const Tin*)f.logits_old + row * f.ld_old;
    const int64_t lead =
        PEEL ? min(V, (int64_t)(((16 - ((uintptr_t)z0 & 15)) & 15) / sizeof(Tin))) : 0;
    const Tin* z = z0 + lead;
    const Tin* zo = zo0 + lead;
    const int64_t nvec = (V - lead) / VEC;
    const int64_t tail0 = nvec * VEC;  // relative to z
    const int64_t ntail = V - lead - tail0;
    const int64_t head = min(nvec, (int64_t)(a.stage_bytes / 16));
    const int idr = id - (int)lead;  // the sampled token relative to z
    Tout* drow0 = a.dlogits ? (Tout*)a.dlogits + row * a.ld_grad : nullptr;
    Tout* drow = drow0 ? drow0 + lead : nullptr;
    if (!(m && id_ok)) {
      if (drow) {
        for (int64_t i = tid; i < nvec; i += NT) OutVecHint<Tout, VEC>::zero(drow + i * VEC, last);
        if ((int64_t)tid < ntail) out_scalar(drow + tail0 + tid, 0.f);
        if (PEEL && (int64_t)tid < lead) out_scalar(drow0 + tid, 0.f);
      }
      if (tid == 0) fused_dropped_outputs(f, row, m, id_ok);
      continue;
    }
    float zy = 0.f, zyo = 0.f, lpm = 0.f, A = 0.f;
    if (tid == 0) {
      zy = Elem<Tin>::load(z0 + id);
      zyo = Elem<Tin>::load(zo0 + id);
      lpm = a.lp_mu[row];
      A = a.adv[row];
    }
    const uint4* zv = reinterpret_cast<const uint4*>(z);
    const uint4* zov = reinterpret_cast<const uint4*>(zo);
    LseAccV acc[2] = {{-INFINITY, 0.f, 0.f}, {-INFINITY, 0.f, 0.f}};
    auto consume = [&](int64_t ii, const uint4& rt, const uint4& ro) {
      if (ii < head) head_sm[ii] = rt;
      float x[VEC], xo[VEC], d[VEC];
      Elem<Tin>::unpack(rt, x);
      Elem<Tin>::unpack(ro, xo);
      if (DIAG) {
#pragma unroll
        for (int q = 0; q < VEC; ++q) d[q] = xo[q] - x[q];
      }
      accv_add<VEC, DIAG>(acc[0], x, x);
      accv_add<VEC, DIAG>(acc[1], xo, d);
    };
    auto consume1 = [&](float xs, float xos) {
      float x1[1] = {xs}, xo1[1] = {xos}, d1[1] = {xos - xs};
      accv_add<1, DIAG>(acc[0], x1, x1);
      accv_add<1, DIAG>(acc[1], xo1, d1);
    };
    // Row walk (GB300, bf16): clamped rounds in the 128-thread tier (V = 32000:
    // 2.03 -> 1.99 ms; 24000: 1.76 -> 1.64 ms) and for peeled rows (V = 50257:
    // 1.94 -> 1.89 ms); one load at a time in the last round for the 256- and
    // 512-thread tiers of aligned rows (V = 50000: 1.82 against 1.84 ms;
    // 151936: 8.28-8.31 ms either way).
    constexpr Walk kW = (NT == 128 || PEEL) ? Walk::kClampAll : Walk::kSerialTail;
    walk_row<kW, U, NT>(
        tid, (int)nvec,
        [&](int j) { return RowPair{ld_hint_v4(zv + j, keep), ld_hint_v4(zov + j, last)}; },
        [&](int j, const RowPair& r) {
          if constexpr (TM) {  // block k of the tensor-memory part: the same for the whole CTA
            const int k = j / NT - kHB;
            if (k >= 0 && k < kTmBlocks) {
              __syncwarp();
              tmem_st16(tmem_warp_base(tmem_sm) + 4u * (uint32_t)k, r.t);
            }
          }
          consume(j, r.t, r.o);
        });
    if constexpr (TM) {
      __syncwarp();
      tmem_wait_st();
    }
    float xt = 0.f, xp = 0.f;
    if ((int64_t)tid < ntail) {
      xt = Elem<Tin>::load(z + tail0 + tid);
      consume1(xt, Elem<Tin>::load(zo + tail0 + tid));
    }
    if (PEEL && (int64_t)tid < lead) {
      xp = Elem<Tin>::load(z0 + tid);
      consume1(xp, Elem<Tin>::load(zo0 + tid));
    }
    float C[2], SV[2];
    float2 S[2];
    block_lse_v2<NT>(acc, red, C, S, SV);
    if (tid < 32) {
      float g, cb;
      fused_token_epilogue(f, C, S, zy, zyo, lpm, A, N, tid, g, cb, tk_sm);
      if (tid == 0) {
        bc_g = g;
        bc_cb = cb;
      }
    }
    __syncthreads();
    if (tid == 0) fused_token_outputs(f, row, tk_sm, S, SV);
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
        const int64_t rb = TM ? (int64_t)(kHB + kTmBlocks) * NT : head;  // first re-read
        const int64_t nre = nvec - rb;
        const uint4* zr = zv + rb;
        walk_row<kW, 8, NT>(  // 8 vectors in flight, whatever the forward pass's U
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

// Any alignment: element loads, old and current rows in one pass, then the
// backward pass over global memory.
template <typename Tin, typename Tout, int NT, bool DIAG>
__global__ void __launch_bounds__(NT) k2_fused_stream(const FusedArgs f) {
  __shared__ FusedRed red;
  __shared__ float bc_g, bc_cb;
  __shared__ FusedTok tk_sm;  // thread 0's token scalars, kept over the broadcast
  const K2Args& a = f.a;
  const int tid = threadIdx.x;
  const int64_t V = a.V;
  const long long N = a.kp.denom > 0 ? a.kp.denom : *a.ws_N;
  for (int64_t row = a.row0 + blockIdx.x; row < a.T; row += gridDim.x) {
    const int id = a.ids[row];
    const bool m = (a.mask == nullptr) || (a.mask[row] != 0);
    const bool id_ok = id >= 0 && (int64_t)id < V;
    Tout* drow = a.dlogits ? (Tout*)a.dlogits + row * a.ld_grad : nullptr;
    if (!(m && id_ok)) {
      if (drow)
        for (int64_t v = tid; v < V; v += NT) out_scalar(drow + v, 0.f);
      if (tid == 0) fused_dropped_outputs(f, row, m, id_ok);
      continue;
    }
    const Tin* z = (const Tin*)a.logits + row * a.ld;
    const Tin* zo = (const Tin*)f.logits_old + row * f.ld_old;
    float zy = 0.f, zyo = 0.f, lpm = 0.f, A = 0.f;
    if (tid == 0) {
      zy = Elem<Tin>::load(z + id);
      zyo = Elem<Tin>::load(zo + id);
      lpm = a.lp_mu[row];
      A = a.adv[row];
    }
    LseAccV acc[2] = {{-INFINITY, 0.f, 0.f}, {-INFINITY, 0.f, 0.f}};
    for (int64_t v0 = tid; v0 < V; v0 += 8 * (int64_t)NT) {
      float x[8], xo[8], xv[8], d[8];  // padding: weight 0 and value 0
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int64_t v = v0 + (int64_t)j * NT;
        x[j] = v < V ? Elem<Tin>::load(z + v) : -INFINITY;
        xo[j] = v < V ? Elem<Tin>::load(zo + v) : -INFINITY;
        xv[j] = v < V ? x[j] : 0.f;
        d[j] = v < V ? xo[j] - x[j] : 0.f;
      }
      accv_add<8, DIAG>(acc[0], x, xv);
      accv_add<8, DIAG>(acc[1], xo, d);
    }
    float C[2], SV[2];
    float2 S[2];
    block_lse_v2<NT>(acc, red, C, S, SV);
    if (tid < 32) {
      float g, cb;
      fused_token_epilogue(f, C, S, zy, zyo, lpm, A, N, tid, g, cb, tk_sm);
      if (tid == 0) {
        bc_g = g;
        bc_cb = cb;
      }
    }
    __syncthreads();
    if (tid == 0) fused_token_outputs(f, row, tk_sm, S, SV);
    if (drow) {
      const float g = bc_g, cb = bc_cb;
      const float sgn = g > 0.f ? -1.f : 1.f;
      for (int64_t v = tid; v < V; v += NT) {
        float dv = 0.f;
        if (g != 0.f) {
          dv = sgn * ex2_approx(fmaf(Elem<Tin>::load(z + v), kLog2e, -cb));
          if (v == id) dv += g;
        }
        out_scalar(drow + v, dv);
      }
    }
    __syncthreads();
  }
}

constexpr int kFusedThreads = 512;
constexpr int kFusedUnroll = 4;

using FusedKern = void (*)(const FusedArgs);

// The diagnostics need two more accumulators and the per-element differences;
// 3 row pairs in flight per thread keep that instantiation free of spills.
constexpr int kFusedUnrollDiag = 3;

template <typename Tin, typename Tout, bool DIAG, bool PEEL>
static FusedKern fused_kernel(int nt) {
  constexpr int U = DIAG ? kFusedUnrollDiag : kFusedUnroll;
  return nt == 128   ? k2_fused_l2<Tin, Tout, 128, U, DIAG, PEEL>
         : nt == 256 ? k2_fused_l2<Tin, Tout, 256, U, DIAG, PEEL>
                     : k2_fused_l2<Tin, Tout, kFusedThreads, U, DIAG, PEEL>;
}

// The tensor-memory tier's instantiation for a CTA size (the plain kernel's
// row pairs in flight).
template <typename Tin, typename Tout, bool DIAG, bool PEEL>
static FusedKern tm_kernel(int nt) {
  constexpr int U = DIAG ? kFusedUnrollDiag : kFusedUnroll;
  return nt == kTmThreads ? k2_fused_l2<Tin, Tout, kTmThreads, U, DIAG, PEEL, true>
         : nt == 256      ? k2_fused_l2<Tin, Tout, 256, U, DIAG, PEEL, true>
                          : k2_fused_l2<Tin, Tout, 128, U, DIAG, PEEL, true>;
}

// Rows off a 16-byte boundary run the vector kernel peeled when the old-logits
// and gradient rows sit at the same byte offsets as the current-logits rows
// (same element size; base addresses and row strides congruent modulo 16
// bytes) and a row holds at least a few vectors.
template <typename Tin, typename Tout>
static bool fused_peel_ok(const FusedArgs& f) {
  const K2Args& a = f.a;
  const int64_t es = (int64_t)sizeof(Tin);
  if (sizeof(Tout) != sizeof(Tin)) return false;
  if (a.V < 16 * Elem<Tin>::kVec || ((uintptr_t)a.logits % es) != 0) return false;
  if ((((uintptr_t)f.logits_old - (uintptr_t)a.logits) % 16) != 0 ||
      (((f.ld_old - a.ld) * es) % 16) != 0)
    return false;
  if (!a.dlogits) return true;
  return (((uintptr_t)a.dlogits - (uintptr_t)a.logits) % 16) == 0 &&
         (((a.ld_grad - a.ld) * es) % 16) == 0;
}

template <typename Tin, typename Tout, bool DIAG>
static occ_status launch_fused(FusedArgs f, bool vec, cudaStream_t s) {
  const int64_t T = f.a.T;
  const int64_t step = 0x7fffffffLL;
  const bool peel = !vec && fused_peel_ok<Tin, Tout>(f);
  if (vec || peel) {
    const int64_t nt_opt = option(OCC_OPT_FUSED_THREADS);
    const int64_t head_opt = option(OCC_OPT_FUSED_HEAD_BYTES);
    // Row-size tiers (measured on GB300, V = 32000 to 151936 bf16): short rows
    // finish in about one load round per CTA, so small CTAs, more of them per
    // SM and no shared-memory head (L2 holds every row in flight) keep the
    // memory system busy; long rows want 512 threads and the largest head
    // with which two CTAs stay in the 164 KB carveout (79 KB for this kernel;
    // at 80 KB it crossed into the 196 KB carveout: 8.38 ms against 8.31 at
    // V = 151936).  OCC_OPT_FUSED_THREADS and OCC_OPT_FUSED_HEAD_BYTES override.
    const size_t row_bytes = (size_t)(f.a.V / Elem<Tin>::kVec) * 16;
    const int nt_auto = row_bytes <= 64 * 1024 ? 128 : row_bytes <= 112 * 1024 ? 256 : kFusedThreads;
    const int nt = nt_opt > 0 ? (int)nt_opt : nt_auto;
    FusedKern kern = fused_kernel<Tin, Tout, DIAG, false>(nt);
    if constexpr (sizeof(Tin) == sizeof(Tout))
      if (peel) kern = fused_kernel<Tin, Tout, DIAG, true>(nt);
    const size_t head_auto =
        nt_auto == kFusedThreads ? two_cta_smem_budget((const void*)kern) : 0;
    size_t head = std::min(head_opt >= 0 ? (size_t)head_opt : head_auto, row_bytes);
    // Aligned rows without diagnostics in the 512- and 128-thread tiers take the
    // tensor-memory tier (GB300, agentic batch V = 151936: 8.06 ms against 8.31 ms, the
    // L2 re-read misses gone) when every tensor-memory block lies in whole rounds of
    // the walk; OCC_OPT_FUSED_TMEM = 0 or a shape option (OCC_OPT_FUSED_THREADS,
    // OCC_OPT_FUSED_HEAD_BYTES) keeps the plain kernel.
    bool tm = false;
    {
      // rows of a peeled call lose up to VEC - 1 elements to their scalar lead
      constexpr int U = DIAG ? kFusedUnrollDiag : kFusedUnroll;
      const int hb = nt == kTmThreads ? kTmHeadBlocks : 0;
      const int64_t nvec_min = (f.a.V - (peel ? Elem<Tin>::kVec - 1 : 0)) / Elem<Tin>::kVec;
      const int64_t full_blocks = nvec_min / ((int64_t)U * nt) * U;
      if ((vec || peel) && (nt == kTmThreads || nt == 256 || nt == 128) &&
          option(OCC_OPT_FUSED_TMEM) != 0 && nt_opt < 0 && head_opt < 0 && T < step &&
          full_blocks >= hb + kTmBlocks) {
        FusedKern kt = tm_kernel<Tin, Tout, DIAG, false>(nt);
        if constexpr (sizeof(Tin) == sizeof(Tout))
          if (peel) kt = tm_kernel<Tin, Tout, DIAG, true>(nt);
        const size_t tm_head = (size_t)hb * nt * 16;
        if (tm_head == 0 || two_cta_smem_budget((const void*)kt) >= tm_head) {
          kern = kt;
          head = tm_head;
          tm = true;
        }
      }
    }
    f.a.stage_bytes = (int64_t)head;
    if (head > 0) {
      cudaError_t e =
          cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)head);
      if (e != cudaSuccess)
        return fail(OCC_ERR_CUDA, "cudaFuncSetAttribute(smem=%zu): %s", head,
                    cudaGetErrorString(e));
    }
    note_kernel(tm ? (peel ? "k2_fused_l2/peel/tmem" : "k2_fused_l2/tmem")
                   : peel ? "k2_fused_l2/peel" : "k2_fused_l2");
    if (tm) {  // persistent: 1024 / nt CTAs per SM (the register limit), rows from the counter
      f.a.row0 = 0;
      const unsigned grid = (unsigned)std::min<int64_t>(T, (int64_t)sm_count() * (1024 / nt));
      kern<<<grid, nt, head, s>>>(f);
    } else {
      for (int64_t r0 = 0; r0 < T; r0 += step) {
        f.a.row0 = r0;
        kern<<<(unsigned)std::min<int64_t>(step, T - r0), nt, head, s>>>(f);
      }
    }
  } else {
    note_kernel("k2_fused_stream");
    for (int64_t r0 = 0; r0 < T; r0 += step) {
      f.a.row0 = r0;
      k2_fused_stream<Tin, Tout, kFusedThreads, DIAG>
          <<<(unsigned)std::min<int64_t>(step, T - r0), kFusedThreads, 0, s>>>(f);
    }
  }
  return check_launch("occ_decoupled_loss_fused");
}

template <typename Tin, typename Tout>
static occ_status launch_fused_any(const FusedArgs& f, bool vec, bool diag, cudaStream_t s) {
  return diag ? launch_fused<Tin, Tout, true>(f, vec, s) : launch_fused<Tin, Tout, false>(f, vec, s);
}

}  // namespace occ

using namespace occ;

extern "C" occ_status occ_decoupled_loss_fused(
    const void* logits, const void* logits_old, occ_dtype dt, int64_t T, int64_t V, int64_t ld,
    int64_t ld_old, const int32_t* ids, const float* logp_mu, const float* adv,
    const uint8_t* loss_mask, const occ_loss_params* p, float* logp_out, float* logp_old_out,
    uint8_t* flags_out, float* entropy_out, float* kl_out, void* dlogits, int64_t ld_grad,
    occ_loss_stats* stats, void* workspace, size_t ws_bytes, void* stream) {
  clear_error();
  FusedArgs f;
  bool vec = false;
  occ_status st = prepare_loss_args(logits, dt, T, V, ld, ids, logp_mu, adv, loss_mask, p,
                                    logp_out, flags_out, dlogits, ld_grad, stats, workspace,
                                    ws_bytes, f.a, vec);
  if (st != OCC_OK) return st;
  if (p->proxy != OCC_PROXY_NONE)
    return fail(OCC_ERR_INVALID_ARG,
                "the fused kernel takes log pi_old from logits_old; proxies are a mode of "
                "occ_decoupled_loss_fwd_bwd");
  const size_t es = dtype_size(dt);
  if (T > 0) {
    if (!logits_old) return fail(OCC_ERR_INVALID_ARG, "null logits_old");
    if (ld_old < V) return fail(OCC_ERR_INVALID_ARG, "ld_old < V");
    if (!aligned(logits_old, es) || (logp_old_out && !aligned(logp_old_out, 4)) ||
        (entropy_out && !aligned(entropy_out, 4)) || (kl_out && !aligned(kl_out, 4)))
      return fail(OCC_ERR_MISALIGNED, "arrays must be aligned to their element size");
    if (dlogits) {
      const size_t es_out = p->dlogits_f32 ? 4 : es;
      const size_t old_bytes = ((size_t)(T - 1) * (size_t)ld_old + (size_t)V) * es;
      const size_t out_bytes = ((size_t)(T - 1) * (size_t)ld_grad + (size_t)V) * es_out;
      if (overlaps(logits_old, old_bytes, dlogits, out_bytes))
        return fail(OCC_ERR_INVALID_ARG, "dlogits overlaps logits_old");
    }
    vec = vec && aligned(logits_old, 16) && ((ld_old * (int64_t)es) % 16 == 0);
  }
  f.logits_old = logits_old;
  f.ld_old = ld_old;
  f.logp_old_out = logp_old_out;
  f.entropy_out = entropy_out;
  f.kl_out = kl_out;
  cudaStream_t s = (cudaStream_t)stream;
  st = launch_k0(f.a, s);
  if (st != OCC_OK) return st;
  if (T > 0) {
    const bool diag = entropy_out || kl_out;
    if (dt == OCC_BF16)
      st = p->dlogits_f32 ? launch_fused_any<bf16_t, float>(f, vec, diag, s)
                          : launch_fused_any<bf16_t, bf16_t>(f, vec, diag, s);
    else
      st = launch_fused_any<float, float>(f, vec, diag, s);
    if (st != OCC_OK) return st;
  }
  return launch_finalize(f.a, stats, s);
}
