// K1 + K2 fused: log pi_old, the decoupled loss and dlogits in one launch,
// with optional per-token diagnostics of the proximal reference.
//
// One CTA per row streams the old (or proxy) logits row and the current
// logits row side by side in the forward pass: log pi_old(y_t) and
// log pi_theta(y_t) come out of the same CTA (Eq. 1 factors), log pi_old stays
// in float64 into the ratio decisions (Eqs. 2-4), and the old row of a dropped
// token is never read.  The backward pass is the K2 one (the current row's
// head from shared memory, the rest re-read from L2).
//
// Diagnostics (optional, no extra HBM bytes): the entropy of pi_theta,
// H = lse - E_p[z], and KL(pi_old || pi_theta) = E_{p_old}[z_old - z] -
// lse_old + lse, which track the reference-policy lag that the revised
// PPO-EWMA is built to limit (Sec. 5.2, Sec. 6.5, App. E).
#include <cstring>

#include "occ_loss_common.cuh"

namespace occ {

struct FusedArgs {
  K2Args a;
  const void* logits_old;
  int64_t ld_old;
  float* logp_old_out;
  float* entropy_out;
  float* kl_out;
};

__device__ __forceinline__ void fused_dropped_outputs(const FusedArgs& f, int64_t row, bool m,
                                                      bool id_ok) {
  dropped_token_outputs(f.a, row, m, id_ok);
  if (f.logp_old_out) f.logp_old_out[row] = id_ok ? 0.f : __int_as_float(0x7fc00000);
  if (f.entropy_out) f.entropy_out[row] = 0.f;
  if (f.kl_out) f.kl_out[row] = 0.f;
}

// Thread 0: token scalars from the two merged rows.  Writes the per-token
// outputs and returns (g, cb) for the backward pass.
__device__ __forceinline__ void fused_token_epilogue(const FusedArgs& f, int64_t row,
                                                     const float (&C)[2], const float2 (&S)[2],
                                                     const float (&SV)[2], float zy, float zyo,
                                                     float lpm, float A, long long N, float& g,
                                                     float& cb) {
  const K2Args& a = f.a;
  const double lse = lse_from(C[0], S[0]);
  const double lse_old = lse_from(C[1], S[1]);
  const double logp_old = (double)zyo - lse_old;
  float loss_t, logp_f;
  uint32_t fl;
  token_math(a.kp, lse, zy, logp_old, lpm, A, N, g, loss_t, fl, logp_f);
  cb = 0.f;
  if (g != 0.f) {
    int e;
    const float fm = frexpf(fabsf(g), &e);
    cb = (float)(lse * (double)kLog2e - (double)e - (double)log2f(fm));
  }
  a.ws_loss[row] = loss_t;
  a.ws_flags[row] = (uint8_t)fl;
  if (a.logp_out) a.logp_out[row] = logp_f;
  if (a.flags_out) a.flags_out[row] = (uint8_t)fl;
  if (f.logp_old_out) f.logp_old_out[row] = (float)logp_old;
  if (f.entropy_out) {
    const double ez = (double)SV[0] / ((double)S[0].x + (double)S[0].y);
    f.entropy_out[row] = (float)(lse - ez);
  }
  if (f.kl_out) {
    const double ed = (double)SV[1] / ((double)S[1].x + (double)S[1].y);
    f.kl_out[row] = (float)(ed - lse_old + lse);
  }
}

// Vector path: 16-byte rows.  U vectors of each row in flight per thread.
template <typename Tin, typename Tout, int NT, int U, bool DIAG>
__global__ void __launch_bounds__(NT, 1024 / NT) k2_fused_l2(const FusedArgs f) {
  constexpr int VEC = Elem<Tin>::kVec;
  extern __shared__ __align__(16) uint4 head_sm[];
  __shared__ FusedRed red;
  __shared__ float bc_g, bc_cb;
  const K2Args& a = f.a;
  const uint64_t keep = l2_policy_evict_last();
  const uint64_t last = l2_policy_evict_first();
  const int tid = threadIdx.x;
  const int64_t V = a.V;
  const int64_t nvec = V / VEC;
  const int64_t tail0 = nvec * VEC;
  const int64_t head = min(nvec, (int64_t)(a.stage_bytes / 16));
  const long long N = a.kp.denom > 0 ? a.kp.denom : *a.ws_N;
  for (int64_t row = a.row0 + blockIdx.x; row < a.T; row += gridDim.x) {
    const int id = a.ids[row];
    const bool m = (a.mask == nullptr) || (a.mask[row] != 0);
    const bool id_ok = id >= 0 && (int64_t)id < V;
    Tout* drow = a.dlogits ? (Tout*)a.dlogits + row * a.ld_grad : nullptr;
    if (!(m && id_ok)) {
      if (drow) {
        for (int64_t i = tid; i < nvec; i += NT) OutVecHint<Tout, VEC>::zero(drow + i * VEC, last);
        if ((int64_t)tid < V - tail0) out_scalar(drow + tail0 + tid, 0.f);
      }
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
    int64_t i = tid;
    for (; i + (int64_t)(U - 1) * NT < nvec; i += (int64_t)U * NT) {
      uint4 rt[U], ro[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        rt[u] = ld_hint_v4(zv + i + u * NT, keep);
        ro[u] = ld_hint_v4(zov + i + u * NT, last);
      }
#pragma unroll
      for (int u = 0; u < U; ++u) consume(i + u * NT, rt[u], ro[u]);
    }
    for (; i < nvec; i += NT) consume(i, ld_hint_v4(zv + i, keep), ld_hint_v4(zov + i, last));
    float xt = 0.f;
    if ((int64_t)tid < V - tail0) {
      xt = Elem<Tin>::load(z + tail0 + tid);
      const float xot = Elem<Tin>::load(zo + tail0 + tid);
      float x1[1] = {xt}, xo1[1] = {xot}, d1[1] = {xot - xt};
      accv_add<1, DIAG>(acc[0], x1, x1);
      accv_add<1, DIAG>(acc[1], xo1, d1);
    }
    float C[2], SV[2];
    float2 S[2];
    block_lse_v2<NT>(acc, red, C, S, SV);
    if (tid == 0) {
      float g, cb;
      fused_token_epilogue(f, row, C, S, SV, zy, zyo, lpm, A, N, g, cb);
      bc_g = g;
      bc_cb = cb;
    }
    __syncthreads();
    if (drow) {
      const float g = bc_g, cb = bc_cb;
      if (g == 0.f) {
        for (int64_t j = tid; j < nvec; j += NT) OutVecHint<Tout, VEC>::zero(drow + j * VEC, last);
        if ((int64_t)tid < V - tail0) out_scalar(drow + tail0 + tid, 0.f);
      } else {
        const float sgn = g > 0.f ? -1.f : 1.f;
        auto emit = [&](int64_t jj, const uint4& r) {
          float x[VEC], d[VEC];
          Elem<Tin>::unpack(r, x);
#pragma unroll
          for (int q = 0; q < VEC; ++q) d[q] = sgn * ex2_approx(fmaf(x[q], kLog2e, -cb));
          if (id >= jj * VEC && id < (jj + 1) * VEC) {
#pragma unroll
            for (int q = 0; q < VEC; ++q)
              if (jj * VEC + q == id) d[q] += g;
          }
          OutVecHint<Tout, VEC>::store(drow + jj * VEC, d, last);
        };
        const int64_t nre = nvec - head;
        int64_t k = tid;
        for (; k + (int64_t)(2 * U - 1) * NT < nre; k += (int64_t)2 * U * NT) {
          uint4 r[2 * U];
#pragma unroll
          for (int u = 0; u < 2 * U; ++u) r[u] = ld_hint_v4(zv + (head + (k + u * NT)), last);
#pragma unroll
          for (int u = 0; u < 2 * U; ++u) emit(head + (k + u * NT), r[u]);
        }
        for (; k < nre; k += NT) emit(head + k, ld_hint_v4(zv + (head + k), last));
#pragma unroll 4
        for (int64_t j = tid; j < head; j += NT) emit(j, head_sm[j]);
        if ((int64_t)tid < V - tail0) {
          float dv = sgn * ex2_approx(fmaf(xt, kLog2e, -cb));
          if (tail0 + tid == id) dv += g;
          out_scalar(drow + tail0 + tid, dv);
        }
      }
    }
    __syncthreads();
  }
}

// Any alignment: element loads, old and current rows in one pass, then the
// backward pass over global memory.
template <typename Tin, typename Tout, int NT, bool DIAG>
__global__ void __launch_bounds__(NT) k2_fused_stream(const FusedArgs f) {
  __shared__ FusedRed red;
  __shared__ float bc_g, bc_cb;
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
    if (tid == 0) {
      float g, cb;
      fused_token_epilogue(f, row, C, S, SV, zy, zyo, lpm, A, N, g, cb);
      bc_g = g;
      bc_cb = cb;
    }
    __syncthreads();
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

// ---------------------------------------------------------------------------
// Persistent TMA-ring variant of the vector path.
//
// One CTA per SM.  A producer thread fetches tokens from a global counter and
// streams their rows through 16 KB cp.async.bulk copies; 16 consumer warps
// reduce them.  The current row's first chunks land in a shared-memory head
// that the backward pass reads back; every other chunk (the old row, the rest
// of the current row, then that rest again for the backward pass, from L2)
// passes through a ring of slots guarded by full / empty mbarriers.  The
// producer runs ahead into the next token while the consumers reduce and write
// dlogits, so the memory system stays busy across row boundaries, and the
// bytes in flight are bounded by the ring rather than by L1.  The consumers
// synchronise through mbarriers only (no bar.sync), and every wait is bounded
// by %globaltimer: a wait that runs out raises a CTA-wide abort, sets
// OCC_DATA_ERR_TIMEOUT, and the producer drains its copies in flight before
// the CTA exits.
namespace ringk {

constexpr int kQ = 4;  // row-queue depth

// Geometry: CW consumer warps + one producer warp, CHK-KB copies, HEADC chunks
// of the current row kept on chip, SLOTS ring slots.
template <int CW, int CHK, int HEADC, int SLOTS>
struct Geo {
  static constexpr int kCW = CW;
  static constexpr int kNC = CW * 32;
  static constexpr int kNT = kNC + 32;
  static constexpr uint32_t kChunk = (uint32_t)CHK * 1024;
  static constexpr int kHead = HEADC;
  static constexpr int kSlots = SLOTS;
  static constexpr size_t kSmem = (size_t)(HEADC + SLOTS) * CHK * 1024;
};

template <int CW, int HEADC, int SLOTS>
struct __align__(16) Shared {
  uint64_t full[SLOTS], empty[SLOTS];
  uint64_t head_full[HEADC], head_free;
  uint64_t q_full[kQ], q_empty[kQ];
  uint64_t red, bc;
  long long q_row[kQ];
  int abort;
  float bc_g, bc_cb;
  float red_c[2][CW];
  float2 red_s[2][CW];
};

__device__ __forceinline__ void arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes,
                                          uint64_t* bar, uint64_t pol) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1], %2, [%3], %4;" ::"r"(smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(pol)
      : "memory");
}
// try_wait with a suspend-time hint: the thread is parked in hardware until the
// phase completes or ~20 us pass, instead of spinning on issue slots.
__device__ __forceinline__ bool try_wait_sleep(uint64_t* bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(done)
      : "r"(smem_u32(bar)), "r"(parity), "r"(20000u)
      : "memory");
  return done != 0;
}
// Waits for phase `parity` of `bar`.  Returns false when another party has
// aborted, or raises the abort itself when `limit_ns` runs out.
__device__ __forceinline__ bool wait(int* abort, uint64_t* bar, uint32_t parity,
                                     uint64_t limit_ns) {
  if (try_wait_sleep(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  while (!try_wait_sleep(bar, parity)) {
    if (*(volatile int*)abort) return false;
    if (globaltimer_ns() - t0 > limit_ns) {
      *(volatile int*)abort = 1;
      return false;
    }
  }
  return true;
}

}  // namespace ringk

template <typename Tin, typename Tout, typename Gm>
__global__ void __launch_bounds__(Gm::kNT, 1) k2_fused_ring(const FusedArgs f) {
  using namespace ringk;
  constexpr int VEC = Elem<Tin>::kVec;
  constexpr int kCW = Gm::kCW, kNC = Gm::kNC, kHead = Gm::kHead, kSlots = Gm::kSlots;
  constexpr uint32_t kChunk = Gm::kChunk;
  constexpr int kPer = (int)(kChunk / 16) / kNC;  // vectors per consumer thread in a full chunk
  static_assert(kPer * kNC * 16 == (int)kChunk, "a chunk splits evenly over the consumers");
  extern __shared__ __align__(128) unsigned char ring_smem[];
  __shared__ Shared<Gm::kCW, Gm::kHead, Gm::kSlots> sh;
  const K2Args& a = f.a;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const int64_t T = a.T, V = a.V;
  const int64_t nvec = V / VEC;
  const int64_t tail0 = nvec * VEC;
  const int64_t nbytes = nvec * 16;
  const int nchunk = (int)((nbytes + kChunk - 1) / kChunk);
  const int nhead = min(nchunk, kHead);
  unsigned char* head = ring_smem;
  unsigned char* slots = ring_smem + (size_t)kHead * kChunk;
  auto chunk_bytes = [&](int k) -> uint32_t {
    return (uint32_t)min((int64_t)kChunk, nbytes - (int64_t)k * kChunk);
  };

  if (tid == 0) {
    for (int s = 0; s < kSlots; ++s) {
      mbar_init(&sh.full[s], 1);
      mbar_init(&sh.empty[s], kCW);
    }
    for (int k = 0; k < kHead; ++k) mbar_init(&sh.head_full[k], 1);
    mbar_init(&sh.head_free, kCW);
    for (int q = 0; q < kQ; ++q) {
      mbar_init(&sh.q_full[q], 1);
      mbar_init(&sh.q_empty[q], kCW);
    }
    mbar_init(&sh.red, kCW);
    mbar_init(&sh.bc, 1);
    sh.abort = 0;
    fence_mbarrier_init();
  }
  __syncthreads();

  if (wid == kCW) {  // ------------------------------------------ producer
    if (lane != 0) return;
    const uint64_t keep = l2_policy_evict_last();
    const uint64_t last = l2_policy_evict_first();
    uint64_t G = 0;       // ring copies issued
    long long jv = 0;     // valid rows whose copies were all issued
    long long rq = 0;     // row-queue entries pushed
    long long hcount[kHead] = {};  // head copies issued, per head slot
    bool ok = true;
    auto ring_copy = [&](const void* src, uint32_t bytes, uint64_t pol) -> bool {
      const int s = (int)(G % kSlots);
      const uint64_t u = G / kSlots;
      if (u >= 1 && !wait(&sh.abort, &sh.empty[s], (uint32_t)((u - 1) & 1), a.wait_ns)) return false;
      fence_proxy_async_smem();
      mbar_arrive_expect_tx(&sh.full[s], bytes);
      bulk_load(slots + (size_t)s * kChunk, src, bytes, &sh.full[s], pol);
      ++G;
      return true;
    };
    while (ok) {
      long long row = (long long)atomicAdd(a.ws_rows, 1ull);
      if (row >= T) row = -1;
      const int q = (int)(rq % kQ);
      const long long uq = rq / kQ;
      if (uq >= 1 && !wait(&sh.abort, &sh.q_empty[q], (uint32_t)((uq - 1) & 1), a.wait_ns)) break;
      sh.q_row[q] = row;
      arrive(&sh.q_full[q]);
      ++rq;
      if (row < 0) break;
      const int id = a.ids[row];
      const bool valid = (a.mask == nullptr || a.mask[row] != 0) && id >= 0 && (int64_t)id < V;
      if (!valid) continue;
      if (jv >= 1 && !wait(&sh.abort, &sh.head_free, (uint32_t)((jv - 1) & 1), a.wait_ns)) break;
      const unsigned char* z = (const unsigned char*)((const Tin*)a.logits + row * a.ld);
      const unsigned char* zo = (const unsigned char*)((const Tin*)f.logits_old + row * f.ld_old);
      for (int k = 0; k < nchunk && ok; ++k) {
        const uint32_t b = chunk_bytes(k);
        const size_t off = (size_t)k * kChunk;
        if (k < nhead) {
          fence_proxy_async_smem();
          mbar_arrive_expect_tx(&sh.head_full[k], b);
          bulk_load(head + off, z + off, b, &sh.head_full[k], last);
          ++hcount[k];
        } else {
          ok = ring_copy(z + off, b, a.dlogits ? keep : last);
        }
        if (ok) ok = ring_copy(zo + off, b, last);
      }
      if (a.dlogits)
        for (int k = nhead; k < nchunk && ok; ++k)
          ok = ring_copy(z + (size_t)k * kChunk, chunk_bytes(k), last);
      if (ok) ++jv;
    }
    // drain: every copy issued must land before the CTA's shared memory goes
    for (int s = 0; s < kSlots; ++s) {
      const uint64_t issued = G / kSlots + ((uint64_t)s < G % kSlots ? 1 : 0);
      if (issued > 0) mbar_wait_bounded(&sh.full[s], (uint32_t)((issued - 1) & 1), a.wait_ns);
    }
    for (int k = 0; k < nhead; ++k)
      if (hcount[k] > 0)
        mbar_wait_bounded(&sh.head_full[k], (uint32_t)((hcount[k] - 1) & 1), a.wait_ns);
    if (*(volatile int*)&sh.abort) atomicOr(a.ws_err, OCC_DATA_ERR_TIMEOUT);
    return;
  }

  // ---------------------------------------------------------------- consumers
  const uint64_t last = l2_policy_evict_first();
  const int ct = tid;  // 0 .. kNC-1
  const long long N = a.kp.denom > 0 ? a.kp.denom : *a.ws_N;
  uint64_t G = 0;
  long long jv = 0, rq = 0;
  while (true) {
    const int q = (int)(rq % kQ);
    if (!wait(&sh.abort, &sh.q_full[q], (uint32_t)((rq / kQ) & 1), a.wait_ns)) break;
    const long long row = sh.q_row[q];
    __syncwarp();
    if (lane == 0) arrive(&sh.q_empty[q]);
    ++rq;
    if (row < 0) break;
    const int id = a.ids[row];
    const bool m = (a.mask == nullptr) || (a.mask[row] != 0);
    const bool id_ok = id >= 0 && (int64_t)id < V;
    Tout* drow = a.dlogits ? (Tout*)a.dlogits + row * a.ld_grad : nullptr;
    if (!(m && id_ok)) {
      if (drow) {
        for (int64_t i = ct; i < nvec; i += kNC) OutVecHint<Tout, VEC>::zero(drow + i * VEC, last);
        if ((int64_t)ct < V - tail0) out_scalar(drow + tail0 + ct, 0.f);
      }
      if (ct == 0) fused_dropped_outputs(f, row, m, id_ok);
      continue;
    }
    const Tin* z = (const Tin*)a.logits + row * a.ld;
    const Tin* zo = (const Tin*)f.logits_old + row * f.ld_old;
    float zy = 0.f, zyo = 0.f, lpm = 0.f, A = 0.f;
    if (ct == 0) {
      zy = Elem<Tin>::load(z + id);
      zyo = Elem<Tin>::load(zo + id);
      lpm = a.lp_mu[row];
      A = a.adv[row];
    }
    // forward: both rows, chunk by chunk
    LseAccV acc[2] = {{-INFINITY, 0.f, 0.f}, {-INFINITY, 0.f, 0.f}};
    bool ok = true;
    for (int k = 0; k < nchunk && ok; ++k) {
      const int nv = (int)(chunk_bytes(k) / 16);
      const uint4* zs;
      int sz = -1;
      if (k < nhead) {
        ok = wait(&sh.abort, &sh.head_full[k], (uint32_t)(jv & 1), a.wait_ns);
        zs = reinterpret_cast<const uint4*>(head + (size_t)k * kChunk);
      } else {
        sz = (int)(G % kSlots);
        ok = wait(&sh.abort, &sh.full[sz], (uint32_t)((G / kSlots) & 1), a.wait_ns);
        zs = reinterpret_cast<const uint4*>(slots + (size_t)sz * kChunk);
        ++G;
      }
      const int so = (int)(G % kSlots);
      ok = ok && wait(&sh.abort, &sh.full[so], (uint32_t)((G / kSlots) & 1), a.wait_ns);
      ++G;
      if (!ok) break;
      const uint4* os = reinterpret_cast<const uint4*>(slots + (size_t)so * kChunk);
      auto fwd = [&](int i) {
        float x[VEC], xo[VEC];
        Elem<Tin>::unpack(zs[i], x);
        accv_add<VEC, false>(acc[0], x, x);
        Elem<Tin>::unpack(os[i], xo);
        accv_add<VEC, false>(acc[1], xo, xo);
      };
      if (nv == kPer * kNC) {  // a full chunk: straight-line, compile-time trip count
        uint4 rz[kPer], ro[kPer];
#pragma unroll
        for (int u = 0; u < kPer; ++u) {
          rz[u] = zs[ct + u * kNC];
          ro[u] = os[ct + u * kNC];
        }
#pragma unroll
        for (int u = 0; u < kPer; ++u) {
          float x[VEC], xo[VEC];
          Elem<Tin>::unpack(rz[u], x);
          accv_add<VEC, false>(acc[0], x, x);
          Elem<Tin>::unpack(ro[u], xo);
          accv_add<VEC, false>(acc[1], xo, xo);
        }
      } else {
        for (int i = ct; i < nv; i += kNC) fwd(i);
      }
      __syncwarp();
      if (lane == 0) {
        if (sz >= 0) arrive(&sh.empty[sz]);
        arrive(&sh.empty[so]);
      }
    }
    if (!ok) break;
    float xt = 0.f;
    if ((int64_t)ct < V - tail0) {
      xt = Elem<Tin>::load(z + tail0 + ct);
      float x1[1] = {xt}, xo1[1] = {Elem<Tin>::load(zo + tail0 + ct)};
      accv_add<1, false>(acc[0], x1, x1);
      accv_add<1, false>(acc[1], xo1, xo1);
    }
    // CTA reduction through mbarriers: warp partials -> consumer thread 0
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      const float wm = warp_max(acc[k].c);
      const float sc = acc[k].c == -INFINITY ? 0.f : exp2f(acc[k].c - wm);
      const float2 v = warp_pair_sum(make_float2(acc[k].s * sc, 0.f));
      if (lane == 0) {
        sh.red_c[k][wid] = wm;
        sh.red_s[k][wid] = v;
      }
    }
    if (lane == 0) arrive(&sh.red);
    if (ct == 0) {
      ok = wait(&sh.abort, &sh.red, (uint32_t)(jv & 1), a.wait_ns);
      float C[2], SV[2];
      float2 S[2];
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        float cm = -INFINITY;
        for (int w = 0; w < kCW; ++w) cm = fmaxf(cm, sh.red_c[k][w]);
        float2 s = make_float2(0.f, 0.f);
        for (int w = 0; w < kCW; ++w) {
          const float cw = sh.red_c[k][w];
          if (cw == -INFINITY) continue;
          const float sc = exp2f(cw - cm);
          const float2 p = sh.red_s[k][w];
          const float hi = p.x * sc;
          s = pair_add(s, make_float2(hi, fmaf(p.x, sc, -hi) + p.y * sc));
        }
        C[k] = cm;
        S[k] = s;
        SV[k] = 0.f;
      }
      float g = 0.f, cb = 0.f;
      if (ok) fused_token_epilogue(f, row, C, S, SV, zy, zyo, lpm, A, N, g, cb);
      sh.bc_g = g;
      sh.bc_cb = cb;
      arrive(&sh.bc);
    }
    if (!ok || !wait(&sh.abort, &sh.bc, (uint32_t)(jv & 1), a.wait_ns)) break;
    const float g = sh.bc_g, cb = sh.bc_cb;
    const float sgn = g > 0.f ? -1.f : 1.f;
    auto emit = [&](int64_t jj, const uint4& r) {
      float x[VEC], d[VEC];
      Elem<Tin>::unpack(r, x);
#pragma unroll
      for (int qq = 0; qq < VEC; ++qq) d[qq] = sgn * ex2_approx(fmaf(x[qq], kLog2e, -cb));
      if (id >= jj * VEC && id < (jj + 1) * VEC) {
#pragma unroll
        for (int qq = 0; qq < VEC; ++qq)
          if (jj * VEC + qq == id) d[qq] += g;
      }
      OutVecHint<Tout, VEC>::store(drow + jj * VEC, d, last);
    };
    auto bwd_chunk = [&](const uint4* zs, int64_t base, int nv) {
      if (g == 0.f) {
        for (int i = ct; i < nv; i += kNC) OutVecHint<Tout, VEC>::zero(drow + (base + i) * VEC, last);
      } else if (nv == kPer * kNC) {
        uint4 r[kPer];
#pragma unroll
        for (int u = 0; u < kPer; ++u) r[u] = zs[ct + u * kNC];
#pragma unroll
        for (int u = 0; u < kPer; ++u) emit(base + ct + u * kNC, r[u]);
      } else {
        for (int i = ct; i < nv; i += kNC) emit(base + i, zs[i]);
      }
    };
    // backward: the head from shared memory, then the re-read chunks
    if (drow) {
      for (int k = 0; k < nhead; ++k) {
        const int nv = (int)(chunk_bytes(k) / 16);
        const uint4* zs = reinterpret_cast<const uint4*>(head + (size_t)k * kChunk);
        const int64_t base = (int64_t)k * (kChunk / 16);
        bwd_chunk(zs, base, nv);
      }
    }
    __syncwarp();
    if (lane == 0) arrive(&sh.head_free);
    if (drow) {
      for (int k = nhead; k < nchunk && ok; ++k) {
        const int nv = (int)(chunk_bytes(k) / 16);
        const int s = (int)(G % kSlots);
        ok = wait(&sh.abort, &sh.full[s], (uint32_t)((G / kSlots) & 1), a.wait_ns);
        ++G;
        if (!ok) break;
        const uint4* zs = reinterpret_cast<const uint4*>(slots + (size_t)s * kChunk);
        const int64_t base = (int64_t)k * (kChunk / 16);
        bwd_chunk(zs, base, nv);
        __syncwarp();
        if (lane == 0) arrive(&sh.empty[s]);
      }
      if (!ok) break;
      if ((int64_t)ct < V - tail0) {
        float dv = 0.f;
        if (g != 0.f) {
          dv = sgn * ex2_approx(fmaf(xt, kLog2e, -cb));
          if (tail0 + ct == id) dv += g;
        }
        out_scalar(drow + tail0 + ct, dv);
      }
    }
    ++jv;
  }
}

constexpr int kFusedThreads = 512;
constexpr int kFusedUnroll = 4;
constexpr size_t kFusedHeadBytes = 80 * 1024;

// OCC_FUSED_VARIANT=ring selects the persistent TMA-ring kernel for the vector
// path without diagnostics.
static bool fused_ring_selected() {
  static const bool v = [] {
    const char* e = getenv("OCC_FUSED_VARIANT");
    return e && strcmp(e, "ring") == 0;
  }();
  return v;
}

template <typename Tin, typename Tout, typename Gm>
static occ_status launch_fused_ring_geo(const FusedArgs& f, cudaStream_t s) {
  auto kern = k2_fused_ring<Tin, Tout, Gm>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)Gm::kSmem);
  if (e != cudaSuccess)
    return fail(OCC_ERR_CUDA, "cudaFuncSetAttribute(smem=%zu): %s", Gm::kSmem,
                cudaGetErrorString(e));
  const unsigned grid = (unsigned)std::min<int64_t>(f.a.T, sm_count());
  kern<<<grid, Gm::kNT, Gm::kSmem, s>>>(f);
  return check_launch("occ_decoupled_loss_fused (ring)");
}

// 16 consumer warps, 16 KB copies, 80 KB head, 8-slot ring (208 KB of shared
// memory).  Measured alternatives: 32 KB copies with a 96 KB head and 4 slots,
// and 24 or 30 consumer warps, were all slower.
template <typename Tin, typename Tout>
static occ_status launch_fused_ring(const FusedArgs& f, cudaStream_t s) {
  return launch_fused_ring_geo<Tin, Tout, ringk::Geo<16, 16, 5, 8>>(f, s);
}

template <typename Tin, typename Tout, bool DIAG>
static occ_status launch_fused(FusedArgs f, bool vec, cudaStream_t s) {
  const int64_t T = f.a.T;
  const int64_t step = 0x7fffffffLL;
  if (vec && !DIAG && f.a.V >= Elem<Tin>::kVec && fused_ring_selected())
    return launch_fused_ring<Tin, Tout>(f, s);
  if (vec) {
    const size_t row_bytes = (size_t)(f.a.V / Elem<Tin>::kVec) * 16;
    const size_t head = std::min(kFusedHeadBytes, row_bytes);
    f.a.stage_bytes = (int64_t)head;
    auto kern = k2_fused_l2<Tin, Tout, kFusedThreads, kFusedUnroll, DIAG>;
    if (head > 0) {
      cudaError_t e =
          cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)head);
      if (e != cudaSuccess)
        return fail(OCC_ERR_CUDA, "cudaFuncSetAttribute(smem=%zu): %s", head,
                    cudaGetErrorString(e));
    }
    for (int64_t r0 = 0; r0 < T; r0 += step) {
      f.a.row0 = r0;
      kern<<<(unsigned)std::min<int64_t>(step, T - r0), kFusedThreads, head, s>>>(f);
    }
  } else {
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
