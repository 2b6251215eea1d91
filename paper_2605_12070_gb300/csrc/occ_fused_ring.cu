// Persistent TMA-ring alternative of the fused loss kernel (selected with the
// option OCC_OPT_FUSED_VARIANT = 1; the default is k2_fused_l2 in occ_fused.cu).
#include "occ_fused_common.cuh"

namespace occ {

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
    // `lost` (test hook): the slot is taken but its copy never issued, so the
    // consumers' wait for it must run out.
    auto ring_copy = [&](const void* src, uint32_t bytes, uint64_t pol, bool lost) -> bool {
      const int s = (int)(G % kSlots);
      const uint64_t u = G / kSlots;
      if (u >= 1 && !wait(&sh.abort, &sh.empty[s], (uint32_t)((u - 1) & 1), a.wait_ns)) return false;
      if (!lost) {
        fence_proxy_async_smem();
        mbar_arrive_expect_tx(&sh.full[s], bytes);
        bulk_load(slots + (size_t)s * kChunk, src, bytes, &sh.full[s], pol);
      }
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
          ok = ring_copy(z + off, b, a.dlogits ? keep : last, false);
        }
        if (ok) ok = ring_copy(zo + off, b, last, k == 0 && row == a.lost_copy_row);
      }
      if (a.dlogits)
        for (int k = nhead; k < nchunk && ok; ++k)
          ok = ring_copy(z + (size_t)k * kChunk, chunk_bytes(k), last, false);
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

template <typename Tin, typename Tout, typename Gm>
static occ_status launch_fused_ring_geo(FusedArgs f, cudaStream_t s) {
  auto kern = k2_fused_ring<Tin, Tout, Gm>;
  // test controls of the bounded waits (off unless a test sets them)
  if (option(OCC_OPT_TEST_LOST_COPY_ROW) >= 0) f.a.lost_copy_row = option(OCC_OPT_TEST_LOST_COPY_ROW);
  if (option(OCC_OPT_TEST_WAIT_NS) > 0) f.a.wait_ns = (uint64_t)option(OCC_OPT_TEST_WAIT_NS);
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)Gm::kSmem);
  if (e != cudaSuccess)
    return fail(OCC_ERR_CUDA, "cudaFuncSetAttribute(smem=%zu): %s", Gm::kSmem,
                cudaGetErrorString(e));
  const unsigned grid = (unsigned)std::min<int64_t>(f.a.T, sm_count());
  note_kernel("k2_fused_ring");
  kern<<<grid, Gm::kNT, Gm::kSmem, s>>>(f);
  return check_launch("occ_decoupled_loss_fused (ring)");
}

// 16 consumer warps, 16 KB copies, 80 KB head, 8-slot ring (208 KB of shared
// memory).  Measured alternatives: 32 KB copies with a 96 KB head and 4 slots,
// and 24 or 30 consumer warps, were all slower.
template <typename Tin, typename Tout>
occ_status launch_fused_ring(const FusedArgs& f, cudaStream_t s) {
  return launch_fused_ring_geo<Tin, Tout, ringk::Geo<16, 16, 5, 8>>(f, s);
}


template occ_status launch_fused_ring<bf16_t, bf16_t>(const FusedArgs&, cudaStream_t);
template occ_status launch_fused_ring<bf16_t, float>(const FusedArgs&, cudaStream_t);
template occ_status launch_fused_ring<float, float>(const FusedArgs&, cudaStream_t);

}  // namespace occ
