// Device building blocks shared by the occ kernels (sm_103a).
//
// The row statistic every kernel needs is the log-partition function
// lse = log sum_v exp(z_v) of a logits row (Eq. 1 ratios are quotients of
// softmax probabilities).  Each thread keeps an online pair (c, s) in base-2
// scaled units: s = sum 2^(z_v * L - c) with L = float(log2 e).  The reference
// exponent c only moves when a new value exceeds it by more than kRescale
// (lazy rescaling), so the inner loop is one FFMA, one MUFU.EX2 and one FADD
// per element.  Partials are merged with one accurate exp2f per thread and a
// compensated (two-float) tree sum, and the row epilogue runs in float-float.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "occ.h"
#include "occ_internal.h"

namespace occ {

constexpr float kLog2e = 1.4426950408889634f;  // float(log2 e)
constexpr double kInvLog2eF = 0.6931471898132927;  // 1 / (double)kLog2e
constexpr float kRescale = 64.f;               // lazy-rescale margin (base-2 exponent units)

// ---------------------------------------------------------------- PTX helpers

__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Streaming 16-byte load: bypass L1, 256-byte L2 prefetch granularity.
__device__ __forceinline__ uint4 ld_stream_v4(const void* p) {
  uint4 r;
  asm volatile("ld.global.L1::no_allocate.L2::256B.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

// L2 eviction policies (createpolicy) and 16-byte accesses that carry them.
__device__ __forceinline__ uint64_t l2_policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint4 ld_hint_v4(const void* p, uint64_t pol) {
  uint4 r;
  asm volatile("ld.global.L1::no_allocate.L2::cache_hint.v4.u32 {%0,%1,%2,%3}, [%4], %5;"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p), "l"(pol));
  return r;
}
__device__ __forceinline__ void st_hint_v4(void* p, uint4 v, uint64_t pol) {
  asm volatile("st.global.L1::no_allocate.L2::cache_hint.v4.u32 [%0], {%1,%2,%3,%4}, %5;" ::"l"(p),
               "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w), "l"(pol)
               : "memory");
}

// Streaming (evict-first) 16-byte store.
__device__ __forceinline__ void st_stream_v4(void* p, uint4 v) {
  asm volatile("st.global.cs.v4.u32 [%0], {%1,%2,%3,%4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z),
               "r"(v.w)
               : "memory");
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  uint32_t d;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
  return d;
}

// Round-to-nearest-even float -> bf16 scalar store to global memory.
__device__ __forceinline__ void st_bf16(void* p, float x) {
  unsigned short h;
  asm("cvt.rn.bf16.f32 %0, %1;" : "=h"(h) : "f"(x));
  asm volatile("st.global.u16 [%0], %1;" ::"l"(p), "h"(h) : "memory");
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// Scalar element access for the two input types.
template <typename T>
struct Elem;
template <>
struct Elem<float> {
  static constexpr int kVec = 4;  // elements per 16-byte vector
  __device__ __forceinline__ static float load(const float* p) { return *(const volatile float*)p; }
  __device__ __forceinline__ static void put(float* p, float x) { *p = x; }
  __device__ __forceinline__ static void unpack(const uint4& r, float (&x)[4]) {
    x[0] = __uint_as_float(r.x);
    x[1] = __uint_as_float(r.y);
    x[2] = __uint_as_float(r.z);
    x[3] = __uint_as_float(r.w);
  }
};
struct bf16_t {
  uint16_t bits;
};
template <>
struct Elem<bf16_t> {
  static constexpr int kVec = 8;
  __device__ __forceinline__ static float load(const bf16_t* p) {
    unsigned short b;
    asm volatile("ld.global.u16 %0, [%1];" : "=h"(b) : "l"(p));
    return __uint_as_float(((uint32_t)b) << 16);
  }
  // Stores a value that is exactly representable in bf16 (its top 16 bits).
  __device__ __forceinline__ static void put(bf16_t* p, float x) {
    p->bits = (uint16_t)(__float_as_uint(x) >> 16);
  }
  __device__ __forceinline__ static void unpack(const uint4& r, float (&x)[8]) {
    x[0] = bf16_lo(r.x); x[1] = bf16_hi(r.x);
    x[2] = bf16_lo(r.y); x[3] = bf16_hi(r.y);
    x[4] = bf16_lo(r.z); x[5] = bf16_hi(r.z);
    x[6] = bf16_lo(r.w); x[7] = bf16_hi(r.w);
  }
};

// ------------------------------------------------------- online log-sum-exp

struct LseAcc {
  float c;  // reference exponent, base-2 scaled units (-inf: nothing finite seen)
  float s;  // sum of 2^(z L - c)
};

__device__ __forceinline__ void acc_init(LseAcc& a) {
  a.c = -INFINITY;
  a.s = 0.f;
}

template <int N>
__device__ __forceinline__ void acc_add(LseAcc& a, const float (&x)[N]) {
  float m = x[0];
#pragma unroll
  for (int j = 1; j < N; ++j) m = fmaxf(m, x[j]);
  const float ms = m * kLog2e;
  if (ms > a.c + kRescale) {  // also taken by the first finite vector (c = -inf)
    a.s *= exp2f(a.c - ms);
    a.c = ms;
  }
  if (a.c != -INFINITY) {
    float t = 0.f;
#pragma unroll
    for (int j = 0; j < N; ++j) t += ex2_approx(fmaf(x[j], kLog2e, -a.c));
    a.s += t;
  }
}

// Same update, fast path: the terms are taken against the current reference
// exponent without a per-vector max; only a group that is not finite or
// exceeds 2^64 (a value far above everything seen so far, or the thread's
// first group) goes through acc_add, which moves the reference.
template <int N>
__device__ __forceinline__ void acc_add_fast(LseAcc& a, const float (&x)[N]) {
  float t = 0.f;
#pragma unroll
  for (int j = 0; j < N; ++j) t += ex2_approx(fmaf(x[j], kLog2e, -a.c));
  if (t <= 1.8446744073709552e19f)  // 2^64; false for inf and NaN
    a.s += t;
  else
    acc_add(a, x);
}

// ------------------------------------------------------- tensor memory (TMEM)

// Tensor memory is the 256 KB per SM (128 lanes x 512 columns of 32 bits) that
// tcgen05 matrix instructions accumulate into.  No step of this path is a
// contraction, so the loss kernels use it as plain on-chip storage for part of
// a logits row.  A warp reaches only its quarter of the lanes (warp % 4); each
// thread owns one lane, and a 32x32b.x4 access moves 16 bytes per thread to or
// from 4 consecutive columns of that lane.  Allocation is per CTA, by one warp.
__device__ __forceinline__ void tmem_alloc(uint32_t* dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   (uint32_t)__cvta_generic_to_shared(dst_smem)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
// Orders tcgen05 work around a CTA barrier (the allocation's address, the
// last accesses before the deallocation).
__device__ __forceinline__ void tmem_fence_before_sync() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tmem_fence_after_sync() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint4& v) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x4.b32 [%0], {%1, %2, %3, %4};" ::"r"(taddr),
               "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
               : "memory");
}
__device__ __forceinline__ uint4 tmem_ld16(uint32_t taddr) {
  uint4 v;
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x4.b32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(taddr)
               : "memory");
  return v;
}
__device__ __forceinline__ void tmem_wait_st() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// The tensor-memory tier of the loss kernels.  A row walks in blocks of NT
// vectors (one per thread); after a shared-memory head of some blocks, the next
// kTmBlocks blocks go to tensor memory and the rest is re-read from L2.  Each
// thread keeps its kTmBlocks vectors in 4 kTmBlocks = 64 columns of its own
// lane; warp w uses the lane quarter w % 4 and columns 64 floor(w / 4) on, so
// a CTA takes NT / 2 columns: 256 for 512 threads (two CTAs per SM), 64 for 128
// threads (eight per SM): the SM's 512 columns either way.  The launchers take
// this tier only for rows whose tensor-memory blocks lie in whole rounds of the
// walk (every thread loads its vector of each such block, so the accesses stay
// warp-converged).
constexpr int kTmThreads = 512;
constexpr int kTmHeadBlocks = 9;  // the 512-thread tier's head: 9 blocks of 512 vectors (72 KB)
constexpr int kTmBlocks = 16;
template <int NT>
constexpr uint32_t tm_cols() {
  return (uint32_t)NT / 2;
}

// This warp's part of the CTA's tensor memory (base from tcgen05.alloc).
__device__ __forceinline__ uint32_t tmem_warp_base(uint32_t base) {
  const uint32_t w = threadIdx.x >> 5;
  return base + ((32u * (w & 3u)) << 16) + (w >> 2) * 64u;
}

// ------------------------------------------------------------ row streaming

// How a thread walks the vectors i = t, t + NT, t + 2 NT, ... < n of a row,
// U loads in flight per round.  The shapes differ only in the last, partial
// round (fewer than U vectors left for the thread):
//   kSerialTail  the partial round takes one load at a time (each waits for
//                the previous vector's use: its latency is paid per vector);
//   kTailRound   full rounds as above, then one round whose loads all issue
//                together, loads past the row's end repeating the last vector
//                (in bounds, from L2) and left unused;
//   kClampAll    every round is that clamped round.
// Which one is fastest depends on the kernel and its CTA size (GB300
// measurements at the launch sites).  Row-local indices are 32-bit: V < 2^31.
enum class Walk { kSerialTail, kTailRound, kClampAll };

// `load(j)` returns the data of vector j (any copyable type), `use(j, d)`
// consumes it.
template <Walk W, int U, int NT, typename Load, typename Use>
__device__ __forceinline__ void walk_row(int t, int n, Load load, Use use) {
  using D = decltype(load(0));
  if constexpr (W == Walk::kClampAll) {
    for (int i = t; i < n; i += U * NT) {
      D r[U];
#pragma unroll
      for (int u = 0; u < U; ++u) r[u] = load(min(i + u * NT, n - 1));
#pragma unroll
      for (int u = 0; u < U; ++u)
        if (i + u * NT < n) use(i + u * NT, r[u]);
    }
  } else {
    int i = t;
    for (; i + (U - 1) * NT < n; i += U * NT) {
      D r[U];
#pragma unroll
      for (int u = 0; u < U; ++u) r[u] = load(i + u * NT);
#pragma unroll
      for (int u = 0; u < U; ++u) use(i + u * NT, r[u]);
    }
    if constexpr (W == Walk::kSerialTail) {
      for (; i < n; i += NT) use(i, load(i));
    } else if (U > 1 && i < n) {
      D r[U > 1 ? U - 1 : 1];
#pragma unroll
      for (int u = 0; u < U - 1; ++u) r[u] = load(min(i + u * NT, n - 1));
#pragma unroll
      for (int u = 0; u < U - 1; ++u)
        if (i + u * NT < n) use(i + u * NT, r[u]);
    }
  }
}

// ------------------------------------------------------------ reductions

// Two-float compensated addition (Knuth TwoSum on the high parts).
__device__ __forceinline__ float2 pair_add(float2 a, float2 b) {
  const float s = a.x + b.x;
  const float bp = s - a.x;
  const float e = (a.x - (s - bp)) + (b.x - bp);
  return make_float2(s, e + (a.y + b.y));
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ float2 warp_pair_sum(float2 v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    float2 w;
    w.x = __shfl_xor_sync(0xffffffffu, v.x, o);
    w.y = __shfl_xor_sync(0xffffffffu, v.y, o);
    v = pair_add(v, w);
  }
  return v;
}

// Shared scratch for block reductions (one slot per warp).
struct RedScratch {
  float c[32];
  float2 s[32];
};

// Merges the per-thread (c, s) of a block with one barrier: each warp scales
// its sum to the warp's largest reference exponent, then warp 0 merges the
// warps' pairs (compensated).  Result (C, S) is valid in every lane of warp 0:
// sum over the block of 2^(z L - C) = S.x + S.y.  Deterministic order.
template <int NT>
__device__ __forceinline__ void block_lse(const LseAcc& a, RedScratch& r, float& C, float2& S) {
  constexpr int NW = NT / 32;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const float wm = warp_max(a.c);
  const float f = a.c == -INFINITY ? 0.f : exp2f(a.c - wm);
  const float2 v = warp_pair_sum(make_float2(a.s * f, 0.f));
  if (lane == 0) {
    r.c[wid] = wm;
    r.s[wid] = v;
  }
  __syncthreads();
  if (wid == 0) {
    const float cw = lane < NW ? r.c[lane] : -INFINITY;
    const float cm = warp_max(cw);
    float2 w = make_float2(0.f, 0.f);
    if (lane < NW && cw != -INFINITY) {
      const float g = exp2f(cw - cm);
      const float2 p = r.s[lane];
      const float hi = p.x * g;
      w = make_float2(hi, fmaf(p.x, g, -hi) + p.y * g);
    }
    S = warp_pair_sum(w);
    C = cm;
  }
}

// ------------------------------------------------------ float-float scalars

// Per-row scalars (log-sum-exp, log-probabilities, log-ratios) are unevaluated
// sums hi + lo of two floats with |lo| <= ulp(hi) / 2: about 48 significant
// bits from float32 operations (Dekker 1971; Knuth, TAOCP vol. 2, 4.2.2, the
// same TwoSum as pair_add).  The row epilogue runs in one thread while the rest
// of the CTA waits, and a float64 instruction issues at a small fraction of the
// float32 rate on GB300: the float64 epilogue of the fused kernel took ~4700
// cycles per row.  Non-finite values carry lo = 0.
struct ff {
  float hi, lo;
};

// a + b = s + e exactly (TwoSum).
__device__ __forceinline__ ff ff_two_sum(float a, float b) {
  const float s = a + b;
  const float bp = s - a;
  const float e = (a - (s - bp)) + (b - bp);
  return {s, isfinite(s) ? e : 0.f};
}
__device__ __forceinline__ ff ff_neg(ff a) { return {-a.hi, -a.lo}; }
__device__ __forceinline__ ff ff_add(ff a, float b) {
  const ff s = ff_two_sum(a.hi, b);
  return ff_two_sum(s.hi, s.lo + a.lo);
}
__device__ __forceinline__ ff ff_sub(ff a, ff b) {
  const ff s = ff_two_sum(a.hi, -b.hi);
  return ff_two_sum(s.hi, s.lo + (a.lo - b.lo));
}
// a b with the exact error of hi * hi from one FMA.
__device__ __forceinline__ ff ff_mul(ff a, ff b) {
  const float p = a.hi * b.hi;
  const float e = fmaf(a.hi, b.hi, -p);
  return ff_two_sum(p, fmaf(a.hi, b.lo, fmaf(a.lo, b.hi, e)));
}
// a <= b for normalised pairs; false when either is NaN.
__device__ __forceinline__ bool ff_le(ff a, ff b) {
  return a.hi < b.hi || (a.hi == b.hi && a.lo <= b.lo);
}
__device__ __forceinline__ float ff_round(ff a) { return a.hi + a.lo; }

// 1 / float(log2 e) as a float-float constant.
constexpr float kInvLog2eHi = (float)kInvLog2eF;
constexpr float kInvLog2eLo = (float)(kInvLog2eF - (double)kInvLog2eHi);

// Row epilogue: log2 of the row's sum of exponentials from the merged (C, S),
// in the base-2 units of the terms 2^(z L - C), L = float(log2 e).
__device__ __forceinline__ ff lse2_from(float C, float2 S) {
  if (!(S.x > 0.f)) return {(S.x == 0.f) ? -INFINITY : __int_as_float(0x7fc00000), 0.f};
  int e;
  const float f = frexpf(S.x, &e);  // S.x = f 2^e, f in [0.5, 1)
  ff l = ff_two_sum(C, (float)e);
  l = ff_add(l, log2f(f));
  return ff_add(l, __fdividef(S.y, S.x) * 1.4426950408889634f);  // a correction ~1e-8 of S.x
}
// The natural-log lse: the base-2 value divided by that same L keeps the error
// at float(log2 e)'s relative error times the row entropy.
__device__ __forceinline__ ff lse_nat(ff l2) { return ff_mul(l2, ff{kInvLog2eHi, kInvLog2eLo}); }

}  // namespace occ
