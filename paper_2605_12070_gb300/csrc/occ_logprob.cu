// K1: vocabulary-streaming log-sum-exp and sampled-token log-probability.
//
// log pi(y_t) = z[t, y_t] - log sum_v exp(z[t, v]) for each row t: the per-token
// factors of the ratios in Eq. 1 (used for pi_old, pi_prox of Eq. 5 or
// pi_async of Table 1).  One CTA (or, for rows of up to 32 KB, one warp)
// streams one row with 16-byte coalesced loads, U vectors in flight per
// thread, and keeps an online (c, s) pair per thread; nothing is staged in
// shared memory because each element is used once.
// HBM traffic is the logits row once: V * sizeof(T) bytes per token.
#include <algorithm>
#include <cstdlib>

#include "occ_common.cuh"

namespace occ {

constexpr int kK1Threads = 512;
constexpr int kK1Unroll = 8;

// PEEL: rows need not start on a 16-byte boundary.  Each row then takes its
// first `lead` elements (up to the boundary) and its last few with scalar
// loads and the aligned body with the vector loop.
template <typename Tin, int NT, int U, bool PEEL>
__global__ void __launch_bounds__(NT, 1024 / NT)
    k1_logprob_vec(const Tin* __restrict__ logits, int64_t T, int64_t V, int64_t ld,
                   const int32_t* __restrict__ ids, float* __restrict__ logp,
                   float* __restrict__ lse_out) {
  constexpr int VEC = Elem<Tin>::kVec;
  __shared__ RedScratch red;
  for (int64_t row = blockIdx.x; row < T; row += gridDim.x) {
    const Tin* z0 = logits + row * ld;
    const int64_t lead =
        PEEL ? min(V, (int64_t)(((16 - ((uintptr_t)z0 & 15)) & 15) / sizeof(Tin))) : 0;
    const Tin* z = z0 + lead;  // 16-byte aligned
    const int64_t nvec = (V - lead) / VEC;
    const int64_t tail0 = nvec * VEC;  // relative to z
    int id = 0;
    float zy = 0.f;
    if (threadIdx.x == 0) {
      id = ids[row];
      if (id >= 0 && id < V) zy = Elem<Tin>::load(z0 + id);
    }
    LseAcc acc;
    acc_init(acc);
    const uint4* zv = reinterpret_cast<const uint4*>(z);
    // Row walk: full rounds, then one round whose loads issue together (GB300:
    // 0.652 -> 0.603 ms at V = 32000 bf16 against one load at a time).
    walk_row<Walk::kTailRound, U, NT>(
        threadIdx.x, (int)nvec, [&](int j) { return ld_stream_v4(zv + j); },
        [&](int, const uint4& r) {
          float x[VEC];
          Elem<Tin>::unpack(r, x);
          acc_add(acc, x);
        });
    if ((int64_t)threadIdx.x < V - lead - tail0) {
      float x[1] = {Elem<Tin>::load(z + tail0 + threadIdx.x)};
      acc_add(acc, x);
    }
    if (PEEL && (int64_t)threadIdx.x < lead) {
      float x[1] = {Elem<Tin>::load(z0 + threadIdx.x)};
      acc_add(acc, x);
    }
    float C;
    float2 S;
    block_lse<NT>(acc, red, C, S);
    if (threadIdx.x == 0) {
      const ff l = lse_nat(lse2_from(C, S));
      logp[row] = (id >= 0 && id < V) ? ff_round(ff_add(ff_neg(l), zy)) : __int_as_float(0x7fc00000);
      if (lse_out) lse_out[row] = ff_round(l);
    }
    __syncthreads();
  }
}

// One warp per row: the same streaming pass, merged with warp shuffles only,
// so a row costs no CTA barrier and the lane-0 epilogue stalls one warp, not a
// whole CTA.  Rows are dealt to warps round-robin over the grid.
template <typename Tin, int NT, int U, bool PEEL>
__global__ void __launch_bounds__(NT, 1024 / NT)
    k1_logprob_warp(const Tin* __restrict__ logits, int64_t T, int64_t V, int64_t ld,
                    const int32_t* __restrict__ ids, float* __restrict__ logp,
                    float* __restrict__ lse_out) {
  constexpr int VEC = Elem<Tin>::kVec;
  constexpr int NW = NT / 32;
  const int lane = threadIdx.x & 31;
  const int64_t warp0 = (int64_t)blockIdx.x * NW + (threadIdx.x >> 5);
  const int64_t nwarps = (int64_t)gridDim.x * NW;
  for (int64_t row = warp0; row < T; row += nwarps) {
    const Tin* z0 = logits + row * ld;
    const int64_t lead =
        PEEL ? min(V, (int64_t)(((16 - ((uintptr_t)z0 & 15)) & 15) / sizeof(Tin))) : 0;
    const Tin* z = z0 + lead;  // 16-byte aligned
    const int64_t nvec = (V - lead) / VEC;
    const int64_t tail0 = nvec * VEC;  // relative to z
    LseAcc acc;
    acc_init(acc);
    const uint4* zv = reinterpret_cast<const uint4*>(z);
    walk_row<Walk::kTailRound, U, 32>(
        lane, (int)nvec, [&](int j) { return ld_stream_v4(zv + j); },
        [&](int, const uint4& r) {
          float x[VEC];
          Elem<Tin>::unpack(r, x);
          acc_add(acc, x);
        });
    if ((int64_t)lane < V - lead - tail0) {
      float x[1] = {Elem<Tin>::load(z + tail0 + lane)};
      acc_add(acc, x);
    }
    if (PEEL && (int64_t)lane < lead) {
      float x[1] = {Elem<Tin>::load(z0 + lane)};
      acc_add(acc, x);
    }
    const float C = warp_max(acc.c);
    const float2 S = warp_pair_sum(
        make_float2((acc.c == -INFINITY) ? 0.f : acc.s * exp2f(acc.c - C), 0.f));
    if (lane == 0) {
      const int id = ids[row];
      const bool ok = id >= 0 && id < V;
      const float zy = ok ? Elem<Tin>::load(z0 + id) : 0.f;
      const ff l = lse_nat(lse2_from(C, S));
      logp[row] = ok ? ff_round(ff_add(ff_neg(l), zy)) : __int_as_float(0x7fc00000);
      if (lse_out) lse_out[row] = ff_round(l);
    }
  }
}

// Any alignment: element loads, consecutive threads on consecutive columns.
template <typename Tin, int NT>
__global__ void __launch_bounds__(NT)
    k1_logprob_scalar(const Tin* __restrict__ logits, int64_t T, int64_t V, int64_t ld,
                      const int32_t* __restrict__ ids, float* __restrict__ logp,
                      float* __restrict__ lse_out) {
  __shared__ RedScratch red;
  for (int64_t row = blockIdx.x; row < T; row += gridDim.x) {
    const Tin* z = logits + row * ld;
    int id = 0;
    float zy = 0.f;
    if (threadIdx.x == 0) {
      id = ids[row];
      if (id >= 0 && id < V) zy = Elem<Tin>::load(z + id);
    }
    LseAcc acc;
    acc_init(acc);
    for (int64_t v0 = threadIdx.x; v0 < V; v0 += 8 * (int64_t)NT) {
      float x[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int64_t v = v0 + (int64_t)j * NT;
        x[j] = v < V ? Elem<Tin>::load(z + v) : -INFINITY;
      }
      acc_add(acc, x);
    }
    float C;
    float2 S;
    block_lse<NT>(acc, red, C, S);
    if (threadIdx.x == 0) {
      const ff l = lse_nat(lse2_from(C, S));
      logp[row] = (id >= 0 && id < V) ? ff_round(ff_add(ff_neg(l), zy)) : __int_as_float(0x7fc00000);
      if (lse_out) lse_out[row] = ff_round(l);
    }
    __syncthreads();
  }
}

template <typename Tin>
static void launch_k1(const void* logits, int64_t T, int64_t V, int64_t ld, const int32_t* ids,
                      float* logp, float* lse, bool vec, cudaStream_t s) {
  const unsigned grid = (unsigned)(T < 0x7fffffffLL ? T : 0x7fffffffLL);
  const int64_t nt_opt = option(OCC_OPT_K1_THREADS);
  if (vec || V >= 16 * Elem<Tin>::kVec) {
    // Row-size tiers (measured on GB300, V = 4096 to 151936): rows up to 32 KB
    // one warp each (V = 8192 bf16: 0.64 against 0.88 ms with 128-thread CTAs:
    // short rows spend much of a CTA's time in its barriers), then CTAs of 128
    // threads up to ~96 KB and 256 beyond (512 left 2-50 % on the table).
    // Rows that are not 16-byte aligned run peeled (scalar head and tail).
    // The options OCC_OPT_K1_WARP (1 / 0) and OCC_OPT_K1_THREADS override.
    const int64_t row_bytes = (V / Elem<Tin>::kVec) * 16;
    const int nt = nt_opt > 0 ? (int)nt_opt : (row_bytes <= 96 * 1024 ? 128 : 256);
    const Tin* z = (const Tin*)logits;
    const int64_t warp_opt = option(OCC_OPT_K1_WARP);
    if (warp_opt == 1 || (warp_opt < 0 && row_bytes <= 32 * 1024)) {
      constexpr int NTW = 256;  // 8 warps, 4 CTAs per SM
      const int64_t want = (T + NTW / 32 - 1) / (NTW / 32);
      const unsigned gw = (unsigned)std::min<int64_t>(want, (int64_t)sm_count() * (1024 / NTW));
      note_kernel(vec ? "k1_logprob_warp" : "k1_logprob_warp/peel");
      if (vec)
        k1_logprob_warp<Tin, NTW, kK1Unroll, false><<<gw, NTW, 0, s>>>(z, T, V, ld, ids, logp, lse);
      else
        k1_logprob_warp<Tin, NTW, kK1Unroll, true><<<gw, NTW, 0, s>>>(z, T, V, ld, ids, logp, lse);
      return;
    }
#define OCC_K1_LAUNCH(NT_, PEEL_) \
  k1_logprob_vec<Tin, NT_, kK1Unroll, PEEL_><<<grid, NT_, 0, s>>>(z, T, V, ld, ids, logp, lse)
    note_kernel(vec ? "k1_logprob_vec" : "k1_logprob_vec/peel");
    if (nt == 128) {
      if (vec) OCC_K1_LAUNCH(128, false); else OCC_K1_LAUNCH(128, true);
    } else if (nt == 256) {
      if (vec) OCC_K1_LAUNCH(256, false); else OCC_K1_LAUNCH(256, true);
    } else {
      if (vec) OCC_K1_LAUNCH(kK1Threads, false); else OCC_K1_LAUNCH(kK1Threads, true);
    }
#undef OCC_K1_LAUNCH
  } else {
    note_kernel("k1_logprob_scalar");
    k1_logprob_scalar<Tin, kK1Threads><<<grid, kK1Threads, 0, s>>>((const Tin*)logits, T, V, ld,
                                                                    ids, logp, lse);
  }
}

}  // namespace occ

using namespace occ;

extern "C" occ_status occ_token_logprob(const void* logits, occ_dtype dt, int64_t T, int64_t V,
                                        int64_t ld, const int32_t* ids, float* logp_out,
                                        float* lse_out, void* stream) {
  clear_error();
  if (dt != OCC_F32 && dt != OCC_BF16) return fail(OCC_ERR_UNSUPPORTED, "dtype %d", (int)dt);
  if (T < 0 || V < 1 || ld < V)
    return fail(OCC_ERR_INVALID_ARG, "need T >= 0, V >= 1, ld >= V (T=%lld V=%lld ld=%lld)",
                (long long)T, (long long)V, (long long)ld);
  if (V > 0x7fffffffLL)  // token ids are int32; row-local indices are 32-bit
    return fail(OCC_ERR_UNSUPPORTED, "V = %lld exceeds 2^31 - 1", (long long)V);
  if (T == 0) return OCC_OK;
  if (!logits || !ids || !logp_out) return fail(OCC_ERR_INVALID_ARG, "null logits/ids/logp_out");
  const size_t es = dtype_size(dt);
  if (!aligned(logits, es) || !aligned(ids, 4) || !aligned(logp_out, 4) ||
      (lse_out && !aligned(lse_out, 4)))
    return fail(OCC_ERR_MISALIGNED, "arrays must be aligned to their element size");
  const bool vec = aligned(logits, 16) && ((ld * (int64_t)es) % 16 == 0);
  cudaStream_t s = (cudaStream_t)stream;
  if (dt == OCC_BF16)
    launch_k1<bf16_t>(logits, T, V, ld, ids, logp_out, lse_out, vec, s);
  else
    launch_k1<float>(logits, T, V, ld, ids, logp_out, lse_out, vec, s);
  return check_launch("occ_token_logprob");
}
