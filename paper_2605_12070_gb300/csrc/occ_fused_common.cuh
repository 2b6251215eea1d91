// Shared by the fused loss kernels (occ_fused.cu): their
// arguments and the per-token epilogue that turns the two merged rows into
// log pi_old, log pi_theta, the Eq. 2-4 decisions and the backward scale.
#pragma once

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

// What the per-token outputs need after the backward pass's scalars are out.
struct FusedTok {
  ff lse, lse_old, logp_old;
  float loss_t, logp_f;
  uint32_t flags;
};

// Warp 0, after the CTA merge (C, S valid in every lane): lanes 0 and 1 form
// the current and the old row's log-sum-exp side by side, then lane 0 the
// token scalars and the backward pass's (g, cb).  Only what the backward pass
// waits for is done here; the outputs follow in fused_token_outputs.
__device__ __forceinline__ void fused_token_epilogue(const FusedArgs& f, const float (&C)[2],
                                                     const float2 (&S)[2], float zy, float zyo,
                                                     float lpm, float A, long long N, int lane,
                                                     float& g, float& cb, FusedTok& tk) {
  const bool old_row = lane == 1;
  const ff l2 = lse2_from(old_row ? C[1] : C[0], old_row ? S[1] : S[0]);
  const ff l = lse_nat(l2);
  const ff lo = {__shfl_sync(0xffffffffu, l.hi, 1), __shfl_sync(0xffffffffu, l.lo, 1)};
  if (lane != 0) return;
  tk.lse = l;
  tk.lse_old = lo;
  tk.logp_old = ff_add(ff_neg(lo), zyo);
  token_math(f.a.kp, l, zy, tk.logp_old, lpm, A, N, g, tk.loss_t, tk.flags, tk.logp_f);
  cb = backward_offset(l2, g);
}

// Thread 0, while the CTA writes dlogits: the per-token outputs.
__device__ __forceinline__ void fused_token_outputs(const FusedArgs& f, int64_t row,
                                                    const FusedTok& tk, const float2 (&S)[2],
                                                    const float (&SV)[2]) {
  const K2Args& a = f.a;
  a.ws_loss[row] = tk.loss_t;
  a.ws_flags[row] = (uint8_t)tk.flags;
  if (a.logp_out) a.logp_out[row] = tk.logp_f;
  if (a.flags_out) a.flags_out[row] = (uint8_t)tk.flags;
  if (f.logp_old_out) f.logp_old_out[row] = ff_round(tk.logp_old);
  if (f.entropy_out) {  // H = lse - E_p[z]
    const float ez = SV[0] / (S[0].x + S[0].y);
    f.entropy_out[row] = ff_round(ff_add(tk.lse, -ez));
  }
  if (f.kl_out) {  // KL = E_{p_old}[z_old - z] - lse_old + lse
    const float ed = SV[1] / (S[1].x + S[1].y);
    f.kl_out[row] = ff_round(ff_add(ff_sub(tk.lse, tk.lse_old), ed));
  }
}

}  // namespace occ
