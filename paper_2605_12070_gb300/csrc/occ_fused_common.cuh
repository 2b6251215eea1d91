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

}  // namespace occ
