/*
 * A plain C caller of the occ C ABI (include/occ.h): no PyTorch, device memory
 * from cudaMalloc, the default stream.  It reads a seeded problem written by
 * tests/test_gpu_c_abi.py, runs
 *   occ_token_logprob            (log pi_old from the old logits),
 *   occ_decoupled_loss_fwd_bwd   (loss, flags, dlogits),
 *   occ_ewma_update              (one PPO-EWMA step with the auto-reset input),
 * and writes the outputs next to the inputs for the test to compare with the
 * oracle.
 *
 * usage: c_abi_caller DIR T V N_PARAMS
 *   DIR/z.f32 z_old.f32 [T*V]  ids.i32 [T]  lmu.f32 adv.f32 [T]  mask.u8 [T]
 *   DIR/theta.f32 theta_prox.f32 [N_PARAMS]
 * writes DIR/logp_old.f32 logp.f32 [T] flags.u8 [T] dlogits.f32 [T*V]
 *        stats.bin (64 bytes) theta_prox_out.f32 [N_PARAMS]
 */
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "occ.h"

static void* read_file(const char* dir, const char* name, size_t bytes) {
  char path[1024];
  snprintf(path, sizeof path, "%s/%s", dir, name);
  FILE* f = fopen(path, "rb");
  if (!f) { fprintf(stderr, "cannot open %s\n", path); exit(2); }
  void* p = malloc(bytes ? bytes : 1);
  if (bytes && fread(p, 1, bytes, f) != bytes) { fprintf(stderr, "short read %s\n", path); exit(2); }
  fclose(f);
  return p;
}

static void write_file(const char* dir, const char* name, const void* p, size_t bytes) {
  char path[1024];
  snprintf(path, sizeof path, "%s/%s", dir, name);
  FILE* f = fopen(path, "wb");
  if (!f || fwrite(p, 1, bytes, f) != bytes) { fprintf(stderr, "cannot write %s\n", path); exit(2); }
  fclose(f);
}

static void* to_device(const void* h, size_t bytes) {
  void* d = NULL;
  if (cudaMalloc(&d, bytes ? bytes : 16) != cudaSuccess) { fprintf(stderr, "cudaMalloc\n"); exit(3); }
  if (bytes) cudaMemcpy(d, h, bytes, cudaMemcpyHostToDevice);
  return d;
}

#define CHECK(call)                                                               \
  do {                                                                            \
    occ_status s_ = (call);                                                       \
    if (s_ != OCC_OK) {                                                           \
      fprintf(stderr, "%s: %s (%s)\n", #call, occ_status_string(s_), occ_last_error()); \
      return 4;                                                                   \
    }                                                                             \
  } while (0)

int main(int argc, char** argv) {
  if (argc != 5) { fprintf(stderr, "usage: %s DIR T V N_PARAMS\n", argv[0]); return 1; }
  const char* dir = argv[1];
  const int64_t T = atoll(argv[2]), V = atoll(argv[3]), n = atoll(argv[4]);
  const size_t tv = (size_t)T * (size_t)V;

  float* z = read_file(dir, "z.f32", tv * 4);
  float* zo = read_file(dir, "z_old.f32", tv * 4);
  int32_t* ids = read_file(dir, "ids.i32", (size_t)T * 4);
  float* lmu = read_file(dir, "lmu.f32", (size_t)T * 4);
  float* adv = read_file(dir, "adv.f32", (size_t)T * 4);
  uint8_t* mask = read_file(dir, "mask.u8", (size_t)T);
  float* th = read_file(dir, "theta.f32", (size_t)n * 4);
  float* tp = read_file(dir, "theta_prox.f32", (size_t)n * 4);

  void* d_z = to_device(z, tv * 4);
  void* d_zo = to_device(zo, tv * 4);
  int32_t* d_ids = to_device(ids, (size_t)T * 4);
  float* d_lmu = to_device(lmu, (size_t)T * 4);
  float* d_adv = to_device(adv, (size_t)T * 4);
  uint8_t* d_mask = to_device(mask, (size_t)T);
  float* d_th = to_device(th, (size_t)n * 4);
  float* d_tp = to_device(tp, (size_t)n * 4);
  float* d_lpo = to_device(NULL, (size_t)T * 4);
  float* d_lp = to_device(NULL, (size_t)T * 4);
  uint8_t* d_flags = to_device(NULL, (size_t)T);
  float* d_dz = to_device(NULL, tv * 4);
  occ_loss_stats* d_stats = to_device(NULL, sizeof(occ_loss_stats));
  occ_ewma_state* d_state = to_device(NULL, sizeof(occ_ewma_state));
  const size_t ws_bytes = occ_loss_workspace_bytes(T, V);
  void* d_ws = to_device(NULL, ws_bytes);

  occ_loss_params p;
  memset(&p, 0, sizeof p);
  p.rd_lo = 0.7;
  p.rd_hi = 1.4;
  p.eps_low = 0.2;
  p.eps_high = 0.28;
  p.grad_scale = 1.0;
  p.denom = 0;
  p.rd_weight = 1;
  p.dlogits_f32 = 1;
  p.proxy = OCC_PROXY_NONE;

  CHECK(occ_token_logprob(d_zo, OCC_F32, T, V, V, d_ids, d_lpo, NULL, NULL));
  CHECK(occ_decoupled_loss_fwd_bwd(d_z, OCC_F32, T, V, V, d_ids, d_lpo, d_lmu, d_adv, d_mask, &p,
                                   d_lp, d_flags, d_dz, V, d_stats, d_ws, ws_bytes, NULL));
  CHECK(occ_ewma_state_init(d_state, 1.0 / (1.0 - 0.75), NULL));
  CHECK(occ_ewma_update(d_tp, d_th, n, 0.75, d_state, d_stats, 0.5, 1, 0, NULL));
  if (cudaDeviceSynchronize() != cudaSuccess) { fprintf(stderr, "sync failed\n"); return 5; }

  float* out_f = malloc(tv * 4);
  cudaMemcpy(out_f, d_lpo, (size_t)T * 4, cudaMemcpyDeviceToHost);
  write_file(dir, "logp_old.f32", out_f, (size_t)T * 4);
  cudaMemcpy(out_f, d_lp, (size_t)T * 4, cudaMemcpyDeviceToHost);
  write_file(dir, "logp.f32", out_f, (size_t)T * 4);
  cudaMemcpy(out_f, d_dz, tv * 4, cudaMemcpyDeviceToHost);
  write_file(dir, "dlogits.f32", out_f, tv * 4);
  uint8_t* out_u8 = malloc((size_t)T);
  cudaMemcpy(out_u8, d_flags, (size_t)T, cudaMemcpyDeviceToHost);
  write_file(dir, "flags.u8", out_u8, (size_t)T);
  occ_loss_stats st;
  cudaMemcpy(&st, d_stats, sizeof st, cudaMemcpyDeviceToHost);
  write_file(dir, "stats.bin", &st, sizeof st);
  float* out_p = malloc((size_t)n * 4);
  cudaMemcpy(out_p, d_tp, (size_t)n * 4, cudaMemcpyDeviceToHost);
  write_file(dir, "theta_prox_out.f32", out_p, (size_t)n * 4);
  printf("occ %d: loss %.9g n_valid %lld n_active %lld\n", occ_version(), st.loss,
         (long long)st.n_valid, (long long)st.n_active);
  return 0;
}
