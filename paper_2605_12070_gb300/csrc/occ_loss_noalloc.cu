// occ_decoupled_loss_fwd_bwd_noalloc: the decoupled loss for callers that
// cannot hand the library a scratch buffer.
//
// Some callers have no way to obtain device memory of their own: a plain C
// plugin loaded into a framework whose caching allocator owns all of the
// GPU's memory, or a latency-critical loop that must not call cudaMalloc /
// cudaFree (both can synchronize the device).  This entry point takes the
// same inputs and outputs as occ_decoupled_loss_fwd_bwd but finds its scratch
// in a fixed-size array that lives in this library's device globals, so the
// caller allocates nothing and the library allocates nothing either.
//
// The array is a file-scope __device__ variable.  Its name, used in host
// code, is only a host-side stand-in for the symbol, not a device address, so
// the device address is looked up once per device with cudaGetSymbolAddress
// (with that device current) and then passed to the kernels like any other
// workspace pointer.
#include <atomic>
#include <mutex>

#include "occ_internal.h"

#define OCC_NOALLOC_SCRATCH_BYTES (4u << 20)

static __device__ __align__(256) unsigned char g_noalloc_scratch[OCC_NOALLOC_SCRATCH_BYTES];

namespace {

constexpr int kMaxDevices = 64;
std::atomic<void*> g_scratch_ptr[kMaxDevices];  // null until resolved on that device
std::mutex g_scratch_mu;

// The device address of the scratch array on the current device `dev`.  A
// failed lookup (for instance inside a stream capture) is not cached: the
// next call tries again.
cudaError_t scratch_on(int dev, void** out) {
  void* ptr = g_scratch_ptr[dev].load(std::memory_order_acquire);
  if (!ptr) {
    std::lock_guard<std::mutex> lk(g_scratch_mu);
    ptr = g_scratch_ptr[dev].load(std::memory_order_relaxed);
    if (!ptr) {
      const cudaError_t e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
      if (e != cudaSuccess || !ptr) {
        cudaGetLastError();
        return e != cudaSuccess ? e : cudaErrorInvalidSymbol;
      }
      g_scratch_ptr[dev].store(ptr, std::memory_order_release);
    }
  }
  *out = ptr;
  return cudaSuccess;
}

}  // namespace

using namespace occ;

extern "C" occ_status occ_decoupled_loss_fwd_bwd_noalloc(
    const void* logits, occ_dtype dt, int64_t T, int64_t V, int64_t ld, const int32_t* ids,
    const float* logp_old, const float* logp_mu, const float* adv, const uint8_t* loss_mask,
    const occ_loss_params* p, float* logp_out, uint8_t* flags_out, void* dlogits,
    int64_t ld_grad, occ_loss_stats* stats, void* stream) {
  clear_error();
  if (!p) return fail(OCC_ERR_INVALID_ARG, "params pointer is null");
  if (T < 0) return fail(OCC_ERR_INVALID_ARG, "need T >= 0 (T=%lld)", (long long)T);
  if (T > OCC_NOALLOC_MAX_TOKENS || occ_loss_workspace_bytes(T, V) > OCC_NOALLOC_SCRATCH_BYTES)
    return fail(OCC_ERR_UNSUPPORTED,
                "occ_decoupled_loss_fwd_bwd_noalloc handles at most %d tokens per call "
                "(got T=%lld); split the batch or use occ_decoupled_loss_fwd_bwd",
                OCC_NOALLOC_MAX_TOKENS, (long long)T);
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(OCC_ERR_CUDA, "cudaGetDevice: %s", cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices)
    return fail(OCC_ERR_UNSUPPORTED, "device ordinal %d >= %d", dev, kMaxDevices);
  // The scratch array used is the current device's: the logits must live there.
  if (T > 0 && logits) {
    cudaPointerAttributes attr;
    e = cudaPointerGetAttributes(&attr, logits);
    if (e != cudaSuccess) {
      cudaGetLastError();
      return fail(OCC_ERR_INVALID_ARG, "cudaPointerGetAttributes(logits): %s",
                  cudaGetErrorString(e));
    }
    if (attr.type == cudaMemoryTypeDevice && attr.device != dev)
      return fail(OCC_ERR_INVALID_ARG,
                  "logits are on device %d but device %d is current; make the device that "
                  "holds the arguments current before the call", attr.device, dev);
  }
  void* scratch = nullptr;
  e = scratch_on(dev, &scratch);
  if (e != cudaSuccess)
    return fail(OCC_ERR_CUDA, "cudaGetSymbolAddress(scratch) on device %d: %s", dev,
                cudaGetErrorString(e));
  return occ_decoupled_loss_fwd_bwd(logits, dt, T, V, ld, ids, logp_old, logp_mu, adv, loss_mask,
                                    p, logp_out, flags_out, dlogits, ld_grad, stats, scratch,
                                    OCC_NOALLOC_SCRATCH_BYTES, stream);
}
