// Status strings, per-thread error messages and device queries of the occ C ABI.
#include <stdarg.h>
#include <stdio.h>

#include <atomic>
#include <mutex>

#include "occ_internal.h"

namespace occ {

static thread_local char g_msg[512] = "";
static thread_local const char* g_kernel = "";

occ_status fail(occ_status s, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_msg, sizeof(g_msg), fmt, ap);
  va_end(ap);
  return s;
}

void clear_error() {
  g_msg[0] = '\0';
  g_kernel = "";
}

void note_kernel(const char* name) { g_kernel = name; }

occ_status check_launch(const char* what) {
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return fail(OCC_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
  return OCC_OK;
}

static std::atomic<int64_t> g_options[OCC_OPT_COUNT_] = {};
static std::once_flag g_options_once;

static void options_init() {
  std::call_once(g_options_once, [] {
    for (auto& o : g_options) o.store(-1);
  });
}

int64_t option(occ_option opt) {
  options_init();
  return (opt >= 0 && opt < OCC_OPT_COUNT_) ? g_options[opt].load(std::memory_order_relaxed) : -1;
}

static bool option_value_ok(occ_option opt, int64_t v) {
  if (v == -1) return true;
  switch (opt) {
    case OCC_OPT_K1_WARP:
    case OCC_OPT_FUSED_TMEM:
    case OCC_OPT_K2_TMEM: return v == 0 || v == 1;
    case OCC_OPT_K1_THREADS:
    case OCC_OPT_K2_THREADS:
    case OCC_OPT_FUSED_THREADS: return v == 128 || v == 256 || v == 512;
    case OCC_OPT_K2_UNROLL: return v == 4 || v == 6 || v == 8;
    case OCC_OPT_K2_HEAD_BYTES:
    case OCC_OPT_FUSED_HEAD_BYTES: return v >= 0 && v <= 227 * 1024 && v % 16 == 0;
    default: return false;
  }
}

int sm_count() {
  static int cached[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 1;
  if (dev >= 0 && dev < 64 && cached[dev]) return cached[dev];
  int n = 1;
  cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  if (dev >= 0 && dev < 64) cached[dev] = n;
  return n;
}

size_t two_cta_smem_budget(const void* kern) {
  constexpr size_t kPerCta = (164 - 1) * 1024 / 2;
  cudaFuncAttributes fa;
  if (cudaFuncGetAttributes(&fa, kern) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  int dev = 0, reserve = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&reserve, cudaDevAttrReservedSharedMemoryPerBlock, dev) !=
          cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  const size_t fixed = ((fa.sharedSizeBytes + 127) & ~(size_t)127) + (size_t)reserve;
  return fixed < kPerCta ? ((kPerCta - fixed) & ~(size_t)511) : 0;
}

}  // namespace occ

extern "C" {

const char* occ_status_string(occ_status s) {
  switch (s) {
    case OCC_OK: return "ok";
    case OCC_ERR_INVALID_ARG: return "invalid argument";
    case OCC_ERR_UNSUPPORTED: return "unsupported dtype or size";
    case OCC_ERR_MISALIGNED: return "misaligned pointer";
    case OCC_ERR_CUDA: return "CUDA error";
    case OCC_ERR_WORKSPACE: return "workspace missing or too small";
  }
  return "unknown status";
}

const char* occ_last_error(void) { return occ::g_msg; }

const char* occ_last_kernel(void) { return occ::g_kernel; }

int occ_version(void) { return OCC_VERSION; }

occ_status occ_set_option(occ_option opt, int64_t value) {
  occ::clear_error();
  if (opt < 0 || opt >= OCC_OPT_COUNT_ || !occ::option_value_ok(opt, value))
    return occ::fail(OCC_ERR_INVALID_ARG, "option %d does not take the value %lld", (int)opt,
                     (long long)value);
  occ::options_init();
  occ::g_options[opt].store(value, std::memory_order_relaxed);
  return OCC_OK;
}

int64_t occ_get_option(occ_option opt) { return occ::option(opt); }

}  // extern "C"
