// Pinned host buffers backed by transparent huge pages.
//
// The inputs of an end-to-end step (both logits tensors, the token arrays and
// the actor parameters: tens of GB) cross the host link every step.  On the
// Grace hosts of GB300 a copy that streams through tens of GB of pinned memory
// spends its time on address translation when the buffer is mapped with base
// pages: cudaHostAlloc memory moved ~100-110 GB/s over a 70 GB working set on
// one box, while the same bytes in huge pages moved ~165 GB/s.  occ_host_alloc
// maps anonymous memory aligned to the transparent-huge-page size (buffers
// smaller than one huge page: to the base page), asks the
// kernel for huge pages (madvise; a kernel that declines gives base pages and
// the buffer still works) and pins it with cudaHostRegister, so device copies
// from it are asynchronous DMA like those from cudaHostAlloc memory.
#include <stdio.h>
#include <sys/mman.h>
#include <unistd.h>

#include "occ_internal.h"

namespace occ {

// Transparent-huge-page size of this host (bytes), else 2 MiB.
static size_t thp_size() {
  static const size_t sz = [] {
    size_t v = 0;
    if (FILE* f = fopen("/sys/kernel/mm/transparent_hugepage/hpage_pmd_size", "r")) {
      unsigned long long x = 0;
      if (fscanf(f, "%llu", &x) == 1) v = (size_t)x;
      fclose(f);
    }
    const size_t page = (size_t)sysconf(_SC_PAGESIZE);
    if (v < page || (v & (v - 1)) != 0) v = (size_t)2 << 20;
    return v;
  }();
  return sz;
}

static size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Granule of a buffer of `bytes`: the huge-page size once the buffer fills at
// least one huge page, else the base page (a small buffer gains nothing from
// huge pages and would pin a whole one).
static size_t granule(size_t bytes) {
  return bytes >= thp_size() ? thp_size() : (size_t)sysconf(_SC_PAGESIZE);
}

}  // namespace occ

using namespace occ;

extern "C" occ_status occ_host_alloc(size_t bytes, void** out) {
  clear_error();
  if (!out) return fail(OCC_ERR_INVALID_ARG, "null output pointer");
  *out = nullptr;
  if (bytes == 0) return fail(OCC_ERR_INVALID_ARG, "bytes == 0");
  const size_t align = granule(bytes);
  const size_t len = round_up(bytes, align);
  if (len < bytes || len + align < len) return fail(OCC_ERR_INVALID_ARG, "size overflow");
  // over-map by one granule and trim, so that the buffer starts on a boundary
  void* raw = mmap(nullptr, len + align, PROT_READ | PROT_WRITE, MAP_PRIVATE | MAP_ANONYMOUS, -1, 0);
  if (raw == MAP_FAILED) return fail(OCC_ERR_INVALID_ARG, "mmap of %zu bytes failed", len + align);
  const uintptr_t base = (uintptr_t)raw;
  const uintptr_t start = round_up(base, align);
  if (start > base) munmap(raw, start - base);
  const size_t tail = (base + len + align) - (start + len);
  if (tail > 0) munmap((void*)(start + len), tail);
  void* p = (void*)start;
  madvise(p, len, MADV_HUGEPAGE);  // advisory: base pages if the kernel declines
  // Fault the range in from the CPU, one write per huge page, before pinning:
  // a first-touch fault in an advised range takes a whole huge page, while the
  // pages the driver faults in while registering are base pages.
  for (size_t off = 0; off < len; off += align) static_cast<volatile char*>(p)[off] = 0;
  const cudaError_t e = cudaHostRegister(p, len, cudaHostRegisterDefault);
  if (e != cudaSuccess) {
    cudaGetLastError();
    munmap(p, len);
    return fail(OCC_ERR_CUDA, "cudaHostRegister(%zu bytes): %s", len, cudaGetErrorString(e));
  }
  *out = p;
  return OCC_OK;
}

extern "C" occ_status occ_host_free(void* ptr, size_t bytes) {
  clear_error();
  if (!ptr) return OCC_OK;
  if (bytes == 0) return fail(OCC_ERR_INVALID_ARG, "bytes == 0");
  const size_t align = granule(bytes);
  if ((uintptr_t)ptr % align != 0)
    return fail(OCC_ERR_INVALID_ARG, "pointer was not returned by occ_host_alloc");
  const size_t len = round_up(bytes, align);
  const cudaError_t e = cudaHostUnregister(ptr);
  munmap(ptr, len);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return fail(OCC_ERR_CUDA, "cudaHostUnregister: %s", cudaGetErrorString(e));
  }
  return OCC_OK;
}
