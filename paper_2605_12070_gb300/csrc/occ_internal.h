// Host-side helpers shared by the occ translation units (not part of the ABI).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "occ.h"

namespace occ {

// Records a printf-style message for occ_last_error() and returns `s`.
occ_status fail(occ_status s, const char* fmt, ...);
// Clears the message and the launched-kernel name of the calling thread.
void clear_error();
// Records `name` (a string literal) for occ_last_kernel().
void note_kernel(const char* name);
// Maps a CUDA error (after a launch) to OCC_ERR_CUDA with a message.
occ_status check_launch(const char* what);

inline bool aligned(const void* p, uintptr_t a) { return ((uintptr_t)p % a) == 0; }

// Byte ranges [a, a+na) and [b, b+nb) intersect.
inline bool overlaps(const void* a, size_t na, const void* b, size_t nb) {
  const uintptr_t x = (uintptr_t)a, y = (uintptr_t)b;
  return na && nb && x < y + nb && y < x + na;
}

inline size_t dtype_size(occ_dtype dt) { return dt == OCC_BF16 ? 2 : 4; }

// Current value of a tuning option (occ_set_option); -1 = automatic.
int64_t option(occ_option opt);

// Multiprocessor count of the current device (cached per device).
int sm_count();

// Dynamic shared memory with which two CTAs of `kern` stay in the 164 KB
// shared-memory carveout of an SM.  Past it the driver takes the 196 KB
// carveout and L1, which holds the loads in flight, shrinks from ~92 KB to
// ~60 KB (the fused kernel: 8.31 ms against 8.38 ms at V = 151936).  Measured
// on GB300 with byte steps: a CTA may take half of 163 KB, counting its static
// shared memory rounded up to 128 bytes and the per-CTA system reservation;
// the result is rounded down to 512 bytes for margin.  0 if a query fails.
size_t two_cta_smem_budget(const void* kern);

}  // namespace occ
