// Device-side bounds checks of the debug build.
//
// Compiled with -DROSETTA_DEBUG, dbg_ok(cond, flag) records a failed check
// in the context's error flag (value 3, reported by rosetta_sync_status as
// ROSETTA_ERR_BOUNDS) and returns false so that the caller skips the access;
// no check traps or stops the kernel, so the GPU context stays usable.  In
// the regular build it is the constant true and costs nothing.
#pragma once
#include <stdint.h>

namespace rosetta {

constexpr uint32_t kErrFlagBounds = 3u;

#ifdef ROSETTA_DEBUG
__device__ __forceinline__ bool dbg_ok(bool ok, uint32_t *flag) {
  if (!ok && flag) atomicExch(flag, kErrFlagBounds);
  return ok;
}
#else
__device__ __forceinline__ constexpr bool dbg_ok(bool, uint32_t *) { return true; }
#endif

}  // namespace rosetta
