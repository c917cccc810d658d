// Device-side index checks of the bounds-checked build (-DBD_CHECKS, built by
// build.py as libbdcommit_checks.so). In that build an index outside its
// buffer skips the access and sets DEV_BOUNDS in the status word
// (bd_get_device_status then returns BD_ERR_BOUNDS); nothing traps. In the
// normal build every check is the constant true and compiles away.
#pragma once

#include <cstdint>

namespace bd {

constexpr uint32_t DEV_BOUNDS = 4u;

#ifdef BD_CHECKS
__device__ __forceinline__ bool index_ok(int64_t i, int64_t n, uint32_t* status) {
  if (i >= 0 && i < n) return true;
  if (status != nullptr) atomicOr(status, DEV_BOUNDS);
  return false;
}
#else
__device__ __forceinline__ bool index_ok(int64_t, int64_t, uint32_t*) { return true; }
#endif

}  // namespace bd
