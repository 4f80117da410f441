// echo_slowdown.cuh -- the duration of an overlapped kernel in the next composition
// (Sec. 2.3: its time grows by its slowdown factor).  Both forms are fp64 with
// explicit round-to-nearest-even steps and no contraction, so they equal the
// oracle's llrint of the same fp64 expression bit for bit.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>

namespace echo {
namespace dev {

// Whole-kernel model: rint(fl(fl(d) * factor)).
__device__ __forceinline__ int64_t slowed(int64_t d, double factor) {
  return __double2ll_rn(__dmul_rn(__ll2double_rn(d), factor));
}

// Proportional model: rint(d + (factor - 1) * len), left to right.
__device__ __forceinline__ int64_t slowed_proportional(int64_t d, double factor, int64_t len) {
  return __double2ll_rn(__dadd_rn(__ll2double_rn(d), __dmul_rn(__dsub_rn(factor, 1.0), __ll2double_rn(len))));
}

}  // namespace dev
}  // namespace echo
