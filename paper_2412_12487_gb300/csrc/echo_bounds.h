// echo_bounds.h -- the index checks of the debug-bounds mode (echo_compose_opts
// debug_bounds).  Every index a composition kernel reads from the graph's index
// arrays (records, programs, candidate and comm lists) is checked with these
// before the access it addresses; a failed check records kDevBounds in the
// status word and the access is skipped, so a bad index never faults the device.
// The header has no CUDA dependency of its own, so the same predicates compile
// for the host and are unit-tested on the CPU.
#pragma once

#include <stdint.h>

#if defined(__CUDACC__)
#define ECHO_HD __host__ __device__ __forceinline__
#else
#define ECHO_HD inline
#endif

namespace echo {

// i is an element of [0, n)
ECHO_HD bool in_range(int64_t i, int64_t n) { return i >= 0 && i < n; }

// [lo, hi) is a (possibly empty) sub-range of [0, n)
ECHO_HD bool range_ok(int64_t lo, int64_t hi, int64_t n) { return 0 <= lo && lo <= hi && hi <= n; }

// the k-th set bit below position t of a 64-bit chain mask, counted from a first
// index `first`, is an element of [0, n): the compact row of a masked chain position
ECHO_HD bool masked_row_ok(int64_t first, uint64_t mask, int64_t n) {
  int64_t bits = 0;
  for (uint64_t m = mask; m; m &= m - 1) ++bits;
  return bits == 0 || range_ok(first, first + bits, n);
}

}  // namespace echo
