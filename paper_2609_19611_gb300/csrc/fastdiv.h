// Division by a run-time constant with one multiply: the quotient of a
// dividend below 2^31 by d is umulhi(x, m) >> s, with m and s from
// Granlund and Montgomery's round-up method for 31-bit dividends
// (l = ceil(log2 d), m = ceil(2^(31 + l) / d) < 2^32, s = l - 1); m = 0
// stands for d = 1.  Host and device; the host form is what the tests
// check against integer division.
#pragma once

#include <cstdint>

#if defined(__CUDACC__)
#define DIRIGO_FD_HD __host__ __device__
#else
#define DIRIGO_FD_HD
#endif

namespace dirigo {

inline void fast_div_make(int64_t d, uint32_t* m, uint32_t* sh) {
  if (d <= 1) {
    *m = 0;
    *sh = 0;
    return;
  }
  int l = 0;
  while ((1ll << l) < d) ++l;
  *m = (uint32_t)(((1ull << (31 + l)) + (uint64_t)d - 1) / (uint64_t)d);
  *sh = (uint32_t)(l - 1);
}

DIRIGO_FD_HD inline uint32_t fast_div(uint32_t x, uint32_t m, uint32_t sh) {
#if defined(__CUDA_ARCH__)
  return m ? (__umulhi(x, m) >> sh) : x;
#else
  return m ? (uint32_t)(((uint64_t)x * m) >> 32) >> sh : x;
#endif
}

}  // namespace dirigo
