// Division of a non-negative 31-bit integer by a divisor fixed at launch time, by one 64-bit
// multiplication and a shift (Granlund and Montgomery, "Division by invariant integers using
// multiplication", PLDI 1994, Theorem 4.2).  With L = ceil(log2 d) and m = floor(2^(31+L) / d) + 1:
//   2^(31+L) < m d <= 2^(31+L) + d <= 2^(31+L) + 2^L,
// so floor(n m / 2^(31+L)) = floor(n / d) for every 0 <= n < 2^31.  m < 2^33 and n < 2^31, so the
// product fits in 64 bits.
//
// The saliency kernel's per-tile bookkeeping uses this instead of the `/` operator: a runtime 32-bit
// division compiles to a conversion and reciprocal sequence on the same pipe as the exponentials, whose
// queue the epilogue keeps full, so every division in a hot loop waits behind it.
#pragma once

#include <stdint.h>

#if defined(__CUDACC__)
#define STEPKV_HD __host__ __device__ __forceinline__
#else
#define STEPKV_HD inline
#endif

namespace stepkv {

struct FastDiv {
  uint64_t m;  // floor(2^k / d) + 1
  uint32_t k;  // 31 + ceil(log2 d)
  int32_t d;   // the divisor (>= 1)
};

// d >= 1.
inline FastDiv make_fastdiv(int32_t d) {
  FastDiv f;
  uint32_t L = 0;
  while ((1ull << L) < (uint64_t)d) ++L;
  f.k = 31u + L;
  f.m = ((1ull << f.k) / (uint64_t)d) + 1ull;
  f.d = d;
  return f;
}

// floor(n / f.d) for 0 <= n < 2^31.
STEPKV_HD int32_t fdiv(int32_t n, const FastDiv& f) {
  return (int32_t)(((uint64_t)(uint32_t)n * f.m) >> f.k);
}

// n mod f.d for 0 <= n < 2^31, with the quotient.
STEPKV_HD int32_t fdivmod(int32_t n, const FastDiv& f, int32_t& rem) {
  const int32_t q = fdiv(n, f);
  rem = n - q * f.d;
  return q;
}

// n mod f.d for 0 <= n < 2^31.
STEPKV_HD int32_t fmodulo(int32_t n, const FastDiv& f) { return n - fdiv(n, f) * f.d; }

}  // namespace stepkv
