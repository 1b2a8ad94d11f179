// Conversion of an fp32 value to the 64-bit fixed point of the least-squares statistics
// without the fp64 pipe. Host and device: the CPU tests check it bit for bit against the fp64
// conversion it replaces.
#pragma once

#include <cmath>
#include <cstdint>

namespace crvq {

__host__ __device__ inline int fx_clz32(uint32_t x) {
#ifdef __CUDA_ARCH__
  return __clz((int)x);
#else
  return x ? __builtin_clz(x) : 32;
#endif
}

// llrint(q * 2^e), rounding half to even, in integer arithmetic: the value that converting the
// exact fp64 product q * 2^e to int64 gives (round to nearest even, saturating at the int64
// range), for every finite q and every e with 2^e a normal fp64 number. Non-finite q gives 0
// (the fixed-point scale's bound check reports those).
__host__ __device__ inline long long fix_rn(float q, int e) {
  uint32_t b;
#ifdef __CUDA_ARCH__
  b = __float_as_uint(q);
#else
  __builtin_memcpy(&b, &q, 4);
#endif
  const int ex = (int)((b >> 23) & 0xffu);
  if (ex == 0xff) return 0;
  const uint32_t m = ex ? ((b & 0x7fffffu) | 0x800000u) : (b & 0x7fffffu);
  const int sh = (ex ? ex : 1) - 150 + e;  // |q| 2^e = m 2^sh
  unsigned long long r = 0;
  if (m != 0 && sh >= 0) {
    if ((31 - fx_clz32(m)) + sh >= 63)
      return (b >> 31) ? (long long)0x8000000000000000ull : 0x7fffffffffffffffll;
    r = (unsigned long long)m << sh;
  } else if (m != 0 && sh >= -31) {
    const int s = -sh;  // 1 .. 31
    const uint32_t q0 = s < 32 ? (m >> s) : 0u;
    const uint32_t rem = m & ((1u << (s - 1)) * 2u - 1u), half = 1u << (s - 1);
    r = q0 + ((rem > half || (rem == half && (q0 & 1u))) ? 1u : 0u);
  }
  return (b >> 31) ? -(long long)r : (long long)r;
}

// llrint(q * 2^e) when 2^e = scale is a normal fp32 number and |q * 2^e| < 2^31 (the
// statistics scale keeps every term below 2^30): the product is exact, or below 2^-126 where
// both give 0, and the conversion rounds half to even. Equals fix_rn(q, e) under those
// conditions, in two instructions (an FMUL and a round-to-nearest F2I) instead of an integer
// sequence with data-dependent branches.
__host__ __device__ inline long long fix_rn_small(float q, float scale) {
#ifdef __CUDA_ARCH__
  return (long long)__float2int_rn(q * scale);
#else
  return (long long)std::lrintf(q * scale);  // default rounding: half to even
#endif
}

}  // namespace crvq
