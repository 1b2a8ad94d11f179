// Host check of crvq::fix_rn and crvq::fix_rn_small (fixed_point.cuh) against the fp64 route
// they replace: llrint of the exact product q * 2^e, saturated to the int64 range. Exit
// status 0 when every case agrees; prints the first disagreements otherwise.
#define __host__
#define __device__
#include <cmath>
#include <cstdint>
#include <cstdio>
#include <cstring>
#include <random>

#include "fixed_point.cuh"

static long long reference(float q, int e) {
  const double x = (double)q * std::ldexp(1.0, e);  // exact: q has 24 significant bits
  if (x >= 9223372036854775808.0) return 0x7fffffffffffffffll;
  if (x < -9223372036854775808.0) return (long long)0x8000000000000000ull;
  return std::llrint(x);  // round half to even (default rounding mode)
}

int main() {
  std::mt19937_64 rng(20241212);
  long long n = 0, bad = 0;
  auto check = [&](float q, int e) {
    if (!std::isfinite(q)) return;
    ++n;
    const long long v = crvq::fix_rn(q, e), r = reference(q, e);
    if (v != r) {
      if (bad < 8) std::printf("q=%a e=%d fix_rn=%lld reference=%lld\n", q, e, v, r);
      ++bad;
    }
  };
  // random bit patterns with exponents placing q * 2^e anywhere from far below 1/2 to beyond
  // the int64 range
  for (int it = 0; it < 2000000; ++it) {
    uint32_t b = (uint32_t)rng();
    float q;
    std::memcpy(&q, &b, 4);
    int ex = (int)((b >> 23) & 0xff);
    int e = (150 - ex) + (int)(rng() % 100) - 40;
    check(q, e);
    check(q, (int)(rng() % 600) - 300);
  }
  // exact halves and their neighbours: q * 2^e = j + 1/2 (ties to even), j +- 1 ulp of q
  for (int it = 0; it < 500000; ++it) {
    const int bits = 1 + (int)(rng() % 23);  // integer part below 2^bits
    const long long j = (long long)(rng() % (1ull << bits));
    const float q0 = (float)((double)j + 0.5);  // exact when j < 2^23
    const int e = (int)(rng() % 60) - 30;
    const float q = std::ldexp(q0, -e);
    check(q, e);
    check(-q, e);
    check(std::nextafter(q, 0.f), e);
    check(std::nextafter(q, 1e30f), e);
  }
  // the saturation edge and denormals
  for (int e = 30; e < 70; ++e) {
    for (float q : {1.f, -1.f, 1.9999999f, -1.9999999f, 0.5f, 1.5f, -2.f})
      check(std::ldexp(q, 63 - e), e), check(std::ldexp(q, 62 - e), e);
  }
  for (int it = 0; it < 100000; ++it) {
    uint32_t b = (uint32_t)(rng() & 0x807fffffu);  // zero exponent: denormals and zeros
    float q;
    std::memcpy(&q, &b, 4);
    check(q, 149 + (int)(rng() % 40) - 20);
  }
  // fix_rn_small, the kernels' form: every e whose 2^e is a normal fp32 number and every q
  // with |q 2^e| < 2^31 (random bit patterns placed in that range, ties and their neighbours)
  auto check_small = [&](float q, int e) {
    if (!std::isfinite(q) || e < -126 || e > 127) return;
    if (std::fabs((double)q * std::ldexp(1.0, e)) >= 2147483648.0) return;
    ++n;
    const long long v = crvq::fix_rn_small(q, std::ldexp(1.f, e)), r = reference(q, e);
    const long long w = crvq::fix_rn(q, e);
    if (v != r || w != r) {
      if (bad < 8) std::printf("q=%a e=%d fix_rn_small=%lld reference=%lld\n", q, e, v, r);
      ++bad;
    }
  };
  for (int it = 0; it < 2000000; ++it) {
    uint32_t b = (uint32_t)rng();
    float q;
    std::memcpy(&q, &b, 4);
    const int ex = (int)((b >> 23) & 0xff);
    check_small(q, (150 - ex) + (int)(rng() % 56) - 40);
  }
  for (int it = 0; it < 500000; ++it) {
    const int bits = 1 + (int)(rng() % 23);
    const long long j = (long long)(rng() % (1ull << bits));
    const float q0 = (float)((double)j + 0.5);
    const int e = (int)(rng() % 120) - 60;
    const float q = std::ldexp(q0, -e);
    check_small(q, e);
    check_small(-q, e);
    check_small(std::nextafter(q, 0.f), e);
    check_small(std::nextafter(q, 1e30f), e);
  }
  std::printf("cases=%lld disagreements=%lld\n", n, bad);
  return bad != 0;
}
