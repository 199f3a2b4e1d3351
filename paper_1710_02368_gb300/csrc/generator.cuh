// Counter-based splitmix64 generator and the variates derived from it.
//
// Definition (Steele, Lea & Flood, OOPSLA 2014; output function of the
// public-domain splitmix64.c):
//   mix(z): z ^= z >> 30; z *= 0xBF58476D1CE4E5B9; z ^= z >> 27;
//           z *= 0x94D049BB133111EB; return z ^ (z >> 31)
//   key(seed, stream) = mix(seed ^ stream * G),  draw(key, i) = mix(key + (i+1) G)
// with G = 0x9E3779B97F4A7C15.  Normal variates use Box-Muller (cos branch)
// with ln and cos evaluated by fixed series from correctly rounded double
// operations only, so host, device and any other implementation of the same
// definition agree bit for bit.  Every double operation below goes through
// dadd/dmul/ddiv/dsqrt: on the device those are the _rn intrinsics, which the
// compiler never fuses; host code is built with -ffp-contract=off.
#pragma once

#include <cstdint>
#include <cmath>

#ifndef AGN_HD
#define AGN_HD __host__ __device__ __forceinline__
#endif

namespace agn {
namespace gen {

constexpr uint64_t kG = 0x9E3779B97F4A7C15ull;
constexpr uint64_t kC1 = 0xBF58476D1CE4E5B9ull;
constexpr uint64_t kC2 = 0x94D049BB133111EBull;

enum Stream : uint64_t {
  kData = 1,
  kTeacher = 2,
  kInit = 3,
  kSchedule = 4,
  kCommitAcc = 5,
  kCommitTheta = 6,
  kCommitOrder = 7,
};

AGN_HD uint64_t mix(uint64_t z) {
  z = (z ^ (z >> 30)) * kC1;
  z = (z ^ (z >> 27)) * kC2;
  return z ^ (z >> 31);
}
AGN_HD uint64_t key(uint64_t seed, uint64_t stream) { return mix(seed ^ (stream * kG)); }
AGN_HD uint64_t draw(uint64_t k, uint64_t i) { return mix(k + (i + 1) * kG); }

AGN_HD double dadd(double a, double b) {
#ifdef __CUDA_ARCH__
  return __dadd_rn(a, b);
#else
  return a + b;
#endif
}
AGN_HD double dsub(double a, double b) {
#ifdef __CUDA_ARCH__
  return __dsub_rn(a, b);
#else
  return a - b;
#endif
}
AGN_HD double dmul(double a, double b) {
#ifdef __CUDA_ARCH__
  return __dmul_rn(a, b);
#else
  return a * b;
#endif
}
AGN_HD double ddiv(double a, double b) {
#ifdef __CUDA_ARCH__
  return __ddiv_rn(a, b);
#else
  return a / b;
#endif
}
AGN_HD double dsqrt(double a) {
#ifdef __CUDA_ARCH__
  return __dsqrt_rn(a);
#else
  return std::sqrt(a);
#endif
}

// U[0,1) in float32 from the top 24 bits (exact), and in float64 from 53 bits.
AGN_HD float uniform_f32(uint64_t d) { return (float)((double)(d >> 40) * 0x1p-24); }
AGN_HD double uniform_f64(uint64_t d) { return (double)(d >> 11) * 0x1p-53; }

// Integer in [0, bound): ((d >> 40) * bound) >> 24.
AGN_HD uint64_t bounded(uint64_t d, uint64_t bound) { return ((d >> 40) * bound) >> 24; }

constexpr double kLn2 = 0.6931471805599453094;
constexpr double kSqrtHalf = 0.70710678118654752440;
constexpr double kPi = 3.14159265358979323846;
constexpr double kTwoPi = 6.28318530717958647692;
constexpr int kLnTerms = 12;
constexpr int kCosTerms = 17;

// ln(x), x in (0, 1]: x = f 2^e, f in [sqrt(1/2), sqrt(2)); ln f = 2 atanh(s),
// s = (f-1)/(f+1), atanh(s)/s = sum_k s^(2k)/(2k+1), Horner from the top.
AGN_HD double ln_series(double x) {
  int e;
  double f = frexp(x, &e);
  if (f < kSqrtHalf) {
    f = dmul(f, 2.0);
    e -= 1;
  }
  double s = ddiv(dsub(f, 1.0), dadd(f, 1.0));
  double s2 = dmul(s, s);
  double p = ddiv(1.0, (double)(2 * (kLnTerms - 1) + 1));
  for (int k = kLnTerms - 2; k >= 0; --k) p = dadd(dmul(p, s2), ddiv(1.0, (double)(2 * k + 1)));
  double lnf = dmul(dmul(2.0, s), p);
  return dadd(dmul((double)e, kLn2), lnf);
}

// cos(2 pi t), t in [0,1): -cos(th), th = 2 pi t - pi, Taylor series in th^2
// with coefficients c_0 = 1, c_k = -c_{k-1} / ((2k-1)(2k)).
AGN_HD double cos2pi_series(double t) {
  double c[kCosTerms];
  c[0] = 1.0;
  for (int k = 1; k < kCosTerms; ++k) c[k] = ddiv(-c[k - 1], (double)((2 * k - 1) * (2 * k)));
  double th = dsub(dmul(t, kTwoPi), kPi);
  double th2 = dmul(th, th);
  double p = c[kCosTerms - 1];
  for (int k = kCosTerms - 2; k >= 0; --k) p = dadd(dmul(p, th2), c[k]);
  return -p;
}

// N(0,1) variate number i of a stream: draws 2i (radius) and 2i+1 (angle).
AGN_HD double normal(uint64_t k, uint64_t i) {
  double u1 = uniform_f64(draw(k, 2 * i));
  double u2 = uniform_f64(draw(k, 2 * i + 1));
  double r = dsqrt(dmul(-2.0, ln_series(dsub(1.0, u1))));
  return dmul(r, cos2pi_series(u2));
}

}  // namespace gen
}  // namespace agn
