// Double-precision exp and log for the replay kernel, written for GB300's FP64
// pipe: a warp's FP64 instruction occupies its scheduler's share of the FP64 unit for
// 64 cycles (2 fused multiply-adds per clock per SM), so range reduction, table indexing,
// exponent scaling and the special-case tests run on the integer pipes and the
// FP64 pipe does only the arithmetic that needs 53-bit precision.
//
// exp: table-driven method of P. T. P. Tang (ACM TOMS 15(2), 1989).  x = (64m + j)
//   ln2/64 + r with |r| <= ln2/128; exp(x) = 2^m 2^(j/64) (1 + p(r)), p the Taylor
//   polynomial of exp(r) - 1 through r^5 (truncation < 4e-17 relative).  The
//   nearest integer 64m + j comes from adding 1.5 * 2^52 (no conversion
//   instruction); 2^m is applied by an integer add to the exponent field.
//   10 FP64 instructions.
// log: table-driven method of P. T. P. Tang (ACM TOMS 16(4), 1990).  x = 2^e m with
//   m in [0.75, 1.5), F = j/128 the nearest table point, f = m - F (exact),
//   u = f / F by a tabulated reciprocal, log x = e ln2 + ln F + log1p(u) with the
//   Taylor polynomial of log1p through u^7 (|u| <= 1/192; truncation < 2e-17
//   relative).  For m near 1, F = 1 and the result is log1p(u) alone, so there is
//   no cancellation.  13 FP64 instructions.
// sin, cos: additive range reduction of W. J. Cody and W. Waite ("Software Manual for
//   the Elementary Functions", 1980) by pi/64: x = n pi/64 + r, |r| <= pi/128, with pi/64
//   in three parts (n times the first two exact for |n| < 2^20), then the addition
//   formulas over a table of sin(k pi/64), k = n mod 128:
//   sin x = S + (S (cos r - 1) + C sin r), cos x = C + (C (cos r - 1) - S sin r),
//   S = sin(k pi/64), C = cos(k pi/64), with sin r through r^7 and cos r - 1 through r^6
//   (truncation below 4e-19 relative at |r| = pi/128).  No branch on the quadrant: every
//   lane of a warp runs the same instructions.  16 FP64 instructions for one of them, 19
//   for both.
// Arguments outside the fast range (|x| >= 708 for exp; x <= 0, subnormal, infinite
// or NaN for log; |x| >= 2^15, infinite or NaN for sin and cos) take CUDA's functions.
// Results are within about 1 ulp (sin and cos: 2 ulp, tested).
#pragma once
#include <cuda_runtime.h>

#include "fmath_tables.h"

namespace ndvm {

// The IEEE bits of x as an integer, through an inline-PTX move that the compiler's front
// end cannot see through.  A test written on the bits of a computed double (x == +-0, a
// range check) can otherwise be turned back into a floating-point compare, which runs on
// the FP64 pipe and costs a full issue slot there; through fbits it stays on the integer
// pipes.  The move itself is a register rename.
__device__ __forceinline__ long long fbits(double x) {
  long long b;
  asm("mov.b64 %0, %1;" : "=l"(b) : "d"(x));
  return b;
}

// The slow paths are calls, not inlined code: a rarely taken branch around inlined library
// code can be compiled to predicated instructions that issue (all lanes off) every time,
// and on GB300's FP64 pipe each of those costs a full slot.
__device__ __noinline__ double slow_exp(double x) { return exp(x); }
__device__ __noinline__ double slow_log(double x) { return log(x); }
__device__ __noinline__ double2 slow_sincos(double x) {
  double2 v;
  sincos(x, &v.x, &v.y);
  return v;
}

__device__ __forceinline__ double fast_exp(double x) {
  const long long bx = fbits(x);
  if ((bx & 0x7fffffffffffffffLL) >= 0x4086200000000000LL) return slow_exp(x);  // |x| >= 708, inf, nan
  const double magic = 0x1.8p52;
  const double t = fma(x, NDVM_64_LN2, magic);
  const int n = __double2loint(t);  // nearest integer to 64 x / ln2
  const double kd = t - magic;
  double r = fma(kd, -NDVM_LN2_64_HI, x);
  r = fma(kd, -NDVM_LN2_64_LO, r);
  double p = fma(r, NDVM_INV120, NDVM_INV24);
  p = fma(r, p, NDVM_INV6);
  p = fma(r, p, 0.5);
  p = fma(r, p, 1.0);
  p = r * p;  // exp(r) - 1
  const double T = kExp2Table[n & 63];
  const double y = fma(T, p, T);
  return __longlong_as_double(fbits(y) + ((long long)(n >> 6) << 52));
}

__device__ __forceinline__ double fast_log(double x) {
  const long long bx = fbits(x);
  if (bx < 0x0010000000000000LL || bx >= 0x7ff0000000000000LL) return slow_log(x);  // <= 0, subnormal, inf, nan
  int e = (int)(bx >> 52) - 1023;
  long long mb = (bx & 0x000fffffffffffffLL) | 0x3ff0000000000000LL;  // m in [1, 2)
  if (mb >= 0x3ff8000000000000LL) {  // m in [1.5, 2): use m/2 in [0.75, 1)
    mb -= 0x0010000000000000LL;
    e += 1;
  }
  // j = nearest integer to 128 m, from the mantissa bits
  const long long mant = mb & 0x000fffffffffffffLL;
  const int j = (mb >= 0x3ff0000000000000LL) ? 128 + (int)((mant + (1LL << 44)) >> 45)
                                              : 64 + (int)((mant + (1LL << 45)) >> 46);
  const int ix = j - 96;
  const double m = __longlong_as_double(mb);
  const double f = m - kLogFv[ix];  // exact
  const double u = f * kLogInvF[ix];
  double t = fma(u, NDVM_INV7, -NDVM_INV6);
  t = fma(u, t, NDVM_INV5);
  t = fma(u, t, -0.25);
  t = fma(u, t, NDVM_INV3);
  t = fma(u, t, -0.5);
  const double p = fma(u * u, t, u);  // log1p(u)
  const double ed = __longlong_as_double(0x4338000000000000LL + e) - 0x1.8p52;  // (double)e, exact
  const double hi = fma(ed, NDVM_LN2_HI, kLogF[ix]);
  const double lo = fma(ed, NDVM_LN2_LO, p);
  return hi + lo;
}

// sin x and cos x; a caller that uses one of them leaves the other's instructions out
__device__ __forceinline__ void fast_sincos(double x, double* s, double* c) {
  const long long bx = fbits(x);
  if ((bx & 0x7fffffffffffffffLL) >= 0x40e0000000000000LL) {  // |x| >= 2^15, inf, nan
    const double2 v = slow_sincos(x);
    *s = v.x;
    *c = v.y;
    return;
  }
  const double magic = 0x1.8p52;
  const double t = fma(x, NDVM_64_PI, magic);
  const int n = __double2loint(t);  // nearest integer to 64 x / pi
  const double kd = t - magic;
  double r = fma(kd, -NDVM_PI_64_1, x);
  r = fma(kd, -NDVM_PI_64_2, r);
  r = fma(kd, -NDVM_PI_64_3, r);
  const double r2 = r * r;
  double ps = fma(r2, -NDVM_INV5040, NDVM_INV120);
  ps = fma(r2, ps, -NDVM_INV6);
  const double sr = fma(r2 * r, ps, r);  // sin r
  double pc = fma(r2, -NDVM_INV720, NDVM_INV24);
  pc = fma(r2, pc, -0.5);
  const double cm = r2 * pc;  // cos r - 1
  const int k = n & 127;
  const double S = kSinTable[k], C = kSinTable[(k + 32) & 127];
  // |x| < 2^-27: sin x rounds to x and cos x to 1 (this also keeps the sign of a zero)
  const bool tiny = (bx & 0x7fffffffffffffffLL) < 0x3e40000000000000LL;
  *s = tiny ? x : S + fma(C, sr, S * cm);
  *c = tiny ? 1.0 : C + fma(-S, sr, C * cm);
}
__device__ __forceinline__ double fast_sin(double x) {
  double s, c;
  fast_sincos(x, &s, &c);
  return s;
}
__device__ __forceinline__ double fast_cos(double x) {
  double s, c;
  fast_sincos(x, &s, &c);
  return c;
}

__device__ __forceinline__ float fast_exp(float x) { return expf(x); }
__device__ __forceinline__ void fast_sincos(float x, float* s, float* c) { sincosf(x, s, c); }
__device__ __forceinline__ float fast_sin(float x) { return sinf(x); }
__device__ __forceinline__ float fast_cos(float x) { return cosf(x); }
__device__ __forceinline__ float fast_log(float x) { return logf(x); }

}  // namespace ndvm
