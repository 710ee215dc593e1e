// devmath.cuh — counter-based RNG and deterministic fp32 elementary functions for
// the device.
//
// Every value that decides an integer in the simulator (event times, thinning,
// request types, sampled actions) must be the same bits on every IEEE-754 machine,
// so these functions use only correctly rounded operations (__fadd_rn, __fmul_rn,
// __fmaf_rn, __fdiv_rn, __fsqrt_rn, rintf, floorf) and integer bit manipulation, in
// a fixed order.  Methods: Philox4x32-10 (Salmon et al., SC'11); Cody-Waite
// argument reduction with a two-part ln 2 (Cody & Waite 1980); the atanh series of
// ln m; Taylor series of e^r, sin and cos; Box-Muller normals (Box & Muller 1958).
#pragma once
#include <cstdint>

namespace simx {

constexpr uint32_t kTimeLimit = 0x7FFFFFFFu;
constexpr uint32_t kNone = 0xFFFFFFFFu;
constexpr uint32_t kEventCap = 1u << 20;
constexpr uint32_t kStTime = 1u, kStEvent = 2u, kStAction = 4u;
enum : uint32_t { kStreamArrival = 1, kStreamPolicy = 2, kStreamSwitch = 3, kStreamInit = 4,
                  kStreamEpoch = 5 };

struct U4 { uint32_t x, y, z, w; };

// Philox4x32-10: ten rounds, multipliers 0xD2511F53 / 0xCD9E8D57, Weyl key bumps.
__device__ __forceinline__ U4 philox(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3,
                                     uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r > 0) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    const uint32_t lo0 = 0xD2511F53u * c0, hi0 = __umulhi(0xD2511F53u, c0);
    const uint32_t lo1 = 0xCD9E8D57u * c2, hi1 = __umulhi(0xCD9E8D57u, c2);
    const uint32_t n0 = hi1 ^ c1 ^ k0;
    const uint32_t n2 = hi0 ^ c3 ^ k1;
    c0 = n0;
    c1 = lo1;
    c2 = n2;
    c3 = lo0;
  }
  return U4{c0, c1, c2, c3};
}

// Two-part ln 2: the high part has 12 significant bits (k * kLn2Hi exact, |k| < 4096).
constexpr float kLn2Hi = 2839.0f / 4096.0f;
constexpr float kLn2Lo = (float)(0.69314718055994530942 - 2839.0 / 4096.0);
constexpr float kLog2e = (float)1.44269504088896340736;
constexpr float kSqrt2 = (float)1.41421356237309504880;
constexpr float kHalfPi = (float)1.57079632679489661923;
constexpr float kTwoM24 = 1.0f / 16777216.0f;

// ln x, x > 0 normal: x = 2^e m, m in [sqrt(1/2), sqrt(2)], ln m = 2 atanh(s),
// s = (m - 1) / (m + 1), odd series through s^11.
__device__ __forceinline__ float det_log(float x) {
  const uint32_t u = __float_as_uint(x);
  int e = (int)((u >> 23) & 0xFFu) - 127;
  float m = __uint_as_float((u & 0x7FFFFFu) | 0x3F800000u);
  if (m > kSqrt2) {
    m = __fmul_rn(m, 0.5f);
    e += 1;
  }
  const float s = __fdiv_rn(__fsub_rn(m, 1.0f), __fadd_rn(m, 1.0f));
  const float z = __fmul_rn(s, s);
  float p = (float)(1.0 / 11.0);
  p = __fmaf_rn(p, z, (float)(1.0 / 9.0));
  p = __fmaf_rn(p, z, (float)(1.0 / 7.0));
  p = __fmaf_rn(p, z, (float)(1.0 / 5.0));
  p = __fmaf_rn(p, z, (float)(1.0 / 3.0));
  const float t = __fadd_rn(s, s);
  const float lnm = __fmaf_rn(__fmul_rn(t, z), p, t);
  const float fe = __int2float_rn(e);
  return __fmaf_rn(fe, kLn2Hi, __fmaf_rn(fe, kLn2Lo, lnm));
}

// e^x: k = rint(x log2 e), r = x - k ln 2, Taylor to r^7, times 2^k.
// x < -87 gives 0, x > 88 gives +inf.
__device__ __forceinline__ float det_exp(float x) {
  if (x < -87.0f) return 0.0f;
  if (x > 88.0f) return __uint_as_float(0x7F800000u);
  const float k = rintf(__fmul_rn(x, kLog2e));
  float r = __fmaf_rn(-k, kLn2Hi, x);
  r = __fmaf_rn(-k, kLn2Lo, r);
  float p = (float)(1.0 / 5040.0);
  p = __fmaf_rn(p, r, (float)(1.0 / 720.0));
  p = __fmaf_rn(p, r, (float)(1.0 / 120.0));
  p = __fmaf_rn(p, r, (float)(1.0 / 24.0));
  p = __fmaf_rn(p, r, (float)(1.0 / 6.0));
  p = __fmaf_rn(p, r, 0.5f);
  p = __fmaf_rn(p, r, 1.0f);
  p = __fmaf_rn(p, r, 1.0f);
  const int ki = (int)k;
  return __fmul_rn(p, __uint_as_float((uint32_t)(ki + 127) << 23));
}

// e^y - 1 for 0 <= y < 0.35 as y (1 + y/2! + ... + y^8/9!).
__device__ __forceinline__ float det_expm1_small(float y) {
  float q = (float)(1.0 / 362880.0);
  q = __fmaf_rn(q, y, (float)(1.0 / 40320.0));
  q = __fmaf_rn(q, y, (float)(1.0 / 5040.0));
  q = __fmaf_rn(q, y, (float)(1.0 / 720.0));
  q = __fmaf_rn(q, y, (float)(1.0 / 120.0));
  q = __fmaf_rn(q, y, (float)(1.0 / 24.0));
  q = __fmaf_rn(q, y, (float)(1.0 / 6.0));
  q = __fmaf_rn(q, y, 0.5f);
  q = __fmaf_rn(q, y, 1.0f);
  return __fmul_rn(q, y);
}

// tanh z = sign(z) (e^{2|z|} - 1) / (e^{2|z|} + 1); |z| >= 10 gives +-1.
__device__ __forceinline__ float det_tanh(float z) {
  const float a = fabsf(z);
  float t;
  if (a >= 10.0f) {
    t = 1.0f;
  } else {
    const float y = __fadd_rn(a, a);
    const float em1 = (y < 0.35f) ? det_expm1_small(y) : __fsub_rn(det_exp(y), 1.0f);
    t = __fdiv_rn(em1, __fadd_rn(em1, 2.0f));
  }
  return copysignf(t, z);
}

// GELU in its tanh form: 0.5 x (1 + tanh(c (x + 0.044715 x^3))), c = sqrt(2/pi), as
// u = fma(0.044715, (x*x)*x, x), t = tanh(c*u), (0.5*x)*(1 + t).
__device__ __forceinline__ float det_gelu(float x) {
  const float x3 = __fmul_rn(__fmul_rn(x, x), x);
  const float u = __fmaf_rn(0.044715f, x3, x);
  const float t = det_tanh(__fmul_rn(0.7978845608028654f, u));
  return __fmul_rn(__fmul_rn(0.5f, x), __fadd_rn(1.0f, t));
}

// GELU of x into g (the same operations as det_gelu) and its derivative
// 0.5 (1 + t) + 0.5 x (1 - t^2) c (1 + 3 a x^2), t = tanh(c (x + a x^3)), into d.
__device__ __forceinline__ void det_gelu_grad(float x, float& g, float& d) {
  const float c = 0.7978845608028654f, a = 0.044715f;
  const float u = __fmaf_rn(a, __fmul_rn(__fmul_rn(x, x), x), x);
  const float t = det_tanh(__fmul_rn(c, u));
  d = 0.5f * (1.0f + t) + 0.5f * x * (1.0f - t * t) * c * (1.0f + 3.0f * a * x * x);
  g = __fmul_rn(__fmul_rn(0.5f, x), __fadd_rn(1.0f, t));
}

// cos(2 pi u), u in [0, 1): quadrant of 4u, reflection to [0, pi/4], Taylor series.
__device__ __forceinline__ float det_cos2pi(float u) {
  const float v = __fmul_rn(u, 4.0f);
  const int q = (int)v;
  float g = __fsub_rn(v, __int2float_rn(q));
  int want_sin = q & 1;
  const float sign = (q == 1 || q == 2) ? -1.0f : 1.0f;
  if (g > 0.5f) {
    g = __fsub_rn(1.0f, g);
    want_sin = !want_sin;
  }
  const float th = __fmul_rn(g, kHalfPi);
  const float w = __fmul_rn(th, th);
  float r;
  if (want_sin) {
    float p = (float)(-1.0 / 39916800.0);
    p = __fmaf_rn(p, w, (float)(1.0 / 362880.0));
    p = __fmaf_rn(p, w, (float)(-1.0 / 5040.0));
    p = __fmaf_rn(p, w, (float)(1.0 / 120.0));
    p = __fmaf_rn(p, w, (float)(-1.0 / 6.0));
    r = __fmaf_rn(__fmul_rn(th, w), p, th);
  } else {
    float p = (float)(1.0 / 479001600.0);
    p = __fmaf_rn(p, w, (float)(-1.0 / 3628800.0));
    p = __fmaf_rn(p, w, (float)(1.0 / 40320.0));
    p = __fmaf_rn(p, w, (float)(-1.0 / 720.0));
    p = __fmaf_rn(p, w, (float)(1.0 / 24.0));
    p = __fmaf_rn(p, w, -0.5f);
    r = __fmaf_rn(w, p, 1.0f);
  }
  return __fmul_rn(sign, r);
}

// Uniforms from the top 24 bits of a Philox word.
__device__ __forceinline__ float u_open0(uint32_t w) {  // (0, 1]
  return __fmul_rn(__uint2float_rn((w >> 8) + 1u), kTwoM24);
}
__device__ __forceinline__ float u_open1(uint32_t w) {  // [0, 1)
  return __fmul_rn(__uint2float_rn(w >> 8), kTwoM24);
}
// Exp(1) by inversion.
__device__ __forceinline__ float expo1(uint32_t w) { return -det_log(u_open0(w)); }

// Standard normal (Box-Muller) from two words.
__device__ __forceinline__ float normal01(uint32_t w0, uint32_t w1) {
  const float r = __fsqrt_rn(__fmul_rn(-2.0f, det_log(u_open0(w0))));
  return __fmul_rn(r, det_cos2pi(u_open1(w1)));
}

// A duration in integer microseconds: round half up, saturated at 2^26.
__device__ __forceinline__ uint32_t duration_us(float x) {
  const float y = __fadd_rn(x, 0.5f);
  if (!(y < 67108864.0f)) return 67108864u;
  return (uint32_t)floorf(y);
}

}  // namespace simx
