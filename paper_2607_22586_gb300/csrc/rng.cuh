// Counter-based normal generator shared by the proxy samplers: Philox4x64-10
// (Salmon, Moraes, Dror, Shaw, SC'11) and the Box-Muller transform (Box and
// Muller 1958) in float32.
#pragma once

#include <stdint.h>

namespace mmshift {
namespace {

// Philox4x64-10 (Salmon et al., SC'11): multipliers and Weyl key increments.
constexpr uint64_t kPhM0 = 0xD2E7470EE14C6C93ull;
constexpr uint64_t kPhM1 = 0xCA5A826395121157ull;
constexpr uint64_t kPhW0 = 0x9E3779B97F4A7C15ull;
constexpr uint64_t kPhW1 = 0xBB67AE8584CAA73Bull;

__device__ __forceinline__ void philox4x64_10(uint64_t c[4], uint64_t k0, uint64_t k1) {
#pragma unroll
  for (int rnd = 0; rnd < 10; ++rnd) {
    if (rnd) { k0 += kPhW0; k1 += kPhW1; }
    const uint64_t hi0 = __umul64hi(kPhM0, c[0]), lo0 = kPhM0 * c[0];
    const uint64_t hi1 = __umul64hi(kPhM1, c[2]), lo1 = kPhM1 * c[2];
    const uint64_t n0 = hi1 ^ c[1] ^ k0, n2 = hi0 ^ c[3] ^ k1;
    c[0] = n0; c[1] = lo1; c[2] = n2; c[3] = lo0;
  }
}

// Uniform in (0, 1) from a 32-bit word: ((w >> 9) + 1/2) 2^-23, exact in float.
__device__ __forceinline__ float uniform_of(uint32_t w) {
  return ((float)(w >> 9) + 0.5f) * 1.1920928955078125e-07f;
}

// ln(u) for a uniform u in (0, 1): u = m 2^e with m in [sqrt(1/2), sqrt(2)),
// ln m = 2 atanh(s) with s = (m - 1) / (m + 1) (|s| <= 0.1716; m - 1 is exact,
// 1 / (m + 1) from the approximate reciprocal and one Newton step, about one
// ulp) from the series 2 (s + s^3/3 + ... + s^13/13), whose truncation is
// below 2e-12 relative, and e ln 2 with ln 2 split into a short leading part
// (its product with e is exact) and the remainder (the argument reduction of
// Cody and Waite, 1980). Rounding leaves about 3 float32 ulp of relative
// error.
__device__ __forceinline__ float ln_uniform(float u) {
  const uint32_t bits = __float_as_uint(u);
  int e = (int)(bits >> 23) - 127;
  float m = __uint_as_float((bits & 0x7FFFFFu) | 0x3F800000u);   // [1, 2)
  if (m > 1.41421356f) { m *= 0.5f; ++e; }
  const float den = m + 1.0f;
  float rcp;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(rcp) : "f"(den));
  rcp = fmaf(rcp, fmaf(-den, rcp, 1.0f), rcp);
  const float s = (m - 1.0f) * rcp;
  const float t = s * s;
  float p = 1.0f / 13.0f;
  p = fmaf(p, t, 1.0f / 11.0f);
  p = fmaf(p, t, 1.0f / 9.0f);
  p = fmaf(p, t, 1.0f / 7.0f);
  p = fmaf(p, t, 1.0f / 5.0f);
  p = fmaf(p, t, 1.0f / 3.0f);
  const float s2 = 2.0f * s;
  const float lnm = fmaf(s2 * t, p, s2);
  const float fe = (float)e;
  return fmaf(fe, 0.693145751953125f, fmaf(fe, 1.4286068203094172e-06f, lnm));
}

// sin(pi x), cos(pi x) for |x| < 1 with x a multiple of 2^-23: x = y + k/2
// with k = rint(2x) and |y| <= 1/4 (both exact), Taylor polynomials of
// sin t and cos t at t = pi y (|t| <= pi/4; truncation below 1e-11), then
// the quarter-turn rotation by k.
__device__ __forceinline__ void sincos_pi(float x, float& sn, float& cs) {
  const float k = rintf(2.0f * x);
  const float y = fmaf(-0.5f, k, x);
  const float t = y * 3.14159265358979323846f;
  const float t2 = t * t;
  float ps = -1.0f / 39916800.0f;                 // -1/11!
  ps = fmaf(ps, t2, 1.0f / 362880.0f);            //  1/9!
  ps = fmaf(ps, t2, -1.0f / 5040.0f);             // -1/7!
  ps = fmaf(ps, t2, 1.0f / 120.0f);               //  1/5!
  ps = fmaf(ps, t2, -1.0f / 6.0f);                // -1/3!
  const float s0 = fmaf(ps * t2, t, t);
  float pc = 1.0f / 479001600.0f;                 //  1/12!
  pc = fmaf(pc, t2, -1.0f / 3628800.0f);          // -1/10!
  pc = fmaf(pc, t2, 1.0f / 40320.0f);             //  1/8!
  pc = fmaf(pc, t2, -1.0f / 720.0f);              // -1/6!
  pc = fmaf(pc, t2, 1.0f / 24.0f);                //  1/4!
  pc = fmaf(pc, t2, -0.5f);                       // -1/2!
  const float c0 = fmaf(pc, t2, 1.0f);
  const int q = ((int)k) & 3;                     // quarter turns
  const float sa = (q & 1) ? c0 : s0, ca = (q & 1) ? s0 : c0;
  sn = (q & 2) ? -sa : sa;
  cs = (q == 1 || q == 2) ? -ca : ca;
}

// Box-Muller: sqrt(-2 ln u) (cos 2 pi v, sin 2 pi v) in float32 from two
// 32-bit words, with 2v reduced to (-1, 1) exactly before the rotation.
__device__ __forceinline__ void box_muller(uint32_t a, uint32_t c, float& z0, float& z1) {
  const float r = sqrtf(-2.0f * ln_uniform(uniform_of(a)));
  const float v2 = 2.0f * uniform_of(c);              // 2v in (0, 2), exact
  const float two_v = v2 >= 1.0f ? v2 - 2.0f : v2;    // exact
  float sv, cv;
  sincos_pi(two_v, sv, cv);
  z0 = r * cv;
  z1 = r * sv;
}

// Eight standard normals from one Philox4x64-10 draw with counter
// (c0, c1, b, layer) and key (k0, k1): its 64-bit outputs split low word first
// into eight uniforms, Box-Muller on consecutive pairs. The query-space
// sampler uses c0 = i * d/8 + q, c1 = query head, key (seed, 0); the
// hidden-space sampler c0 = i * d_model/8 + q, c1 = 0, key (seed, 1).
__device__ __forceinline__ void normals8_at(uint64_t c0, uint64_t c1, int b, int layer,
                                            uint64_t k0, uint64_t k1, float (&z)[8]) {
  uint64_t c[4] = {c0, c1, (uint64_t)b, (uint64_t)(int64_t)layer};
  philox4x64_10(c, k0, k1);
  box_muller((uint32_t)c[0], (uint32_t)(c[0] >> 32), z[0], z[1]);
  box_muller((uint32_t)c[1], (uint32_t)(c[1] >> 32), z[2], z[3]);
  box_muller((uint32_t)c[2], (uint32_t)(c[2] >> 32), z[4], z[5]);
  box_muller((uint32_t)c[3], (uint32_t)(c[3] >> 32), z[6], z[7]);
}

}  // namespace
}  // namespace mmshift
