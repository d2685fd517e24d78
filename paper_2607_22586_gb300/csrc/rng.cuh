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

// ln(u) for a uniform u = ((w >> 9) + 1/2) 2^-23. Near 1, with c = 1 - u
// (exact) below 1/16, the series ln(1 - c) = -(c + c^2/2 + ... + c^8/8)
// (truncation below 1e-11 relative); elsewhere log2(u) from the MUFU times
// ln 2, whose absolute error (about 2^-22) is small against |ln u| >= 0.064.
__device__ __forceinline__ float ln_uniform(float u) {
  const float c = 1.0f - u;
  float lg;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(lg) : "f"(u));
  const float far = lg * 0.6931471805599453f;
  float p = 1.0f / 8.0f;
  p = fmaf(p, c, 1.0f / 7.0f);
  p = fmaf(p, c, 1.0f / 6.0f);
  p = fmaf(p, c, 1.0f / 5.0f);
  p = fmaf(p, c, 1.0f / 4.0f);
  p = fmaf(p, c, 1.0f / 3.0f);
  p = fmaf(p, c, 0.5f);
  p = fmaf(p, c, 1.0f);
  const float near = -c * p;
  return c < 0.0625f ? near : far;
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
