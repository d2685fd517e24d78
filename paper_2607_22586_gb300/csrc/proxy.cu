// Step 1: variance-expanded query proxies (Section 3.2.1; Appendix A.4), packed
// per KV head in the row order the scoring kernels consume.
//
// One CTA per (query head, request, layer). It computes the per-dimension
// mean and unbiased std of the W window queries of its head, draws the
// normals with Philox4x64-10 + Box-Muller, forms mu + gamma * sigma * z,
// optionally rotates it to the first decode position, rounds to the input
// dtype and writes (one Philox draw per thread and proxy gives the eight
// normals of dims [4q, 4q+4) and [d/2+4q, d/2+4q+4), the RoPE pairs):
//   - the packed block [Prows_pad][d] of its KV head: group-major rows
//     (group g holds the g-th slice of every query head of the KV head), the
//     last window query of each query head as anchor rows, zero padding;
//   - optionally the caller-layout copy [Hq][N][d].
#include "common.cuh"

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

// Eight standard normals for dims 4q..4q+3 (z[0..3]) and d/2+4q..d/2+4q+3
// (z[4..7]) of proxy i of query head hq: one Philox4x64-10 draw, its 64-bit
// outputs split low word first into eight uniforms, Box-Muller on pairs.
__device__ __forceinline__ void normals8(const Problem& P, int i, int q, int hq, int b, int layer,
                                         float (&z)[8]) {
  uint64_t c[4] = {(uint64_t)i * (uint64_t)(P.d / 8) + (uint64_t)q, (uint64_t)hq, (uint64_t)b,
                   (uint64_t)(int64_t)layer};
  philox4x64_10(c, P.seed, 0ull);
  box_muller((uint32_t)c[0], (uint32_t)(c[0] >> 32), z[0], z[1]);
  box_muller((uint32_t)c[1], (uint32_t)(c[1] >> 32), z[2], z[3]);
  box_muller((uint32_t)c[2], (uint32_t)(c[2] >> 32), z[4], z[5]);
  box_muller((uint32_t)c[3], (uint32_t)(c[3] >> 32), z[6], z[7]);
}

// Four consecutive values rounded to T, one vector store.
__device__ __forceinline__ void store4(__nv_bfloat16* dst, float a, float b, float c, float d) {
  __nv_bfloat162 lo = __floats2bfloat162_rn(a, b), hi = __floats2bfloat162_rn(c, d);
  uint2 u;
  u.x = *reinterpret_cast<uint32_t*>(&lo);
  u.y = *reinterpret_cast<uint32_t*>(&hi);
  *reinterpret_cast<uint2*>(dst) = u;
}
__device__ __forceinline__ void store4(float* dst, float a, float b, float c, float d) {
  *reinterpret_cast<float4*>(dst) = make_float4(a, b, c, d);
}

// Proxies of one query head are spread over kProxyChunks CTAs.
constexpr int kProxyChunks = 8;

template <typename T, int D>
__global__ void __launch_bounds__(256) proxy_pack_kernel(Problem P, Buffers bf, const T* qwin) {
  const int hq = blockIdx.x / kProxyChunks, chunk = blockIdx.x % kProxyChunks;
  const int b = blockIdx.y, l = blockIdx.z;
  const int h = hq / P.r, j = hq - h * P.r;
  __shared__ float mu[D], sg[D], rc[D / 2], rs[D / 2];
  constexpr int RPT = 256 / D;               // threads per dimension
  __shared__ float part[RPT][D];
  const T* q = qwin ? qwin + (size_t)l * P.ls_q + ((size_t)b * P.W * P.Hq + hq) * D : nullptr;
  const size_t qstride = (size_t)P.Hq * D;
  if (bf.stats_in) {
    // given statistics (e.g. over the whole prefill): [L][B][2][Hq][D]
    const float* st = bf.stats_in + (((size_t)l * P.B + b) * 2 * P.Hq + hq) * D;
    for (int k = threadIdx.x; k < D; k += blockDim.x) {
      mu[k] = st[k];
      sg[k] = st[(size_t)P.Hq * D + k];
    }
  } else {
    // mean and unbiased std over the W window rows: thread (k, rg) sums rows
    // rg, rg + RPT, ... of dimension k; loads are independent and unrolled
    const int k = threadIdx.x % D, rg = threadIdx.x / D;
    float s = 0.f;
#pragma unroll 8
    for (int w = rg; w < P.W; w += RPT) s += to_f32(q[w * qstride + k]);
    part[rg][k] = s;
    __syncthreads();
    float tot = 0.f;
#pragma unroll
    for (int g = 0; g < RPT; ++g) tot += part[g][k];
    const float m = tot / (float)P.W;
    __syncthreads();
    float v = 0.f;
#pragma unroll 8
    for (int w = rg; w < P.W; w += RPT) {
      const float dv = to_f32(q[w * qstride + k]) - m;
      v = fmaf(dv, dv, v);
    }
    part[rg][k] = v;
    __syncthreads();
    if (rg == 0) {
      float vt = 0.f;
#pragma unroll
      for (int g = 0; g < RPT; ++g) vt += part[g][k];
      mu[k] = m;
      sg[k] = sqrtf(vt / (float)(P.W - 1));
    }
  }
  const bool rope = P.rope_theta > 0.f && !bf.proxies_in;
  if (rope) {
    // angle = pos * theta^(-2k/d), reduced modulo 2*pi in double once per block
    const double pos = (double)(P.req[b].t_len + P.rope_off);
    for (int k = threadIdx.x; k < D / 2; k += blockDim.x) {
      const double ang = pos * pow((double)P.rope_theta, -2.0 * k / (double)D);
      const double red = ang - 6.283185307179586 * rint(ang / 6.283185307179586);
      float sv, cv;
      sincosf((float)red, &sv, &cv);
      rc[k] = cv; rs[k] = sv;
    }
  }
  __syncthreads();

  const int layer = P.layer_id0 + l;
  T* packed = bf.packed ? (T*)bf.packed + ((((size_t)l * P.B + b) * P.Hkv + h) * P.Prows_pad) * D
                        : nullptr;
  const size_t user_off = ((((size_t)l * P.B + b) * P.Hq + hq) * P.Np) * D;
  const T* pin = bf.proxies_in ? (const T*)bf.proxies_in + user_off : nullptr;
  T* pout = bf.proxies_out ? (T*)bf.proxies_out + user_off : nullptr;
  constexpr int NQ8 = D / 8;  // threads per proxy: dims [4qq, 4qq+4) and [D/2+4qq, +4)
  const int per = (P.Np + kProxyChunks - 1) / kProxyChunks;
  const int i0 = chunk * per, i1 = min(P.Np, i0 + per);
  // independent iterations unrolled so several Philox chains are in flight
#pragma unroll 4
  for (int e = i0 * NQ8 + threadIdx.x; e < i1 * NQ8; e += blockDim.x) {
    const int i = e / NQ8, qq = e - i * NQ8;
    float v[8];
    if (pin) {
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        v[k] = to_f32(pin[(size_t)i * D + 4 * qq + k]);
        v[4 + k] = to_f32(pin[(size_t)i * D + D / 2 + 4 * qq + k]);
      }
    } else {
      float z[8];
      normals8(P, i, qq, hq, b, layer, z);
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int d0 = 4 * qq + k, d1 = D / 2 + 4 * qq + k;
        v[k] = fmaf(P.gamma * sg[d0], z[k], mu[d0]);
        v[4 + k] = fmaf(P.gamma * sg[d1], z[4 + k], mu[d1]);
      }
      if (rope) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int f = 4 * qq + k;
          const float a = v[k], c = v[4 + k];
          v[k] = a * rc[f] - c * rs[f];
          v[4 + k] = c * rc[f] + a * rs[f];
        }
      }
    }
    const int g = i / P.gs, ii = i - g * P.gs;
    if (packed) {
      T* dst = packed + ((size_t)g * P.RG + (size_t)j * P.gs + ii) * D;
      store4(dst + 4 * qq, v[0], v[1], v[2], v[3]);
      store4(dst + D / 2 + 4 * qq, v[4], v[5], v[6], v[7]);
    }
    if (pout) {
      store4(pout + (size_t)i * D + 4 * qq, v[0], v[1], v[2], v[3]);
      store4(pout + (size_t)i * D + D / 2 + 4 * qq, v[4], v[5], v[6], v[7]);
    }
  }
  if (!packed || chunk != 0) return;
  // anchor row of this query head: the last window query as given
  T* arow = packed + (size_t)(P.n_group_rows + j) * D;
  for (int k = threadIdx.x; k < D; k += blockDim.x) arow[k] = q[(size_t)(P.W - 1) * qstride + k];
  // padding rows (the tail of each group's rows, of the anchor rows and of
  // the block) are zeroed by the first query head of the KV head
  if (j == 0) {
    const int gpad = P.RG - P.r * P.gs;                  // per group
    const int apad = P.anchor_rows - P.r;                // after the anchor rows
    const int tail = P.Prows_pad - P.Prows;              // after the last block row
    const int n_pad = P.G * gpad + apad + tail;
    for (int e = threadIdx.x; e < n_pad * D; e += blockDim.x) {
      const int pr = e / D, k = e - pr * D;
      int row;
      if (pr < P.G * gpad) {
        row = (pr / gpad) * P.RG + P.r * P.gs + pr % gpad;
      } else if (pr < P.G * gpad + apad) {
        row = P.n_group_rows + P.r + (pr - P.G * gpad);
      } else {
        row = P.Prows + (pr - P.G * gpad - apad);
      }
      packed[(size_t)row * D + k] = from_f32<T>(0.f);
    }
  }
}

template <typename T, int D>
cudaError_t launch_t(const Problem& P, const Buffers& bf, cudaStream_t st, const void* qwin) {
  dim3 grid(P.Hq * kProxyChunks, P.B, P.L);
  proxy_pack_kernel<T, D><<<grid, 256, 0, st>>>(P, bf, (const T*)qwin);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_proxy_pack(const Problem& P, const Buffers& bf, cudaStream_t st,
                              const void* qwin) {
  if (P.dtype == MMSHIFT_BF16)
    return P.d == 128 ? launch_t<__nv_bfloat16, 128>(P, bf, st, qwin)
                      : launch_t<__nv_bfloat16, 64>(P, bf, st, qwin);
  return P.d == 128 ? launch_t<float, 128>(P, bf, st, qwin) : launch_t<float, 64>(P, bf, st, qwin);
}

}  // namespace mmshift
