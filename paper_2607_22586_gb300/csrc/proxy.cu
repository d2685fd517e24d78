// Step 1: variance-expanded query proxies (Section 3.2.1; Appendix A.4), packed
// per KV head in the row order the scoring kernels consume.
//
// One CTA per (query head, request, layer). It computes the per-dimension
// mean and unbiased std of the W window queries of its head, draws the
// normals with Philox4x64-10 + Box-Muller, forms mu + gamma * sigma * z,
// optionally rotates it to the first decode position, rounds to the input
// dtype and writes:
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

// Box-Muller on two Philox words a, c: with u = ((a >> 11) + 1/2) 2^-53 and
// v = ((c >> 11) + 1/2) 2^-53, returns sqrt(-2 ln u) (cos 2 pi v, sin 2 pi v).
// Evaluated in float32 without losing the precision the 53-bit uniforms carry
// where it matters: ln u for u >= 1/2 is log1p(-(1 - u)) with 1 - u taken from
// the integer complement, and the angle is first reduced to (-1/2, 1/2] turn in
// integer arithmetic, so sin/cos near their zeros keep full relative precision.
__device__ __forceinline__ void box_muller(uint64_t a, uint64_t c, float& z0, float& z1) {
  constexpr float k2m53 = 1.1102230246251565e-16f;  // 2^-53
  constexpr float k2m52 = 2.220446049250313e-16f;   // 2^-52
  const uint64_t ma = a >> 11;
  float lnu;
  if (ma < (1ull << 52)) {
    lnu = logf((__ull2float_rn(ma) + 0.5f) * k2m53);
  } else {
    const uint64_t comp = ((1ull << 53) - 1) - ma;
    lnu = log1pf(-(__ull2float_rn(comp) + 0.5f) * k2m53);
  }
  const float r = sqrtf(-2.0f * lnu);
  const uint64_t mc = c >> 11;
  const int64_t cen = (int64_t)mc - (mc >= (1ull << 52) ? (int64_t)(1ull << 53) : 0);
  const float two_v = (__ll2float_rn(cen) + 0.5f) * k2m52;  // 2v reduced to (-1, 1]
  float sv, cv;
  sincospif(two_v, &sv, &cv);
  z0 = r * cv;
  z1 = r * sv;
}

// Four standard normals for dims 4q..4q+3 of proxy i of query head hq.
__device__ __forceinline__ void normals4(const Problem& P, int i, int q, int hq, int b,
                                         int layer, float& z0, float& z1, float& z2, float& z3) {
  uint64_t c[4] = {(uint64_t)i * (uint64_t)(P.d / 4) + (uint64_t)q, (uint64_t)hq,
                   (uint64_t)b, (uint64_t)(int64_t)layer};
  philox4x64_10(c, P.seed, 0ull);
  box_muller(c[0], c[1], z0, z1);
  box_muller(c[2], c[3], z2, z3);
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
  const T* q = qwin + (size_t)l * P.ls_q + ((size_t)b * P.W * P.Hq + hq) * D;
  const size_t qstride = (size_t)P.Hq * D;
  for (int k = threadIdx.x; k < D; k += blockDim.x) {
    float s = 0.f;
    for (int w = 0; w < P.W; ++w) s += to_f32(q[w * qstride + k]);
    const float m = s / (float)P.W;
    float v = 0.f;
    for (int w = 0; w < P.W; ++w) {
      const float dv = to_f32(q[w * qstride + k]) - m;
      v = fmaf(dv, dv, v);
    }
    mu[k] = m;
    sg[k] = sqrtf(v / (float)(P.W - 1));
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
      normals4(P, i, qq, hq, b, layer, z[0], z[1], z[2], z[3]);
      normals4(P, i, qq + NQ8, hq, b, layer, z[4], z[5], z[6], z[7]);
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
  // padding rows are written by the first query head of the KV head
  if (j == 0) {
    for (int p = 0; p < P.Prows_pad; ++p) {
      if (row_kind(P, p).group >= 0) continue;
      for (int k = threadIdx.x; k < D; k += blockDim.x) packed[(size_t)p * D + k] = from_f32<T>(0.f);
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
