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
#include <algorithm>

#include "common.cuh"
#include "rng.cuh"

namespace mmshift {
namespace {

// Eight standard normals for dims 4q..4q+3 (z[0..3]) and d/2+4q..d/2+4q+3
// (z[4..7]) of proxy i of query head hq: one Philox4x64-10 draw, its 64-bit
// outputs split low word first into eight uniforms, Box-Muller on pairs.
__device__ __forceinline__ void normals8(const Problem& P, int i, int q, int hq, int b, int layer,
                                         float (&z)[8]) {
  normals8_at((uint64_t)i * (uint64_t)(P.d / 8) + (uint64_t)q, (uint64_t)hq, b, layer, P.seed, 0ull,
              z);
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

// Proxies of one query head are spread over up to kProxyChunks CTAs, about
// 1024 Philox draws each (few proxies: one CTA per query head).
constexpr int kProxyChunks = 8;

template <typename T, int D>
__global__ void __launch_bounds__(256) proxy_pack_kernel(Problem P, Buffers bf, const T* qwin,
                                                         int nch) {
  const int hq = blockIdx.x / nch, chunk = blockIdx.x % nch;
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
  const int per = (P.Np + nch - 1) / nch;
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
  const int draws = P.Np * (D / 8);
  const int nch = draws <= 0 ? 1 : std::min(kProxyChunks, (draws + 1023) / 1024);
  dim3 grid(P.Hq * nch, P.B, P.L);
  proxy_pack_kernel<T, D><<<grid, 256, 0, st>>>(P, bf, (const T*)qwin, nch);
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
