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
//
// bf16 proxies equal the bf16 rounding of the exact (real-number) value of
// mu + gamma * sigma * z, rotated: the float32 evaluation is within a bound
// of that value (2^-20 of the magnitudes involved, 2^-19 rotated; below), so
// it rounds to the same bf16 unless a rounding boundary lies within the bound.
// Such elements (about four in ten thousand) are recomputed in float64 -- the
// window statistics from their exact sums, the normal (log, sin, cos of the
// same 24-bit uniforms), the sum and the rotation -- and rounded from there by
// refine_kernel, from a list in the workspace. A call without a workspace
// (mmshift_build_proxies), or whose list overflowed, has every element
// recomputed in float64.
//
// Window statistics: per (query head, dimension) the sums of d = x - x0 and
// d^2 over the W rows (x0 the first row's value) are kept as unevaluated
// float32 pairs by error-free additions and products (Knuth's TwoSum,
// Dekker's product through an FMA), so they are exact up to about 2^-43;
// mean = x0 + S1/W and variance (S2 - S1^2/W)/(W-1) follow in pairs too,
// each then rounded once to float32.
#include <algorithm>
#include <type_traits>

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

// (hi, lo) += x: the rounding error of hi + x (Knuth's TwoSum) goes into lo.
__device__ __forceinline__ void df_add(float& hi, float& lo, float x) {
  const float t = hi + x;
  const float bp = t - hi;
  lo += (hi - (t - bp)) + (x - bp);
  hi = t;
}

// Per (query head, dimension) window sums of a thread or a block: x0 and the
// pairs S1 = sum (x - x0), S2 = sum (x - x0)^2.
struct WinSums {
  float s1h, s1l, s2h, s2l;
};

// Adds row value x (d = x - x0 is exact in float32 for bf16 and float32 data
// of the same scale; d^2 is split exactly into d*d and its FMA remainder).
__device__ __forceinline__ void win_add(WinSums& w, float x, float x0) {
  const float d = x - x0;
  df_add(w.s1h, w.s1l, d);
  const float p = d * d;
  df_add(w.s2h, w.s2l, p);
  w.s2l += fmaf(d, d, -p);
}

// Mean and unbiased std (float32) of W rows from their sums; |mean - x0| in
// *dev (it enters the error bound of the mean). S1^2 / W is formed as a pair
// (Dekker's product, then the exact remainder of the rounded quotient), so
// the cancellation in S2 - S1^2 / W costs no accuracy.
__device__ __forceinline__ void win_stats(const WinSums& w, float x0, int W, float& mu, float& sg,
                                          float& dev) {
  const float fw = (float)W;
  const float m1 = (w.s1h + w.s1l) / fw;
  mu = x0 + m1;
  dev = fabsf(m1);
  const float p = w.s1h * w.s1h;
  const float e = fmaf(w.s1h, w.s1h, -p) + 2.0f * w.s1h * w.s1l;
  const float q = p / fw;
  const float ql = (fmaf(-q, fw, p) + e) / fw;
  float nh = w.s2h, nl = w.s2l;
  df_add(nh, nl, -q);
  const float var = (nh + (nl - ql)) / (float)(W - 1);
  sg = sqrtf(fmaxf(var, 0.f));
}

// Bound on |float32 value - exact value| of a proxy element relative to the
// magnitudes it is made of: |mu| + |mean - x0| + |gamma sigma z|, summed over
// the RoPE pair when rotated. Unrotated the float32 path stays within about
// 9 ulp of them: the normal about 4.8 (log 3, square root 0.5, sine / cosine
// 2), sigma and gamma sigma 1.8, the mean 1, the FMA 0.5. Rotated, the
// table's sine / cosine (2 ulp) and the rotation's roundings add about 3.5.
constexpr float kRefineRel = 1.0f / 1048576.0f;      // 2^-20
constexpr float kRefineRelRope = 1.0f / 524288.0f;   // 2^-19

// Whether rounding to bf16 is decided by the float32 value v within +-err
// (both ends rounded by one paired conversion).
__device__ __forceinline__ bool bf16_undecided(float v, float err) {
  const __nv_bfloat162 r = __floats2bfloat162_rn(v - err, v + err);
  const uint32_t u = *reinterpret_cast<const uint32_t*>(&r);
  return (u & 0xFFFFu) != (u >> 16);
}

// Packed row of proxy i of local query head j (group-major rows).
__device__ __forceinline__ size_t packed_row(const Problem& P, int i, int j) {
  const int g = i / P.gs, ii = i - g * P.gs;
  return (size_t)g * P.RG + (size_t)j * P.gs + ii;
}

// Window mean and std of (request b of call layer l, query head hq, dim dd)
// in float64: from the exact sums the sampler stored (rs: [L][B][Hq][5][D]
// = x0, S1 hi / lo, S2 hi / lo), or, without them, from the W rows summed in
// row order.
template <int D>
__device__ void win_stats_f64(const Problem& P, const float* rs, const __nv_bfloat16* qwin, int l,
                              int b, int hq, int dd, double& mu, double& sig) {
  const double fw = (double)P.W;
  if (rs) {
    const float* r = rs + ((((size_t)l * P.B + b) * P.Hq + hq) * 5) * D + dd;
    const double x0 = r[0], s1 = (double)r[D] + (double)r[2 * D],
                 s2 = (double)r[3 * D] + (double)r[4 * D];
    mu = x0 + s1 / fw;
    sig = sqrt(fmax((s2 - s1 * s1 / fw) / (double)(P.W - 1), 0.0));
    return;
  }
  const __nv_bfloat16* q = qwin + (size_t)l * P.ls_q + ((size_t)b * P.W * P.Hq + hq) * D + dd;
  const size_t qs = (size_t)P.Hq * D;
  // rows in blocks of eight independent loads, added in row order
  double sum = 0.0;
  for (int w0 = 0; w0 < P.W; w0 += 8) {
    float x[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) x[k] = w0 + k < P.W ? __bfloat162float(q[(size_t)(w0 + k) * qs]) : 0.f;
#pragma unroll
    for (int k = 0; k < 8; ++k)
      if (w0 + k < P.W) sum = __dadd_rn(sum, (double)x[k]);
  }
  mu = __ddiv_rn(sum, fw);
  double var = 0.0;
  for (int w0 = 0; w0 < P.W; w0 += 8) {
    float x[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) x[k] = w0 + k < P.W ? __bfloat162float(q[(size_t)(w0 + k) * qs]) : 0.f;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      if (w0 + k < P.W) {
        const double dv = __dadd_rn((double)x[k], -mu);
        var = __dadd_rn(var, __dmul_rn(dv, dv));
      }
    }
  }
  sig = __dsqrt_rn(__ddiv_rn(var, (double)(P.W - 1)));
}

// Proxy element (request b of call layer l, query head hq, proxy i, dim dd)
// before rotation, in float64: mu + (gamma sigma) z with z from the same
// Philox words as the float32 path.
template <int D>
__device__ double proxy_f64(const Problem& P, const float* rs, const __nv_bfloat16* qwin, int l,
                            int b, int hq, int i, int dd) {
  double mu, sig;
  win_stats_f64<D>(P, rs, qwin, l, b, hq, dd, mu, sig);
  const int half = D / 2;
  const int qq = dd < half ? dd / 4 : (dd - half) / 4;
  const int k = dd < half ? dd % 4 : 4 + (dd - half) % 4;    // normal k of the draw
  uint64_t c[4] = {(uint64_t)i * (uint64_t)(D / 8) + (uint64_t)qq, (uint64_t)hq, (uint64_t)b,
                   (uint64_t)(int64_t)(P.layer_id0 + l)};
  philox4x64_10(c, P.seed, 0ull);
  const uint64_t w64 = c[k / 2];
  const double u1 = ((double)((uint32_t)w64 >> 9) + 0.5) * 1.1920928955078125e-07;
  const double u2 = ((double)((uint32_t)(w64 >> 32) >> 9) + 0.5) * 1.1920928955078125e-07;
  const double rad = sqrt(-2.0 * log(u1));
  const double z = __dmul_rn(rad, (k & 1) ? sinpi(2.0 * u2) : cospi(2.0 * u2));
  return __dadd_rn(mu, __dmul_rn(__dmul_rn((double)P.gamma, sig), z));
}

// Recompute element (l, b, hq, i, dd) in float64 and store its bf16 rounding
// in the packed block and the caller-layout copy.
template <int D>
__device__ void refine_element(const Problem& P, const Buffers& bf, const __nv_bfloat16* qwin,
                               int l, int b, int hq, int i, int dd) {
  const int half = D / 2;
  double v;
  if (P.rope_theta > 0.f) {
    const int f = dd % half;
    const double a = proxy_f64<D>(P, bf.refine_stats, qwin, l, b, hq, i, f);
    const double c = proxy_f64<D>(P, bf.refine_stats, qwin, l, b, hq, i, f + half);
    const double pos = (double)(P.req[b].t_len + P.rope_off);
    const double ang = pos * pow((double)P.rope_theta, -2.0 * f / (double)D);
    double sn, cs;
    sincos(ang, &sn, &cs);
    v = dd < half ? __dadd_rn(__dmul_rn(a, cs), -__dmul_rn(c, sn))
                  : __dadd_rn(__dmul_rn(c, cs), __dmul_rn(a, sn));
  } else {
    v = proxy_f64<D>(P, bf.refine_stats, qwin, l, b, hq, i, dd);
  }
  const __nv_bfloat16 o = __double2bfloat16(v);
  const int h = hq / P.r, j = hq - h * P.r;
  if (bf.packed) {
    __nv_bfloat16* packed = (__nv_bfloat16*)bf.packed +
                            ((((size_t)l * P.B + b) * P.Hkv + h) * P.Prows_pad) * D;
    packed[packed_row(P, i, j) * D + dd] = o;
  }
  if (bf.proxies_out)
    ((__nv_bfloat16*)bf.proxies_out)[((((size_t)l * P.B + b) * P.Hq + hq) * P.Np + i) * D + dd] = o;
}

// Appends the undecided elements (bit k: element k of the thread's draw) of
// proxy i to the refinement list. The count keeps growing past the list's
// capacity, which tells refine_kernel to redo the whole call.
template <int D>
__device__ __noinline__ void enlist(const Problem& P, const Buffers& bf, int l, int b, int hq,
                                    int i, int qq, uint32_t undecided) {
  while (undecided) {
    const int k = __ffs(undecided) - 1;
    undecided &= undecided - 1;
    const int dd = k < 4 ? 4 * qq + k : D / 2 + 4 * qq + (k - 4);
    const int slot = atomicAdd(bf.refine_count, 1);
    if (slot < bf.refine_cap) bf.refine_items[slot] = make_int4(l * P.B + b, hq, i, dd);
  }
}

// Proxies of one query head are spread over up to kProxyChunks CTAs, about
// 1024 Philox draws each (few proxies: one CTA per query head).
constexpr int kProxyChunks = 8;

template <typename T, int D>
__global__ void __launch_bounds__(256, 6) proxy_pack_kernel(Problem P, Buffers bf, const T* qwin,
                                                         int nch) {
  const int hq = blockIdx.x / nch, chunk = blockIdx.x % nch;
  const int b = blockIdx.y, l = blockIdx.z;
  const int h = hq / P.r, j = hq - h * P.r;
  // mean, std, and |mean| + |mean - x0| (the mean's part of the error bound)
  __shared__ float mu[D], sg[D], mmag[D], rc[D / 2], rs[D / 2];
  constexpr int RPT = 256 / D;               // threads per dimension
  __shared__ WinSums part[RPT][D];
  const T* q = qwin ? qwin + (size_t)l * P.ls_q + ((size_t)b * P.W * P.Hq + hq) * D : nullptr;
  const size_t qstride = (size_t)P.Hq * D;
  if (bf.stats_in) {
    // given statistics (e.g. over the whole prefill): [L][B][2][Hq][D]
    const float* st = bf.stats_in + (((size_t)l * P.B + b) * 2 * P.Hq + hq) * D;
    for (int k = threadIdx.x; k < D; k += blockDim.x) {
      mu[k] = st[k];
      sg[k] = st[(size_t)P.Hq * D + k];
      mmag[k] = fabsf(mu[k]);
    }
  } else {
    // exact window sums: thread (k, rg) takes rows rg, rg + RPT, ... of
    // dimension k (independent, unrolled loads); the block adds the partials
    const int k = threadIdx.x % D, rg = threadIdx.x / D;
    const float x0 = to_f32(q[k]);
    WinSums w{0.f, 0.f, 0.f, 0.f};
#pragma unroll 8
    for (int r = rg; r < P.W; r += RPT) win_add(w, to_f32(q[r * qstride + k]), x0);
    part[rg][k] = w;
    __syncthreads();
    if (rg == 0) {
      WinSums t = part[0][k];
#pragma unroll
      for (int g = 1; g < RPT; ++g) {
        df_add(t.s1h, t.s1l, part[g][k].s1h);
        t.s1l += part[g][k].s1l;
        df_add(t.s2h, t.s2l, part[g][k].s2h);
        t.s2l += part[g][k].s2l;
      }
      float dev;
      win_stats(t, x0, P.W, mu[k], sg[k], dev);
      mmag[k] = fabsf(mu[k]) + dev;
      if (bf.refine_stats && chunk == 0) {
        // the exact sums, for the float64 recomputation of undecided elements
        float* rsd = bf.refine_stats + ((((size_t)l * P.B + b) * P.Hq + hq) * 5) * D + k;
        rsd[0] = x0;
        rsd[D] = t.s1h;
        rsd[2 * D] = t.s1l;
        rsd[3 * D] = t.s2h;
        rsd[4 * D] = t.s2l;
      }
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
      uint32_t undecided = 0;
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int d0 = 4 * qq + k, d1 = D / 2 + 4 * qq + k;
        const float g0 = P.gamma * sg[d0], g1 = P.gamma * sg[d1];
        float a = fmaf(g0, z[k], mu[d0]), c = fmaf(g1, z[4 + k], mu[d1]);
        float ma = mmag[d0] + fabsf(g0 * z[k]), mc = mmag[d1] + fabsf(g1 * z[4 + k]);
        if (rope) {
          const float ar = a * rc[d0] - c * rs[d0];
          c = c * rc[d0] + a * rs[d0];
          a = ar;
          ma = mc = ma + mc;
        }
        v[k] = a;
        v[4 + k] = c;
          if constexpr (std::is_same<T, __nv_bfloat16>::value) {
          const float rel = rope ? kRefineRelRope : kRefineRel;
          undecided |= (bf16_undecided(a, rel * ma) ? 1u : 0u) << k;
          undecided |= (bf16_undecided(c, rel * mc) ? 1u : 0u) << (4 + k);
        }
      }
      if (undecided && bf.refine_items && !bf.stats_in) enlist<D>(P, bf, l, b, hq, i, qq, undecided);
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

// Elements the sampler found undecided, recomputed in float64, one thread
// per list entry. A call whose entries overflowed the list, or that has no
// list (all = true), has every element recomputed.
template <int D>
__global__ void __launch_bounds__(128) refine_kernel(Problem P, Buffers bf, const __nv_bfloat16* qwin,
                                                     bool all) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t t0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (!all) {
    const int cnt = *bf.refine_count;
    if (cnt <= bf.refine_cap) {
      for (int64_t e = t0; e < cnt; e += stride) {
        const int4 it = bf.refine_items[e];
        const int l = it.x / P.B, b = it.x - l * P.B;
        refine_element<D>(P, bf, qwin, l, b, it.y, it.z, it.w);
      }
      return;
    }
  }
  const int64_t n = (int64_t)P.L * P.B * P.Hq * P.Np * D;
  for (int64_t e = t0; e < n; e += stride) {
    int64_t r = e;
    const int dd = (int)(r % D); r /= D;
    const int i = (int)(r % P.Np); r /= P.Np;
    const int hq = (int)(r % P.Hq); r /= P.Hq;
    const int b = (int)(r % P.B);
    const int l = (int)(r / P.B);
    refine_element<D>(P, bf, qwin, l, b, hq, i, dd);
  }
}

// Whether a call samples bf16 proxies (then refine_kernel follows the
// sampler), and whether it has a refinement list.
bool samples_bf16(const Problem& P, const Buffers& bf) {
  return P.dtype == MMSHIFT_BF16 && P.Np > 0 && !bf.proxies_in && !bf.stats_in;
}
bool has_refine_list(const Buffers& bf) {
  return bf.refine_items && bf.refine_count && bf.refine_cap > 0;
}

template <typename T, int D>
cudaError_t launch_t(const Problem& P, const Buffers& bf, cudaStream_t st, const void* qwin) {
  const int draws = P.Np * (D / 8);
  const int nch = draws <= 0 ? 1 : std::min(kProxyChunks, (draws + 1023) / 1024);
  const bool refine = samples_bf16(P, bf);
  Buffers b2 = bf;
  if (!has_refine_list(bf)) {
    b2.refine_items = nullptr;
    b2.refine_count = nullptr;
    b2.refine_cap = 0;
    b2.refine_stats = nullptr;
  }
  cudaError_t e;
  if (refine && b2.refine_items &&
      (e = cudaMemsetAsync(b2.refine_count, 0, sizeof(int), st)) != cudaSuccess)
    return e;
  dim3 grid(P.Hq * nch, P.B, P.L);
  proxy_pack_kernel<T, D><<<grid, 256, 0, st>>>(P, b2, (const T*)qwin, nch);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  if (refine) {
    int dev = 0, nsm = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
      return e;
    const bool all = b2.refine_items == nullptr;
    refine_kernel<D><<<8 * std::max(nsm, 1), 128, 0, st>>>(
        P, b2, (const __nv_bfloat16*)qwin, all);
    e = cudaGetLastError();
  }
  return e;
}

}  // namespace

int64_t proxy_refine_capacity(const Problem& P) {
  const int64_t elems = (int64_t)P.L * P.B * P.Hq * P.Np * P.d;
  return std::min<int64_t>(elems / 256 + 4096, (int64_t)1 << 30);
}

int proxy_launches(const Problem& P, const Buffers& bf) { return samples_bf16(P, bf) ? 2 : 1; }

cudaError_t launch_proxy_pack(const Problem& P, const Buffers& bf, cudaStream_t st,
                              const void* qwin) {
  if (P.dtype == MMSHIFT_BF16)
    return P.d == 128 ? launch_t<__nv_bfloat16, 128>(P, bf, st, qwin)
                      : launch_t<__nv_bfloat16, 64>(P, bf, st, qwin);
  return P.d == 128 ? launch_t<float, 128>(P, bf, st, qwin) : launch_t<float, 64>(P, bf, st, qwin);
}

}  // namespace mmshift
