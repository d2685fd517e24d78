// Proxy statistics over the whole prefill (Section 3.2.1: mean and standard
// deviation of the prompt's features across all prompt tokens; read in query
// space, per (query head, dimension) over the T prompt queries of a request,
// with the unbiased T - 1 estimator).
//
// A streaming reduction over Q [L][total_T][Hq][d]: every byte of Q is read
// once, in coalesced 16-byte vectors, so the pass is bounded by HBM.
//  - stats_partial_kernel: one CTA per chunk of kStatsChunk prompt queries of
//    one request and layer, one thread per 8 consecutive columns (q-head,
//    dimension) up to 1024 threads; a thread keeps, per column, the sums of
//    (x - x0) and (x - x0)^2 in fp32, x0 being the chunk's first query (the
//    shift keeps the second sum free of cancellation), with eight rows' loads
//    in flight.
//  - stats_merge_kernel: one thread per column merges the chunks in order with
//    the pairwise update of Chan, Golub and LeVeque (count, mean, sum of
//    squared deviations), then writes mean and std.
#include <algorithm>

#include "common.cuh"

namespace mmshift {
namespace {

constexpr int kStatsRows = 8;      // rows of loads in flight per thread
constexpr int kMergeAhead = 8;     // chunks of partial sums loaded ahead in the merge

template <typename T>
__device__ __forceinline__ void load8(const T* p, float (&x)[8]);
template <>
__device__ __forceinline__ void load8<__nv_bfloat16>(const __nv_bfloat16* p, float (&x)[8]) {
  const uint4 v = __ldg(reinterpret_cast<const uint4*>(p));
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    x[2 * i] = __uint_as_float(w[i] << 16);
    x[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
  }
}
template <>
__device__ __forceinline__ void load8<float>(const float* p, float (&x)[8]) {
  const float4 a = __ldg(reinterpret_cast<const float4*>(p));
  const float4 b = __ldg(reinterpret_cast<const float4*>(p) + 1);
  x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w;
  x[4] = b.x; x[5] = b.y; x[6] = b.z; x[7] = b.w;
}

// part: [L][B][nchunk][3][ncol] (x0, sum of x - x0, sum of (x - x0)^2)
template <typename T>
__global__ void __launch_bounds__(1024) stats_partial_kernel(StatsJob J, const T* Q, float* part) {
  const int c = blockIdx.x, b = blockIdx.y, l = blockIdx.z;
  const int t_len = J.t_len[b];
  const int t0 = c * kStatsChunk;
  if (t0 >= t_len) return;
  const int t1 = min(t_len, t0 + kStatsChunk);
  const T* q = Q + (size_t)l * J.ls + ((size_t)J.tok_off[b] + t0) * J.ncol;
  float* out = part + (((size_t)l * J.B + b) * J.nchunk + c) * 3 * J.ncol;
  for (int cg = threadIdx.x; cg < J.ncol / 8; cg += blockDim.x) {
    const T* col = q + (size_t)cg * 8;
    float x0[8], s1[8], s2[8];
    load8(col, x0);
#pragma unroll
    for (int k = 0; k < 8; ++k) { s1[k] = 0.f; s2[k] = 0.f; }
    int t = 1;
    // kStatsRows independent rows in flight
    for (; t + kStatsRows <= t1 - t0; t += kStatsRows) {
      float x[kStatsRows][8];
#pragma unroll
      for (int u = 0; u < kStatsRows; ++u) load8(col + (size_t)(t + u) * J.ncol, x[u]);
#pragma unroll
      for (int u = 0; u < kStatsRows; ++u)
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const float dv = x[u][k] - x0[k];
          s1[k] += dv;
          s2[k] = fmaf(dv, dv, s2[k]);
        }
    }
    for (; t < t1 - t0; ++t) {
      float x[8];
      load8(col + (size_t)t * J.ncol, x);
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const float dv = x[k] - x0[k];
        s1[k] += dv;
        s2[k] = fmaf(dv, dv, s2[k]);
      }
    }
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      out[cg * 8 + k] = x0[k];
      out[J.ncol + cg * 8 + k] = s1[k];
      out[2 * J.ncol + cg * 8 + k] = s2[k];
    }
  }
}

// stats: [L][B][2][ncol] (mean, std)
__global__ void __launch_bounds__(256) stats_merge_kernel(StatsJob J, const float* part,
                                                          float* stats) {
  const int col = blockIdx.x * blockDim.x + threadIdx.x;
  const int b = blockIdx.y, l = blockIdx.z;
  if (col >= J.ncol) return;
  const int t_len = J.t_len[b];
  const float* in = part + ((size_t)l * J.B + b) * J.nchunk * 3 * J.ncol + col;
  float n = 0.f, mean = 0.f, m2 = 0.f;
  const int nch = (t_len + kStatsChunk - 1) / kStatsChunk;
  for (int c0 = 0; c0 < nch; c0 += kMergeAhead) {
    // the loads of kMergeAhead chunks first, then the merges in chunk order
    float v[kMergeAhead][3];
#pragma unroll
    for (int u = 0; u < kMergeAhead; ++u)
      if (c0 + u < nch)
#pragma unroll
        for (int q = 0; q < 3; ++q) v[u][q] = in[((size_t)(c0 + u) * 3 + q) * J.ncol];
#pragma unroll
    for (int u = 0; u < kMergeAhead; ++u) {
      const int c = c0 + u;
      if (c >= nch) break;
      const float nb = (float)(min(t_len, (c + 1) * kStatsChunk) - c * kStatsChunk);
      const float x0 = v[u][0], s1 = v[u][1], s2 = v[u][2];
      const float mb = x0 + s1 / nb;
      const float m2b = fmaxf(s2 - s1 * (s1 / nb), 0.f);
      const float nab = n + nb;
      const float delta = mb - mean;
      mean += delta * (nb / nab);
      m2 += m2b + delta * delta * (n * nb / nab);
      n = nab;
    }
  }
  float* out = stats + ((size_t)l * J.B + b) * 2 * J.ncol;
  out[col] = mean;
  out[J.ncol + col] = t_len > 1 ? sqrtf(m2 / (float)(t_len - 1)) : 0.f;
}

}  // namespace

cudaError_t launch_prefill_stats(const StatsJob& J, const void* Q, float* part, float* stats,
                                 cudaStream_t st, bool bf16) {
  dim3 g1(J.nchunk, J.B, J.L);
  const int threads = std::min(1024, (J.ncol / 8 + 31) / 32 * 32);
  if (bf16)
    stats_partial_kernel<__nv_bfloat16><<<g1, threads, 0, st>>>(J, (const __nv_bfloat16*)Q, part);
  else
    stats_partial_kernel<float><<<g1, threads, 0, st>>>(J, (const float*)Q, part);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  dim3 g2((J.ncol + 255) / 256, J.B, J.L);
  stats_merge_kernel<<<g2, 256, 0, st>>>(J, part, stats);
  return cudaGetLastError();
}

}  // namespace mmshift
