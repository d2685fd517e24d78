// Quality metric: attention-mass coverage of a kept set (Section 1, Fig. 1b:
// the share of decode-time attention probability that falls on the prompt
// entries kept after prefill). The decode queries run through steps 2-4 as
// n_dec groups of one proxy each, so the group masses hold, per (layer, KV
// head, decode query, key), the attention probability summed over the r query
// heads; coverage_kernel divides the masses of the kept keys by the masses of
// all T_b keys (r up to rounding).
#include "common.cuh"

namespace mmshift {
namespace {

constexpr int kCovThreads = 256;

__device__ __forceinline__ float block_sum(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float s = 0.f;
  if (warp == 0) {
    s = lane < kCovThreads / 32 ? red[lane] : 0.f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  }
  __syncthreads();
  return s;   // valid in thread 0
}

// One CTA per (decode query g, KV head h, layer x request); fixed-order sums.
__global__ void __launch_bounds__(kCovThreads) coverage_kernel(Problem P, const float* gmass,
                                                               const int32_t* idx, float* cov,
                                                               int* status) {
  __shared__ float red[kCovThreads / 32];
  const int g = blockIdx.x, h = blockIdx.y;
  const int l = blockIdx.z / P.B, b = blockIdx.z % P.B;
  const ReqInfo R = P.req[b];
  const float* row = gmass + (((size_t)l * P.Hkv + h) * P.G + g) * P.total_T + R.tok_off;
  const int32_t* id = idx + ((size_t)l * P.R + R.out_off) * P.Hkv + h;
  float kept = 0.f, tot = 0.f;
  bool bad = false;
  for (int c = threadIdx.x; c < R.keep; c += kCovThreads) {
    const int t = id[(size_t)c * P.Hkv];
    if ((unsigned)t < (unsigned)R.t_len) kept += row[t];
    else if (t != -1) bad = true;   // -1: padding row of a head with a smaller budget
  }
  for (int t = threadIdx.x; t < R.t_len; t += kCovThreads) tot += row[t];
  if (bad) set_status(status, kStatusBadIndex);
  kept = block_sum(kept, red);
  tot = block_sum(tot, red);
  if (threadIdx.x == 0)
    cov[(((size_t)l * P.B + b) * P.Hkv + h) * P.G + g] = tot > 0.f ? kept / tot : 0.f;
}

}  // namespace

cudaError_t launch_coverage(const Problem& P, const Buffers& bf, const int32_t* idx, float* cov,
                            cudaStream_t st) {
  if (P.G == 0 || P.R == 0) return cudaSuccess;
  dim3 grid(P.G, P.Hkv, P.L * P.B);
  coverage_kernel<<<grid, kCovThreads, 0, st>>>(P, bf.gmass, idx, cov, bf.status);
  return cudaGetLastError();
}

}  // namespace mmshift
