// Steps 2-4 on CUDA cores (fp32 FMA): proxy logits, row softmax over the whole
// prompt and group-mass aggregation (Section 3.2.2; Appendix B).
//
// This path serves float32 inputs, for which the tensor cores would round the
// operands (TF32), and head dims or shapes the tcgen05 path does not cover.
//
// Pass 1: CTA = (layer, KV head, key split, 64 packed proxy rows). It streams
//   the keys of its split through shared memory and keeps, per proxy row, an
//   online (max, sum of exp2) pair of the log2-scaled logits x = s * alpha,
//   alpha = softmax_scale * log2(e).
// Merge: combines the partials of each row (one per key split, two on the
//   tensor-core path) in a fixed order into c = m + log2(Z) (the log2
//   normaliser), +inf for padding rows so they weigh nothing.
// Pass 2: CTA = (layer, KV head, 64 keys). It streams every packed proxy row,
//   recomputes the logits and adds exp2(x - c) into per-(group, key) sums in a
//   fixed order, then writes the group masses and the anchor (mean over the r
//   anchor rows).
#include "common.cuh"

namespace mmshift {
namespace {

constexpr int TILE = 64;

__device__ __forceinline__ void find_split(const Problem& P, int s, int& b, int& sl) {
  b = 0;
  while (b + 1 < P.B && P.req[b + 1].split_off <= s) ++b;
  sl = s - P.req[b].split_off;
}

// 64x64 logits tile: acc[i][j] = A_row(ty*4+i) . B_row(tx*4+j) over D dims,
// A and B in shared memory with row stride D+1.
template <int D>
__device__ __forceinline__ void tile_dot(const float* A, const float* Bm, int ty, int tx,
                                         float acc[4][4]) {
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
#pragma unroll 4
  for (int k = 0; k < D; ++k) {
    float a[4], bv[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) a[i] = A[(ty * 4 + i) * (D + 1) + k];
#pragma unroll
    for (int j = 0; j < 4; ++j) bv[j] = Bm[(tx * 4 + j) * (D + 1) + k];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], bv[j], acc[i][j]);
  }
}


template <typename T, int D>
__global__ void __launch_bounds__(256) pass1_simt(Problem P, Buffers bf, const T* K) {
  extern __shared__ float sm[];
  float* Ps = sm;                    // [64][D+1] proxy rows
  float* Ks = Ps + TILE * (D + 1);   // [64][D+1] keys
  float* Ls = Ks + TILE * (D + 1);   // [64][65] scaled logits
  const int n_rt = P.Prows_pad / TILE;
  int u = blockIdx.x;
  const int rt = u % n_rt; u /= n_rt;
  const int s = u % P.total_splits; u /= P.total_splits;
  const int h = u, l = blockIdx.y;
  int b, sl;
  find_split(P, s, b, sl);
  const ReqInfo R = P.req[b];
  const int t0 = sl * P.split_len, t1 = min(R.t_len, t0 + P.split_len);
  const int tid = threadIdx.x, ty = tid / 16, tx = tid % 16;

  const T* pk = (const T*)bf.packed +
                ((((size_t)l * P.B + b) * P.Hkv + h) * P.Prows_pad + (size_t)rt * TILE) * D;
  for (int e = tid; e < TILE * D; e += 256) Ps[(e / D) * (D + 1) + e % D] = to_f32(pk[e]);
  const T* kb = K + (size_t)l * P.ls_kv + ((size_t)R.tok_off * P.Hkv + h) * D;
  const size_t kstride = (size_t)P.Hkv * D;

  float run_m = -INFINITY, run_z = 0.f;
  const int row = tid / 4, part = tid % 4;
  for (int kt = t0; kt < t1; kt += TILE) {
    __syncthreads();
    for (int e = tid; e < TILE * D; e += 256) {
      const int kk = e / D, c = e - kk * D, t = kt + kk;
      Ks[kk * (D + 1) + c] = t < t1 ? to_f32(kb[(size_t)t * kstride + c]) : 0.f;
    }
    __syncthreads();
    float acc[4][4];
    tile_dot<D>(Ps, Ks, ty, tx, acc);
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int kk = tx * 4 + j;
        Ls[(ty * 4 + i) * (TILE + 1) + kk] = (kt + kk < t1) ? acc[i][j] * P.alpha : -INFINITY;
      }
    __syncthreads();
    float m = -INFINITY;
    for (int c = part * 16; c < part * 16 + 16; ++c) m = fmaxf(m, Ls[row * (TILE + 1) + c]);
    float z = 0.f;
    if (m != -INFINITY)
      for (int c = part * 16; c < part * 16 + 16; ++c) z += fast_exp2(Ls[row * (TILE + 1) + c] - m);
#pragma unroll
    for (int off = 1; off < 4; off <<= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
      const float z2 = __shfl_xor_sync(0xffffffffu, z, off);
      merge_ms(m, z, m2, z2);
    }
    merge_ms(run_m, run_z, m, z);
  }
  if (part == 0)
    bf.part[(((size_t)l * P.Hkv + h) * P.total_splits + s) * P.part_slots * P.Prows_pad +
            rt * TILE + row] = make_float2(run_m, run_z);
}

// SUB threads per row (four when a row has at least 128 partials, else one):
// thread q of a row merges the row's partials q, q + SUB, q + 2 SUB, ... in
// order (eight loads issued ahead), then the SUB results are merged by xor
// shuffles; for a given SUB the order is fixed, and SUB depends only on the
// call's shape.
template <int kMergeSub>
__global__ void merge_kernel(Problem P, Buffers bf) {
  const int q = threadIdx.x % kMergeSub;
  const int p = blockIdx.x * (blockDim.x / kMergeSub) + threadIdx.x / kMergeSub;
  const int bh = blockIdx.y, l = blockIdx.z;
  const int b = bh / P.Hkv, h = bh - b * P.Hkv;
  // with anchor_split the softmax pass has no partials for the anchor rows
  const int rows = P.anchor_split ? P.n_group_rows : P.Prows_pad;
  const bool live = p < rows;
  const ReqInfo R = P.req[b];
  float m = -INFINITY, z = 0.f;
  const float2* src = bf.part +
                      (((size_t)l * P.Hkv + h) * P.total_splits + R.split_off) * P.part_slots * P.Prows_pad +
                      (live ? p : 0);
  const int ns = live ? R.nsplit * P.part_slots : 0;
  constexpr int A = 8;
  for (int s0 = q; s0 < ns; s0 += A * kMergeSub) {
    float2 v[A];
#pragma unroll
    for (int u = 0; u < A; ++u) {
      const int si = s0 + u * kMergeSub;
      v[u] = si < ns ? src[(size_t)si * P.Prows_pad] : make_float2(-INFINITY, 0.f);
    }
#pragma unroll
    for (int u = 0; u < A; ++u)
      if (s0 + u * kMergeSub < ns) merge_ms(m, z, v[u].x, v[u].y);
  }
#pragma unroll
  for (int off = 1; off < kMergeSub; off <<= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
    const float z2 = __shfl_xor_sync(0xffffffffu, z, off);
    merge_ms(m, z, m2, z2);
  }
  if (!live || q) return;
  const bool valid = row_kind(P, p).group >= 0;
  bf.cvals[(((size_t)l * P.B + b) * P.Hkv + h) * P.Prows_pad + p] =
      valid ? m + __log2f(z) : INFINITY;
}

template <typename T, int D>
__global__ void __launch_bounds__(256) pass2_simt(Problem P, Buffers bf, const T* K) {
  extern __shared__ float sm[];
  float* Ks = sm;                    // [64][D+1] keys (stationary)
  float* Ps = Ks + TILE * (D + 1);   // [64][D+1] proxy rows
  float* Ls = Ps + TILE * (D + 1);   // [64][65] exp2(x - c)
  float* cs = Ls + TILE * (TILE + 1);// [64]
  float* gacc = cs + TILE;           // [G+1][64]
  int u = blockIdx.x;
  const int l = blockIdx.y;
  const int h = u % P.Hkv;
  u /= P.Hkv;
  int b = 0;
  for (; b < P.B; ++b) {
    const int nt = (P.req[b].t_len + TILE - 1) / TILE;
    if (u < nt) break;
    u -= nt;
  }
  const ReqInfo R = P.req[b];
  const int kt = u * TILE;
  const int tid = threadIdx.x, ty = tid / 16, tx = tid % 16;
  const T* kb = K + (size_t)l * P.ls_kv + ((size_t)R.tok_off * P.Hkv + h) * D;
  const size_t kstride = (size_t)P.Hkv * D;
  for (int e = tid; e < TILE * D; e += 256) {
    const int kk = e / D, c = e - kk * D, t = kt + kk;
    Ks[kk * (D + 1) + c] = t < R.t_len ? to_f32(kb[(size_t)t * kstride + c]) : 0.f;
  }
  for (int e = tid; e < (P.G + 1) * TILE; e += 256) gacc[e] = 0.f;
  const T* pk = (const T*)bf.packed + ((((size_t)l * P.B + b) * P.Hkv + h) * P.Prows_pad) * D;
  const float* cv = bf.cvals + (((size_t)l * P.B + b) * P.Hkv + h) * P.Prows_pad;
  const int key = tid % TILE, ch = tid / TILE;
  for (int pt = 0; pt < P.Prows_pad / TILE; ++pt) {
    __syncthreads();
    for (int e = tid; e < TILE * D; e += 256)
      Ps[(e / D) * (D + 1) + e % D] = to_f32(pk[(size_t)pt * TILE * D + e]);
    if (tid < TILE) cs[tid] = cv[pt * TILE + tid];
    __syncthreads();
    float acc[4][4];
    tile_dot<D>(Ps, Ks, ty, tx, acc);
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int pr = ty * 4 + i;
        Ls[pr * (TILE + 1) + tx * 4 + j] = fast_exp2(fmaf(acc[i][j], P.alpha, -cs[pr]));
      }
    __syncthreads();
    float csum = 0.f;
    for (int rr = 0; rr < kChunk; ++rr) csum += Ls[(ch * kChunk + rr) * (TILE + 1) + key];
    const int g = chunk_group(P, pt * (TILE / kChunk) + ch);
    for (int c = 0; c < TILE / kChunk; ++c) {
      if (ch == c) gacc[g * TILE + key] += csum;
      __syncthreads();
    }
  }
  __syncthreads();
  const int t = kt + key;
  if (t < R.t_len) {
    const size_t col = (size_t)R.tok_off + t;
    for (int g = ch; g < P.G; g += 256 / TILE)
      bf.gmass[(((size_t)l * P.Hkv + h) * P.G + g) * P.total_T + col] = gacc[g * TILE + key];
    if (ch == 0)
      bf.anchor[((size_t)l * P.Hkv + h) * P.total_T + col] = gacc[P.G * TILE + key] / (float)P.r;
  }
}

template <typename T, int D>
cudaError_t launch_t(const Problem& P, const Buffers& bf, cudaStream_t st, const void* K,
                     cudaEvent_t* ev) {
  const size_t sm1 = (2 * TILE * (D + 1) + TILE * (TILE + 1)) * sizeof(float);
  const size_t sm2 = sm1 + (TILE + (size_t)(P.G + 1) * TILE) * sizeof(float);
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(pass1_simt<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)sm1)) != cudaSuccess) return e;
  if ((e = cudaFuncSetAttribute(pass2_simt<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)sm2)) != cudaSuccess) return e;
  dim3 g1(P.Hkv * P.total_splits * (P.Prows_pad / TILE), P.L);
  if (ev && (e = cudaEventRecord(ev[1], st)) != cudaSuccess) return e;
  pass1_simt<T, D><<<g1, 256, sm1, st>>>(P, bf, (const T*)K);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  if (ev && (e = cudaEventRecord(ev[2], st)) != cudaSuccess) return e;
  if ((e = launch_merge(P, bf, st)) != cudaSuccess) return e;
  if (ev && (e = cudaEventRecord(ev[3], st)) != cudaSuccess) return e;
  int tiles = 0;
  for (int b = 0; b < P.B; ++b) tiles += (P.req[b].t_len + TILE - 1) / TILE;
  dim3 g2(P.Hkv * tiles, P.L);
  pass2_simt<T, D><<<g2, 256, sm2, st>>>(P, bf, (const T*)K);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_merge(const Problem& P, const Buffers& bf, cudaStream_t st) {
  int max_ns = 0;
  for (int b = 0; b < P.B; ++b) max_ns = max(max_ns, P.req[b].nsplit * P.part_slots);
  const int rows = P.anchor_split ? P.n_group_rows : P.Prows_pad;
  if (max_ns >= 128) {
    constexpr int threads = 256, rows_per_block = threads / 4;
    dim3 grid((rows + rows_per_block - 1) / rows_per_block, P.B * P.Hkv, P.L);
    merge_kernel<4><<<grid, threads, 0, st>>>(P, bf);
  } else {
    constexpr int threads = 128;
    dim3 grid((rows + threads - 1) / threads, P.B * P.Hkv, P.L);
    merge_kernel<1><<<grid, threads, 0, st>>>(P, bf);
  }
  return cudaGetLastError();
}

cudaError_t launch_score_simt(const Problem& P, const Buffers& bf, cudaStream_t st,
                              const void* K, cudaEvent_t* ev) {
  if (P.dtype == MMSHIFT_BF16)
    return P.d == 128 ? launch_t<__nv_bfloat16, 128>(P, bf, st, K, ev)
                      : launch_t<__nv_bfloat16, 64>(P, bf, st, K, ev);
  return P.d == 128 ? launch_t<float, 128>(P, bf, st, K, ev)
                    : launch_t<float, 64>(P, bf, st, K, ev);
}

}  // namespace mmshift
