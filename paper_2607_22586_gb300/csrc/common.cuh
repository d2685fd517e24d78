// Internal definitions shared by the kernels and the host entry points.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "mmshift.h"

namespace mmshift {

constexpr float kLog2e = 1.4426950408889634f;
constexpr int kChunk = 16;       // proxy rows per packing chunk (one group id)
constexpr int kRowTile = 256;    // proxy rows are padded to a multiple of this
constexpr int kMaxSplitAnchor = 8;  // anchor_split needs r <= this (one warp per anchor row)
constexpr int kUmmaPartSlots = 4; // softmax partials per (row, split) of the tensor-core pass

// Status bits the kernels OR into the workspace status word.
enum : int {
  kStatusTimeout = 1,   // a bounded wait gave up
  kStatusBadIndex = 2,  // gather saw an index outside [0, T_b)
  kStatusBadBudget = 4, // a per-head budget outside [1, C_b] (clamped)
};

struct ReqInfo {
  int32_t t_len;     // T_b
  int32_t tok_off;   // cu_seqlens[b]
  int32_t out_off;   // sum_{b' < b} keep_{b'}
  int32_t keep;      // min(C_b, T_b)
  int32_t budget;    // C_b
  int32_t word_off;  // offset of the request in a coverage bitmap row (32-bit words)
  int32_t split_off; // first key split of the request in the softmax partials
  int32_t nsplit;    // key splits of the request
};

// Everything a kernel needs to know about one call, passed by value.
struct Problem {
  int32_t B, L, Hq, Hkv, r, d, W, dtype;
  int32_t Np, G, gs;
  int32_t RG;          // packed rows per group: roundup(r * gs, 16)
  int32_t n_group_rows;// G * RG
  int32_t anchor_rows; // roundup(r, 16)
  int32_t Prows;       // n_group_rows + anchor_rows
  int32_t Prows_pad;   // roundup(Prows, kRowTile)
  int32_t part_slots;  // softmax partials per (row, key split): 1 (CUDA cores) or kUmmaPartSlots
  int32_t total_T, R, total_words, total_splits, split_len;
  int64_t ls_kv, ls_q;
  float scale, alpha, gamma, tau, lambda;
  int32_t mode;
  uint64_t seed;
  int32_t layer_id0;
  float rope_theta;
  int32_t rope_off;
  int32_t use_umma;    // steps 2-4 on the tensor cores (set per call)
  // tensor-core path whose anchor rows would fill a 256-row softmax block of
  // their own (the group rows end on a block boundary): the softmax pass
  // leaves them out, the mass pass writes their scaled logits to alog and
  // anchor_part_kernel / anchor_final_kernel normalise them (set per call)
  int32_t anchor_split;
  // expected total of one group's masses over a request (its proxy rows:
  // each row's softmax sums to 1) when the coverage vote reads masses this
  // library computed, else 0 (set per call); only a hint, checked in use
  float cover_hint;
  int32_t test_stuck_wait; // test only: see mmshift_debug.test_stuck_wait
  ReqInfo req[MMSHIFT_MAX_BATCH];
};

// Device buffers of one call (carved out of the caller's workspace, or the
// caller's own debug buffers where given).
struct Buffers {
  int* status;
  void* packed;       // [L][B][Hkv][Prows_pad][d] proxies, group-major rows
  float2* part;       // [L][Hkv][total_splits][part_slots][Prows_pad] (max, sum) partials
  float* cvals;       // [L][B][Hkv][Prows_pad] log2 normaliser of each row
  float* gmass;       // [L][Hkv][G][T]
  float* anchor;      // [L][Hkv][T]
  float* alog;        // [L][Hkv][r][T] scaled anchor logits (anchor_split only)
  float2* apart;      // [L][Hkv][total_splits][kMaxSplitAnchor] their (max, sum) per key split
  uint32_t* bits;     // [L][Hkv][G][total_words] coverage bitmaps
  float* scores;      // [L][Hkv][T]
  int32_t scores_out; // the caller asked for the scores (else the top-k writes them only when it reads them back)
  float* mass;        // [L][Hkv][T] or null
  void* proxies_out;  // [L][B][Hq][Np][d] or null
  const void* proxies_in; // [L][B][Hq][Np][d] or null
  const float* stats_in;  // [L][B][2][Hq][d] mean / std of the proxies, or null (window's)
  const int32_t* head_budget; // [L][B][Hkv] budgets C_{l,b,h} in [1, C_b], or null (C_b for all)
  int32_t* out_count;         // [L][B][Hkv] kept rows per head, or null
  // bf16 proxies whose float32 value lies too close to a rounding boundary
  // are recomputed in float64 (proxy.cu): the sampler appends them here and a
  // second kernel redoes them; without a list (null) the sampler redoes them
  // itself
  int* refine_count;          // entries appended (may exceed refine_cap)
  int4* refine_items;         // [refine_cap] (layer * B + request, query head, proxy, dim)
  float* refine_stats;        // [L][B][Hq][5][d] exact window sums (x0, S1 hi / lo, S2 hi / lo)
  int32_t refine_cap;
};

// Whole-prefill statistics job (stats.cu).
constexpr int kStatsChunk = 512;   // prompt queries per partial
struct StatsJob {
  int32_t L, B, ncol, nchunk;        // ncol = Hq * d; nchunk = max chunks per request
  int64_t ls;                        // elements between layers of Q
  int32_t t_len[MMSHIFT_MAX_BATCH];
  int32_t tok_off[MMSHIFT_MAX_BATCH];
};

// Hidden-space proxy job (hidden.cu): per (layer, request) N proxy hidden
// states sampled in d_model dims and projected by W_Q [F = Hq*d][d_model].
struct HiddenJob {
  int32_t L, B, Hq, d, F, DM, N, Npad;  // Npad = roundup(N, 128)
  int32_t NT, MT, NTL, tiles;           // feature tile width, proxy / feature tiles, total tiles
  float gamma, rope_theta;
  uint64_t seed;
  int32_t layer_id0;
  int32_t pos[MMSHIFT_MAX_BATCH];       // RoPE position of each request's proxies
  const float* hstats;                  // [L][B][2][DM] mean, std of the hidden states
  const __nv_bfloat16* bias;            // [L][F] or null
  float* rope;                          // [B][d/2][2] cos, sin (scratch) or null
  __nv_bfloat16* hs;                    // [L][B][Npad][DM] sampled hidden states (scratch)
  __nv_bfloat16* out;                   // [L][B][Hq][N][d] proxies
  int* status;
};

// Row p of the packed proxy block of KV head h: which group / query head /
// proxy it holds, or that it is padding.
struct RowKind {
  int group;   // 0..G-1 proxy group, G = anchor, -1 = padding
  int j;       // local query head (0..r-1)
  int i;       // proxy index within the query head (groups only)
};

__host__ __device__ inline RowKind row_kind(const Problem& P, int p) {
  RowKind k{-1, 0, 0};
  if (p < P.n_group_rows) {
    int g = p / P.RG, q = p - g * P.RG;
    if (q < P.r * P.gs) { k.group = g; k.j = q / P.gs; k.i = g * P.gs + (q % P.gs); }
  } else {
    int q = p - P.n_group_rows;
    if (q < P.r) { k.group = P.G; k.j = q; }
  }
  return k;
}

__host__ __device__ inline int chunk_group(const Problem& P, int chunk) {
  int p = chunk * kChunk;
  return p < P.n_group_rows ? p / P.RG : P.G;
}

template <typename T> __device__ __forceinline__ float to_f32(T x);
template <> __device__ __forceinline__ float to_f32<float>(float x) { return x; }
template <> __device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 x) {
  return __bfloat162float(x);
}
template <typename T> __device__ __forceinline__ T from_f32(float x);
template <> __device__ __forceinline__ float from_f32<float>(float x) { return x; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float x) {
  return __float2bfloat16_rn(x);
}

__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// (m, z) += (m2, z2) for partial softmax normalisers: the sum of exp2(x - m)
// over the union, relative to the larger reference max.
__device__ __forceinline__ void merge_ms(float& m, float& z, float m2, float z2) {
  const float mn = fmaxf(m, m2);
  if (mn == -INFINITY) return;
  z = z * fast_exp2(m - mn) + z2 * fast_exp2(m2 - mn);
  m = mn;
}

__device__ __forceinline__ void set_status(int* status, int bit) {
  if (status) atomicOr(status, bit);
}

// Host-side launchers (one translation unit each).
cudaError_t launch_prefill_stats(const StatsJob& J, const void* Q, float* part, float* stats,
                                 cudaStream_t st, bool bf16);
cudaError_t launch_proxy_pack(const Problem& P, const Buffers& bf, cudaStream_t st,
                              const void* qwin);
// Proxy elements the list of bf holds for a call's shape: at most this many
// are refined by the second kernel, the rest by the sampler itself.
int64_t proxy_refine_capacity(const Problem& P);
// Kernels launch_proxy_pack enqueues for P and bf.
int proxy_launches(const Problem& P, const Buffers& bf);
// ev (nullable): stage events 1 (softmax pass), 2 (merge) and 3 (mass pass)
// are recorded just before the corresponding launch.
cudaError_t launch_score_simt(const Problem& P, const Buffers& bf, cudaStream_t st,
                              const void* K, cudaEvent_t* ev);
cudaError_t launch_score_umma(const Problem& P, const Buffers& bf, cudaStream_t st,
                              const void* K, cudaEvent_t* ev);
bool umma_supported(const Problem& P);
// Scratch of launch_hidden_proxies (sampled hidden states, RoPE table) and
// the launch itself: sampling kernel, then the projection GEMM.
size_t hidden_scratch_bytes(const HiddenJob& J);
cudaError_t launch_hidden_proxies(HiddenJob J, void* scratch, const void* W, int64_t w_layer_stride,
                                  cudaStream_t st);
// Tiled TMA descriptor of a 3-D bf16 tensor (dims d0 innermost): boxes of
// 64 x box1 x 1 elements, 128-byte swizzle; false if the driver's encoder is
// unavailable or rejects the layout.
bool make_tmap_bf16_3d(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2,
                       uint64_t stride1_bytes, uint64_t stride2_bytes, uint32_t box1);
bool tmap_encoder_available();
int umma_launches(const Problem& P);
cudaError_t launch_anchor_split(const Problem& P, const Buffers& bf, cudaStream_t st);
cudaError_t launch_merge(const Problem& P, const Buffers& bf, cudaStream_t st);
// Attention-mass coverage of the kept set idx from the group masses in bf.
cudaError_t launch_coverage(const Problem& P, const Buffers& bf, const int32_t* idx, float* cov,
                            cudaStream_t st);
cudaError_t launch_cover(const Problem& P, const Buffers& bf, cudaStream_t st);
cudaError_t launch_mass_sum(const Problem& P, const Buffers& bf, cudaStream_t st);
cudaError_t launch_topk(const Problem& P, const Buffers& bf, cudaStream_t st,
                        int32_t* out_idx, bool from_scores);
cudaError_t launch_gather(const Problem& P, const Buffers& bf, cudaStream_t st,
                          const void* K, const void* V, const int32_t* idx,
                          void* outK, void* outV);

}  // namespace mmshift
