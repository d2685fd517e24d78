// Step 5: tau-coverage votes and the budgeted top-k (Sections 3.2.2-3.2.3;
// Algorithm 1, last steps). Step 6: the gather into the compact cache
// (Appendix B).
//
// Both selections are radix selects on order-preserving 32-bit keys of the
// non-negative float values -- no full sort. Digits: the 8 exponent bits, then
// 8, 8 and 7 mantissa bits. Each warp owns a private 256-bin histogram in
// shared memory (counts, and for the weighted select a 64-bit fixed-point
// weight kept as two 32-bit words whose carry is detected from the atomic's
// return value), so atomics only contend inside a warp; after the first digit
// only the few keys matching the prefix are counted and warps without any skip
// the pass.
//  - cover_kernel: one CTA per (layer, request, KV head, group). Weighted
//    select: the smallest prefix of keys in (mass desc, t asc) order whose
//    mass reaches tau * total. Masses are summed in 64-bit fixed point (2^-S
//    units, S <= 40, chosen per group so the total cannot overflow), so sums
//    are exact and order-independent. Output: the cover set as a bitmap.
//  - topk_kernel: one CTA per (layer, request, KV head). Builds S_t (votes
//    counted from the bitmaps with warp ballots, plus lambda * anchor; or the
//    summed mass), then a count select of the C-1 largest among t < T-1
//    (ties: lower t) and an ordered compaction with warp ballots that writes
//    the kept indices ascending with T-1 last.
#include "common.cuh"

namespace mmshift {
namespace {

constexpr int NT = 512;           // threads per selection CTA
constexpr int NW = NT / 32;
constexpr int NBIN = 256;
constexpr int kMaxStaged = 40960; // keys staged in shared memory (160 KB)
constexpr int HIST_WORDS = 3 * NW * NBIN;  // per-warp count / weight-lo / weight-hi

__device__ __forceinline__ uint32_t ordered_key(float x) {
  uint32_t u = __float_as_uint(x + 0.0f);  // -0 -> +0
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float key_value(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}
// Keys of non-negative values (negatives and NaN are clamped to +0).
__device__ __forceinline__ uint32_t nonneg_key(float x) {
  return ordered_key(fmaxf(x, 0.f));
}

struct SelShared {
  unsigned long long total;
  unsigned long long wsum[NW];
  unsigned int wcnt[NW];
  unsigned long long cum_w;
  unsigned int cum_n;
  unsigned int digit;
  unsigned int prefix;
  unsigned int n_theta;
  int aux;
  float fsum;
};

// Key source: shared memory when staged, else recomputed from global floats.
struct KeySrc {
  const uint32_t* smem;
  const float* gmem;
  __device__ __forceinline__ uint32_t operator()(int i) const {
    return smem ? smem[i] : nonneg_key(gmem[i]);
  }
};

__device__ __forceinline__ unsigned long long fx_weight(uint32_t key, int shift) {
  const float x = fmaxf(key_value(key), 0.f);
  return __float2ull_rn(ldexpf(x, shift));
}

// Block-wide exclusive scan of one unsigned per warp (warp totals in S.wcnt).
__device__ __forceinline__ unsigned warp_excl_prefix(SelShared& S, unsigned mine) {
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) S.wcnt[w] = mine;
  __syncthreads();
  unsigned before = 0;
  for (int i = 0; i < w; ++i) before += S.wcnt[i];
  __syncthreads();
  return before;
}

// Smallest prefix of the (key desc, index asc) order whose cumulative weight
// is >= target_w and whose length is >= target_n (all keys >= 0x80000000,
// i.e. of non-negative values). On return S.prefix is the key theta of the
// prefix's last element, S.cum_w / S.cum_n the weight / count of keys above
// theta and S.n_theta the number of keys equal to theta. `hist` is
// HIST_WORDS words of shared memory.
//
// Weighted mode: target_w is derived from the exact fixed-point total, summed in
// the first pass: target_w = min(total, ceil(tau * total)); S.total holds it.
template <bool WEIGHTED>
__device__ void radix_select(const KeySrc& get, int n, unsigned long long target_w,
                             unsigned target_n, int shift, float tau, SelShared& S,
                             uint32_t* hist) {
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  uint32_t* hn = hist + w * NBIN;
  uint32_t* hlo = hist + (NW + w) * NBIN;
  uint32_t* hhi = hist + (2 * NW + w) * NBIN;
  if (tid == 0) { S.cum_w = 0; S.cum_n = 0; }
  uint32_t prefix = 0x80000000u;
  constexpr int kSh[4] = {23, 15, 7, 0};
  constexpr int kWid[4] = {8, 8, 8, 7};
#pragma unroll 1
  for (int pass = 0; pass < 4; ++pass) {
    const int sh = kSh[pass], hs = sh + kWid[pass];
    const uint32_t dmask = (1u << kWid[pass]) - 1u;
    for (int i = lane; i < NBIN; i += 32) {
      hn[i] = 0;
      if (WEIGHTED) { hlo[i] = 0; hhi[i] = 0; }
    }
    __syncwarp();
    unsigned long long tot = 0;
    for (int base = 0; base < n; base += NT) {
      const int i = base + tid;
      const uint32_t k = i < n ? get(i) : 0u;
      const bool take = i < n && (k >> hs) == (prefix >> hs);
      if (pass > 0 && !__any_sync(0xffffffffu, take)) continue;
      if (take) {
        const uint32_t d = (k >> sh) & dmask;
        atomicAdd(&hn[d], 1u);
        if (WEIGHTED) {
          const unsigned long long wt = fx_weight(k, shift);
          if (pass == 0) tot += wt;
          const uint32_t lo = (uint32_t)wt;
          uint32_t hi = (uint32_t)(wt >> 32);
          if (lo) {
            const uint32_t old = atomicAdd(&hlo[d], lo);
            hi += (old + lo < old) ? 1u : 0u;   // carry out of the low word
          }
          if (hi) atomicAdd(&hhi[d], hi);
        }
      }
    }
    if (WEIGHTED && pass == 0) {
      for (int off = 16; off; off >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, off);
      if (lane == 0) S.wsum[w] = tot;
    }
    __syncthreads();
    if (WEIGHTED && pass == 0) {
      unsigned long long total = 0;
      for (int i = 0; i < NW; ++i) total += S.wsum[i];
      unsigned long long t = (unsigned long long)ceil((double)tau * (double)total);
      target_w = t > total ? total : t;
      if (tid == 0) S.total = total;
    }
    if (tid < 32) {
      // lane L owns digits 255-8L .. 248-8L, scanned from the top
      unsigned long long bw[8];
      unsigned bn[8];
      unsigned long long sw = 0;
      unsigned sn = 0;
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int d = 255 - 8 * lane - k;
        unsigned long long wsum = 0;
        unsigned nsum = 0;
        for (int ww = 0; ww < NW; ++ww) {
          nsum += hist[ww * NBIN + d];
          if (WEIGHTED)
            wsum += (unsigned long long)hist[(NW + ww) * NBIN + d] +
                    ((unsigned long long)hist[(2 * NW + ww) * NBIN + d] << 32);
        }
        bw[k] = wsum;
        bn[k] = nsum;
        sw += wsum;
        sn += nsum;
      }
      unsigned long long iw = sw;
      unsigned in = sn;
      for (int off = 1; off < 32; off <<= 1) {
        const unsigned long long tw = __shfl_up_sync(0xffffffffu, iw, off);
        const unsigned tn = __shfl_up_sync(0xffffffffu, in, off);
        if (lane >= off) { iw += tw; in += tn; }
      }
      const unsigned long long cw = S.cum_w;
      const unsigned cn = S.cum_n;
      const bool hit = (!WEIGHTED || cw + iw >= target_w) && cn + in >= target_n;
      const unsigned ball = __ballot_sync(0xffffffffu, hit);
      const int f = ball ? __ffs(ball) - 1 : 31;
      if (lane == f) {
        unsigned long long c_w = cw + iw - sw;
        unsigned c_n = cn + in - sn;
        int chosen = 7;
        unsigned n_ch = bn[7];
        bool found = false;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          if (!found) {
            if ((!WEIGHTED || c_w + bw[k] >= target_w) && c_n + bn[k] >= target_n) {
              chosen = k;
              n_ch = bn[k];
              found = true;
            } else if (k < 7) {
              c_w += bw[k];
              c_n += bn[k];
            }
          }
        }
        S.cum_w = c_w;
        S.cum_n = c_n;
        S.digit = (unsigned)(255 - 8 * lane - chosen);
        S.n_theta = n_ch;
      }
    }
    __syncthreads();
    prefix |= (S.digit & dmask) << sh;
    __syncthreads();
  }
  if (tid == 0) S.prefix = prefix;
  __syncthreads();
}

__global__ void __launch_bounds__(NT, 1) cover_kernel(Problem P, Buffers bf) {
  extern __shared__ uint32_t dyn[];
  uint32_t* hist = dyn;
  uint32_t* keys_sm = dyn + HIST_WORDS;
  __shared__ SelShared S;
  const int g = blockIdx.x % P.G, h = blockIdx.x / P.G, b = blockIdx.y, l = blockIdx.z;
  const ReqInfo R = P.req[b];
  const int n = R.t_len, tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  const size_t row = ((size_t)l * P.Hkv + h) * P.G + g;
  const float* m = bf.gmass + row * P.total_T + R.tok_off;
  const bool staged = n <= kMaxStaged;
  // stage keys and sum the masses (float, only to choose the fixed point)
  float fs = 0.f;
  for (int i = tid; i < n; i += NT) {
    const float x = fmaxf(m[i], 0.f);
    if (staged) keys_sm[i] = ordered_key(x);
    fs += x;
  }
  for (int off = 16; off; off >>= 1) fs += __shfl_xor_sync(0xffffffffu, fs, off);
  if (lane == 0) S.wsum[w] = __float_as_uint(fs);
  __syncthreads();
  if (tid == 0) {
    float t = 0.f;
    for (int i = 0; i < NW; ++i) t += __uint_as_float((unsigned)S.wsum[i]);
    S.fsum = t;
  }
  __syncthreads();
  int e = 0;
  frexpf(S.fsum + 1.0f, &e);               // S.fsum + 1 < 2^e
  const int shift = max(0, min(40, 60 - e));
  KeySrc get{staged ? keys_sm : nullptr, m};
  radix_select<true>(get, n, 0ull, 1u, shift, P.tau, S, hist);
  const uint32_t theta = S.prefix;
  const unsigned n_theta = S.n_theta;
  const unsigned long long target = min(S.total, (unsigned long long)ceil((double)P.tau * (double)S.total));
  const unsigned long long wth = fx_weight(theta, shift);
  const unsigned long long need_w = target > S.cum_w ? target - S.cum_w : 0ull;
  unsigned n_tie = 1;
  if (need_w > 0 && wth > 0) n_tie = (unsigned)((need_w + wth - 1) / wth);
  if (n_tie > n_theta) n_tie = n_theta;
  if (tid == 0) S.aux = n;  // every key equal to theta is in
  if (n_tie < n_theta) {
    // t* = index of the n_tie-th key equal to theta (ascending t); warp segments
    const int seg = ((n + NW * 32 - 1) / (NW * 32)) * 32;
    const int lo = w * seg, hi = min(n, lo + seg);
    unsigned cnt = 0;
    for (int base = lo; base < hi; base += 32) {
      const int i = base + lane;
      cnt += __popc(__ballot_sync(0xffffffffu, i < hi && get(i) == theta));
    }
    const unsigned before = warp_excl_prefix(S, cnt);
    if (before < n_tie && before + cnt >= n_tie) {
      unsigned seen = before;
      for (int base = lo; base < hi; base += 32) {
        const int i = base + lane;
        const unsigned bal = __ballot_sync(0xffffffffu, i < hi && get(i) == theta);
        if (seen + __popc(bal) >= n_tie) {
          const unsigned want = n_tie - seen;   // 1-based rank inside this word
          unsigned bb = bal;
          for (unsigned k = 1; k < want; ++k) bb &= bb - 1;
          if (lane == 0) S.aux = base + __ffs(bb) - 1;
          break;
        }
        seen += __popc(bal);
      }
    }
  }
  __syncthreads();
  const int tstar = S.aux;
  uint32_t* bits = bf.bits + row * P.total_words + R.word_off;
  for (int base = w * 32; base < n; base += NT) {
    const int i = base + lane;
    bool mem = false;
    if (i < n) {
      const uint32_t k = get(i);
      mem = k > theta || (k == theta && i <= tstar);
    }
    const unsigned word = __ballot_sync(0xffffffffu, mem);
    if (lane == 0) bits[base >> 5] = word;
  }
}

// from_scores: S comes from bf.scores as given; otherwise it is built here.
__global__ void __launch_bounds__(NT, 1) topk_kernel(Problem P, Buffers bf, int32_t* out_idx,
                                                  int from_scores) {
  extern __shared__ uint32_t dyn[];
  uint32_t* hist = dyn;
  uint32_t* keys_sm = dyn + HIST_WORDS;
  __shared__ SelShared S;
  const int h = blockIdx.x, b = blockIdx.y, l = blockIdx.z;
  const ReqInfo R = P.req[b];
  const int n = R.t_len, tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  const size_t hrow = ((size_t)l * P.Hkv + h) * P.total_T + R.tok_off;
  float* sc = bf.scores + hrow;
  const bool staged = n <= kMaxStaged;
  if (!from_scores) {
    const float* an = bf.anchor + hrow;
    const uint32_t* bw = bf.bits + ((size_t)l * P.Hkv + h) * P.G * P.total_words + R.word_off;
    // each warp takes 32 consecutive keys at a time
    for (int base = w * 32; base < n; base += NT) {
      const int i = base + lane;
      float s;
      if (P.mode == MMSHIFT_SCORE_VOTE) {
        // lane g holds the coverage word of group g for these 32 keys; the
        // vote of key base+j is the number of lanes whose bit j is set
        unsigned vote = 0;
        for (int g0 = 0; g0 < P.G; g0 += 32) {
          const int g = g0 + lane;
          const uint32_t word = g < P.G ? bw[(size_t)g * P.total_words + (base >> 5)] : 0u;
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const unsigned c = __popc(__ballot_sync(0xffffffffu, (word >> j) & 1u));
            if (lane == j) vote += c;
          }
        }
        s = i < n ? __fadd_rn((float)vote, __fmul_rn(P.lambda, an[i])) : 0.f;  // no contraction
      } else {
        float ms = 0.f;
        if (i < n)
          for (int g = 0; g < P.G; ++g)
            ms += bf.gmass[(((size_t)l * P.Hkv + h) * P.G + g) * P.total_T + R.tok_off + i];
        s = ms;
      }
      if (i < n) {
        sc[i] = s;
        if (staged) keys_sm[i] = nonneg_key(s);
      }
    }
  } else if (staged) {
    for (int i = tid; i < n; i += NT) keys_sm[i] = nonneg_key(sc[i]);
  }
  __syncthreads();
  int32_t* out = out_idx + ((size_t)l * P.R + R.out_off) * P.Hkv + h;
  const int keep = R.keep;
  if (keep >= n) {
    for (int i = tid; i < n; i += NT) out[(size_t)i * P.Hkv] = i;
    return;
  }
  if (keep == 1) {
    if (tid == 0) out[0] = n - 1;
    return;
  }
  KeySrc get{staged ? keys_sm : nullptr, sc};
  const int nc = n - 1;  // candidates t < T-1
  radix_select<false>(get, nc, 0ull, (unsigned)(keep - 1), 0, 0.f, S, hist);
  const uint32_t theta = S.prefix;
  const unsigned n_tie = (unsigned)(keep - 1) - S.cum_n;
  // ordered compaction over warp segments
  const int seg = ((nc + NW * 32 - 1) / (NW * 32)) * 32;
  const int lo = w * seg, hi = min(nc, lo + seg);
  unsigned c_gt = 0, c_tie = 0;
  for (int base = lo; base < hi; base += 32) {
    const int i = base + lane;
    const uint32_t k = i < hi ? get(i) : 0u;
    c_gt += __popc(__ballot_sync(0xffffffffu, i < hi && k > theta));
    c_tie += __popc(__ballot_sync(0xffffffffu, i < hi && k == theta));
  }
  const unsigned gt_before = warp_excl_prefix(S, c_gt);
  unsigned tie_before = warp_excl_prefix(S, c_tie);
  unsigned pos = gt_before + min(tie_before, n_tie);
  const unsigned lt = (1u << lane) - 1u;
  for (int base = lo; base < hi; base += 32) {
    const int i = base + lane;
    const uint32_t k = i < hi ? get(i) : 0u;
    const bool is_tie = i < hi && k == theta;
    const unsigned tie_m = __ballot_sync(0xffffffffu, is_tie);
    const unsigned my_rank = tie_before + __popc(tie_m & lt);
    const bool sel = i < hi && (k > theta || (is_tie && my_rank < n_tie));
    const unsigned sel_m = __ballot_sync(0xffffffffu, sel);
    if (sel) out[(size_t)(pos + __popc(sel_m & lt)) * P.Hkv] = i;
    pos += __popc(sel_m);
    tie_before += __popc(tie_m);
  }
  if (tid == 0) out[(size_t)(keep - 1) * P.Hkv] = n - 1;
}

// mass[l][h][t] = sum over g (ascending) of gmass[l][h][g][t].
__global__ void mass_sum_kernel(Problem P, Buffers bf) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  const int h = blockIdx.y, l = blockIdx.z;
  if (t >= P.total_T) return;
  float ms = 0.f;
  for (int g = 0; g < P.G; ++g) ms += bf.gmass[(((size_t)l * P.Hkv + h) * P.G + g) * P.total_T + t];
  bf.mass[((size_t)l * P.Hkv + h) * P.total_T + t] = ms;
}

// One output row (c, h) per group of 16-byte lanes.
template <int ROWB>
__global__ void __launch_bounds__(256) gather_kernel(Problem P, Buffers bf, const uint8_t* K,
                                                     const uint8_t* V, const int32_t* idx,
                                                     uint8_t* oK, uint8_t* oV) {
  constexpr int LPR = ROWB / 16;  // lanes per row
  const int l = blockIdx.y;
  const long long q = (long long)blockIdx.x * (256 / LPR) + threadIdx.x / LPR;
  const int part = threadIdx.x % LPR;
  if (q >= (long long)P.R * P.Hkv) return;
  const int c = (int)(q / P.Hkv), h = (int)(q % P.Hkv);
  int b = 0;
  while (b + 1 < P.B && P.req[b + 1].out_off <= c) ++b;
  const ReqInfo R = P.req[b];
  const int t = idx[(size_t)l * P.R * P.Hkv + q];
  const size_t esz = ROWB / P.d;
  uint4* dk = (uint4*)(oK + (((size_t)l * P.R * P.Hkv + q) * ROWB)) + part;
  uint4* dv = (uint4*)(oV + (((size_t)l * P.R * P.Hkv + q) * ROWB)) + part;
  if (t < 0 || t >= R.t_len) {
    *dk = make_uint4(0, 0, 0, 0);
    *dv = make_uint4(0, 0, 0, 0);
    if (part == 0) set_status(bf.status, kStatusBadIndex);
    return;
  }
  const size_t src = (size_t)l * P.ls_kv * esz + (((size_t)R.tok_off + t) * P.Hkv + h) * ROWB;
  *dk = __ldg((const uint4*)(K + src) + part);
  *dv = __ldg((const uint4*)(V + src) + part);
}

}  // namespace

cudaError_t launch_mass_sum(const Problem& P, const Buffers& bf, cudaStream_t st) {
  if (!bf.mass || P.total_T == 0) return cudaSuccess;
  dim3 grid((P.total_T + 255) / 256, P.Hkv, P.L);
  mass_sum_kernel<<<grid, 256, 0, st>>>(P, bf);
  return cudaGetLastError();
}

cudaError_t launch_cover(const Problem& P, const Buffers& bf, cudaStream_t st) {
  if (P.G == 0) return cudaSuccess;
  int maxT = 0;
  for (int b = 0; b < P.B; ++b) maxT = max(maxT, P.req[b].t_len);
  const size_t smem = (size_t)(HIST_WORDS + min(maxT, kMaxStaged)) * sizeof(uint32_t);
  cudaError_t e = cudaFuncSetAttribute(cover_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)((HIST_WORDS + kMaxStaged) * sizeof(uint32_t)));
  if (e != cudaSuccess) return e;
  dim3 grid(P.Hkv * P.G, P.B, P.L);
  cover_kernel<<<grid, NT, smem, st>>>(P, bf);
  return cudaGetLastError();
}

cudaError_t launch_topk(const Problem& P, const Buffers& bf, cudaStream_t st, int32_t* out_idx,
                        bool from_scores) {
  int maxT = 0;
  for (int b = 0; b < P.B; ++b) maxT = max(maxT, P.req[b].t_len);
  const size_t smem = (size_t)(HIST_WORDS + min(maxT, kMaxStaged)) * sizeof(uint32_t);
  cudaError_t e = cudaFuncSetAttribute(topk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)((HIST_WORDS + kMaxStaged) * sizeof(uint32_t)));
  if (e != cudaSuccess) return e;
  dim3 grid(P.Hkv, P.B, P.L);
  topk_kernel<<<grid, NT, smem, st>>>(P, bf, out_idx, from_scores ? 1 : 0);
  return cudaGetLastError();
}

cudaError_t launch_gather(const Problem& P, const Buffers& bf, cudaStream_t st, const void* K,
                          const void* V, const int32_t* idx, void* outK, void* outV) {
  const int rowb = P.d * (P.dtype == MMSHIFT_BF16 ? 2 : 4);
  const long long rows = (long long)P.R * P.Hkv;
  if (rows == 0) return cudaSuccess;
#define MMSHIFT_GATHER(RB)                                                                   \
  {                                                                                          \
    constexpr int LPR = RB / 16;                                                             \
    dim3 grid((unsigned)((rows + (256 / LPR) - 1) / (256 / LPR)), P.L);                      \
    gather_kernel<RB><<<grid, 256, 0, st>>>(P, bf, (const uint8_t*)K, (const uint8_t*)V, idx, \
                                            (uint8_t*)outK, (uint8_t*)outV);                 \
    return cudaGetLastError();                                                               \
  }
  switch (rowb) {
    case 128: MMSHIFT_GATHER(128)
    case 256: MMSHIFT_GATHER(256)
    case 512: MMSHIFT_GATHER(512)
    default: return cudaErrorInvalidValue;
  }
#undef MMSHIFT_GATHER
}

}  // namespace mmshift
