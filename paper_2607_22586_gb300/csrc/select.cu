// Step 5: tau-coverage votes and the budgeted top-k (Sections 3.2.2-3.2.3;
// Algorithm 1, last steps). Step 6: the gather into the compact cache
// (Appendix B).
//
// Both selections are radix selects on order-preserving 32-bit keys of the
// float values, 8 bits per pass from the top, with warp-aggregated histogram
// updates (__match_any_sync groups lanes with the same digit; the group leader
// adds the group's count, and its weight summed with __reduce_add_sync). No
// full sort is done.
//  - cover_kernel: one CTA per (layer, request, KV head, group). Weighted
//    select: the smallest prefix of keys in (mass desc, t asc) order whose
//    mass reaches tau * total. Masses are summed in 64-bit fixed point (2^-S
//    units, S <= 40, chosen per group so the total cannot overflow), so the
//    sums are exact and order-independent. Output: the cover set as a bitmap
//    (one bit per key).
//  - topk_kernel: one CTA per (layer, request, KV head). Builds S_t (votes
//    from the bitmaps plus lambda * anchor, or the summed mass), then a count
//    select of the C-1 largest among t < T-1 (ties: lower t), and an ordered
//    compaction with warp ballots that writes the kept indices ascending with
//    T-1 last.
#include "common.cuh"

namespace mmshift {
namespace {

constexpr int NT = 1024;          // threads per selection CTA
constexpr int NW = NT / 32;
constexpr int kMaxStaged = 49152; // keys staged in shared memory (192 KB)

__device__ __forceinline__ uint32_t ordered_key(float x) {
  uint32_t u = __float_as_uint(x + 0.0f);  // -0 -> +0
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float key_value(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

struct SelShared {
  unsigned long long hw[256];
  unsigned int hn[256];
  unsigned long long wsum[NW];
  unsigned int wcnt[NW];
  unsigned long long cum_w;
  unsigned int cum_n;
  unsigned int digit;
  unsigned int prefix;
  int aux;
  float fsum;
};

// Key source: shared memory when staged, else recomputed from global floats.
struct KeySrc {
  const uint32_t* smem;
  const float* gmem;
  __device__ __forceinline__ uint32_t operator()(int i) const {
    return smem ? smem[i] : ordered_key(gmem[i]);
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
// is >= target_w and whose length is >= target_n. On return S.prefix is the
// key theta of the prefix's last element, S.cum_w / S.cum_n the weight / count
// of keys > theta, and the return value is the number of keys equal to theta.
template <bool WEIGHTED>
__device__ unsigned radix_select(const KeySrc& get, int n, unsigned long long target_w,
                                 unsigned target_n, int shift, SelShared& S) {
  const int tid = threadIdx.x, lane = tid & 31;
  uint32_t prefix = 0, mask = 0;
  if (tid == 0) { S.cum_w = 0; S.cum_n = 0; }
  unsigned n_theta = 0;
  for (int pass = 0; pass < 4; ++pass) {
    const int sh = 24 - 8 * pass;
    for (int i = tid; i < 256; i += NT) { S.hw[i] = 0; S.hn[i] = 0; }
    __syncthreads();
    for (int base = 0; base < n; base += NT) {
      const int i = base + tid;
      const uint32_t k = i < n ? get(i) : 0u;
      const bool take = i < n && (k & mask) == prefix;
      const unsigned dig = take ? ((k >> sh) & 255u) : 256u;
      const unsigned peers = __match_any_sync(0xffffffffu, dig);
      const bool leader = take && lane == (__ffs(peers) - 1);
      if (WEIGHTED) {
        const unsigned long long w = take ? fx_weight(k, shift) : 0ull;
        const unsigned s0 = __reduce_add_sync(peers, (unsigned)(w & 0x1fffffull));
        const unsigned s1 = __reduce_add_sync(peers, (unsigned)((w >> 21) & 0x1fffffull));
        const unsigned s2 = __reduce_add_sync(peers, (unsigned)(w >> 42));
        if (leader)
          atomicAdd(&S.hw[dig], (unsigned long long)s0 + ((unsigned long long)s1 << 21) +
                                    ((unsigned long long)s2 << 42));
      }
      if (leader) atomicAdd(&S.hn[dig], (unsigned)__popc(peers));
    }
    __syncthreads();
    if (tid < 32) {
      // lane L owns digits 255-8L .. 248-8L, scanned from the top
      unsigned long long sw = 0;
      unsigned sn = 0;
      for (int k = 0; k < 8; ++k) {
        const int d = 255 - 8 * lane - k;
        sw += S.hw[d];
        sn += S.hn[d];
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
        int chosen = 255 - 8 * lane - 7;
        for (int k = 0; k < 8; ++k) {
          const int d = 255 - 8 * lane - k;
          if ((!WEIGHTED || c_w + S.hw[d] >= target_w) && c_n + S.hn[d] >= target_n) {
            chosen = d;
            break;
          }
          if (k < 7) { c_w += S.hw[d]; c_n += S.hn[d]; }
        }
        S.cum_w = c_w;
        S.cum_n = c_n;
        S.digit = (unsigned)chosen;
      }
    }
    __syncthreads();
    prefix |= S.digit << sh;
    mask |= 255u << sh;
    n_theta = S.hn[S.digit];
    __syncthreads();
  }
  if (tid == 0) S.prefix = prefix;
  __syncthreads();
  return n_theta;
}

__global__ void __launch_bounds__(NT) cover_kernel(Problem P, Buffers bf) {
  extern __shared__ uint32_t keys_sm[];
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
    const float x = m[i];
    if (staged) keys_sm[i] = ordered_key(x);
    fs += fmaxf(x, 0.f);
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
  // exact fixed-point total
  unsigned long long tw = 0;
  for (int i = tid; i < n; i += NT) tw += fx_weight(get(i), shift);
  for (int off = 16; off; off >>= 1) tw += __shfl_xor_sync(0xffffffffu, tw, off);
  __syncthreads();
  if (lane == 0) S.wsum[w] = tw;
  __syncthreads();
  unsigned long long total = 0;
  for (int i = 0; i < NW; ++i) total += S.wsum[i];
  __syncthreads();
  unsigned long long target = (unsigned long long)ceil((double)P.tau * (double)total);
  if (target > total) target = total;
  const unsigned n_theta = radix_select<true>(get, n, target, 1u, shift, S);
  const uint32_t theta = S.prefix;
  const unsigned long long wth = fx_weight(theta, shift);
  const unsigned long long need_w = target > S.cum_w ? target - S.cum_w : 0ull;
  unsigned n_tie = 1;
  if (need_w > 0 && wth > 0) n_tie = (unsigned)((need_w + wth - 1) / wth);
  if (n_tie > n_theta) n_tie = n_theta;
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
__global__ void __launch_bounds__(NT) topk_kernel(Problem P, Buffers bf, int32_t* out_idx,
                                                  int from_scores) {
  extern __shared__ uint32_t keys_sm[];
  __shared__ SelShared S;
  const int h = blockIdx.x, b = blockIdx.y, l = blockIdx.z;
  const ReqInfo R = P.req[b];
  const int n = R.t_len, tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  const size_t hrow = ((size_t)l * P.Hkv + h) * P.total_T + R.tok_off;
  float* sc = bf.scores + hrow;
  const bool staged = n <= kMaxStaged;
  if (!from_scores) {
    const float* an = bf.anchor + hrow;
    for (int i = tid; i < n; i += NT) {
      float s;
      if (P.mode == MMSHIFT_SCORE_VOTE) {
        unsigned vote = 0;
        const uint32_t* bw = bf.bits + ((size_t)l * P.Hkv + h) * P.G * P.total_words + R.word_off + (i >> 5);
        for (int g = 0; g < P.G; ++g) vote += (bw[(size_t)g * P.total_words] >> (i & 31)) & 1u;
        s = __fadd_rn((float)vote, __fmul_rn(P.lambda, an[i]));  // no contraction
      } else {
        float ms = 0.f;
        for (int g = 0; g < P.G; ++g)
          ms += bf.gmass[(((size_t)l * P.Hkv + h) * P.G + g) * P.total_T + R.tok_off + i];
        s = ms;
      }
      sc[i] = s;
      if (staged) keys_sm[i] = ordered_key(s);
    }
  } else if (staged) {
    for (int i = tid; i < n; i += NT) keys_sm[i] = ordered_key(sc[i]);
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
  radix_select<false>(get, nc, 0ull, (unsigned)(keep - 1), 0, S);
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
  const size_t smem = (size_t)min(maxT, kMaxStaged) * sizeof(uint32_t);
  cudaError_t e = cudaFuncSetAttribute(cover_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)(kMaxStaged * sizeof(uint32_t)));
  if (e != cudaSuccess) return e;
  dim3 grid(P.Hkv * P.G, P.B, P.L);
  cover_kernel<<<grid, NT, smem, st>>>(P, bf);
  return cudaGetLastError();
}

cudaError_t launch_topk(const Problem& P, const Buffers& bf, cudaStream_t st, int32_t* out_idx,
                        bool from_scores) {
  int maxT = 0;
  for (int b = 0; b < P.B; ++b) maxT = max(maxT, P.req[b].t_len);
  const size_t smem = (size_t)min(maxT, kMaxStaged) * sizeof(uint32_t);
  cudaError_t e = cudaFuncSetAttribute(topk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)(kMaxStaged * sizeof(uint32_t)));
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
