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

constexpr int kTopkCand = 4096;   // first-digit candidates a top-k CTA keeps in shared memory
constexpr int kCoverCand = 3072;  // first-digit candidates (key, index) a coverage CTA keeps in shared memory
constexpr int NBIN = 256;
constexpr int kMaxStaged = 40960; // top-k keys staged in shared memory (160 KB)

// per-warp histograms: counts, and for the weighted select weight lo / hi
template <int NTH, bool WEIGHTED>
__host__ __device__ constexpr int hist_words() { return (WEIGHTED ? 3 : 1) * (NTH / 32) * NBIN; }

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

template <int NTH>
struct SelShared {
  unsigned long long total;
  unsigned long long wsum[NTH / 32];
  unsigned int wcnt[NTH / 32];
  unsigned long long bin_w[NBIN];
  unsigned int bin_n[NBIN];
  unsigned long long cum_w;
  unsigned int cum_n;
  unsigned int digit;
  unsigned int prefix;
  unsigned int n_theta;
  unsigned int ncand;
  unsigned int rend;
  int aux;
};

// Key sources, chosen at compile time: keys staged in shared memory, or
// recomputed from global floats (read four at a time where aligned).
struct SmemKeys {
  static constexpr bool kGlobal = false;
  const uint32_t* smem;
  __device__ __forceinline__ uint32_t operator()(int i) const { return smem[i]; }
};
struct GlobalFloats {
  static constexpr bool kGlobal = true;
  const float* gmem;
  __device__ __forceinline__ uint32_t operator()(int i) const { return nonneg_key(__ldg(gmem + i)); }
};

// Weight of a key (of a non-negative float x) in 2^-shift units: x * 2^shift
// rounded to the nearest integer, ties to even, saturated at 2^64 - 1 (what
// a float-to-integer conversion of the exact product gives), in integer
// arithmetic without branches: x = mant * 2^(e - 150) with the 24-bit
// significand mant, so the weight is mant shifted left by s = e - 150 +
// shift, or right by r = -s as (mant + 2^(r-1) - 1 + (bit r of mant)) >> r,
// which rounds half to even (r >= 25 gives 0; r is clamped to 31, which
// also makes zero and the subnormals weigh 0).
__device__ __forceinline__ unsigned long long fx_weight(uint32_t key, int shift) {
  const uint32_t u = key & 0x7FFFFFFFu;
  const int e = (int)(u >> 23);
  const uint32_t mant = (u & 0x7FFFFFu) | 0x800000u;
  const int s = e - 150 + shift;
  const int r = min(max(-s, 1), 31);
  const uint32_t small = (mant + ((1u << (r - 1)) - 1u) + ((mant >> r) & 1u)) >> r;
  const unsigned long long big = (unsigned long long)mant << min(max(s, 0), 40);
  const unsigned long long wt = s >= 0 ? big : (unsigned long long)small;
  return (e == 255 || s > 40) ? ~0ull : wt;      // at least 2^64, infinity, NaN
}

// Add a 64-bit weight to a histogram bin held as two 32-bit words (low,
// high): the carry out of the low word is detected from the atomic's return.
__device__ __forceinline__ void add_weight(uint32_t* lo_w, uint32_t* hi_w, unsigned long long wt) {
  const uint32_t lo = (uint32_t)wt;
  uint32_t hi = (uint32_t)(wt >> 32);
  if (lo) {
    const uint32_t old = atomicAdd(lo_w, lo);
    hi += (old + lo < old) ? 1u : 0u;
  }
  if (hi) atomicAdd(hi_w, hi);
}

// 32 x 32 bit-matrix transpose across a warp: on entry lane i holds row i
// (bit j = element (i, j)), on return lane j holds column j (bit i = element
// (i, j)). Five rounds swap the off-diagonal s x s blocks (s = 16 .. 1)
// between lanes i and i ^ s.
__device__ __forceinline__ uint32_t warp_transpose32(uint32_t x) {
  const int lane = threadIdx.x & 31;
  uint32_t m = 0x0000FFFFu;
#pragma unroll
  for (int s = 16; s > 0; s >>= 1, m ^= m << s) {
    const uint32_t y = __shfl_xor_sync(0xffffffffu, x, s);
    x = (lane & s) ? ((x & ~m) | ((y >> s) & m)) : ((x & m) | ((y & m) << s));
  }
  return x;
}

// Block-wide exclusive scan of one unsigned per warp (warp totals in S.wcnt).
template <int NTH>
__device__ __forceinline__ unsigned warp_excl_prefix(SelShared<NTH>& S, unsigned mine) {
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) S.wcnt[w] = mine;
  __syncthreads();
  unsigned before = 0;
  for (int i = 0; i < w; ++i) before += S.wcnt[i];
  __syncthreads();
  return before;
}

// One digit pass: per-warp histograms of the keys matching `prefix` above
// bit `hs`, digit = bits [sh, hs). Weighted: also the weights, and in the
// first pass the exact total (returned through S.wsum) and the largest key.
// ONE: every warp adds into one CTA-wide histogram (for the few candidate
// keys of the later digits, where combining per-warp copies would cost more
// than the atomics' contention).
template <bool WEIGHTED, int NTH, class Src, bool ONE = false>
__device__ __forceinline__ void digit_histogram(const Src& get, int n, uint32_t prefix, int sh,
                                                int hs, uint32_t dmask, int shift, bool first,
                                                SelShared<NTH>& S, uint32_t* hist) {
  constexpr int NWH = ONE ? 1 : NTH / 32;
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  const int hw = ONE ? 0 : w;
  uint32_t* hn = hist + hw * NBIN;
  uint32_t* hlo = hist + (NWH + hw) * NBIN;
  uint32_t* hhi = hist + (2 * NWH + hw) * NBIN;
  if (ONE) {
    for (int i = tid; i < NBIN; i += NTH) {
      hn[i] = 0;
      if (WEIGHTED) { hlo[i] = 0; hhi[i] = 0; }
    }
    __syncthreads();
  } else {
    for (int i = lane; i < NBIN; i += 32) {
      hn[i] = 0;
      if (WEIGHTED) { hlo[i] = 0; hhi[i] = 0; }
    }
    __syncwarp();
  }
  unsigned long long tot = 0;
  uint32_t kmax = 0;
  const uint32_t wmin = ordered_key(__int_as_float((126 - shift) << 23)) + 1u;
  auto count = [&](uint32_t k, bool valid) {
    const bool take = valid && (k >> hs) == (prefix >> hs);
    if (!first && !__any_sync(0xffffffffu, take)) return;
    if (take) {
      const uint32_t d = (k >> sh) & dmask;
      atomicAdd(&hn[d], 1u);
      if (WEIGHTED) {
        // keys at or below 2^-(shift+1) weigh 0 units: no conversion
        const unsigned long long wt = k >= wmin ? fx_weight(k, shift) : 0ull;
        if (first) { tot += wt; kmax = max(kmax, k); }
        add_weight(&hlo[d], &hhi[d], wt);
      }
    }
  };
  int done = 0;
  if constexpr (Src::kGlobal) if ((reinterpret_cast<uintptr_t>(get.gmem) & 15) == 0) {
    // 16-byte loads of four keys, four loads in flight per thread
    constexpr int U4 = 4;
    const float4* g4 = reinterpret_cast<const float4*>(get.gmem);
    const int n4 = n >> 2;
    for (int base = 0; base < n4; base += U4 * NTH) {
      float4 f[U4];
#pragma unroll
      for (int j = 0; j < U4; ++j) {
        const int i4 = base + j * NTH + tid;
        f[j] = i4 < n4 ? __ldg(g4 + i4) : make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int j = 0; j < U4; ++j) {
        const bool valid = base + j * NTH + tid < n4;
        count(nonneg_key(f[j].x), valid);
        count(nonneg_key(f[j].y), valid);
        count(nonneg_key(f[j].z), valid);
        count(nonneg_key(f[j].w), valid);
      }
    }
    done = n4 << 2;
  }
  constexpr int U = 8;  // independent loads in flight per thread
  for (int base = done; base < n; base += U * NTH) {
    uint32_t kk[U];
#pragma unroll
    for (int j = 0; j < U; ++j) {
      const int i = base + j * NTH + tid;
      kk[j] = i < n ? get(i) : 0u;
    }
#pragma unroll
    for (int j = 0; j < U; ++j) count(kk[j], base + j * NTH + tid < n);
  }
  if (WEIGHTED && first) {
    for (int off = 16; off; off >>= 1) {
      tot += __shfl_xor_sync(0xffffffffu, tot, off);
      kmax = max(kmax, __shfl_xor_sync(0xffffffffu, kmax, off));
    }
    if (lane == 0) { S.wsum[w] = tot; S.wcnt[w] = kmax; }
  }
  __syncthreads();
  // combine the per-warp histograms: bin totals in shared memory
  for (int d = tid; d < NBIN; d += NTH) {
    unsigned long long wsum = 0;
    unsigned nsum = 0;
    for (int ww = 0; ww < NWH; ++ww) {
      nsum += hist[ww * NBIN + d];
      if (WEIGHTED)
        wsum += (unsigned long long)hist[(NWH + ww) * NBIN + d] +
                ((unsigned long long)hist[(2 * NWH + ww) * NBIN + d] << 32);
    }
    S.bin_n[d] = nsum;
    S.bin_w[d] = wsum;
  }
  __syncthreads();
}

// Pick the digit where the (key desc) cumulative weight / count first reaches
// the targets; warp 0 only. Lane L owns digits 255-8L .. 248-8L.
template <bool WEIGHTED, int NTH>
__device__ __forceinline__ void digit_scan(unsigned long long target_w, unsigned target_n,
                                           SelShared<NTH>& S) {
  const int lane = threadIdx.x & 31;
  unsigned long long sw = 0;
  unsigned sn = 0;
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const int d = 255 - 8 * lane - k;
    sw += S.bin_w[d];
    sn += S.bin_n[d];
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
      if ((!WEIGHTED || c_w + S.bin_w[d] >= target_w) && c_n + S.bin_n[d] >= target_n) {
        chosen = d;
        break;
      }
      if (k < 7) { c_w += S.bin_w[d]; c_n += S.bin_n[d]; }
    }
    S.cum_w = c_w;
    S.cum_n = c_n;
    S.digit = (unsigned)chosen;
    S.n_theta = S.bin_n[chosen];
  }
}

// Digit passes [p0, p1) of a radix select for the smallest prefix of the
// (key desc, index asc) order whose cumulative weight is >= target_w and
// whose length is >= target_n (all keys are of non-negative values). Pass 0
// starts from prefix 0x80000000; each pass appends its chosen digit to
// `prefix`. After the last pass, prefix is the key theta of the prefix's last
// element, S.cum_w / S.cum_n the weight / count of keys above theta and
// S.n_theta the number of keys equal to theta; after pass 0, S.n_theta is
// the number of keys that share the chosen first digit (the only keys the
// later passes look at). Weighted mode: pass 0 sets target_w to
// min(total, ceil(tau * total)) of the exact fixed-point total (S.total) and
// lowers *shift (redoing the pass) if 2^shift units could overflow 64 bits,
// unless pass0_total is false (target_w and *shift then stand as given).
// `hist` is hist_words<NTH, WEIGHTED>() words of shared memory.
template <bool WEIGHTED, int NTH, class Src, bool ONE = false>
__device__ void radix_passes(const Src& get, int n, int p0, int p1, uint32_t& prefix,
                             unsigned long long& target_w, unsigned target_n, int* shift,
                             float tau, SelShared<NTH>& S, uint32_t* hist,
                             bool pass0_total = true) {
  constexpr int NWH = NTH / 32;
  const int tid = threadIdx.x;
  if (p0 == 0 && tid == 0) { S.cum_w = 0; S.cum_n = 0; }
#pragma unroll 1
  for (int pass = p0; pass < p1; ++pass) {
    // digits: bits 23-30 (the exponent), 15-22, 7-14, 0-6
    const int wid = pass == 3 ? 7 : 8;
    const int sh = pass == 3 ? 0 : 23 - 8 * pass, hs = sh + wid;
    const uint32_t dmask = (1u << wid) - 1u;
    digit_histogram<WEIGHTED, NTH, Src, ONE>(get, n, prefix, sh, hs, dmask, WEIGHTED ? *shift : 0,
                                             pass == 0, S, hist);
    if (WEIGHTED && pass == 0 && pass0_total) {
      uint32_t kmax = 0;
      for (int i = 0; i < NWH; ++i) kmax = max(kmax, S.wcnt[i]);
      int e = 0;
      frexpf(key_value(kmax), &e);              // values < 2^e
      int lg = 0;
      while ((1 << lg) < n) ++lg;               // n <= 2^lg
      if (e + lg + *shift > 63) {               // n * max * 2^shift could overflow
        *shift = max(0, 63 - e - lg);
        __syncthreads();
        digit_histogram<WEIGHTED, NTH, Src, ONE>(get, n, prefix, sh, hs, dmask, *shift, true, S, hist);
      }
      unsigned long long total = 0;
      for (int i = 0; i < NWH; ++i) total += S.wsum[i];
      const unsigned long long t = (unsigned long long)ceil((double)tau * (double)total);
      target_w = t > total ? total : t;
      if (tid == 0) S.total = total;
    }
    if (tid < 32) digit_scan<WEIGHTED, NTH>(target_w, target_n, S);
    __syncthreads();
    prefix |= (S.digit & dmask) << sh;
    __syncthreads();
  }
}

// Copies the keys of get[0, n) whose bits at and above `hs` equal those of
// `prefix` into cand (in no particular order) and returns their number to
// every thread. Used after the first digit pass, when the keys sharing the
// chosen first digit fit in shared memory: the later passes then read only
// them. Each warp appends a ballot's worth at a time.
template <int NTH, class Src>
__device__ int compact_prefix(const Src& get, int n, uint32_t prefix, int hs, uint32_t* cand,
                              SelShared<NTH>& S) {
  const int tid = threadIdx.x, lane = tid & 31;
  if (tid == 0) S.ncand = 0;
  __syncthreads();
  const uint32_t want = prefix >> hs;
  const unsigned below = (1u << lane) - 1u;
  // a batch of keys per lane: the warp's candidates of the whole batch take
  // one atomic on the counter, then each key its place from the ballots
  auto put_batch = [&](const uint32_t* k, const bool* valid, int nb) {
    unsigned bal[16];
    unsigned tot = 0;
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      if (j < nb) {
        bal[j] = __ballot_sync(0xffffffffu, valid[j] && (k[j] >> hs) == want);
        tot += __popc(bal[j]);
      }
    }
    if (!tot) return;
    unsigned at = 0;
    if (lane == 0) at = atomicAdd(&S.ncand, tot);
    at = __shfl_sync(0xffffffffu, at, 0);
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      if (j < nb) {
        if ((bal[j] >> lane) & 1u) cand[at + __popc(bal[j] & below)] = k[j];
        at += __popc(bal[j]);
      }
    }
  };
  int done = 0;
  if constexpr (Src::kGlobal) if ((reinterpret_cast<uintptr_t>(get.gmem) & 15) == 0) {
    constexpr int U4 = 4;
    const float4* g4 = reinterpret_cast<const float4*>(get.gmem);
    const int n4 = n >> 2;
    for (int base = 0; base < n4; base += U4 * NTH) {
      float4 f[U4];
#pragma unroll
      for (int j = 0; j < U4; ++j) {
        const int i4 = base + j * NTH + tid;
        f[j] = i4 < n4 ? __ldg(g4 + i4) : make_float4(0.f, 0.f, 0.f, 0.f);
      }
      uint32_t kk[4 * U4];
      bool va[4 * U4];
#pragma unroll
      for (int j = 0; j < U4; ++j) {
        const bool valid = base + j * NTH + tid < n4;
        kk[4 * j] = nonneg_key(f[j].x); kk[4 * j + 1] = nonneg_key(f[j].y);
        kk[4 * j + 2] = nonneg_key(f[j].z); kk[4 * j + 3] = nonneg_key(f[j].w);
        va[4 * j] = va[4 * j + 1] = va[4 * j + 2] = va[4 * j + 3] = valid;
      }
      put_batch(kk, va, 4 * U4);
    }
    done = n4 << 2;
  }
  constexpr int U = 8;
  for (int base = done; base < n; base += U * NTH) {
    uint32_t kk[U];
    bool va[U];
#pragma unroll
    for (int j = 0; j < U; ++j) {
      const int i = base + j * NTH + tid;
      va[j] = i < n;
      kk[j] = va[j] ? get(i) : 0u;
    }
    put_batch(kk, va, U);
  }
  __syncthreads();
  return (int)S.ncand;
}

// Per-thread asynchronous 16-byte copies global -> shared (completion waited
// for by the issuing thread with cp.async.wait_group).
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                   (uint32_t)__cvta_generic_to_shared(smem)),
               "l"(gmem)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// Stages of the shared-memory ring of a streaming pass: NTH quads each, so
// the ring is exactly the size of the weighted per-warp histograms it
// shares memory with.
constexpr int kRingStages = 6;
static_assert(hist_words<512, true>() * 4 == kRingStages * 512 * 16 &&
                  hist_words<256, true>() * 4 == kRingStages * 256 * 16,
              "the streaming ring fills the weighted histograms exactly");

// One pass over m[0, n): the exact total weight (2^-shift units) and the
// largest key, returned to every thread, and the keys at or above kspec
// with their indices appended to (cand, cidx) (S.ncand, 0 on entry, counts
// them all; only the first cap are stored; kspec = ~0 appends none).
// The quads after a scalar head up to the first 16-byte boundary stream
// through `ring` (kRingStages * NTH quads of shared memory): thread t
// copies quads t, t + NTH, ... with cp.async, kRingStages ahead, and reads
// back only its own copies, so no barrier is needed between the stages.
template <int NTH>
__device__ void total_and_max(const float* m, int n, int shift, uint32_t kspec, uint32_t* cand,
                              uint32_t* cidx, int cap, float4* ring, SelShared<NTH>& S,
                              unsigned long long& total, uint32_t& kmax) {
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  // keys at or below 2^-(shift+1) weigh 0 units: no conversion
  const uint32_t wmin = ordered_key(__int_as_float((126 - shift) << 23)) + 1u;
  unsigned long long tot = 0;
  uint32_t km = 0;
  auto append = [&](uint32_t k, int i) {
    const unsigned o = atomicAdd(&S.ncand, 1u);
    if (o < (unsigned)cap) { cand[o] = k; cidx[o] = (uint32_t)i; }
  };
  auto add1 = [&](float x, int i) {
    const uint32_t k = nonneg_key(x);
    km = max(km, k);
    if (k >= wmin) tot += fx_weight(k, shift);
    if (k >= kspec) append(k, i);
  };
  const int head = min(n, (int)(((16u - (uint32_t)(reinterpret_cast<uintptr_t>(m) & 15)) & 15u) >> 2));
  if (tid < head) add1(__ldg(m + tid), tid);
  const float4* g4 = reinterpret_cast<const float4*>(m + head);
  const int n4 = (n - head) >> 2;
#pragma unroll
  for (int s = 0; s < kRingStages; ++s) {
    const int i4 = s * NTH + tid;
    if (i4 < n4) cp_async16(ring + s * NTH + tid, g4 + i4);
    cp_async_commit();
  }
  int slot = 0;
  for (int c = 0; c * NTH < n4; ++c) {
    cp_async_wait<kRingStages - 1>();
    const int i4 = c * NTH + tid;
    if (i4 < n4) {
      const float4 f = ring[slot * NTH + tid];
      const uint32_t k0 = nonneg_key(f.x), k1 = nonneg_key(f.y), k2 = nonneg_key(f.z),
                     k3 = nonneg_key(f.w);
      km = max(max(km, max(k0, k1)), max(k2, k3));
      const unsigned long long w0 = k0 >= wmin ? fx_weight(k0, shift) : 0ull;
      const unsigned long long w1 = k1 >= wmin ? fx_weight(k1, shift) : 0ull;
      const unsigned long long w2 = k2 >= wmin ? fx_weight(k2, shift) : 0ull;
      const unsigned long long w3 = k3 >= wmin ? fx_weight(k3, shift) : 0ull;
      tot += (w0 + w1) + (w2 + w3);
      if (max(max(k0, k1), max(k2, k3)) >= kspec) {   // rare
        const int i0 = head + 4 * i4;
        if (k0 >= kspec) append(k0, i0);
        if (k1 >= kspec) append(k1, i0 + 1);
        if (k2 >= kspec) append(k2, i0 + 2);
        if (k3 >= kspec) append(k3, i0 + 3);
      }
    }
    // the quad this thread just read is in registers: its slot takes the
    // copy kRingStages chunks ahead
    const int nx = (c + kRingStages) * NTH + tid;
    if (nx < n4) cp_async16(ring + slot * NTH + tid, g4 + nx);
    cp_async_commit();
    if (++slot == kRingStages) slot = 0;
  }
  cp_async_wait<0>();
  for (int i = head + (n4 << 2) + tid; i < n; i += NTH) add1(__ldg(m + i), i);
  for (int off = 16; off; off >>= 1) {
    tot += __shfl_xor_sync(0xffffffffu, tot, off);
    km = max(km, __shfl_xor_sync(0xffffffffu, km, off));
  }
  if (lane == 0) { S.wsum[w] = tot; S.wcnt[w] = km; }
  __syncthreads();
  total = 0;
  kmax = 0;
  for (int i = 0; i < NTH / 32; ++i) { total += S.wsum[i]; kmax = max(kmax, S.wcnt[i]); }
  __syncthreads();
}

// Smallest key (of a non-negative float) whose weight in 2^-shift units is
// at least wt >= 1 (weights do not decrease with the key).
__device__ __forceinline__ uint32_t key_of_weight(unsigned long long wt, int shift) {
  uint32_t lo = 0x80000001u, hi = 0xFF7FFFFFu;   // the largest finite float weighs >= 2^63
  while (lo < hi) {
    const uint32_t mid = lo + ((hi - lo) >> 1);
    if (fx_weight(mid, shift) >= wt) hi = mid; else lo = mid + 1u;
  }
  return lo;
}

// Appends the keys of m[0, n) at or above klb (> the key of 0) with their
// indices to (cand, cidx), in no particular order, and returns their number
// to every thread (also when it exceeds cap: only the first cap are kept).
// S.ncand must be 0 on entry. Each warp takes one atomic per batch of loads.
template <int NTH>
__device__ int compact_above(const float* m, int n, uint32_t klb, uint32_t* cand, uint32_t* cidx,
                             int cap, SelShared<NTH>& S) {
  const int tid = threadIdx.x, lane = tid & 31;
  const unsigned below = (1u << lane) - 1u;
  const int head = min(n, (int)(((16u - (uint32_t)(reinterpret_cast<uintptr_t>(m) & 15)) & 15u) >> 2));
  const float4* g4 = reinterpret_cast<const float4*>(m + head);
  const int n4 = (n - head) >> 2;
  constexpr int U4 = 4;
  for (int base = 0; base < n4; base += U4 * NTH) {   // the same trip count in every warp
    float4 f[U4];
#pragma unroll
    for (int j = 0; j < U4; ++j) {
      const int i4 = base + j * NTH + tid;
      f[j] = i4 < n4 ? __ldg(g4 + i4) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    uint32_t kk[4 * U4];
    unsigned bal[4 * U4];
    unsigned tot = 0;
#pragma unroll
    for (int j = 0; j < U4; ++j) {
      kk[4 * j] = nonneg_key(f[j].x); kk[4 * j + 1] = nonneg_key(f[j].y);
      kk[4 * j + 2] = nonneg_key(f[j].z); kk[4 * j + 3] = nonneg_key(f[j].w);
    }
#pragma unroll
    for (int j = 0; j < 4 * U4; ++j) {
      bal[j] = __ballot_sync(0xffffffffu, kk[j] >= klb);
      tot += __popc(bal[j]);
    }
    if (!tot) continue;   // the usual case: one atomic per warp and batch otherwise
    unsigned at = 0;
    if (lane == 0) at = atomicAdd(&S.ncand, tot);
    at = __shfl_sync(0xffffffffu, at, 0);
#pragma unroll
    for (int j = 0; j < 4 * U4; ++j) {
      if ((bal[j] >> lane) & 1u) {
        const unsigned o = at + __popc(bal[j] & below);
        if (o < (unsigned)cap) {
          cand[o] = kk[j];
          cidx[o] = (uint32_t)(head + 4 * (base + (j >> 2) * NTH + tid) + (j & 3));
        }
      }
      at += __popc(bal[j]);
    }
  }
  if (tid < 32) {  // the head and the tail: at most 3 + 3 keys, warp 0
    const int tail0 = head + (n4 << 2);
    const int i = tid < head ? tid : tail0 + (tid - 3);
    const bool has = tid < head || (tid >= 3 && tid < 6 && i < n);
    const bool in = has && nonneg_key(__ldg(m + i)) >= klb;
    const unsigned bl = __ballot_sync(0xffffffffu, in);
    if (bl) {
      unsigned at = 0;
      if (lane == 0) at = atomicAdd(&S.ncand, __popc(bl));
      at = __shfl_sync(0xffffffffu, at, 0) + __popc(bl & below);
      if (in && at < (unsigned)cap) { cand[at] = nonneg_key(__ldg(m + i)); cidx[at] = (uint32_t)i; }
    }
  }
  __syncthreads();
  return (int)S.ncand;
}

// The cover set's keys among the candidates (cand, cidx)[0, nc): every key
// ranked before them in (key desc, index asc) order weighs S.cum_w in all,
// every key ranked after them is below all of them, and the last digits
// from p0 on are still open (prefix holds the chosen ones). The set is the
// shortest prefix of that order whose weight reaches target_w; its bits are
// ORed into the bitmap. Up to NTH candidates: each thread ranks one against
// all the others. More: the remaining digit passes among them, then the
// keys equal to the last key theta by index.
template <int NTH>
__device__ void cover_among(const uint32_t* cand, const uint32_t* cidx, int nc, int p0,
                            uint32_t prefix, unsigned long long target_w, int shift, float tau,
                            SelShared<NTH>& S, uint32_t* hist, uint32_t* bits) {
  const int tid = threadIdx.x;
  if (nc <= NTH) {
    // (key << 32 | ~index, weight) per candidate: a larger first word ranks
    // earlier
    ulonglong2* cw = reinterpret_cast<ulonglong2*>(hist);
    if (tid == 0) S.rend = 0xFFFFFFFFu;
    if (tid < nc)
      cw[tid] = make_ulonglong2(((unsigned long long)cand[tid] << 32) | (uint32_t)~cidx[tid],
                                fx_weight(cand[tid], shift));
    __syncthreads();
    const unsigned long long above = S.cum_w;
    unsigned rank = 0;
    unsigned long long me = 0;
    if (tid < nc) {
      const ulonglong2 x = cw[tid];
      me = x.x;
      unsigned long long before = 0;
      int e = 0;
      for (; e + 4 <= nc; e += 4) {
        const ulonglong2 y0 = cw[e], y1 = cw[e + 1], y2 = cw[e + 2], y3 = cw[e + 3];
        rank += (y0.x > me) + (y1.x > me) + (y2.x > me) + (y3.x > me);
        before += (y0.x > me ? y0.y : 0ull) + (y1.x > me ? y1.y : 0ull) +
                  (y2.x > me ? y2.y : 0ull) + (y3.x > me ? y3.y : 0ull);
      }
      for (; e < nc; ++e) {
        const ulonglong2 y = cw[e];
        rank += y.x > me;
        before += y.x > me ? y.y : 0ull;
      }
      if (above + before + x.y >= target_w) atomicMin(&S.rend, rank);
    }
    __syncthreads();
    if (tid < nc && rank <= S.rend) {
      const uint32_t ix = ~(uint32_t)me;
      atomicOr(bits + (ix >> 5), 1u << (ix & 31));
    }
    return;
  }
  radix_passes<true, NTH, SmemKeys, true>(SmemKeys{cand}, nc, p0, 4, prefix, target_w, 1u, &shift,
                                          tau, S, hist, false);
  const uint32_t theta = prefix;
  const unsigned n_theta = S.n_theta;
  const unsigned long long wth = fx_weight(theta, shift);
  const unsigned long long need_w = target_w > S.cum_w ? target_w - S.cum_w : 0ull;
  unsigned n_tie = 1;
  if (need_w > 0 && wth > 0) n_tie = (unsigned)((need_w + wth - 1) / wth);
  if (n_tie > n_theta) n_tie = n_theta;
  // a key equal to theta is in if fewer than n_tie equal keys precede it
  for (int c = tid; c < nc; c += NTH) {
    const uint32_t k = cand[c], i = cidx[c];
    bool in = k > theta;
    if (k == theta) {
      unsigned rank = 0;
      if (n_tie < n_theta)
        for (int e = 0; e < nc; ++e) rank += (cand[e] == theta && cidx[e] < i) ? 1u : 0u;
      in = rank < n_tie;
    }
    if (in) atomicOr(bits + (i >> 5), 1u << (i & 31));
  }
}

template <int NTH>
__global__ void __launch_bounds__(NTH, 1024 / NTH) cover_kernel(Problem P, Buffers bf) {
  extern __shared__ uint32_t dyn[];
  uint32_t* hist = dyn;
  uint32_t* cand = dyn + hist_words<NTH, true>();   // kCoverCand keys, then their indices
  uint32_t* cidx = cand + kCoverCand;
  __shared__ SelShared<NTH> S;
  constexpr int NWC = NTH / 32;
  const int g = blockIdx.x % P.G, h = blockIdx.x / P.G, b = blockIdx.y, l = blockIdx.z;
  const ReqInfo R = P.req[b];
  const int n = R.t_len, tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  if (n <= 0) return;
  const size_t row = ((size_t)l * P.Hkv + h) * P.G + g;
  const float* m = bf.gmass + row * P.total_T + R.tok_off;
  uint32_t* bits = bf.bits + row * P.total_words + R.word_off;
  const GlobalFloats get{m};

  // Only keys of weight >= lb can be in the cover set or tie with its last
  // key theta, where lb = (total - target + 1) / n: the keys ranked before
  // theta weigh at most target - 1 (else the cover would end earlier) and
  // the at most n - 1 after it at most w_theta each, so total <= target - 1
  // + n * w_theta. With few such keys the cover is decided among them
  // alone, every other bit being 0. When the masses are softmax sums of a
  // known number of rows (P.cover_hint), the keys above half the bound that
  // total implies are collected in the same pass as the total; the
  // collection stands if its bound is at most lb, else a second pass
  // collects the keys of weight >= lb.
  int shift = 40;
  unsigned long long gspec = 0;
  if (P.cover_hint > 0.f) {
    const double g = ((1.0 - (double)P.tau) * 0.5 * (double)P.cover_hint * 1099511627776.0 - 1.0) /
                     (double)n;                       // 2^40 units
    gspec = g >= 1.0 ? (unsigned long long)g : 0ull;
  }
  if (tid == 0) {
    S.prefix = gspec ? key_of_weight(gspec, shift) : 0xFFFFFFFFu;
    S.ncand = 0;
    S.cum_w = 0;
    S.cum_n = 0;
  }
  for (int i = tid; i < (n + 31) / 32; i += NTH) bits[i] = 0u;
  __syncthreads();
  unsigned long long total = 0;
  uint32_t kmax = 0;
  total_and_max<NTH>(m, n, shift, S.prefix, cand, cidx, kCoverCand,
                     reinterpret_cast<float4*>(hist), S, total, kmax);
  int nc = (int)S.ncand;
  {
    // the 2^-shift unit is lowered where n * max * 2^shift could overflow 64 bits
    int e = 0;
    frexpf(key_value(kmax), &e);              // values < 2^e
    int lg = 0;
    while ((1 << lg) < n) ++lg;               // n <= 2^lg
    if (e + lg + shift > 63) {
      shift = max(0, 63 - e - lg);
      gspec = 0;
      total_and_max<NTH>(m, n, shift, 0xFFFFFFFFu, cand, cidx, kCoverCand,
                         reinterpret_cast<float4*>(hist), S, total, kmax);
    }
  }
  const unsigned long long tt = (unsigned long long)ceil((double)P.tau * (double)total);
  unsigned long long target_w = tt > total ? total : tt;
  const unsigned long long lb = (total - target_w + 1) / (unsigned long long)n;
  if (lb > 0) {
    if (!(gspec > 0 && gspec <= lb && nc <= kCoverCand)) {
      __syncthreads();   // every thread has read S.ncand
      if (tid == 0) {
        S.prefix = key_of_weight(lb, shift);
        S.ncand = 0;
      }
      __syncthreads();
      nc = compact_above<NTH>(m, n, S.prefix, cand, cidx, kCoverCand, S);
    }
    if (nc > 0 && nc <= kCoverCand) {
      cover_among<NTH>(cand, cidx, nc, 0, 0x80000000u, target_w, shift, P.tau, S, hist, bits);
      return;
    }
  }

  // Many keys above the bound: the first digit pass over the masses (from
  // L2), then, when the keys that share the chosen first digit fit in shared
  // memory, one more pass writes the bitmap words of the keys above that
  // digit and copies the keys sharing it; the last three digits and the ties
  // are resolved among those.
  uint32_t prefix = 0x80000000u;
  radix_passes<true, NTH>(get, n, 0, 1, prefix, target_w, 1u, &shift, P.tau, S, hist);
  constexpr int U = 8;
  if (S.n_theta <= (unsigned)kCoverCand) {
    if (tid == 0) S.ncand = 0;
    __syncthreads();
    const uint32_t d0 = prefix >> 23;
    const unsigned below = (1u << lane) - 1u;
    for (int base = w * 32; base < n; base += U * NTH) {
      uint32_t kk[U];
#pragma unroll
      for (int j = 0; j < U; ++j) {
        const int i = base + j * NTH + lane;
        kk[j] = i < n ? get(i) : 0u;
      }
      unsigned cb[U];
      unsigned tot = 0;
#pragma unroll
      for (int j = 0; j < U; ++j) {
        const int i = base + j * NTH + lane;
        const bool in = i < n && (kk[j] >> 23) > d0;
        const unsigned word = __ballot_sync(0xffffffffu, in);
        if (lane == 0 && base + j * NTH < n) bits[(base + j * NTH) >> 5] = word;
        cb[j] = __ballot_sync(0xffffffffu, i < n && (kk[j] >> 23) == d0);
        tot += __popc(cb[j]);
      }
      if (tot) {   // the batch's candidates: one atomic for the warp
        unsigned at = 0;
        if (lane == 0) at = atomicAdd(&S.ncand, tot);
        at = __shfl_sync(0xffffffffu, at, 0);
#pragma unroll
        for (int j = 0; j < U; ++j) {
          if ((cb[j] >> lane) & 1u) {
            const unsigned o = at + __popc(cb[j] & below);
            cand[o] = kk[j];
            cidx[o] = (uint32_t)(base + j * NTH + lane);
          }
          at += __popc(cb[j]);
        }
      }
    }
    __syncthreads();
    cover_among<NTH>(cand, cidx, (int)S.ncand, 1, prefix, target_w, shift, P.tau, S, hist, bits);
    return;
  }
  radix_passes<true, NTH>(get, n, 1, 4, prefix, target_w, 1u, &shift, P.tau, S, hist);
  if (tid == 0) S.prefix = prefix;
  __syncthreads();
  const uint32_t theta = S.prefix;
  const unsigned n_theta = S.n_theta;
  const unsigned long long wth = fx_weight(theta, shift);
  const unsigned long long need_w = target_w > S.cum_w ? target_w - S.cum_w : 0ull;
  unsigned n_tie = 1;
  if (need_w > 0 && wth > 0) n_tie = (unsigned)((need_w + wth - 1) / wth);
  if (n_tie > n_theta) n_tie = n_theta;
  if (tid == 0) S.aux = n;  // every key equal to theta is in
  __syncthreads();
  if (n_tie < n_theta) {
    // t* = index of the n_tie-th key equal to theta (ascending t); warp segments
    const int seg = ((n + NWC * 32 - 1) / (NWC * 32)) * 32;
    const int lo = w * seg, hi = min(n, lo + seg);
    unsigned cnt = 0;
    for (int base = lo; base < hi; base += 32) {
      const int i = base + lane;
      cnt += __popc(__ballot_sync(0xffffffffu, i < hi && get(i) == theta));
    }
    const unsigned before = warp_excl_prefix<NTH>(S, cnt);
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
  for (int base = w * 32; base < n; base += U * NTH) {
    uint32_t kk[U];
#pragma unroll
    for (int j = 0; j < U; ++j) {
      const int i = base + j * NTH + lane;
      kk[j] = i < n ? get(i) : 0u;
    }
#pragma unroll
    for (int j = 0; j < U; ++j) {
      const int i = base + j * NTH + lane;
      const bool mem = i < n && (kk[j] > theta || (kk[j] == theta && i <= tstar));
      const unsigned word = __ballot_sync(0xffffffffu, mem);
      if (lane == 0 && base + j * NTH < n) bits[(base + j * NTH) >> 5] = word;
    }
  }
}

// The keep - 1 largest keys among t < n - 1 (ties: lower t), written to out
// (stride ostride) in ascending t, then n - 1 last. The first digit is taken
// over all candidates, the later digits over the keys that share it, copied
// to shared memory when they fit (cand, kTopkCand keys).
template <int NT, class Src>
__device__ void select_kept(const Src& get, int n, int keep, int32_t* out, int ostride,
                            SelShared<NT>& S, uint32_t* hist, uint32_t* cand) {
  constexpr int NW = NT / 32;
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  const int nc = n - 1;  // candidates t < T-1
  uint32_t theta = 0x80000000u;
  unsigned long long no_w = 0;
  radix_passes<false, NT, Src>(get, nc, 0, 1, theta, no_w, (unsigned)(keep - 1), nullptr, 0.f, S,
                               hist);
  if (S.n_theta <= (unsigned)kTopkCand) {
    const int ncand = compact_prefix<NT, Src>(get, nc, theta, 23, cand, S);
    radix_passes<false, NT, SmemKeys, true>(SmemKeys{cand}, ncand, 1, 4, theta, no_w,
                                            (unsigned)(keep - 1), nullptr, 0.f, S, hist);
  } else {
    radix_passes<false, NT, Src>(get, nc, 1, 4, theta, no_w, (unsigned)(keep - 1), nullptr, 0.f, S,
                                 hist);
  }
  const unsigned n_tie = (unsigned)(keep - 1) - S.cum_n;
  // ordered compaction over warp segments, four 32-key chunks' loads at a time
  constexpr int UC = 4;
  const int seg = ((nc + NW * 32 - 1) / (NW * 32)) * 32;
  const int lo = w * seg, hi = min(nc, lo + seg);
  unsigned c_gt = 0, c_tie = 0;
  for (int base = lo; base < hi; base += UC * 32) {
    uint32_t kk[UC];
#pragma unroll
    for (int u = 0; u < UC; ++u) {
      const int i = base + u * 32 + lane;
      kk[u] = i < hi ? get(i) : 0u;
    }
#pragma unroll
    for (int u = 0; u < UC; ++u) {
      const bool in = base + u * 32 + lane < hi;
      c_gt += __popc(__ballot_sync(0xffffffffu, in && kk[u] > theta));
      c_tie += __popc(__ballot_sync(0xffffffffu, in && kk[u] == theta));
    }
  }
  // both exclusive prefixes over the warps at once (counts < 2^32 each)
  if (lane == 0) S.wsum[w] = (unsigned long long)c_gt | ((unsigned long long)c_tie << 32);
  __syncthreads();
  unsigned long long before = 0;
  for (int i = 0; i < w; ++i) before += S.wsum[i];
  __syncthreads();
  const unsigned gt_before = (unsigned)before;
  unsigned tie_before = (unsigned)(before >> 32);
  unsigned pos = gt_before + min(tie_before, n_tie);
  const unsigned lt = (1u << lane) - 1u;
  for (int base = lo; base < hi; base += UC * 32) {
    uint32_t kk[UC];
#pragma unroll
    for (int u = 0; u < UC; ++u) {
      const int i = base + u * 32 + lane;
      kk[u] = i < hi ? get(i) : 0u;
    }
#pragma unroll
    for (int u = 0; u < UC; ++u) {
      const int i = base + u * 32 + lane;
      const bool is_tie = i < hi && kk[u] == theta;
      const unsigned tie_m = __ballot_sync(0xffffffffu, is_tie);
      const unsigned my_rank = tie_before + __popc(tie_m & lt);
      const bool sel = i < hi && (kk[u] > theta || (is_tie && my_rank < n_tie));
      const unsigned sel_m = __ballot_sync(0xffffffffu, sel);
      if (sel) out[(size_t)(pos + __popc(sel_m & lt)) * ostride] = i;
      pos += __popc(sel_m);
      tie_before += __popc(tie_m);
    }
  }
  if (tid == 0) out[(size_t)(keep - 1) * ostride] = n - 1;
}

// The keep - 1 largest of the staged keys[0, n - 1) (ties: lower t), written
// to out (stride ostride) in ascending t, then n - 1 last, with a 12-bit
// first digit (the exponent and the top four significand bits): one
// CTA-wide histogram of 4096 bins (hist_built: already counted over keys
// [0, n - 1) by the caller), a block scan for the digit d0 where the
// count from the top reaches keep - 1, the keys of digit d0 copied to shared
// memory with their indices while the bitmap of the keys above d0 is
// written, the kept ones among them added to it (ranked one per thread when
// few, else by the last three digit passes and the ties' indices), then a
// block scan over the bitmap's words places the kept indices. Returns false (before writing any
// output) when more than kFineCand keys share d0.
constexpr int kFineCand = 1024;
template <int NT>
__device__ bool select_kept_fine(const uint32_t* keys, int n, int keep, int32_t* out, int ostride,
                                 SelShared<NT>& S, uint32_t* hist, uint32_t* cand,
                                 bool hist_built) {
  constexpr int NW = NT / 32;
  constexpr int BPT = 4096 / NT;                       // histogram bins per thread
  constexpr int WPL = (kMaxStaged / (NW * 32) + 31) / 32 + 1;   // kept words per lane
  static_assert(hist_words<NT, false>() >= 4096, "12-bit histogram in the per-warp histograms' room");
  static_assert(2 * kFineCand + kMaxStaged / 32 <= kTopkCand, "candidates and kept bits in cand");
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  const int nc = n - 1;                 // candidates t < n - 1
  const unsigned k = (unsigned)(keep - 1);   // 1 <= k < nc
  uint32_t* ck = cand;                  // keys of digit d0
  uint32_t* ci = cand + kFineCand;      // their indices
  uint32_t* kbits = cand + 2 * kFineCand;    // kept keys of digit d0, by index
  const int nwords = (nc + 31) >> 5;
  if (!hist_built) {
    for (int i = tid; i < 4096; i += NT) hist[i] = 0u;
    __syncthreads();
    for (int i = tid; i < nc; i += NT) atomicAdd(&hist[(keys[i] >> 19) & 0xFFFu], 1u);
  }
  if (tid == 0) S.ncand = 0;
  __syncthreads();
  // thread t owns digits 4095 - BPT t down to 4096 - BPT (t + 1): inclusive
  // scan of their counts in thread order is the count from the top
  unsigned c = 0;
#pragma unroll
  for (int j = 0; j < BPT; ++j) c += hist[4095 - BPT * tid - j];
  unsigned incl = c;
  for (int off = 1; off < 32; off <<= 1) {
    const unsigned t = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += t;
  }
  if (lane == 31) S.wcnt[w] = incl;
  __syncthreads();
  for (int i = 0; i < w; ++i) incl += S.wcnt[i];
  const unsigned excl = incl - c;
  if (excl < k && incl >= k) {
    unsigned cum = excl;
    for (int j = 0; j < BPT; ++j) {
      const int d = 4095 - BPT * tid - j;
      const unsigned b = hist[d];
      if (cum + b >= k) {
        S.digit = (unsigned)d;
        S.cum_n = cum;
        S.n_theta = b;
        break;
      }
      cum += b;
    }
  }
  __syncthreads();
  const uint32_t d0 = S.digit;
  const unsigned above = S.cum_n, nd = S.n_theta;
  if (nd > (unsigned)kFineCand) {
    __syncthreads();   // every thread has read S before the caller's select rewrites it
    return false;
  }
  // the keys of digit d0 with their indices, and the kept-bitmap words of
  // the keys above d0 (every word of [0, nc) is written here); a warp's 32
  // consecutive keys, four chunks at a time, take one atomic
  const unsigned below = (1u << lane) - 1u;
  for (int base = w * 128; base < nc; base += NT * 4) {
    bool in[4];
    unsigned bal[4], tot = 0;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int i = base + 32 * u + lane;
      const uint32_t d = i < nc ? (keys[i] >> 19) & 0xFFFu : 0u;
      in[u] = i < nc && d == d0;
      bal[u] = __ballot_sync(0xffffffffu, in[u]);
      tot += __popc(bal[u]);
      const unsigned gt = __ballot_sync(0xffffffffu, i < nc && d > d0);
      if (lane == 0 && base + 32 * u < nc) kbits[(base + 32 * u) >> 5] = gt;
    }
    if (!tot) continue;
    unsigned at = 0;
    if (lane == 0) at = atomicAdd(&S.ncand, tot);
    at = __shfl_sync(0xffffffffu, at, 0);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      if (in[u]) {
        const unsigned o = at + __popc(bal[u] & below);
        const int i = base + 32 * u + lane;
        ck[o] = keys[i];
        ci[o] = (uint32_t)i;
      }
      at += __popc(bal[u]);
    }
  }
  __syncthreads();
  const unsigned need = k - above;      // kept keys of digit d0, 1 <= need <= nd
  if (nd <= (unsigned)NT) {
    // (key << 32 | ~index) ranks earlier when larger
    unsigned long long* comp = reinterpret_cast<unsigned long long*>(hist);
    if (tid < (int)nd) comp[tid] = ((unsigned long long)ck[tid] << 32) | (uint32_t)~ci[tid];
    __syncthreads();
    if (tid < (int)nd) {
      const unsigned long long me = comp[tid];
      unsigned rank = 0;
      int e = 0;
      for (; e + 4 <= (int)nd; e += 4)
        rank += (comp[e] > me) + (comp[e + 1] > me) + (comp[e + 2] > me) + (comp[e + 3] > me);
      for (; e < (int)nd; ++e) rank += comp[e] > me;
      if (rank < need) {
        const uint32_t i = ~(uint32_t)me;
        atomicOr(&kbits[i >> 5], 1u << (i & 31));
      }
    }
  } else {
    uint32_t theta = ck[0] & 0xFFF80000u;   // bits 19-31 are d0's
    unsigned long long no_w = 0;
    radix_passes<false, NT, SmemKeys, true>(SmemKeys{ck}, (int)nd, 1, 4, theta, no_w, k, nullptr,
                                            0.f, S, hist);
    const unsigned n_tie = k - S.cum_n;   // keys equal to theta kept, lowest indices first
    for (int c2 = tid; c2 < (int)nd; c2 += NT) {
      const uint32_t kk = ck[c2], i = ci[c2];
      bool kept = kk > theta;
      if (kk == theta) {
        unsigned r = 0;
        for (int e = 0; e < (int)nd; ++e) r += (ck[e] == theta && ci[e] < i) ? 1u : 0u;
        kept = r < n_tie;
      }
      if (kept) atomicOr(&kbits[i >> 5], 1u << (i & 31));
    }
  }
  __syncthreads();
  // kept words (the bitmap above): warp w owns words [w0, w0 + wpw); lane j
  // of row q holds word w0 + 32 q + j
  const int wpw = (nwords + NW - 1) / NW;
  const int w0 = w * wpw;
  const int nww = max(0, min(wpw, nwords - w0));   // words of this warp
  uint32_t word[WPL];
  unsigned row_tot[WPL], row_excl[WPL];
  unsigned wtot = 0;
#pragma unroll
  for (int q = 0; q < WPL; ++q) {
    const int wi = 32 * q + lane;
    word[q] = wi < nww ? kbits[w0 + wi] : 0u;
    const unsigned cnt = __popc(word[q]);
    unsigned inc = cnt;
    for (int off = 1; off < 32; off <<= 1) {
      const unsigned t = __shfl_up_sync(0xffffffffu, inc, off);
      if (lane >= off) inc += t;
    }
    row_excl[q] = inc - cnt;
    row_tot[q] = __shfl_sync(0xffffffffu, inc, 31);
    wtot += row_tot[q];
  }
  if (lane == 0) S.wcnt[w] = wtot;
  __syncthreads();
  unsigned pos = 0;
  for (int i = 0; i < w; ++i) pos += S.wcnt[i];
  // the kept indices go to shared memory (the histograms' room) in order,
  // then out in one coalesced sweep; directly when they do not fit
  int32_t* staging = reinterpret_cast<int32_t*>(hist);
  const bool via_smem = k <= (unsigned)hist_words<NT, false>();
#pragma unroll
  for (int q = 0; q < WPL; ++q) {
    unsigned p = pos + row_excl[q];
    uint32_t m = word[q];
    const int i0 = (w0 + 32 * q + lane) * 32;
    while (m) {
      const int bit = __ffs(m) - 1;
      m &= m - 1u;
      if (via_smem) staging[p++] = i0 + bit;
      else out[(size_t)(p++) * ostride] = i0 + bit;
    }
    pos += row_tot[q];
  }
  if (via_smem) {
    __syncthreads();
    for (int i = tid; i < (int)k; i += NT) out[(size_t)i * ostride] = staging[i];
  }
  if (tid == 0) out[(size_t)(keep - 1) * ostride] = n - 1;
  return true;
}

// from_scores: S comes from bf.scores as given; otherwise it is built here.
// NT threads per CTA (512, or 1024 when the units are fewer than the SMs).
template <int NT>
__global__ void __launch_bounds__(NT, NT >= 1024 ? 1 : 2) topk_kernel(Problem P, Buffers bf, int32_t* out_idx,
                                                     int from_scores, int staged_cap) {
  constexpr int NW = NT / 32;
  extern __shared__ uint32_t dyn[];
  uint32_t* hist = dyn;
  uint32_t* cand = dyn + hist_words<NT, false>();     // kTopkCand first-digit candidates
  uint32_t* keys_sm = cand + kTopkCand;               // staged_cap keys
  __shared__ SelShared<NT> S;
  const int h = blockIdx.x, b = blockIdx.y, l = blockIdx.z;
  const ReqInfo R = P.req[b];
  const int n = R.t_len, tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  const size_t hrow = ((size_t)l * P.Hkv + h) * P.total_T + R.tok_off;
  float* sc = bf.scores + hrow;
  const bool staged = n <= staged_cap;
  // scores go to global memory when the selection reads them from there or
  // the caller asked for them
  const bool write_sc = !staged || bf.scores_out;
  // staged keys are counted by their 12-bit first digit as they are written
  // (select_kept_fine), the last key excepted
  if (staged) {
    for (int i = tid; i < 4096; i += NT) hist[i] = 0u;
    __syncthreads();
  }
  auto count12 = [&](uint32_t key, int i) {
    if (i < n - 1) atomicAdd(&hist[(key >> 19) & 0xFFFu], 1u);
  };
  if (!from_scores) {
    const float* an = bf.anchor + hrow;
    const uint32_t* bw = bf.bits + ((size_t)l * P.Hkv + h) * P.G * P.total_words + R.word_off;
    int done = 0;
    if (P.mode == MMSHIFT_SCORE_VOTE && P.G <= 8 && staged &&
        ((reinterpret_cast<uintptr_t>(an) | reinterpret_cast<uintptr_t>(sc)) & 15) == 0) {
      // four keys per lane: 16-byte loads of the anchors and stores of the
      // scores (if written) and keys; a lane's keys 4j .. 4j+3 are bits
      // (4j mod 32) .. +3 of coverage word 4j / 32 (one word serves eight
      // lanes)
      constexpr int UB4 = 4;
      const float4* an4 = reinterpret_cast<const float4*>(an);
      float4* sc4 = reinterpret_cast<float4*>(sc);
      uint4* ks4 = reinterpret_cast<uint4*>(keys_sm);
      const int n4 = (n >> 5) << 3;   // whole 32-key words only: the rest goes below
      for (int b4 = w * 32; b4 < n4; b4 += UB4 * NT) {
        float4 a[UB4];
        uint32_t vt[UB4];   // four 8-bit vote counters per lane
#pragma unroll
        for (int u = 0; u < UB4; ++u) {
          const int j4 = b4 + u * NT + lane;
          a[u] = j4 < n4 ? __ldg(an4 + j4) : make_float4(0.f, 0.f, 0.f, 0.f);
          vt[u] = 0;
        }
        for (int g = 0; g < P.G; ++g) {
#pragma unroll
          for (int u = 0; u < UB4; ++u) {
            const int j4 = b4 + u * NT + lane;
            const uint32_t word =
                j4 < n4 ? __ldg(bw + (size_t)g * P.total_words + (j4 >> 3)) : 0u;
            const uint32_t nib = (word >> ((j4 & 7) * 4)) & 0xFu;
            // spread the nibble's bits into the bytes of vt
            vt[u] += (nib & 1u) | ((nib & 2u) << 7) | ((nib & 4u) << 14) | ((nib & 8u) << 21);
          }
        }
#pragma unroll
        for (int u = 0; u < UB4; ++u) {
          const int j4 = b4 + u * NT + lane;
          if (j4 < n4) {
            float4 sv;
            sv.x = __fadd_rn((float)(vt[u] & 255u), __fmul_rn(P.lambda, a[u].x));
            sv.y = __fadd_rn((float)((vt[u] >> 8) & 255u), __fmul_rn(P.lambda, a[u].y));
            sv.z = __fadd_rn((float)((vt[u] >> 16) & 255u), __fmul_rn(P.lambda, a[u].z));
            sv.w = __fadd_rn((float)(vt[u] >> 24), __fmul_rn(P.lambda, a[u].w));
            if (write_sc) sc4[j4] = sv;
            const uint4 kq = make_uint4(nonneg_key(sv.x), nonneg_key(sv.y), nonneg_key(sv.z),
                                        nonneg_key(sv.w));
            ks4[j4] = kq;
            count12(kq.x, 4 * j4); count12(kq.y, 4 * j4 + 1);
            count12(kq.z, 4 * j4 + 2); count12(kq.w, 4 * j4 + 3);
          }
        }
      }
      done = n4 << 2;
    }
    // each warp takes 32 consecutive keys at a time, UB chunks of them with
    // their loads in flight together (the keys the 16-byte path left, if any)
    constexpr int UB = NT >= 1024 ? 4 : 8;
    for (int base0 = done + w * 32; base0 < n; base0 += UB * NT) {
      float sv[UB];
      if (P.mode == MMSHIFT_SCORE_VOTE) {
        // lane g holds the coverage word of group g for a chunk of 32 keys;
        // after the transpose lane j holds the bits of key base+j over the
        // groups, and its vote is their count
        unsigned vote[UB];
        float av[UB];
#pragma unroll
        for (int u = 0; u < UB; ++u) {
          vote[u] = 0;
          const int i = base0 + u * NT + lane;
          av[u] = i < n ? __ldg(an + i) : 0.f;
        }
        if (P.G <= 8) {
          // few groups: every lane reads the chunk's word of each group (one
          // broadcast load) and takes its own bit
          for (int g = 0; g < P.G; ++g) {
            uint32_t word[UB];
#pragma unroll
            for (int u = 0; u < UB; ++u) {
              const int base = base0 + u * NT;
              word[u] = base < n ? __ldg(bw + (size_t)g * P.total_words + (base >> 5)) : 0u;
            }
#pragma unroll
            for (int u = 0; u < UB; ++u) vote[u] += (word[u] >> lane) & 1u;
          }
        } else {
          for (int g0 = 0; g0 < P.G; g0 += 32) {
            const int g = g0 + lane;
            uint32_t word[UB];
#pragma unroll
            for (int u = 0; u < UB; ++u) {
              const int base = base0 + u * NT;
              word[u] = (g < P.G && base < n) ? __ldg(bw + (size_t)g * P.total_words + (base >> 5)) : 0u;
            }
#pragma unroll
            for (int u = 0; u < UB; ++u) vote[u] += __popc(warp_transpose32(word[u]));
          }
        }
#pragma unroll
        for (int u = 0; u < UB; ++u)
          sv[u] = __fadd_rn((float)vote[u], __fmul_rn(P.lambda, av[u]));  // no contraction
      } else {
#pragma unroll
        for (int u = 0; u < UB; ++u) sv[u] = 0.f;
        for (int g = 0; g < P.G; ++g) {
          const float* gm = bf.gmass + (((size_t)l * P.Hkv + h) * P.G + g) * P.total_T + R.tok_off;
#pragma unroll
          for (int u = 0; u < UB; ++u) {
            const int i = base0 + u * NT + lane;
            if (i < n) sv[u] += __ldg(gm + i);
          }
        }
      }
#pragma unroll
      for (int u = 0; u < UB; ++u) {
        const int i = base0 + u * NT + lane;
        if (i < n) {
          if (write_sc) sc[i] = sv[u];
          if (staged) {
            const uint32_t kq = nonneg_key(sv[u]);
            keys_sm[i] = kq;
            count12(kq, i);
          }
        }
      }
    }
  } else if (staged) {
    for (int i = tid; i < n; i += NT) {
      const uint32_t kq = nonneg_key(sc[i]);
      keys_sm[i] = kq;
      count12(kq, i);
    }
  }
  __syncthreads();
  int32_t* out = out_idx + ((size_t)l * P.R + R.out_off) * P.Hkv + h;
  int keep = R.keep;
  if (bf.head_budget) {
    // this head's own budget; its rows past the kept ones are padding (-1)
    int c = bf.head_budget[((size_t)l * P.B + b) * P.Hkv + h];
    if (c < 1 || c > R.budget) {
      if (tid == 0) set_status(bf.status, kStatusBadBudget);
      c = min(max(c, 1), R.budget);
    }
    keep = min(c, n);
    for (int i = keep + tid; i < R.keep; i += NT) out[(size_t)i * P.Hkv] = -1;
  }
  if (bf.out_count && tid == 0) bf.out_count[((size_t)l * P.B + b) * P.Hkv + h] = keep;
  if (keep >= n) {
    for (int i = tid; i < n; i += NT) out[(size_t)i * P.Hkv] = i;
    return;
  }
  if (keep == 1) {
    if (tid == 0) out[0] = n - 1;
    return;
  }
  if (staged) {
    if (!select_kept_fine<NT>(keys_sm, n, keep, out, P.Hkv, S, hist, cand, true))
      select_kept<NT>(SmemKeys{keys_sm}, n, keep, out, P.Hkv, S, hist, cand);
  }
  else {
    select_kept<NT>(GlobalFloats{sc}, n, keep, out, P.Hkv, S, hist, cand);
  }
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
    // zero rows: padding of a head with its own smaller budget (-1), or a bad index
    *dk = make_uint4(0, 0, 0, 0);
    *dv = make_uint4(0, 0, 0, 0);
    if (part == 0 && !(bf.head_budget && t == -1)) set_status(bf.status, kStatusBadIndex);
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
  dim3 grid(P.Hkv * P.G, P.B, P.L);
  // few units (the few-proxy setting): 512 threads each, all resident at
  // two per SM; many units: 256 threads each, four per SM
  int dev = 0, nsm = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  const long long units = (long long)grid.x * grid.y * grid.z;
#define MMSHIFT_COVER(NTH)                                                                    \
  {                                                                                          \
    const size_t smem = (size_t)(hist_words<NTH, true>() + 2 * kCoverCand) * sizeof(uint32_t); \
    if ((e = cudaFuncSetAttribute(cover_kernel<NTH>,                                         \
                                  cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) != \
        cudaSuccess)                                                                         \
      return e;                                                                              \
    cover_kernel<NTH><<<grid, NTH, smem, st>>>(P, bf);                                       \
    return cudaGetLastError();                                                               \
  }
  if (units <= 2LL * nsm) MMSHIFT_COVER(512)
  MMSHIFT_COVER(256)
#undef MMSHIFT_COVER
}

cudaError_t launch_topk(const Problem& P, const Buffers& bf, cudaStream_t st, int32_t* out_idx,
                        bool from_scores) {
  int maxT = 0;
  for (int b = 0; b < P.B; ++b) maxT = max(maxT, P.req[b].t_len);
  int dev = 0, nsm = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  dim3 grid(P.Hkv, P.B, P.L);
  const long long units = (long long)grid.x * grid.y * grid.z;
  const int staged = min(maxT, kMaxStaged);
#define MMSHIFT_TOPK(NTT)                                                                        \
  {                                                                                             \
    const size_t smem = (size_t)(hist_words<NTT, false>() + kTopkCand + staged) * sizeof(uint32_t); \
    if ((e = cudaFuncSetAttribute(topk_kernel<NTT>, cudaFuncAttributeMaxDynamicSharedMemorySize,  \
                                  (int)smem)) != cudaSuccess)                                   \
      return e;                                                                                 \
    topk_kernel<NTT><<<grid, NTT, smem, st>>>(P, bf, out_idx, from_scores ? 1 : 0, staged);      \
    return cudaGetLastError();                                                                  \
  }
  if (units <= nsm) MMSHIFT_TOPK(1024)
  MMSHIFT_TOPK(512)
#undef MMSHIFT_TOPK
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
