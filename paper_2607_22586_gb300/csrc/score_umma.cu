// Steps 2-4 on the 5th-generation tensor cores (tcgen05 + TMA + TMEM), bf16:
// proxy logits, row softmax over the whole prompt and group-mass aggregation
// (Section 3.2.2; Appendix B). Two persistent, warp-specialised kernels of
// 576 threads, one CTA per SM:
//   warp 0      TMA producer (stationary proxy rows, a ring of K tiles);
//   warp 1      TMEM allocator and MMA issuer (one thread);
//   warps 2-17  epilogue (four warpgroups): tcgen05.ld of the accumulators,
//               exp2 and reductions in registers, outputs to global memory.
// Work units are (layer, request, KV head, key split of 1024 keys, proxy
// block). Teams of one CTA (softmax: one CTA pair) per proxy block walk
// contiguous ranges of key splits, so the team reads each K tile together
// (DRAM once, then L2) and a stationary block changes only with the (layer,
// request, head). Where the SMs are not a multiple of the blocks, the teams
// take a little less and the CTAs left over share the teams' remaining
// splits block by block (work lists, below), so no SM idles. The split
// boundaries (and so the merge order of the softmax partials) are those of
// the CUDA-core path.
//
// Softmax pass (softmax_pair_kernel): CTA pairs and 2-SM MMAs, below. The
//   accumulator lane is a proxy row, so each thread keeps its row's running
//   (max, sum of exp2) without any cross-thread reduction. Each split starts
//   from the max of its first 32-key chunk; after that the max is only raised
//   when a chunk's sum would exceed 2^100, so the common path is one FFMA, one
//   MUFU.EX2 and one FADD per logit (packed in pairs). Every split's partials
//   start afresh and land in fixed slots, so a split's results are the same
//   whichever CTA runs it: a stack of layers in one call gives the same bits
//   as the layers called one by one.
// Mass pass (mass_umma_kernel): K tile = M operand (128 keys), stationary =
//   up to 256 proxy rows holding whole groups as the N operand; the
//   accumulator lane is a key, so each thread sums exp2(x - c_row) over the
//   columns of a group in registers and writes one group mass per key
//   (coalesced along keys).
// Every wait is bounded; a CTA that gives up raises the timeout status bit and
// stops issuing work. Before it frees its tensor memory and exits, its
// producer waits (bounded) for every TMA load it armed and its MMA issuer for
// every MMA it issued, so no copy or MMA lands in memory the CTA gave back.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <mutex>

#include "common.cuh"
#include "umma.cuh"
#include "work_lists.h"

namespace mmshift {
namespace {

using namespace umma;

constexpr int BK = 128;          // keys per K tile
constexpr int SROWS = 256;       // stationary proxy rows per block
constexpr int NSTAGE = 4;        // K-tile ring depth
constexpr int NTHREADS = 576;
constexpr int EPI_WARP0 = 2;
constexpr int NEPI = 512;        // epilogue threads: 4 warpgroups
constexpr int TMEM_COLS = 512;
constexpr int ACC_STRIDE = 256;  // TMEM columns per accumulator buffer

struct Sched {
  int32_t uoff[MMSHIFT_MAX_BATCH + 1];  // per-layer units, prefix over requests
  int32_t ntiles;                        // stationary blocks per (request, KV head)
  int32_t units;                         // total units of the launch
  int32_t last_groups;                   // mass pass: groups of the last block (see mass_block)
  // per-worker lists (work_lists.h); a worker is a CTA (mass pass) or a CTA
  // pair (softmax pass)
  WorkLists wl;
};

// A worker's walk over its list, one split row at a time. The plain team
// schedule is resolved once: a = the worker's first split row, c = its
// block. A list is followed segment by segment: c = current segment, a =
// split rows of the worker before it. LISTS (a template argument of both
// kernels) selects the list form at compile time, so the plain-team kernels
// carry no list walk.
struct Walk {
  int n;      // split rows of the worker
  int a, c;
};

template <bool LISTS>
__device__ __forceinline__ Walk walk_begin(const Sched& S, int w, int nw) {
  Walk k;
  if (LISTS) {
    k.n = 0;
    for (int i = 0; i < S.wl.nseg[w]; ++i) k.n += S.wl.seg[w][i].e - (S.wl.seg[w][i].bt >> 8);
    k.a = 0;
    k.c = 0;
  } else {
    const int nteams = nw / S.ntiles, team = w / S.ntiles;
    const int rows = S.units / S.ntiles;
    k.a = (int)((long long)team * rows / nteams);
    k.n = (int)((long long)(team + 1) * rows / nteams) - k.a;
    k.c = w % S.ntiles;
  }
  return k;
}

// Unit index of the worker's i-th split row; i grows by one per call.
template <bool LISTS>
__device__ __forceinline__ int walk_unit(const Sched& S, int w, Walk& k, int i) {
  if (!LISTS) return (k.a + i) * S.ntiles + k.c;
  for (;;) {
    const PackedSeg p = S.wl.seg[w][k.c];
    const int b = p.bt >> 8, len = p.e - b;
    if (i - k.a < len) return (b + i - k.a) * S.ntiles + (p.bt & 255);
    k.a += len;
    ++k.c;
  }
}

struct Unit {
  int l, b, h, tile, split, t0, t1;
};

__device__ __forceinline__ Unit decode(const Problem& P, const Sched& S, int u) {
  Unit x;
  const int per_layer = S.uoff[P.B];
  x.l = u / per_layer;
  int r = u - x.l * per_layer;
  int b = 0;
  while (b + 1 < P.B && S.uoff[b + 1] <= r) ++b;
  x.b = b;
  r -= S.uoff[b];
  const int ns = P.req[b].nsplit;
  x.tile = r % S.ntiles;
  r /= S.ntiles;
  x.split = r % ns;
  x.h = r / ns;
  x.t0 = x.split * P.split_len;
  x.t1 = min(P.req[b].t_len, x.t0 + P.split_len);
  return x;
}

// Rows of stationary block t of the mass pass. Blocks hold whole groups;
// the last block also holds the anchor rows (they follow the last group's
// rows in the packed layout) and takes S.last_groups groups, as many as fit
// beside them; blocks 0 .. ntiles-2 share the other groups as evenly as
// possible. A group's masses do not depend on the block it lands in.
struct Block {
  int row0, rows, g0, ng, anchor;
};

__host__ __device__ inline Block mass_block(const Problem& P, const Sched& S, int t) {
  Block k;
  if (t < S.ntiles - 1) {
    const int nb = S.ntiles - 1, rest = P.G - S.last_groups;
    const int base = rest / nb, rem = rest % nb;
    k.ng = base + (t < rem ? 1 : 0);
    k.g0 = t * base + min(t, rem);
    k.anchor = 0;
  } else {
    k.g0 = P.G - S.last_groups;
    k.ng = S.last_groups;
    k.anchor = 1;
  }
  k.row0 = k.g0 * P.RG;
  k.rows = k.ng * P.RG + (k.anchor ? P.anchor_rows : 0);
  return k;
}

__device__ __forceinline__ long long block_key(const Problem& P, const Sched& S, const Unit& x) {
  return ((long long)(x.l * P.B + x.b) * P.Hkv + x.h) * S.ntiles + x.tile;
}

template <int D>
struct Smem {
  static constexpr int CH = D / 64;                         // 128-byte K chunks
  static constexpr int STAT_BYTES = CH * SROWS * 128;
  static constexpr int STAGE_BYTES = CH * BK * 128;
  static constexpr int RING_BYTES = NSTAGE * STAGE_BYTES;
  static constexpr int CS_BYTES = (NEPI / 32) * SROWS * 4;    // per-warp normaliser copies
  static constexpr int DYN_BYTES = 1024 + STAT_BYTES + RING_BYTES + CS_BYTES;
};

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  tmem_ld16(taddr, *reinterpret_cast<float(*)[16]>(v));
  tmem_ld16(taddr + 16, *reinterpret_cast<float(*)[16]>(v + 16));
}

// Online (max, sum of exp2) update of one row over 32 logits v (columns past
// the end of the split are set to -inf beforehand by mask_tail).
// m is the running max of the log2-scaled logits, z the sum of exp2(x - m).
// The max is only raised when the chunk's sum relative to it would exceed
// 2^100 (or while it is still -inf), so the common path is FFMA + EX2 + FADD; z
// stays below 2^127 over the 32 chunks of a key split.
__device__ __noinline__ void mask_tail(float (&v)[32], int c0, int nvalid) {
#pragma unroll
  for (int j = 0; j < 32; ++j)
    if (c0 + j >= nvalid) v[j] = -INFINITY;
}

// Sum over 32 logits of exp2(v * alpha - m) into four interleaved partial
// sums (column j feeds sum j mod 4), then (s0 + s1) + (s2 + s3). The scale
// and the additions run as packed pairs.
__device__ __forceinline__ float exp2_sum32(const float (&v)[32], uint64_t al2, float m) {
  const uint64_t nm2 = pk2(-m, -m);
  uint64_t s01 = 0, s23 = 0;       // the bit pattern 0 is (+0, +0)
#pragma unroll
  for (int j = 0; j < 32; j += 4) {
    float y0, y1, y2, y3;
    upk2(ffma2(pk2(v[j], v[j + 1]), al2, nm2), y0, y1);
    upk2(ffma2(pk2(v[j + 2], v[j + 3]), al2, nm2), y2, y3);
    s01 = fadd2(s01, pk2(fast_exp2(y0), fast_exp2(y1)));
    s23 = fadd2(s23, pk2(fast_exp2(y2), fast_exp2(y3)));
  }
  float s0, s1, s2, s3;
  upk2(s01, s0, s1);
  upk2(s23, s2, s3);
  return (s0 + s1) + (s2 + s3);
}

__device__ __forceinline__ void softmax_chunk(float (&v)[32], float alpha, float& m, float& z) {
  const uint64_t al2 = pk2(alpha, alpha);
  float zc = exp2_sum32(v, al2, m);
  if (!(zc <= 1.2676506e30f)) {  // first chunk, sum above 2^100 or NaN: raise the max
    float cm = -INFINITY;
#pragma unroll
    for (int j = 0; j < 32; ++j) cm = fmaxf(cm, v[j] * alpha);
    const float mn = fmaxf(m, cm);
    if (mn == -INFINITY) {
      zc = 0.f;
    } else {
      z *= fast_exp2(m - mn);
      m = mn;
      zc = exp2_sum32(v, al2, mn);
    }
  }
  z += zc;
}

// First chunk of a split: the reference is the chunk's own max (ALU only, so
// the exponentials are evaluated once); z starts from this chunk's sum.
__device__ __forceinline__ void softmax_first(const float (&v)[32], float alpha, float& m, float& z) {
  float c0 = -INFINITY, c1 = -INFINITY;
#pragma unroll
  for (int j = 0; j < 32; j += 2) {
    c0 = fmaxf(c0, v[j] * alpha);
    c1 = fmaxf(c1, v[j + 1] * alpha);
  }
  m = fmaxf(c0, c1);
  if (m == -INFINITY) return;      // every column masked: nothing to add
  z = exp2_sum32(v, pk2(alpha, alpha), m);
}

// 16 consecutive negated row normalisers (-c) from the warp's shared-memory
// copy, as 8 packed pairs.
__device__ __forceinline__ void load_nc16(const float* nc, uint64_t (&ncv)[8]) {
  const ulonglong2* c2 = reinterpret_cast<const ulonglong2*>(nc);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const ulonglong2 t = c2[i];
    ncv[2 * i] = t.x; ncv[2 * i + 1] = t.y;
  }
}

// a01 += (e_j, e_j+1), a23 += (e_j+2, e_j+3) over 16 columns, e_j =
// exp2(v_j * alpha - c_j): column j feeds partial sum j mod 4.
__device__ __forceinline__ void mass_chunk(const float (&v)[16], const uint64_t (&ncv)[8],
                                           uint64_t al2, uint64_t& a01, uint64_t& a23) {
#pragma unroll
  for (int j = 0; j < 16; j += 4) {
    float y0, y1, y2, y3;
    upk2(ffma2(pk2(v[j], v[j + 1]), al2, ncv[j / 2]), y0, y1);
    upk2(ffma2(pk2(v[j + 2], v[j + 3]), al2, ncv[j / 2 + 1]), y2, y3);
    a01 = fadd2(a01, pk2(fast_exp2(y0), fast_exp2(y1)));
    a23 = fadd2(a23, pk2(fast_exp2(y2), fast_exp2(y3)));
  }
}

// Sum over the ncols (multiple of 8) accumulator columns of one group:
// sum_j exp2(acc_j * alpha - c_j), four partial sums added in a fixed order.
// nc points at the warp's shared-memory copy of the block's negated normalisers.
__device__ __forceinline__ float group_sum(uint32_t tcol, const float* nc, int ncols, float alpha) {
  const uint64_t al2 = pk2(alpha, alpha);
  uint64_t a01 = 0, a23 = 0;       // (+0, +0)
  int cc = 0;
#pragma unroll 1
  for (; cc + 32 <= ncols; cc += 32) {
    float v[32];
    uint64_t ncv[8];
    tmem_ld32(tcol + cc, v);
    load_nc16(nc + cc, ncv);
    tmem_wait_ld();
    mass_chunk(*reinterpret_cast<float(*)[16]>(v), ncv, al2, a01, a23);
    load_nc16(nc + cc + 16, ncv);
    mass_chunk(*reinterpret_cast<float(*)[16]>(v + 16), ncv, al2, a01, a23);
  }
  if (cc + 16 <= ncols) {
    float v[16];
    uint64_t ncv[8];
    tmem_ld16(tcol + cc, v);
    load_nc16(nc + cc, ncv);
    tmem_wait_ld();
    mass_chunk(v, ncv, al2, a01, a23);
    cc += 16;
  }
  if (cc < ncols) {   // an 8-column tail (the anchor rows, r <= 8)
    float v[8];
    tmem_ld8(tcol + cc, v);
    const ulonglong2* c2 = reinterpret_cast<const ulonglong2*>(nc + cc);
    const ulonglong2 n0 = c2[0], n1 = c2[1];
    tmem_wait_ld();
    float y0, y1, y2, y3;
    upk2(ffma2(pk2(v[0], v[1]), al2, n0.x), y0, y1);
    upk2(ffma2(pk2(v[2], v[3]), al2, n0.y), y2, y3);
    a01 = fadd2(a01, pk2(fast_exp2(y0), fast_exp2(y1)));
    a23 = fadd2(a23, pk2(fast_exp2(y2), fast_exp2(y3)));
    upk2(ffma2(pk2(v[4], v[5]), al2, n1.x), y0, y1);
    upk2(ffma2(pk2(v[6], v[7]), al2, n1.y), y2, y3);
    a01 = fadd2(a01, pk2(fast_exp2(y0), fast_exp2(y1)));
    a23 = fadd2(a23, pk2(fast_exp2(y2), fast_exp2(y3)));
  }
  float a0, a1, a2, a3;
  upk2(a01, a0, a1);
  upk2(a23, a2, a3);
  return (a0 + a1) + (a2 + a3);
}

template <int D, bool LISTS>
__global__ void __launch_bounds__(NTHREADS, 1)
    mass_umma_kernel(const __grid_constant__ CUtensorMap kmap,
                      const __grid_constant__ CUtensorMap pmap, const __grid_constant__ Problem P,
                      const __grid_constant__ Sched S, Buffers bf) {
  using SM = Smem<D>;
  extern __shared__ unsigned char smraw[];
  unsigned char* sm =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smraw) + 1023) & ~uintptr_t(1023));
  unsigned char* stat = sm;
  unsigned char* ring_buf = sm + SM::STAT_BYTES;
  float* cs_all = reinterpret_cast<float*>(ring_buf + SM::RING_BYTES);
  __shared__ uint64_t full[NSTAGE], empty[NSTAGE], sfull, sempty, tfull[2], tempty[2];
  __shared__ uint64_t drain, never;
  __shared__ uint32_t tbase;
  __shared__ int abort_flag;
  volatile int* abort_ = &abort_flag;

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  // Work list of this CTA (Sched). In a team (one CTA per stationary block)
  // all CTAs walk the same key splits (over layers, requests and heads) at the
  // same time, so each K tile comes from DRAM once and from L2 for the others;
  // a CTA reloads its stationary block only when the (layer, request, head)
  // or the block changes. The three roles walk the same list.
  const int wk = blockIdx.x;
  Walk walk = walk_begin<LISTS>(S, wk, gridDim.x);

  if (threadIdx.x == 0) {
    abort_flag = 0;
    for (int s = 0; s < NSTAGE; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(&sfull, 1);
    mbar_init(&sempty, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], NEPI / 2);   // drained by a pair of warpgroups
    }
    mbar_init(&drain, 1);
    mbar_init(&never, 1);                // nothing arrives here (test_stuck_wait)
    fence_barrier_init();
    prefetch_tmap(&kmap);
    prefetch_tmap(&pmap);
  }
  if (warp == 1) {
    tmem_alloc(&tbase, TMEM_COLS);
    tmem_relinquish();
  }
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = tbase;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0, sphase = 0;
      ArmedStages armed_k, armed_s;
      long long prev = -1;
      bool ok = true;
      for (int i = 0; i < walk.n && ok; ++i) {
        const int u = walk_unit<LISTS>(S, wk, walk, i);
        const Unit x = decode(P, S, u);
        const long long key = block_key(P, S, x);
        if (key != prev) {
          if (!mbar_wait(&sempty, sphase ^ 1u, abort_)) { ok = false; break; }
          const Block k = mass_block(P, S, x.tile);
          const int row0 = k.row0, rows = k.rows;
          mbar_expect_tx(&sfull, (uint32_t)(rows * D * 2));
          armed_s.arm(0, sphase);
          const int zc = (x.l * P.B + x.b) * P.Hkv + x.h;
          for (int c = 0; c < SM::CH; ++c)
            for (int r = 0; r < rows; r += 16)
              tma_load_3d(stat + c * SROWS * 128 + r * 128, &pmap, &sfull, c * 64, row0 + r, zc);
          sphase ^= 1u;
          prev = key;
        }
        const int kbase = P.req[x.b].tok_off;
        for (int kt = x.t0; kt < x.t1; kt += BK) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_)) { ok = false; break; }
          mbar_expect_tx(&full[stage], (uint32_t)SM::STAGE_BYTES);
          armed_k.arm(stage, phase);
          for (int c = 0; c < SM::CH; ++c)
            tma_load_3d(ring_buf + stage * SM::STAGE_BYTES + c * BK * 128, &kmap, &full[stage],
                        x.h * D + c * 64, kbase + kt, x.l);
          if (++stage == NSTAGE) { stage = 0; phase ^= 1u; }
        }
      }
      // every load issued has landed before the CTA's shared memory goes
      if (!(armed_k.drain(full) && armed_s.drain(&sfull))) *abort_ = 1;
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0, bphase = 0, sphase = 0;   // bphase: one phase bit per accumulator
      long long prev = -1;
      uint32_t idesc = 0;
      bool ok = true, issued = false;
      for (int i = 0; i < walk.n && ok; ++i) {
        const int u = walk_unit<LISTS>(S, wk, walk, i);
        const Unit x = decode(P, S, u);
        const long long key = block_key(P, S, x);
        if (key != prev) {
          if (prev != -1) mma_commit(&sempty);   // old block free once its MMAs finish
          if (!mbar_wait(&sfull, sphase, abort_)) { ok = false; break; }
          sphase ^= 1u;
          fence_after();
          idesc = idesc_bf16_f32(128, mass_block(P, S, x.tile).rows);
          prev = key;
        }
        // accumulator = parity of the tile's index within its split, so a
        // split's tiles reach the same epilogue warpgroups whatever ran before
        for (int kt = x.t0, j = 0; kt < x.t1; kt += BK, ++j) {
          const int buf = j & 1;
          if (!mbar_wait(&full[stage], phase, abort_) ||
              !mbar_wait(&tempty[buf], ((bphase >> buf) & 1u) ^ 1u, abort_)) { ok = false; break; }
          fence_after();
          const uint32_t ks_base = smem_u32(ring_buf + stage * SM::STAGE_BYTES);
          const uint32_t st_base = smem_u32(stat);
          const uint32_t dcol = tmem + (uint32_t)(buf * ACC_STRIDE);
#pragma unroll
          for (int ks = 0; ks < D / 16; ++ks) {
            const int c = ks / 4, w = ks % 4;
            const uint64_t kd = sdesc_k_sw128(ks_base + c * BK * 128 + w * 32);
            const uint64_t pd = sdesc_k_sw128(st_base + c * SROWS * 128 + w * 32);
            mma_bf16(dcol, kd, pd, idesc, ks > 0 ? 1u : 0u);
          }
          mma_commit(&empty[stage]);
          mma_commit(&tfull[buf]);
          issued = true;
          if (++stage == NSTAGE) { stage = 0; phase ^= 1u; }
          bphase ^= 1u << buf;
        }
      }
      // every MMA issued has finished before the CTA's tensor memory goes
      if (issued) {
        mma_commit(&drain);
        if (!mbar_wait_drain(&drain, 0)) *abort_ = 1;
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue
    // Warpgroups 0,1 drain accumulator 0 and 2,3 accumulator 1 (every other
    // key tile), the two warpgroups of a pair splitting the groups of the
    // stationary block; each accumulator has one fixed pair of consumers
    // that waits for each of its phases in turn.
    const int ew = warp - EPI_WARP0;      // 0..15
    const int wg = ew / 4;                // warpgroup 0..3
    const int par = wg >> 1, sub = wg & 1;  // accumulator / half of the block's groups
    const int q = warp % 4;               // TMEM lane quarter this warp may access
    const int lrow = q * 32 + lane;       // accumulator lane: a key of the tile
    const float alpha = P.alpha;
    uint32_t bphase = 0;                  // one phase bit per accumulator
    long long prev_blk = -1;
    bool ok = true;
    // test only: the first epilogue warp of CTA 0 waits on a barrier that
    // nothing arrives on, gives up after a few polls and aborts the CTA
    if (P.test_stuck_wait && blockIdx.x == 0 && ew == 0)
      ok = mbar_wait(&never, 0, abort_, kTestSpinLimit);
    for (int i = 0; i < walk.n && ok; ++i) {
      const int u = walk_unit<LISTS>(S, wk, walk, i);
      const Unit x = decode(P, S, u);
      const ReqInfo R = P.req[x.b];
      const long long key = block_key(P, S, x);
      const Block blk = mass_block(P, S, x.tile);
      const float* cv = cs_all + ew * SROWS;   // this warp's copy of the block's negated normalisers
      if (key != prev_blk) {
        const float* src = bf.cvals + (((size_t)x.l * P.B + x.b) * P.Hkv + x.h) * P.Prows_pad + blk.row0;
        __syncwarp();
        for (int i = lane; i < blk.rows; i += 32) cs_all[ew * SROWS + i] = -src[i];
        __syncwarp();
        prev_blk = key;
      }
      for (int kt = x.t0, j = 0; kt < x.t1; kt += BK, ++j) {
        const int buf = j & 1;
        if (buf != par) continue;
        const uint32_t ph = (bphase >> buf) & 1u;
        bphase ^= 1u << buf;
        if (!mbar_wait(&tfull[buf], ph, abort_)) { ok = false; break; }
        fence_after();
        const uint32_t tacc = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * ACC_STRIDE);
        const int t = kt + lrow;
        const bool valid = t < x.t1;
        const size_t col = (size_t)R.tok_off + t;
        const int ng0 = (blk.ng + 1) / 2;
        const int gb = sub == 0 ? 0 : ng0, ge = sub == 0 ? ng0 : blk.ng;
        for (int gi = gb; gi < ge; ++gi) {
          const float sm = group_sum(tacc + (uint32_t)(gi * P.RG), cv + gi * P.RG, P.RG, alpha);
          if (valid)
            bf.gmass[(((size_t)x.l * P.Hkv + x.h) * P.G + blk.g0 + gi) * P.total_T + col] = sm;
        }
        const bool my_anchor = blk.anchor && (blk.ng == 0 ? sub == 0 : sub == 1);
        if (my_anchor) {
          const int a0 = blk.ng * P.RG;
          if (P.anchor_split) {
            // no normalisers yet: the scaled logits go to alog, row by row
            // (coalesced along keys), for anchor_part_kernel / anchor_final_kernel
            float v[kMaxSplitAnchor];
            tmem_ld8(tacc + (uint32_t)a0, v);
            tmem_wait_ld();
            if (valid) {
              float* dst = bf.alog + ((size_t)x.l * P.Hkv + x.h) * P.r * P.total_T + col;
#pragma unroll
              for (int a = 0; a < kMaxSplitAnchor; ++a)
                if (a < P.r) dst[(size_t)a * P.total_T] = v[a] * alpha;
            }
          } else {
            // the r anchor rows, in 8-column steps (the padding rows up to 16
            // would add exp2(-inf) = 0)
            const float sm = group_sum(tacc + (uint32_t)a0, cv + a0, (P.r + 7) & ~7, alpha);
            if (valid)
              bf.anchor[((size_t)x.l * P.Hkv + x.h) * P.total_T + col] = sm / (float)P.r;
          }
        }
        fence_before();
        mbar_arrive(&tempty[buf]);
      }
    }
  }

  fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, TMEM_COLS);
  if (threadIdx.x == 0 && abort_flag) set_status(bf.status, kStatusTimeout);
}

// ---------------------------------------------------------------- softmax pass on CTA pairs
// Each cluster of two CTAs (a pair) owns one 256-row stationary block: the
// leader (rank 0) holds rows 0-127, the peer rows 128-255. K tiles have 256
// keys; each CTA stages 128 of them (leader keys 0-127, peer 128-255). The
// leader issues M = 256 x N = 256 pair MMAs, so per 16-deep K step each SM
// reads 4 KB of its proxy rows and 4 KB of its keys from shared memory (half
// of what a one-SM MMA pair of the same work reads); TMA completions of both
// CTAs land on the leader's barriers, and its commits arrive on both CTAs'.
// Each CTA's accumulator holds its 128 rows x 256 keys: warpgroup g drains
// keys 64g .. 64g+63 of every tile, keeping one (max, sum) partial per row,
// warpgroup and split (kUmmaPartSlots = 4 slots, merged in a fixed order).
// Every epilogue warp of both CTAs releases the accumulator on the leader's
// barrier once its tensor-memory reads have completed (tcgen05.wait::ld),
// with a relaxed arrival.
constexpr int PBK = 256;          // keys per K tile of the pair softmax pass
constexpr int PROWS = 128;        // stationary rows per CTA of a pair
constexpr int PNSTAGE = 6;        // K ring depth (each stage: 128 keys)

template <int D>
struct PairSmem {
  static constexpr int CH = D / 64;
  static constexpr int STAT_BYTES = CH * PROWS * 128;
  static constexpr int STAGE_BYTES = CH * (PBK / 2) * 128;
  static constexpr int RING_BYTES = PNSTAGE * STAGE_BYTES;
  static constexpr int DYN_BYTES = 1024 + STAT_BYTES + RING_BYTES;
};

template <int D, bool LISTS>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(NTHREADS, 1)
    softmax_pair_kernel(const __grid_constant__ CUtensorMap kmap,
                        const __grid_constant__ CUtensorMap pmap, const __grid_constant__ Problem P,
                        const __grid_constant__ Sched S, Buffers bf) {
  using SM = PairSmem<D>;
  extern __shared__ unsigned char smraw[];
  unsigned char* sm =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smraw) + 1023) & ~uintptr_t(1023));
  unsigned char* stat = sm;
  unsigned char* ring = sm + SM::STAT_BYTES;
  // full / sfull / tempty count on the leader's copies; empty / sempty /
  // tfull receive the leader's multicast commits in both CTAs
  __shared__ uint64_t full[PNSTAGE], empty[PNSTAGE], sfull, sempty, tfull[2], tempty[2];
  __shared__ uint64_t drain;
  __shared__ uint32_t tbase;
  __shared__ int abort_flag;
  volatile int* abort_ = &abort_flag;

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const uint32_t rank = cluster_rank();
  // work lists as in the one-SM kernel, one per pair
  const int wk = blockIdx.x >> 1;
  Walk walk = walk_begin<LISTS>(S, wk, gridDim.x >> 1);

  if (threadIdx.x == 0) {
    abort_flag = 0;
    for (int s = 0; s < PNSTAGE; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(&sfull, 1);
    mbar_init(&sempty, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], 2 * (NEPI / 32));   // every epilogue warp of both CTAs
    }
    mbar_init(&drain, 1);
    fence_barrier_init();
    prefetch_tmap(&kmap);
    prefetch_tmap(&pmap);
  }
  if (warp == 1) {
    tmem_alloc_pair(&tbase, TMEM_COLS);
    tmem_relinquish_pair();
  }
  fence_before();
  __syncthreads();
  cluster_sync();   // both CTAs' barriers exist before any remote arrival
  fence_after();
  const uint32_t tmem = tbase;

  if (warp == 0) {
    // ------------------------------------------------------------ producer (both CTAs)
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0, sphase = 0;
      ArmedStages armed_k, armed_s;   // the leader's barriers count both CTAs' loads
      long long prev = -1;
      bool ok = true;
      for (int i = 0; i < walk.n && ok; ++i) {
        const Unit x = decode(P, S, walk_unit<LISTS>(S, wk, walk, i));
        const long long key = block_key(P, S, x);
        if (key != prev) {
          if (!mbar_wait(&sempty, sphase ^ 1u, abort_)) { ok = false; break; }
          if (rank == 0) {
            mbar_expect_tx(&sfull, (uint32_t)(2 * PROWS * D * 2));
            armed_s.arm(0, sphase);
          }
          const uint32_t bar = mapa(smem_u32(&sfull), 0);
          const int zc = (x.l * P.B + x.b) * P.Hkv + x.h;
          const int row0 = x.tile * SROWS + (int)rank * PROWS;
          for (int c = 0; c < SM::CH; ++c)
            for (int r = 0; r < PROWS; r += 16)
              tma_load_3d_pair(stat + c * PROWS * 128 + r * 128, &pmap, bar, c * 64, row0 + r, zc);
          sphase ^= 1u;
          prev = key;
        }
        const int kbase = P.req[x.b].tok_off + (int)rank * (PBK / 2);
        for (int kt = x.t0; kt < x.t1; kt += PBK) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_)) { ok = false; break; }
          if (rank == 0) {
            mbar_expect_tx(&full[stage], (uint32_t)(2 * SM::STAGE_BYTES));
            armed_k.arm(stage, phase);
          }
          const uint32_t bar = mapa(smem_u32(&full[stage]), 0);
          for (int c = 0; c < SM::CH; ++c)
            tma_load_3d_pair(ring + stage * SM::STAGE_BYTES + c * (PBK / 2) * 128, &kmap, bar,
                             x.h * D + c * 64, kbase + kt, x.l);
          if (++stage == PNSTAGE) { stage = 0; phase ^= 1u; }
        }
      }
      // the leader waits for every load of both CTAs it armed (the pair's
      // final cluster barrier keeps the peer until then)
      if (rank == 0 && !(armed_k.drain(full) && armed_s.drain(&sfull))) *abort_ = 1;
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer (leader)
    if (lane == 0 && rank == 0) {
      int stage = 0;
      uint32_t phase = 0, bphase = 0, sphase = 0;
      long long prev = -1;
      const uint32_t idesc = idesc_bf16_f32(2 * PROWS, PBK);
      bool ok = true, issued = false;
      for (int i = 0; i < walk.n && ok; ++i) {
        const Unit x = decode(P, S, walk_unit<LISTS>(S, wk, walk, i));
        const long long key = block_key(P, S, x);
        if (key != prev) {
          if (prev != -1) mma_commit_pair(&sempty, 0x3);   // old block free once its MMAs finish
          if (!mbar_wait(&sfull, sphase, abort_)) { ok = false; break; }
          sphase ^= 1u;
          fence_after();
          prev = key;
        }
        for (int kt = x.t0, j = 0; kt < x.t1; kt += PBK, ++j) {
          const int buf = j & 1;
          if (!mbar_wait(&full[stage], phase, abort_) ||
              !mbar_wait(&tempty[buf], ((bphase >> buf) & 1u) ^ 1u, abort_)) { ok = false; break; }
          fence_after();
          const uint32_t ks_base = smem_u32(ring + stage * SM::STAGE_BYTES);
          const uint32_t st_base = smem_u32(stat);
          const uint32_t dcol = tmem + (uint32_t)(buf * PBK);
#pragma unroll
          for (int ks = 0; ks < D / 16; ++ks) {
            const int c = ks / 4, w = ks % 4;
            mma_bf16_pair(dcol, sdesc_k_sw128(st_base + c * PROWS * 128 + w * 32),
                          sdesc_k_sw128(ks_base + c * (PBK / 2) * 128 + w * 32), idesc,
                          ks > 0 ? 1u : 0u);
          }
          mma_commit_pair(&empty[stage], 0x3);
          mma_commit_pair(&tfull[buf], 0x3);
          issued = true;
          if (++stage == PNSTAGE) { stage = 0; phase ^= 1u; }
          bphase ^= 1u << buf;
        }
      }
      // every pair MMA issued has finished before either CTA's tensor memory goes
      if (issued) {
        mma_commit_pair(&drain, 0x1);
        if (!mbar_wait_drain(&drain, 0)) *abort_ = 1;
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue (both CTAs)
    const int ew = warp - EPI_WARP0;
    const int wg = ew / 4;                  // warpgroup: keys 64 wg .. of each tile
    const int q = warp % 4;                 // TMEM lane quarter this warp may access
    const int lrow = q * 32 + lane;         // accumulator lane: this CTA's proxy row
    const float alpha = P.alpha;
    const int c_lo = wg * (PBK / 4);
    const uint32_t tempty_lead[2] = {mapa(smem_u32(&tempty[0]), 0), mapa(smem_u32(&tempty[1]), 0)};
    uint32_t bphase = 0;
    bool ok = true;
    for (int i = 0; i < walk.n && ok; ++i) {
      const Unit x = decode(P, S, walk_unit<LISTS>(S, wk, walk, i));
      const ReqInfo R = P.req[x.b];
      // (reference max, sum of exp2(x - max)) of this thread's row over its
      // quarter of every tile of the split, restarted per split
      float m_run = -INFINITY, z_run = 0.f;
      bool first = true;
      for (int kt = x.t0, j = 0; kt < x.t1; kt += PBK, ++j) {
        const int buf = j & 1;
        const uint32_t ph = (bphase >> buf) & 1u;
        bphase ^= 1u << buf;
        if (!mbar_wait(&tfull[buf], ph, abort_)) { ok = false; break; }
        fence_after();
        const uint32_t tcol =
            tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * PBK + c_lo);
        const int nvalid = min(PBK, x.t1 - kt) - c_lo;
        if (nvalid >= PBK / 4) {         // every tile but the last of a short split
#pragma unroll 1
          for (int c0 = 0; c0 < PBK / 4; c0 += 32) {
            float v[32];
            tmem_ld32(tcol + c0, v);
            tmem_wait_ld();
            if (first) {
              softmax_first(v, alpha, m_run, z_run);
              first = false;
            } else {
              softmax_chunk(v, alpha, m_run, z_run);
            }
          }
        } else {
#pragma unroll 1
          for (int c0 = 0; c0 < PBK / 4; c0 += 32) {
            float v[32];
            tmem_ld32(tcol + c0, v);
            tmem_wait_ld();
            mask_tail(v, c0, nvalid);
            if (first) {
              softmax_first(v, alpha, m_run, z_run);
              first = false;
            } else {
              softmax_chunk(v, alpha, m_run, z_run);
            }
          }
        }
        fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster_relaxed(tempty_lead[buf]);
      }
      if (!ok) break;
      const int prow = x.tile * SROWS + (int)rank * PROWS + lrow;
      bf.part[((((size_t)x.l * P.Hkv + x.h) * P.total_splits + R.split_off + x.split) * kUmmaPartSlots +
               wg) * P.Prows_pad + prow] = make_float2(m_run, z_run);
    }
  }

  fence_before();
  __syncthreads();
  cluster_sync();   // no CTA leaves while the other may still reach its memory
  if (warp == 1) tmem_dealloc_pair(tmem, TMEM_COLS);
  if (threadIdx.x == 0 && abort_flag) set_status(bf.status, kStatusTimeout);
}

// ---------------------------------------------------------------- anchor rows (anchor_split)
// The anchor is the last window query's attention over the request's keys,
// averaged over the r query heads of the KV head (Section 3.2.3). With
// anchor_split the mass pass writes its logits (alog, log2 units). Then, per
// (key split, KV head, layer): anchor_part_kernel takes each anchor row's
// (max, sum of exp2(y - max)) over the split's keys (apart), and
// anchor_final_kernel merges the request's partials in split order into c_j =
// log2 sum_t exp2(y_jt) and writes anchor_t = (sum_j exp2(y_jt - c_j)) / r
// for the split's keys. All reductions run in a fixed order, so the result
// does not depend on the other requests or layers of the call.
constexpr int ANT = 256;

__device__ __forceinline__ int split_request(const Problem& P, int s) {
  int b = 0;
  while (b + 1 < P.B && P.req[b + 1].split_off <= s) ++b;
  return b;
}

// warp j: anchor row j over the split's keys, 32 keys per round
__global__ void __launch_bounds__(ANT) anchor_part_kernel(const __grid_constant__ Problem P,
                                                          Buffers bf) {
  const int s = blockIdx.x, h = blockIdx.y, l = blockIdx.z;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  if (w >= P.r) return;
  const ReqInfo R = P.req[split_request(P, s)];
  const int t0 = (s - R.split_off) * P.split_len, t1 = min(R.t_len, t0 + P.split_len);
  const float* y = bf.alog + (((size_t)l * P.Hkv + h) * P.r + w) * P.total_T + R.tok_off;
  constexpr int U = 8;
  float m = -INFINITY, z = 0.f;
  for (int base = t0; base < t1; base += U * 32) {
    float v[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int t = base + u * 32 + lane;
      v[u] = t < t1 ? y[t] : -INFINITY;
    }
    float cm = v[0];
#pragma unroll
    for (int u = 1; u < U; ++u) cm = fmaxf(cm, v[u]);
    if (cm == -INFINITY) continue;
    if (cm > m) {
      z *= fast_exp2(m - cm);       // 0 while m is still -inf
      m = cm;
    }
#pragma unroll
    for (int u = 0; u < U; ++u) z += fast_exp2(v[u] - m);
  }
  for (int off = 16; off; off >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
    const float z2 = __shfl_xor_sync(0xffffffffu, z, off);
    merge_ms(m, z, m2, z2);
  }
  if (lane == 0)
    bf.apart[(((size_t)l * P.Hkv + h) * P.total_splits + s) * kMaxSplitAnchor + w] = make_float2(m, z);
}

__global__ void __launch_bounds__(ANT) anchor_final_kernel(const __grid_constant__ Problem P,
                                                           Buffers bf) {
  const int s = blockIdx.x, h = blockIdx.y, l = blockIdx.z;
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  const ReqInfo R = P.req[split_request(P, s)];
  const int t0 = (s - R.split_off) * P.split_len, t1 = min(R.t_len, t0 + P.split_len);
  __shared__ float cs[kMaxSplitAnchor];
  if (w < P.r) {
    const float2* src =
        bf.apart + (((size_t)l * P.Hkv + h) * P.total_splits + R.split_off) * kMaxSplitAnchor + w;
    float m = -INFINITY, z = 0.f;
    for (int i = lane; i < R.nsplit; i += 32) {
      const float2 v = src[(size_t)i * kMaxSplitAnchor];
      merge_ms(m, z, v.x, v.y);
    }
    for (int off = 16; off; off >>= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
      const float z2 = __shfl_xor_sync(0xffffffffu, z, off);
      merge_ms(m, z, m2, z2);
    }
    if (lane == 0) cs[w] = m + __log2f(z);
  }
  __syncthreads();
  const float* y0 = bf.alog + ((size_t)l * P.Hkv + h) * P.r * P.total_T + R.tok_off;
  float* out = bf.anchor + ((size_t)l * P.Hkv + h) * P.total_T + R.tok_off;
  for (int t = t0 + tid; t < t1; t += ANT) {
    float sm = 0.f;
    for (int j = 0; j < P.r; ++j) sm += fast_exp2(y0[(size_t)j * P.total_T + t] - cs[j]);
    out[t] = sm / (float)P.r;
  }
}

// ---------------------------------------------------------------- host side
Sched make_sched(const Problem& P, int pass) {
  Sched s;
  memset(&s, 0, sizeof(s));
  if (pass == 1) {
    // with anchor_split the anchor rows stay out (they would fill a block alone)
    s.ntiles = (P.anchor_split ? P.n_group_rows : P.Prows_pad) / SROWS;
  } else {
    // fewest blocks of whole groups, the last one with the anchor rows
    const int per_block = SROWS / P.RG;                      // >= 1 (RG <= SROWS)
    const int per_last = (SROWS - P.anchor_rows) / P.RG;     // >= 0
    s.last_groups = min(per_last, P.G);
    s.ntiles = 1 + (P.G - s.last_groups + per_block - 1) / per_block;
  }
  int acc = 0;
  for (int b = 0; b < P.B; ++b) {
    s.uoff[b] = acc;
    acc += P.Hkv * s.ntiles * P.req[b].nsplit;
  }
  s.uoff[P.B] = acc;
  s.units = acc * P.L;
  return s;
}

int sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  return n;
}

// the scoring kernels take two tensor maps, Problem, Sched and Buffers by value
static_assert(2 * sizeof(CUtensorMap) + sizeof(Problem) + sizeof(Sched) + sizeof(Buffers) <= 32764,
              "kernel parameters above the 32,764-byte limit");

template <int D>
cudaError_t launch_d(const Problem& P, const Buffers& bf, cudaStream_t st, const void* K,
                     cudaEvent_t* ev) {
  using SM = Smem<D>;
  CUtensorMap kmap, pmap;
  const uint64_t ls = P.L > 1 ? (uint64_t)P.ls_kv : (uint64_t)P.total_T * P.Hkv * D;
  if (!make_tmap_bf16_3d(&kmap, K, (uint64_t)P.Hkv * D, (uint64_t)P.total_T, (uint64_t)P.L,
                   (uint64_t)P.Hkv * D * 2, ls * 2, BK))
    return cudaErrorInvalidValue;
  if (!make_tmap_bf16_3d(&pmap, bf.packed, D, (uint64_t)P.Prows_pad, (uint64_t)P.L * P.B * P.Hkv,
                   (uint64_t)D * 2, (uint64_t)P.Prows_pad * D * 2, 16))
    return cudaErrorInvalidValue;
  const int nsm = sm_count();
  if (nsm <= 0) return cudaErrorInvalidDevice;
  cudaError_t e;
  for (auto f : {softmax_pair_kernel<D, false>, softmax_pair_kernel<D, true>})
    if ((e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  PairSmem<D>::DYN_BYTES)) != cudaSuccess) return e;
  for (auto f : {mass_umma_kernel<D, false>, mass_umma_kernel<D, true>})
    if ((e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  SM::DYN_BYTES)) != cudaSuccess) return e;
  Sched s1 = make_sched(P, 1), s2 = make_sched(P, 2);
  if (ev && (e = cudaEventRecord(ev[1], st)) != cudaSuccess) return e;
  if (s1.units) {
    // softmax pass: workers are CTA pairs (clusters of two), one per two SMs
    const int pairs = nsm / 2;
    if (balance_workers(s1.wl, s1.ntiles, s1.units / s1.ntiles, pairs)) {
      softmax_pair_kernel<D, true><<<2 * pairs, NTHREADS, PairSmem<D>::DYN_BYTES, st>>>(
          kmap, pmap, P, s1, bf);
    } else {
      // whole teams of ntiles pairs
      const int rows = s1.units / s1.ntiles;
      const int grid_pairs = std::max(1, std::min(pairs / s1.ntiles, rows)) * s1.ntiles;
      softmax_pair_kernel<D, false><<<2 * grid_pairs, NTHREADS, PairSmem<D>::DYN_BYTES, st>>>(
          kmap, pmap, P, s1, bf);
    }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  if (ev && (e = cudaEventRecord(ev[2], st)) != cudaSuccess) return e;
  if ((e = launch_merge(P, bf, st)) != cudaSuccess) return e;
  if (ev && (e = cudaEventRecord(ev[3], st)) != cudaSuccess) return e;
  if (s2.units) {
    // mass pass: workers are CTAs, one per SM
    if (balance_workers(s2.wl, s2.ntiles, s2.units / s2.ntiles, nsm)) {
      mass_umma_kernel<D, true><<<nsm, NTHREADS, SM::DYN_BYTES, st>>>(kmap, pmap, P, s2, bf);
    } else {
      const int rows = s2.units / s2.ntiles;
      const int grid = std::max(1, std::min(nsm / s2.ntiles, rows)) * s2.ntiles;
      mass_umma_kernel<D, false><<<grid, NTHREADS, SM::DYN_BYTES, st>>>(kmap, pmap, P, s2, bf);
    }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace

static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static std::once_flag once;
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

bool make_tmap_bf16_3d(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2,
                       uint64_t stride1_bytes, uint64_t stride2_bytes, uint32_t box1) {
  auto fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[3] = {d0, d1, d2};
  const cuuint64_t strides[2] = {stride1_bytes, stride2_bytes};
  const cuuint32_t box[3] = {64, box1, 1};
  const cuuint32_t es[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool tmap_encoder_available() { return encode_fn() != nullptr; }

bool umma_supported(const Problem& P) {
  if (P.dtype != MMSHIFT_BF16 || (P.d != 64 && P.d != 128)) return false;
  if (P.RG > SROWS || P.anchor_rows > SROWS || P.Prows_pad % SROWS) return false;
  if (P.L > 1 && (P.ls_kv % 8)) return false;   // TMA strides: multiples of 16 bytes
  int dev = 0, major = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess)
    return false;
  return major == 10 && tmap_encoder_available();
}

int umma_launches(const Problem& P) { return P.anchor_split ? 5 : 3; }

// The anchor rows of an anchor_split call, after the mass pass (their own
// stage, so that the mass pass is timed alone).
cudaError_t launch_anchor_split(const Problem& P, const Buffers& bf, cudaStream_t st) {
  if (!P.anchor_split || !P.total_T) return cudaSuccess;
  anchor_part_kernel<<<dim3(P.total_splits, P.Hkv, P.L), ANT, 0, st>>>(P, bf);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  anchor_final_kernel<<<dim3(P.total_splits, P.Hkv, P.L), ANT, 0, st>>>(P, bf);
  return cudaGetLastError();
}

cudaError_t launch_score_umma(const Problem& P, const Buffers& bf, cudaStream_t st,
                              const void* K, cudaEvent_t* ev) {
  if (reinterpret_cast<uintptr_t>(K) & 15) return cudaErrorMisalignedAddress;
  return P.d == 128 ? launch_d<128>(P, bf, st, K, ev) : launch_d<64>(P, bf, st, K, ev);
}

}  // namespace mmshift
