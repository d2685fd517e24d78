// Work lists of the persistent scoring kernels (host side, plain C++).
//
// The scoring passes split their work into units (layer, request, KV head,
// key split, stationary proxy block). A "split row" is one key split of one
// (layer, request, KV head) over all T stationary blocks; there are R split
// rows, so T * R units. A worker (a CTA, or a CTA pair) processes units one
// block at a time; workers that hold the same block range read the same K
// tiles, so teams of one worker per block that walk the same split rows read
// each K tile from DRAM once and from L2 for the rest of the team.
//
// With C workers and C not a multiple of T, whole teams alone leave C mod T
// workers idle. balance_workers() then gives every worker an explicit list:
// nt = C / T teams take L = ceil(R * T / C) split rows each, and the other
// E = C - nt * T workers share the rest -- the split rows [nt * L, R) of every
// block -- in equal parts of a block-by-block walk. Adjacent parts meet at
// the same integer position, so each unit is taken exactly once.
#ifndef MMSHIFT_WORK_LISTS_H_
#define MMSHIFT_WORK_LISTS_H_

#include <stdint.h>

#include <algorithm>

namespace mmshift {

constexpr int kMaxWorkers = 160;  // workers that can hold their own list
constexpr int kMaxSeg = 4;        // segments per list (block switches of a worker)

// Split rows [bt >> 8, e) of stationary block bt & 255.
struct PackedSeg {
  int32_t bt, e;
};

// nworkers == 0: no lists (whole teams of T workers, team j = workers
// [j * T, (j + 1) * T), worker w on block w % T, the teams splitting the R
// split rows evenly). Otherwise worker w takes its nseg[w] segments in turn.
struct WorkLists {
  int32_t nworkers;
  int32_t nseg[kMaxWorkers];
  PackedSeg seg[kMaxWorkers][kMaxSeg];
};

// Fills `wl` for T blocks, R split rows and C workers. Returns false (and
// nworkers = 0) where whole teams already use every worker, where they do as
// well as the lists, where there are more blocks than workers, where the
// packed segments cannot hold the sizes, or where a list would need more
// than kMaxSeg segments.
inline bool balance_workers(WorkLists& wl, int T, int R, int C) {
  wl.nworkers = 0;
  if (T < 1 || T > 256 || R < 1 || R >= (1 << 23) || C > kMaxWorkers || C < T) return false;
  const int nt = C / T, E = C - nt * T;
  if (E == 0) return false;
  int L = (int)(((long long)R * T + C - 1) / C);
  if ((long long)L * nt > R) L = R / nt;
  int w = 0;
  for (int j = 0; j < nt; ++j)
    for (int t = 0; t < T; ++t, ++w) {
      wl.nseg[w] = L > 0 ? 1 : 0;
      wl.seg[w][0] = PackedSeg{(j * L) << 8 | t, (j + 1) * L};
    }
  // the rest, block by block: block t's split rows [b0, R) are the positions
  // [t * rest, (t + 1) * rest) of the walk; worker k takes [k * Wr / E,
  // (k + 1) * Wr / E)
  const int b0 = nt * L, rest = R - b0;
  const long long Wr = (long long)rest * T;
  long long worst = L;
  for (int k = 0; k < E; ++k, ++w) {
    const long long lo = Wr * k / E, hi = Wr * (k + 1) / E;
    int n = 0;
    for (int t = 0; t < T; ++t) {
      const long long a = std::max(lo, (long long)t * rest);
      const long long z = std::min(hi, (long long)(t + 1) * rest);
      if (z <= a) continue;
      if (n == kMaxSeg) return false;
      wl.seg[w][n++] = PackedSeg{(int)(b0 + a - (long long)t * rest) << 8 | t,
                                 (int)(b0 + z - (long long)t * rest)};
    }
    wl.nseg[w] = n;
    worst = std::max(worst, hi - lo);
  }
  // keep the whole teams unless the lists shorten the longest worker
  const int nt_plain = std::max(1, std::min(C / T, R));
  if (worst >= (R + nt_plain - 1) / nt_plain) return false;
  wl.nworkers = C;
  return true;
}

}  // namespace mmshift

#endif  // MMSHIFT_WORK_LISTS_H_
