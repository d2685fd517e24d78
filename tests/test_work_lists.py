"""Host logic of the scoring kernels' work lists (csrc/work_lists.h).

balance_workers() decides which (split row, stationary block) units each
persistent CTA or CTA pair of the two scoring passes processes. A unit that
no worker takes leaves group masses unwritten, and a unit taken twice races
on them, so the lists must cover every unit exactly once. This test compiles
the header with the host C++ compiler and checks that over a sweep of shapes,
together with the balance the lists promise: no worker gets more than the
longest worker of whole teams, and the ideal share is met to within one
split row.
"""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "paper_2607_22586_gb300", "csrc", "work_lists.h")

HARNESS = r"""
#include "work_lists.h"
#include <cstdio>
#include <cstring>
#include <vector>
using namespace mmshift;

// 0: lists valid (or whole teams kept); prints "T R C lists maxwork" per shape
static int check(int T, int R, int C) {
  static WorkLists wl;
  std::memset(&wl, 0xff, sizeof(wl));
  const bool ok = balance_workers(wl, T, R, C);
  if (!ok) {
    if (wl.nworkers != 0) { std::printf("nworkers not reset\n"); return 1; }
    std::printf("%d %d %d 0 0\n", T, R, C);
    return 0;
  }
  if (wl.nworkers != C) { std::printf("nworkers %d != %d\n", wl.nworkers, C); return 1; }
  std::vector<int> cnt((size_t)T * R, 0);
  long long maxw = 0;
  for (int w = 0; w < C; ++w) {
    if (wl.nseg[w] < 0 || wl.nseg[w] > kMaxSeg) { std::printf("nseg %d\n", wl.nseg[w]); return 1; }
    long long work = 0;
    for (int i = 0; i < wl.nseg[w]; ++i) {
      const int t = wl.seg[w][i].bt & 255, b = wl.seg[w][i].bt >> 8, e = wl.seg[w][i].e;
      if (t >= T || b < 0 || e > R || b >= e) { std::printf("bad segment\n"); return 1; }
      for (int r = b; r < e; ++r) cnt[(size_t)r * T + t]++;
      work += e - b;
    }
    if (work > maxw) maxw = work;
  }
  for (size_t u = 0; u < cnt.size(); ++u)
    if (cnt[u] != 1) { std::printf("unit %zu taken %d times\n", u, cnt[u]); return 1; }
  std::printf("%d %d %d 1 %lld\n", T, R, C, maxw);
  return 0;
}

int main() {
  const int Rs[] = {1, 2, 3, 7, 16, 33, 100, 257, 896, 1000, 3584, 48000};
  const int Cs[] = {1, 2, 7, 64, 75, 76, 150, 152, 160, 161};
  for (int T = 1; T <= 40; ++T)
    for (int R : Rs)
      for (int C : Cs)
        if (check(T, R, C)) { std::printf("FAIL %d %d %d\n", T, R, C); return 1; }
  return 0;
}
"""


def _compiler():
    for c in ("g++", "c++", "clang++"):
        if shutil.which(c):
            return c
    return None


@pytest.fixture(scope="module")
def sweep(tmp_path_factory):
    cxx = _compiler()
    if cxx is None:
        pytest.skip("no host C++ compiler")
    d = tmp_path_factory.mktemp("work_lists")
    src, exe = d / "harness.cpp", d / "harness"
    src.write_text(HARNESS)
    subprocess.run([cxx, "-std=c++17", "-O1", "-I", os.path.dirname(HEADER), str(src), "-o", str(exe)],
                   check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True)
    assert out.returncode == 0, out.stdout[-2000:]
    rows = {}
    for line in out.stdout.split("\n"):
        if line:
            T, R, C, lists, maxw = map(int, line.split())
            rows[(T, R, C)] = (lists, maxw)
    return rows


def test_every_unit_taken_exactly_once(sweep):
    # the harness exits non-zero on any unit taken zero or two times
    assert len(sweep) == 40 * 12 * 10
    assert sum(v[0] for v in sweep.values()) > 1000   # lists were built for many shapes


def test_lists_never_slower_than_whole_teams(sweep):
    for (T, R, C), (lists, maxw) in sweep.items():
        if not lists:
            continue
        teams = max(1, min(C // T, R))
        assert maxw < -(-R // teams), (T, R, C)          # strictly shorter longest worker
        assert maxw <= -(-R * T // C) + 1, (T, R, C)     # ideal share, within one split row


def test_no_lists_where_teams_fill_the_workers(sweep):
    for (T, R, C), (lists, _) in sweep.items():
        if C % T == 0 or C < T or C > 160:
            assert not lists, (T, R, C)


def test_benchmark_shapes_use_lists():
    # 28-layer 32K stack (R = 28 * 4 * 32): the mass pass's 16 blocks over 152
    # CTAs use lists; the softmax pass's 15 blocks over 76 pairs would need 15
    # block switches for the one spare pair and keep whole teams. 72B-class
    # batch (R = 80 * 8 * 75): 17 blocks over 76 pairs and over 152 CTAs.
    cxx = _compiler()
    if cxx is None:
        pytest.skip("no host C++ compiler")
    import tempfile
    prog = r"""
#include "work_lists.h"
#include <cstdio>
using namespace mmshift;
int main() {
  static WorkLists wl;
  const int cases[][3] = {{16, 3584, 152}, {15, 3584, 76}, {17, 48000, 76}, {17, 48000, 152}};
  for (auto& c : cases) std::printf("%d ", (int)balance_workers(wl, c[0], c[1], c[2]));
  return 0;
}
"""
    with tempfile.TemporaryDirectory() as d:
        src, exe = os.path.join(d, "p.cpp"), os.path.join(d, "p")
        with open(src, "w") as f:
            f.write(prog)
        subprocess.run([cxx, "-std=c++17", "-I", os.path.dirname(HEADER), src, "-o", exe], check=True)
        out = subprocess.run([exe], capture_output=True, text=True, check=True).stdout.split()
    assert out == ["1", "0", "1", "1"]
