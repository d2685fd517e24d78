"""Host logic of the mass pass's stationary blocks (csrc/score_umma.cu).

The tensor-core mass pass holds up to 256 proxy rows per CTA: whole proxy
groups, plus the anchor rows in the last block (in the packed proxy layout
they follow the last group's rows). make_sched() picks the number of blocks
and mass_block() the rows of each. A group left out of every block has no
masses; a group in two blocks is written twice; a block of more than 256 rows
overflows the accumulator. This test compiles the two host functions (the
library source with nvcc, host side only run) and checks, over a sweep of
head ratios, group sizes and group counts, that the blocks cover every group
once and in order, end with the anchor rows, stay within 256 rows in
multiples of 16, and are as few as whole groups allow.
"""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2607_22586_gb300", "csrc")

HARNESS = r"""
#include "score_umma.cu"
#include <cstdio>
// the merge launcher lives in another translation unit of the library
namespace mmshift { cudaError_t launch_merge(const Problem&, const Buffers&, cudaStream_t) { return cudaSuccess; } }
using namespace mmshift;

int main() {
  int checked = 0;
  for (int r : {1, 2, 4, 7, 8, 16})
    for (int gs : {1, 2, 4, 8, 16, 32, 64, 128, 256})
      for (int G : {0, 1, 2, 3, 5, 8, 16, 31, 32, 64}) {
        Problem P;
        memset(&P, 0, sizeof(P));
        P.G = G; P.r = r; P.RG = ((r * gs + 15) / 16) * 16; P.n_group_rows = G * P.RG;
        P.anchor_rows = ((r + 15) / 16) * 16;
        if (P.RG > SROWS) continue;          // such shapes take the CUDA-core path
        P.B = 1; P.L = 1; P.Hkv = 1; P.req[0].nsplit = 1;
        const Sched s = make_sched(P, 2);
        int g = 0, row = 0;
        for (int t = 0; t < s.ntiles; ++t) {
          const Block k = mass_block(P, s, t);
          if (k.g0 != g || k.row0 != row || k.ng < 0 || k.rows <= 0 || k.rows > SROWS || k.rows % 16 ||
              k.rows != k.ng * P.RG + (k.anchor ? P.anchor_rows : 0) || k.anchor != (t == s.ntiles - 1)) {
            std::printf("FAIL block r=%d gs=%d G=%d t=%d\n", r, gs, G, t);
            return 1;
          }
          g += k.ng;
          row += k.rows;
        }
        if (g != G || row != P.n_group_rows + P.anchor_rows) {
          std::printf("FAIL cover r=%d gs=%d G=%d\n", r, gs, G);
          return 1;
        }
        // fewest blocks: with one block less, whole groups plus the anchor rows do not fit
        const int per_block = SROWS / P.RG, per_last = (SROWS - P.anchor_rows) / P.RG;
        if (s.ntiles > 1 && (s.ntiles - 2) * per_block + per_last >= G) {
          std::printf("FAIL fewest r=%d gs=%d G=%d\n", r, gs, G);
          return 1;
        }
        ++checked;
      }
  std::printf("checked %d\n", checked);
  // the benchmark shapes: r = 7 and 8, 16 proxies per group, G = 32 and 2
  for (int r : {7, 8})
    for (int G : {32, 2}) {
      Problem P;
      memset(&P, 0, sizeof(P));
      P.G = G; P.r = r; P.RG = r * 16; P.n_group_rows = G * P.RG; P.anchor_rows = 16;
      P.B = 1; P.L = 1; P.Hkv = 1; P.req[0].nsplit = 1;
      const Sched s = make_sched(P, 2);
      std::printf("r%dG%d", r, G);
      for (int t = 0; t < s.ntiles; ++t) std::printf(" %d", mass_block(P, s, t).rows);
      std::printf("\n");
    }
  return 0;
}
"""


@pytest.fixture(scope="module")
def output(tmp_path_factory):
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(nvcc):
        pytest.skip("nvcc not found")
    d = tmp_path_factory.mktemp("mass_layout")
    src, exe = d / "harness.cu", d / "harness"
    src.write_text(HARNESS)
    subprocess.run([nvcc, "-std=c++17", "-O1", "-gencode", "arch=compute_103a,code=sm_103a",
                    "--expt-relaxed-constexpr", "-I", CSRC, "-I", os.path.join(ROOT, "include"),
                    str(src), "-o", str(exe)], check=True, capture_output=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True)
    assert out.returncode == 0, out.stdout[-2000:]
    return out.stdout


def test_blocks_cover_groups_once_and_fit(output):
    checked = int(output.split("checked ")[1].split()[0])
    assert checked > 400


def test_benchmark_shapes(output):
    lines = dict(line.split(" ", 1) for line in output.strip().split("\n")[1:])
    assert lines["r7G32"] == " ".join(["224"] * 15 + ["240"])    # anchor on the last of 16 blocks
    assert lines["r7G2"] == "240"
    assert lines["r8G32"] == " ".join(["256"] * 15 + ["128", "144"])
    assert lines["r8G2"] == "128 144"                            # no anchor-only block
