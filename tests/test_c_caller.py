"""The C ABI from a plain C program (no Python, no torch).

include/mmshift.h is meant for C and C++ callers that link libmmshift.so
directly. This test compiles a C11 program against the header with the host
C compiler, links it with the in-tree library and runs the host-side entry
points (defaults, output rows, workspace size, validation, status strings),
which need no GPU. It checks that the header is valid C, that the exported
names link, and that the values match the documented ones.
"""
import ctypes
import os
import shutil
import subprocess

import pytest

from paper_2607_22586_gb300 import _lib as L
from paper_2607_22586_gb300 import build as B

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

PROGRAM = r"""
#include <stddef.h>
#include <stdio.h>
#include <string.h>
#include "mmshift.h"

int main(void) {
  mmshift_params p;
  mmshift_default_params(&p);
  printf("params %d %d %.3f %.3f %.3f %d\n", p.n_proxies, p.n_groups, p.gamma, p.tau, p.lambda,
         p.score_mode);

  /* two requests of 1000 and 300 tokens, budgets 128 and 512 (the second keeps all 300) */
  const int32_t cu[3] = {0, 1000, 1300};
  const int32_t budgets[2] = {128, 512};
  mmshift_shape s;
  memset(&s, 0, sizeof(s));
  s.batch = 2; s.n_q_heads = 28; s.n_kv_heads = 4; s.head_dim = 128; s.window = 32;
  s.dtype = MMSHIFT_BF16; s.cu_seqlens = cu; s.budgets = budgets; s.n_layers = 1;
  s.layer_stride_kv = 1300 * 4 * 128; s.layer_stride_q = 2 * 32 * 28 * 128;
  int64_t rows = -1;
  mmshift_status st = mmshift_output_rows(&s, &rows);
  printf("rows %d %lld\n", (int)st, (long long)rows);
  size_t ws = 0;
  st = mmshift_workspace_size(&s, &p, &ws);
  printf("workspace %d %d\n", (int)st, ws > 0 && ws % 256 == 0);

  /* invalid shapes are refused before anything is enqueued */
  s.head_dim = 96;
  printf("bad_head_dim %d\n", (int)mmshift_workspace_size(&s, &p, &ws));
  s.head_dim = 128;
  s.window = 1;
  printf("bad_window %d\n", (int)mmshift_workspace_size(&s, &p, &ws));
  s.window = 32;
  printf("null_select %d\n", (int)mmshift_select(&s, NULL, NULL, NULL, NULL, &p, NULL, NULL, NULL,
                                                 NULL, NULL, 0, NULL));
  printf("status %s\n", mmshift_status_string(MMSHIFT_ERR_WORKSPACE));
  printf("sizes %d %d %d %d\n", (int)sizeof(mmshift_params), (int)sizeof(mmshift_shape),
         (int)sizeof(mmshift_debug), (int)offsetof(mmshift_debug, test_stuck_wait));
  return 0;
}
"""


def _cc():
    for c in ("cc", "gcc", "clang"):
        if shutil.which(c):
            return c
    return None


def test_plain_c_program_links_and_runs(tmp_path):
    cc = _cc()
    if cc is None:
        pytest.skip("no host C compiler")
    lib = B.build()
    src, exe = tmp_path / "caller.c", tmp_path / "caller"
    src.write_text(PROGRAM)
    libdir = os.path.dirname(lib)
    subprocess.run([cc, "-std=c11", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"), str(src),
                    "-o", str(exe), "-L", libdir, "-lmmshift", "-Wl,-rpath," + libdir],
                   check=True, capture_output=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout
    got = dict(line.split(" ", 1) for line in out.strip().split("\n"))
    assert got["params"] == "512 32 10.000 0.950 1.000 0"        # Section 4.1 defaults, VOTE
    assert got["rows"] == "0 428"                                  # min(128, 1000) + min(512, 300)
    assert got["workspace"] == "0 1"
    assert got["bad_head_dim"] == "2"                              # MMSHIFT_ERR_UNSUPPORTED
    assert got["bad_window"] == "1"                                # MMSHIFT_ERR_INVALID_ARG
    assert got["null_select"] == "1"
    assert got["status"].strip() != ""
    # the ctypes binding lays the structs out as the C compiler does
    assert got["sizes"] == (f"{ctypes.sizeof(L.Params)} {ctypes.sizeof(L.Shape)} "
                            f"{ctypes.sizeof(L.Debug)} {L.Debug.test_stuck_wait.offset}")
