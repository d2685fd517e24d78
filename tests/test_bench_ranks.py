"""The benchmark's multi-rank host logic on CPU: two ``gloo`` ranks started
the way torchrun starts them (environment variables, 127.0.0.1 rendezvous).

Each rank must run its own replica (different seeded inputs), meet the
others at the barriers, agree on the maximum of the per-rank step times and
report the whole-job value from it; under ``--impl reference`` only rank 0
runs and prints.
"""
import argparse
import io
import json
import os
import socket
import contextlib

import numpy as np
import torch.multiprocessing as tmp

import bench
from paper_2607_22586_gb300 import synth as S


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    ranks = bench.Ranks("gloo")
    res = {"rank": ranks.rank, "world": ranks.world}
    # replica inputs: the workload's seed offset by the rank
    wl = S.WORKLOADS["tiny-f32"].replace(n_layers=2)
    K, V, Q = bench.gen_workload(wl, ranks.rank, 1)
    res["k_sum"] = float(np.asarray(K, dtype=np.float64).sum())
    ranks.barrier()
    # per-rank step times 1.5 ms and 2.5 ms: every rank sees the slower one
    res["ms_max"] = ranks.max(1.5 + ranks.rank)
    res["value"] = bench.job_value(1000.0, ranks.world, res["ms_max"])
    # reference arm: rank 0 alone prints a line
    buf = io.StringIO()
    args = argparse.Namespace(proxies="few", steps=1, warmup=3, ref_seconds=0.0, gpus=world)
    with contextlib.redirect_stdout(buf):
        rc = bench.run_reference(args, wl.replace(n_layers=1))
    res["ref_rc"] = rc
    res["ref_out"] = buf.getvalue()
    ranks.close()
    with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
        json.dump(res, f)


def test_two_gloo_ranks(tmp_path):
    world, port = 2, _free_port()
    tmp.start_processes(_rank_main, args=(world, port, str(tmp_path)), nprocs=world, join=True,
                        start_method="spawn")
    res = [json.load(open(tmp_path / f"rank{r}.json")) for r in range(world)]
    assert [r["rank"] for r in res] == [0, 1] and all(r["world"] == 2 for r in res)
    assert res[0]["k_sum"] != res[1]["k_sum"], "ranks must run different replicas"
    assert all(r["ms_max"] == 2.5 for r in res)
    assert all(abs(r["value"] - 1000.0 * 2 / 2.5e-3) < 1e-6 for r in res)
    assert all(r["ref_rc"] == 0 for r in res)
    line = json.loads(res[0]["ref_out"].strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["cpu_baseline"]["kind"] == "oracle"
    assert line["e2e"]["h2d_bytes_per_step"] == 0
    assert res[1]["ref_out"] == "", "only rank 0 runs the reference arm"


def test_single_rank_needs_no_group():
    for k in ("WORLD_SIZE", "RANK", "LOCAL_RANK"):
        os.environ.pop(k, None)
    r = bench.Ranks("gloo")
    assert r.world == 1 and r.dist is None
    assert r.max(3.25) == 3.25
    r.barrier()
    r.close()
    assert bench.job_value(500.0, 1, 2.0) == 500.0 / 2e-3
