"""The multi-rank logic of bench.py, run as two gloo ranks on the CPU.

Replicas are independent, so under torchrun the ranks split the replicas of
the one plan into contiguous ranges (strong scaling, no data-path collective)
and meet only to take the slowest rank's time.  Checked here: the ranks'
ranges cover the plan exactly once and each rank's replicas are the plan's
(same traces, seeds and parameters), the timing reduction is the maximum over
ranks, and a rank other than 0 prints nothing.
"""
import contextlib
import io
import json
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank: int, world: int, port: int, out_dir: str):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        p, lo, hi = bench._plan("grid", rank, world, n_req=50)
        # rank r's step time is r + 1 ms, its end-to-end time 10 - r s
        ms, e2e = bench._max_over_ranks([rank + 1.0, 10.0 - rank], "cpu")
        buf = io.StringIO()
        with contextlib.redirect_stdout(buf):
            if rank != 0:
                bench.run_reference(type("A", (), {"steps": 1, "warmup": 0, "workload": "tiny"})())
        rec = {"range": [lo, hi],
               "reps": [(p.trace_seeds[r.trace], r.seed, r.C, r.policy, r.omega, r.tau, r.n_req)
                        for r in p.replicas],
               "max": [ms, e2e], "printed": buf.getvalue()}
        with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
            json.dump(rec, f)
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_shard_replicas_and_take_max_time(tmp_path):
    mp = pytest.importorskip("torch.multiprocessing")
    world = 2
    port = _free_port()
    ctx = mp.get_context("spawn")
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, str(tmp_path)))
             for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=180)
    for p in procs:
        if p.is_alive():
            p.kill()
    assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
    r0 = json.loads((tmp_path / "rank0.json").read_text())
    r1 = json.loads((tmp_path / "rank1.json").read_text())
    # the ranks' ranges partition the plan, and hold exactly its replicas
    sys.path.insert(0, ROOT)
    from paper_2606_17081_gb300 import workloads as wk
    full = wk.plan("grid", n_req=50)
    assert r0["range"][0] == 0 and r0["range"][1] == r1["range"][0]
    assert r1["range"][1] == len(full.replicas) and r0["range"][1] > 0
    want = [[full.trace_seeds[r.trace], r.seed, r.C, r.policy, r.omega, r.tau, r.n_req]
            for r in full.replicas]
    assert [list(x) for x in r0["reps"] + r1["reps"]] == want
    # the reported times are the slowest rank's
    assert r0["max"] == r1["max"] == [2.0, 10.0]
    # the reference arm prints only on rank 0
    assert r1["printed"] == ""


def test_profiling_subsets():
    # --replicas N keeps the plan's first N replicas; per-trace keeps the
    # first replica of every trace (one hash launch over every trace)
    import bench
    from paper_2606_17081_gb300 import workloads as wk
    full = wk.plan("grid", n_req=50)
    assert bench._subset(full, "5") == [0, 1, 2, 3, 4]
    idx = bench._subset(full, "per-trace")
    assert len(idx) == len(full.trace_seeds)
    assert sorted({full.replicas[k].trace for k in idx}) == list(range(len(full.trace_seeds)))
    p, lo, hi = bench._plan("grid", n_req=50, subset="per-trace")
    assert (lo, hi) == (0, len(idx)) and len(p.trace_seeds) == len(idx)


def test_profile_commands_are_bench_options():
    # every bench command a profile summary gives parses with the bench's
    # own options, and its replica subset selects replicas of the plan
    import glob
    import re
    import shlex
    import bench
    from paper_2606_17081_gb300 import workloads as wk
    cmds = []
    for md in glob.glob(os.path.join(ROOT, "profiles", "*.md")):
        text = open(md).read().replace("\\\n", " ")
        cmds += [m.group(1) for m in re.finditer(r"python bench\.py([^\n]*)", text)]
    assert cmds
    for cmd in cmds:
        args = bench.arg_parser().parse_args(shlex.split(cmd))
        if args.replicas is not None:
            full = wk.plan(args.workload, n_req=50)
            idx = bench._subset(full, args.replicas)
            assert idx and max(idx) < len(full.replicas)
