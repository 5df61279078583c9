"""The N>1 path of bench.py on CPU: two gloo ranks, as torchrun would start them.

Each rank times a different (fake) step; the job time must be the maximum over ranks on every
rank, the whole-job rate the per-rank units times the world size over that maximum, and only
rank 0 may print a reference-arm line.
"""
import io
import json
import os
import socket
import sys
from contextlib import redirect_stdout

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port),
                       "RANK": str(rank), "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank)})
    sys.path.insert(0, ROOT)
    import bench
    d = bench.Dist()
    assert (d.rank, d.world) == (rank, world)
    d.init("gloo")
    local_s = 0.010 * (rank + 1)                 # rank r "took" 10(r+1) ms
    d.barrier()
    job_s = d.max(local_s)
    rate = bench.job_rate(1.0e9, job_s, d.world)
    buf = io.StringIO()
    with redirect_stdout(buf):
        # The reference arm does all its work on rank 0; other ranks return at once.
        if rank != 0:
            bench.reference_arm(None, d)
    d.barrier()
    d.close()
    with open(os.path.join(out_dir, "rank%d.json" % rank), "w") as f:
        json.dump({"job_s": job_s, "rate": rate, "printed": buf.getvalue()}, f)


def test_two_gloo_ranks_max_and_rate(tmp_path):
    import torch.multiprocessing as mp
    world = 2
    mp.start_processes(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world,
                       join=True, start_method="spawn")
    res = [json.load(open(tmp_path / ("rank%d.json" % r))) for r in range(world)]
    for r in res:
        assert r["job_s"] == pytest.approx(0.020)          # slowest rank
        assert r["rate"] == pytest.approx(1.0e9 * 2 / 0.020)
    assert res[1]["printed"] == ""


def test_job_rate_single():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.job_rate(3.0, 1.5, 1) == pytest.approx(2.0)
    assert bench.job_rate(3.0, 1.5, 4) == pytest.approx(8.0)
