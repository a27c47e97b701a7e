"""The replicas-only multi-GPU plumbing of bench.py, on CPU with world-size-2 gloo ranks.

bench.py runs one independent pass per rank (no data-path collective); what the ranks share is
the barrier around the timed region, the max over ranks of the elapsed time, the sum over
ranks of the bytes moved, and rank-0-only reporting.  These are exercised here with the gloo
backend; the reference arm (the C oracle) must print one line on rank 0 and nothing elsewhere.
"""
import io
import json
import os
import socket
import sys
from contextlib import redirect_stdout

import pytest
import torch.multiprocessing as mp

from tests.conftest import ROOT


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out_q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        bench.barrier(world)
        mx = bench.max_over_ranks(world, float(rank + 1) * 1.5)
        sm = bench.sum_over_ranks(world, float(10 * (rank + 1)))
        # reference arm: rank 0 prints one JSON line, the others nothing
        sys.argv = ["bench.py", "--impl", "reference", "--gpus", str(world), "--steps", "2",
                    "--warmup", "1"]
        a = bench.parse()
        buf = io.StringIO()
        with redirect_stdout(buf):
            bench.run_reference(a, world, rank)
        out_q.put((rank, mx, sm, buf.getvalue()))
    finally:
        dist.destroy_process_group()


@pytest.fixture(scope="module")
def oracle_built():
    from oracle import build
    build.build()


def test_two_gloo_ranks(oracle_built):
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    results = sorted(q.get(timeout=240) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, mx0, sm0, out0), (r1, mx1, sm1, out1) = results
    assert mx0 == mx1 == 3.0          # max of 1.5, 3.0
    assert sm0 == sm1 == 30.0         # 10 + 20
    assert out1 == ""
    line = json.loads(out0.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["n_gpus"] == world
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["d2h_bytes_per_step"] == 0
    assert line["cpu_baseline"]["kind"] == "oracle" and line["value"] > 0
