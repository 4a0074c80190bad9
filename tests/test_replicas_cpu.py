"""The multi-GPU path of the bench is N independent replicas (the step does not
shard): its only collectives are the barriers and the maximum of the ranks'
times, and the reference arm runs on rank 0 alone. Checked here with two gloo
ranks on the CPU."""
import io
import json
import os
import socket
import sys
from contextlib import redirect_stdout
from types import SimpleNamespace

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        ms = [12.0, 20.0][rank]                   # the ranks' own timed regions
        dist.barrier()
        ms_max = bench.max_over_ranks(ms, world, "cpu")
        rate = bench.aggregate_rate(32, world, ms_max)
        buf = io.StringIO()
        args = SimpleNamespace(workload="tiny", steps=1, warmup=0, gpus=world)
        with redirect_stdout(buf):
            bench.run_reference(args, rank, world)
        dist.barrier()
        out.put((rank, ms_max, rate, buf.getvalue()))
    finally:
        dist.destroy_process_group()


def test_two_replicas_take_the_slowest_rank_and_rank0_reports():
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    res = {}
    for _ in range(2):
        r, ms_max, rate, text = out.get(timeout=600)
        res[r] = (ms_max, rate, text)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for r in (0, 1):
        assert res[r][0] == pytest.approx(20.0)                 # the slower rank's time
        assert res[r][1] == pytest.approx(2 * 32 / 0.020)       # all ranks' steps / that time
    assert res[1][2] == ""                                      # the reference arm: rank 0 only
    line = json.loads(res[0][2].strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["value"] > 0 and line["e2e"]["value"] == line["value"]
