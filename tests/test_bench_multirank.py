"""bench.py's multi-process host logic on CPU: two gloo ranks (127.0.0.1).
The max-over-ranks reduction, the whole-job throughput and the rule that only
rank 0 runs and prints the reference arm."""

import io
import os
import socket
import sys
from contextlib import redirect_stdout

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    got = bench.max_over_ranks([1.0 + rank, 10.0 - rank, 5.0])
    # the reference arm: rank 0 alone runs and prints (run_reference stubbed)
    bench.run_reference = lambda args: {"impl": "reference", "rank": rank}
    sys.argv = ["bench.py", "--impl", "reference", "--gpus", str(world)]
    buf = io.StringIO()
    with redirect_stdout(buf):
        bench.main()
    dist.barrier()
    out.put((rank, got, buf.getvalue()))
    dist.destroy_process_group()


def test_two_gloo_ranks():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = {}
    for _ in range(world):
        rank, got, printed = q.get(timeout=120)
        res[rank] = (got, printed)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank in range(world):
        assert res[rank][0] == [2.0, 10.0, 5.0]            # element-wise maximum on every rank
    assert '"impl": "reference"' in res[0][1] and res[1][1] == ""


def test_job_throughput_counts_every_rank():
    import bench
    gbs1, tok1 = bench.job_throughput(2_000_000_000, 1, 1, 1, 2.0)
    gbs2, tok2 = bench.job_throughput(2_000_000_000, 1, 1, 2, 2.0)
    assert gbs1 == pytest.approx(1000.0) and tok1 == pytest.approx(500.0)
    assert gbs2 == pytest.approx(2 * gbs1) and tok2 == pytest.approx(2 * tok1)
    assert bench.max_over_ranks([3.0, 1.5]) == [3.0, 1.5]   # no process group: the values themselves
