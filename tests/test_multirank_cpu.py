"""The multi-rank path of bench.py on the CPU: two gloo ranks on 127.0.0.1.

The decode path shards by sequence (each rank runs its own replica of the
layer, no collective on the data path); the only cross-rank steps are the
timing reductions, which these tests run as real two-process all-reduces."""
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    if ROOT not in sys.path:
        sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank-dependent totals: the job time is the slowest rank's, the e2e rate the slowest rank's
        slow = bench.cross_rank([1.0 + rank, 10.0 - rank], "max")
        fast = bench.cross_rank([3.0 + rank], "min")
        out.put((rank, slow, fast))
    finally:
        dist.destroy_process_group()


def test_cross_rank_reductions_two_gloo_ranks():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(out.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, slow, fast in res:
        assert slow == [2.0, 10.0]          # max over ranks of each total
        assert fast == [3.0]                # min over ranks


def test_cross_rank_single_process_is_identity():
    import bench
    assert bench.cross_rank([1.5, 2.5], "max") == [1.5, 2.5]


def test_job_throughput_counts_every_rank():
    import bench
    # each of 4 ranks decodes 1000 tokens; the slowest took 0.5 s
    assert bench.job_throughput(1000, 4, 0.5) == 8000.0


def test_reference_arm_prints_only_on_rank_zero(capsys, monkeypatch):
    import bench
    monkeypatch.setattr(sys, "argv", ["bench.py", "--impl", "reference", "--steps", "1", "--warmup", "0"])
    args = bench.parse()
    bench.run_reference(args, rank=1, world=2)
    assert capsys.readouterr().out == ""
