"""bench.py under torchrun runs one independent replica per GPU (the path does
not shard: "replicas only"); the job's line takes the slowest rank's times and
the sum of all ranks' tokens.  This checks that aggregation with two gloo ranks
on the CPU."""
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank: int, world: int, port: int, out):
    import torch
    import torch.distributed as dist

    sys.path.insert(0, ROOT)
    import bench

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank r: ms, tokens, e2e_s, generated, verify_ms
        mine = torch.tensor([10.0 + rank, 7.0 * (rank + 1), 2.0 - rank, 3.0 + rank, 1.5 + 0.5 * rank],
                            dtype=torch.float64)
        job = bench.combine_rank_stats(mine, world, "cpu")
        out[rank] = [float(x) for x in job]
    finally:
        dist.destroy_process_group()


def test_two_rank_aggregation():
    torch = pytest.importorskip("torch")
    mp = torch.multiprocessing.get_context("spawn")
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        procs = [mp.Process(target=_rank, args=(r, 2, port, out)) for r in range(2)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(120)
            assert p.exitcode == 0
        res = dict(out)
    # max over ranks for times, sum for counts; every rank sees the job's values
    want = [11.0, 7.0 + 14.0, 2.0, 3.0 + 4.0, 2.0]
    assert res[0] == want and res[1] == want


def test_single_rank_is_identity():
    torch = pytest.importorskip("torch")
    sys.path.insert(0, ROOT)
    import bench

    mine = torch.tensor([1.0, 2.0, 3.0, 4.0, 5.0], dtype=torch.float64)
    assert bench.combine_rank_stats(mine, 1, "cpu").tolist() == mine.tolist()
