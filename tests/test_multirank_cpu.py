"""The bench's N > 1 path on CPU: two gloo ranks (independent replicas, weak scaling) agree on the
slowest rank's step time and report the whole job's tokens/s.  No GPU."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, ms_of_rank, out):
    import sys
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms = bench.slowest_rank_ms(ms_of_rank[rank], torch.device("cpu"))
    out[rank] = (ms, bench.whole_job_tokens_per_s(8, world, ms))
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_step():
    import torch.multiprocessing as mp
    world = 2
    ms_of_rank = [3.25, 4.5]
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_rank, args=(world, _free_port(), ms_of_rank, out), nprocs=world, join=True)
        got = dict(out)
    for r in range(world):
        ms, tps = got[r]
        assert ms == 4.5
        assert tps == pytest.approx(8 * 2 / 4.5e-3)


def test_one_rank_is_unchanged():
    import bench
    assert bench.slowest_rank_ms(2.0, torch.device("cpu")) == 2.0
    assert bench.whole_job_tokens_per_s(8, 1, 2.0) == pytest.approx(4000.0)
