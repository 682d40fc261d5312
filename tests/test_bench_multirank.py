"""The N > 1 host logic of bench.py on CPU: two gloo ranks, each a replica
of the workload with its own seed, time = max over ranks, value = the units
all ranks processed / that time (weak scaling, no data-path collective)."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank_main(rank, world, port, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    ws, r, local = bench.dist_env()
    my_ms = 10.0 + 5.0 * rank                     # rank 1 is the slow one
    worst = bench.max_over_ranks(my_ms)
    bench.barrier()
    rate = bench.whole_job_rate(1000.0, 4, ws, worst)
    out[rank] = (ws, r, local, bench.rank_seed(20262, r), worst, rate)
    dist.destroy_process_group()


def test_two_rank_weak_scaling_aggregation():
    world = 2
    port = _free_port()
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
    a, b = out[0], out[1]
    assert a[0] == b[0] == 2 and (a[1], b[1]) == (0, 1)
    assert a[3] != b[3], "each replica must draw its own inputs"
    assert a[4] == b[4] == 15.0, "step time is the max over ranks"
    assert a[5] == pytest.approx(1000.0 * 4 * 2 / 0.015)


def test_single_process_defaults(monkeypatch):
    import bench
    for k in ("WORLD_SIZE", "RANK", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)
    assert bench.dist_env() == (1, 0, 0)
    assert bench.max_over_ranks(3.5) == 3.5
