"""Multi-rank logic of bench.py on CPU: two gloo ranks (one replica per GPU in the real run,
weak scaling, no data-path collective): the job time is the max over ranks and the whole-job
rate counts every rank's units."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, ws, port, q):
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port), "RANK": str(rank),
                       "WORLD_SIZE": str(ws), "LOCAL_RANK": str(rank)})
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    got_ws, got_rank = bench._dist()
    vals = bench.max_over_ranks([1.0 + rank, 10.0 - rank, 3.5], got_ws)
    dist.barrier()
    dist.destroy_process_group()
    q.put((got_rank, got_ws, vals))


def test_two_gloo_ranks_take_the_max_and_count_all_units():
    ws, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, ws, port, q)) for r in range(ws)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in range(ws))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[0] for r in res] == [0, 1] and all(r[1] == 2 for r in res)
    for _, _, vals in res:
        assert vals == [2.0, 10.0, 3.5]


def test_whole_job_rate_is_weak_scaling():
    import bench
    assert bench.whole_job_rate(25_000_000, 1, 20.0) == pytest.approx(1.25e9)
    assert bench.whole_job_rate(25_000_000, 4, 20.0) == pytest.approx(5.0e9)
    assert bench.max_over_ranks([3.0, 4.0], 1) == [3.0, 4.0]
