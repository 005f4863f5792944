"""The multi-GPU path of bench.py on CPU: two gloo ranks.  Each rank prunes
its own scenes (disjoint seeds, weak scaling, no collective on the data
path); the step time is the max over ranks and the rate is the whole job's."""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    import torch
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    seeds = bench.rank_seeds(rank)
    local_ms = 100.0 + 50.0 * rank  # the slower rank decides the job's time
    ms_max = bench.reduce_max(local_ms, dist, torch.device("cpu"))
    q.put((rank, seeds, ms_max, bench.whole_job_rate(len(seeds), world, ms_max)))
    dist.barrier()
    dist.destroy_process_group()


def test_two_ranks_shard_scenes_and_take_the_slowest_time():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    out.sort()
    seeds0, seeds1 = out[0][1], out[1][1]
    assert len(seeds0) == len(seeds1) == 32
    assert set(seeds0).isdisjoint(seeds1) and sorted(seeds0 + seeds1) == list(range(64))
    for _, _, ms_max, rate in out:
        assert ms_max == 150.0
        assert rate == pytest.approx(64 / 0.150)


def test_single_process_needs_no_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.reduce_max(12.5, None, None) == 12.5
    assert bench.rank_seeds(0)[:3] == [0, 1, 2]
