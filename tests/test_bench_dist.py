"""Host logic of the multi-rank benchmark on CPU: two gloo ranks agree on
the slowest rank's time and the whole-job rate (requests are sharded by
rank, so no data-path collective exists to test)."""
import os
import socket

import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    r, w, _ = bench.dist_env()
    assert (r, w) == (rank, world)
    bench.init_dist(world, "gloo")
    bench.barrier(world)
    mx = bench.allreduce_max(1.0 + rank * 0.5, world, "cpu")
    out[rank] = (mx, bench.whole_job_rate(64 * 10, world, mx))
    import torch.distributed as dist
    dist.destroy_process_group()


def test_two_rank_gloo_aggregation():
    world = 2
    port = _free_port()
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
    assert out[0] == out[1]
    mx, rate = out[0]
    assert mx == 1.5
    assert rate == 640 * 2 / 1.5


def test_single_rank_defaults():
    for k in ("WORLD_SIZE", "RANK", "LOCAL_RANK"):
        os.environ.pop(k, None)
    assert bench.dist_env() == (0, 1, 0)
    assert bench.allreduce_max(3.0, 1, "cpu") == 3.0
    assert bench.whole_job_rate(100, 1, 2.0) == 50.0
