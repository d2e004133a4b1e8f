"""World-size-2 gloo check of the benchmark's multi-rank host logic (CPU only):
max-over-ranks timing and the weak-scaling whole-job value."""
import os
import socket

import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, ws, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(ws),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    assert bench.dist_env() == (ws, rank, rank)
    ms = 2.0 + rank            # rank 1 is the slow one
    bench.barrier(ws)
    t = bench.max_over_ranks(ms, ws)
    q.put((rank, t, bench.weak_scaling_value(1e12, t, ws)))
    dist.destroy_process_group()


def test_two_rank_max_and_weak_scaling():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=10) for _ in range(2))
    for rank, t, v in got:
        assert t == 3.0                       # max over ranks
        assert abs(v - 2 * 1e12 / 3e-3 / 1e12) < 1e-9
