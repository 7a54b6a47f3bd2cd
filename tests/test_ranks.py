"""The N > 1 host path of bench.py on CPU: two gloo ranks (replicas) reduce their timings the
way the GPU run does (the slowest rank's time, the tokens and end-to-end rates of all)."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms, tok = bench.aggregate_ranks(100.0 + 10 * rank, 128 + rank)
    e2e = bench.sum_over_ranks(150.0 + rank)
    dist.barrier()
    dist.destroy_process_group()
    q.put((rank, ms, tok, e2e))


def test_two_gloo_ranks_aggregate_like_the_gpu_run():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, ms, tok, e2e in got:
        assert ms == 110.0          # the slowest rank's time
        assert tok == 128 + 129     # every rank's tokens
        assert e2e == 301.0         # replicas: rates add up
