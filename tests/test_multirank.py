"""Host-side logic of bench.py's multi-rank path, on CPU with gloo (world size 2).

Each rank runs its own parameter shard; the only inter-rank operations are
the host-side barrier and the max over ranks of the timed region, which is
what these tests exercise.
"""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    import sys
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    import bench
    import workloads as W
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        r, w, local = bench.dist_env()
        assert (r, w, local) == (rank, world, rank)
        dist.barrier()
        mine = 1.0 + rank            # rank 1 is the slower one
        slowest = bench.max_over_ranks(mine, world)
        hp = bench.shard_hparams(W.WORKLOADS["gpt2s"].hp, rank)
        value = bench.whole_job_value(W.WORKLOADS["gpt2s"].d, world, 10, slowest)
        q.put((rank, slowest, hp.seed, value))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_time_and_distinct_shards():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    out = sorted(q.get(timeout=10) for _ in range(world))
    import workloads as W
    d = W.WORKLOADS["gpt2s"].d
    for rank, slowest, seed, value in out:
        assert slowest == 2.0                       # max over ranks
        assert seed == W.WORKLOADS["gpt2s"].hp.seed + rank
        assert value == pytest.approx(2 * d * 10 / 2.0)
    assert out[0][2] != out[1][2]                   # each rank its own inputs


def test_single_rank_is_unchanged():
    import bench
    assert bench.max_over_ranks(3.5, 1) == 3.5
    assert bench.whole_job_value(100, 1, 4, 2.0) == 200.0
