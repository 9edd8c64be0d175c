"""The multi-GPU path's host logic, on CPU: parameter shards of one model (gloo, world size 2).

Every step of Algorithm 1 is elementwise, so G processes can each run a
contiguous range of one model's parameters with no communication on the
data path (paper_2411_17866_gb300/shard.py).  These tests check that the
shards partition the model exactly, that a shard run with its
``first_element`` computes what the whole-model run computes on that range
(both oracles), and, with two gloo ranks, that gathering the shards' states
and summing their statistics over the ranks gives the one-process run of
the whole model: states bit for bit, counts exactly, sums to rounding.
Also the benchmark's rank arithmetic (max over ranks, whole-job params/s)
and its choice of shard per rank.
"""
import dataclasses
import os
import socket

import numpy as np
import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

import workloads as W  # noqa: E402
from oracle import cxx_oracle as C  # noqa: E402
from oracle import dsm_oracle as O  # noqa: E402
from paper_2411_17866_gb300 import shard as S  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
MODEL = (W.Tensor("a", 7, W.KIND_WEIGHT, 1e-2), W.Tensor("b", 2049, W.KIND_WEIGHT, 1e-3),
         W.Tensor("c", 8, W.KIND_BIAS, 1e-3, wd=0), W.Tensor("d", 5000, W.KIND_LN_W, 1e-3),
         W.Tensor("e", 0, W.KIND_WEIGHT, 1e-3), W.Tensor("f", 4096, W.KIND_WEIGHT, 1e-2),
         W.Tensor("g", 77, W.KIND_LN_B, 1e-4), W.Tensor("h", 3333, W.KIND_WEIGHT, 1e-3))
HP = dataclasses.replace(W.HParams(), sign_mode=W.RSIGN_PM, rsign_B=0.5, grad_dtype=W.BF16, seed=9)
HP_SGDM = dataclasses.replace(W.SGDM_HP, seed=4)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _bits(a):
    return np.ascontiguousarray(a, dtype=np.float32).view(np.uint32)


@pytest.mark.parametrize("world", [1, 2, 3, 5])
def test_shards_partition_the_model(world):
    d = sum(t.numel for t in MODEL)
    starts = np.cumsum([0] + [t.numel for t in MODEL])
    covered = 0
    for r in range(world):
        sh = S.shard_layout(MODEL, world, r)
        assert sh.first_element == covered and sh.first_element % 64 == 0
        assert sum(p.numel for p in sh.pieces) == sh.count
        e = sh.first_element
        for p in sh.pieces:   # each piece is the range of its tensor it claims, with the tensor's properties
            t = MODEL[p.tensor]
            assert starts[p.tensor] + p.offset == e and 0 < p.numel and p.offset + p.numel <= t.numel
            assert (p.kind, p.grad_scale, p.wd) == (t.kind, t.grad_scale, t.wd)
            e += p.numel
        covered += sh.count
    assert covered == d


@pytest.mark.parametrize("hp", [HP, HP_SGDM], ids=["adamw-bf16-rsignpm", "sgdm-rsign0"])
@pytest.mark.parametrize("impl", ["numpy", "cxx"])
def test_shard_run_equals_the_whole_model_on_its_range(hp, impl):
    """A shard run (its pieces as the layout, first_element set) equals the whole-model run restricted to
    the shard's elements, bit for bit, over two rounds: the synthetic gradients, the initial model and the
    randomized signs are those of the whole model."""
    Run = O.OracleRun if impl == "numpy" else C.CxxOracleRun
    n, tau, world = 3, 2, 3
    for r in range(world):
        sh = S.shard_layout(MODEL, world, r)
        part = Run(sh.tensors, n, tau, hp, first_element=sh.first_element)
        whole = Run(MODEL, n, tau, hp, elems=np.arange(sh.first_element, sh.first_element + sh.count))
        for _ in range(2):
            part.run_round()
            whole.run_round()
            for a, b in ((part.x, whole.x), (part.m, whole.m), (part.opt_m[1], whole.opt_m[1])):
                assert np.array_equal(_bits(a), _bits(b))


def _rank_main(rank, world, port, q):
    import sys
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        r, w, local = bench.dist_env()
        assert (r, w, local) == (rank, world, rank)
        # the benchmark's timing arithmetic: the slowest rank's time, the whole job's parameters
        slowest = bench.max_over_ranks(1.0 + rank, world)
        value = bench.whole_job_value(W.WORKLOADS["gpt2s"].d, world, 10, slowest)
        bench_shard = bench.rank_shard(W.WORKLOADS["gpt2s"], world, rank)
        # one model over two ranks: this rank's shard, run by the oracle as the library runs it on a GPU
        n, tau = 3, 2
        sh = S.shard_layout(MODEL, world, rank)
        run = C.CxxOracleRun(sh.tensors, n, tau, HP, first_element=sh.first_element, with_stats=True)
        per_round = []
        for _ in range(2):
            run.run_round()
            mine = S.stats_by_tensor(sh, run.last_stats, len(MODEL))
            per_round.append(S.all_reduce_stats(mine))
        states = [None] * world
        dist.all_gather_object(states, (sh.first_element, run.x, run.m, run.X, run.opt_m, run.opt_v))
        q.put((rank, slowest, value, bench_shard.first_element, bench_shard.count,
               [p.tensor for p in bench_shard.pieces], per_round, states if rank == 0 else None))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_compute_one_model():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = sorted((q.get(timeout=300) for _ in range(world)), key=lambda o: o[0])
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    wl = W.WORKLOADS["gpt2s"]
    for rank, slowest, value, first, count, tensors, _, _ in out:
        assert slowest == 2.0                                   # max over ranks
        assert value == pytest.approx(2 * wl.d * 10 / 2.0)      # every rank's d parameters
        assert (first, count) == (rank * wl.d, wl.d)            # rank r holds copy r of the tensor list
        assert tensors == list(range(rank * len(wl.tensors), (rank + 1) * len(wl.tensors)))
    # the one-process run of the whole model
    whole = C.CxxOracleRun(MODEL, 3, 2, HP, with_stats=True)
    for t in range(2):
        whole.run_round()
        for rank in range(world):      # every rank holds the same reduced statistics
            got = out[rank][6][t]
            for g, w in zip(got, whole.last_stats):
                for k in S.STAT_COUNTS:
                    assert g[k] == w[k], (t, k)
                for k in S.STAT_SUMS:   # the ranks' partial sums add in another order
                    assert g[k] == pytest.approx(w[k], rel=1e-12, abs=0.0), (t, k)
    states = sorted(out[0][7], key=lambda s: s[0])
    x = np.concatenate([s[1] for s in states])
    m = np.concatenate([s[2] for s in states])
    X = np.concatenate([s[3] for s in states], axis=1)
    om = np.concatenate([s[4] for s in states], axis=1)
    ov = np.concatenate([s[5] for s in states], axis=1)
    for a, b in ((x, whole.x), (m, whole.m), (X, whole.X), (om, whole.opt_m), (ov, whole.opt_v)):
        assert np.array_equal(_bits(a), _bits(b))


def test_single_rank_is_unchanged():
    import bench
    assert bench.max_over_ranks(3.5, 1) == 3.5
    assert bench.whole_job_value(100, 1, 4, 2.0) == 200.0
    sh = bench.rank_shard(W.WORKLOADS["gpt2xl"], 1, 0)
    assert sh.first_element == 0 and sh.count == W.WORKLOADS["gpt2xl"].d
    assert [p.numel for p in sh.pieces] == [t.numel for t in W.WORKLOADS["gpt2xl"].tensors if t.numel]
