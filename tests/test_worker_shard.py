"""Worker-sharded rounds (paper_2411_17866_gb300/worker_shard.py) on CPU with gloo ranks.

Each rank holds a group of the n workers and computes with the oracle (the compute backend below):
its workers' local steps with their synthetic gradients (global worker indices), and the global step
on the parameter range it owns, from the n models that the all-to-all brings it.  After two rounds
every rank's x, every worker's model and base-optimizer state, the owners' momentum ranges and the
all-reduced statistics must equal the one-process oracle run: states bit for bit (the owner adds the
n differences in worker order 0..n-1, as one process does), counts exactly, sums to rounding.
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
from oracle import dsm_oracle as O  # noqa: E402
from paper_2411_17866_gb300 import shard as S  # noqa: E402
from paper_2411_17866_gb300 import worker_shard as WS  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
MODEL = (W.Tensor("a", 7, W.KIND_WEIGHT, 1e-2), W.Tensor("b", 2049, W.KIND_WEIGHT, 1e-3),
         W.Tensor("c", 8, W.KIND_BIAS, 1e-3, wd=0), W.Tensor("d", 5000, W.KIND_LN_W, 1e-3),
         W.Tensor("e", 4096, W.KIND_WEIGHT, 1e-2), W.Tensor("f", 333, W.KIND_LN_B, 1e-4))
CASES = {
    "adamw-bf16-rsignpm": dataclasses.replace(W.HParams(), sign_mode=W.RSIGN_PM, rsign_B=0.5, grad_dtype=W.BF16,
                                              seed=5),
    "sgdm-rsign0": dataclasses.replace(W.SGDM_HP, seed=2),
}


class OracleWorkers:
    """The compute backend of one rank, from the oracle's functions: the rank's workers are an OracleRun of
    their own (its x is the rank's copy of the global model) fed their own synthetic gradients; the owned
    range's global step is the oracle's global step on the n models of the range."""

    def __init__(self, tensors, n, tau, hp, group):
        self.hp, self.tau, self.group = hp, tau, group
        self.run = O.OracleRun(tensors, group.count, tau, hp)
        self.m_shard = None

    def local_steps(self, t):
        run = self.run
        for k in range(self.tau):
            step = t * self.tau + k
            grads = [O.synthetic_grad(run.elems, run.scale, self.hp.seed, step, self.group.first_worker + i,
                                      self.hp.grad_dtype) for i in range(self.group.count)]
            run.local_step(grads)

    def replicas(self):
        return torch.from_numpy(np.stack(self.run.X))

    def global_step(self, shard, X_shard, t):
        a, b = shard.first_element, shard.first_element + shard.count
        run, hp = self.run, self.hp
        if self.m_shard is None:
            self.m_shard = np.zeros(shard.count, dtype=np.float32)
        elems = np.arange(a, b)
        r = O.philox_uniform(elems, hp.seed, t) if hp.sign_mode != 0 else None
        x_new, m_new, inter = O.global_step(run.x[a:b], self.m_shard, [row for row in X_shard.numpy()], run.gamma,
                                            hp.g_b1, hp.g_b2, hp.g_eta, run.wd_global[a:b], hp.sign_mode,
                                            hp.rsign_B, r, run.dt)
        self.m_shard = m_new
        piece_of = np.repeat(np.arange(len(shard.pieces)), [p.numel for p in shard.pieces])
        stats = O.round_stats(inter, piece_of, len(shard.pieces), hp.sign_mode, hp.rsign_B)
        return torch.from_numpy(x_new), stats

    def restart(self, x):
        run = self.run
        run.x = x.numpy().copy()
        run.X = [run.x.copy() for _ in range(run.n)]
        run.t += 1
        run.k = 0


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, case, n, tau, q):
    import sys
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        hp = CASES[case]
        groups = WS.worker_groups(n, world)
        backend = OracleWorkers(MODEL, n, tau, hp, groups[rank])
        driver = WS.WorkerShardedRound(MODEL, n, backend)
        stats = [driver.run_round(with_stats=True) for _ in range(2)]
        run = backend.run
        q.put((rank, run.x, np.stack(run.X), np.stack(run.opt_m),
               None if run.opt_v is None else np.stack(run.opt_v), driver.shard.first_element, backend.m_shard,
               stats))
    finally:
        dist.destroy_process_group()


def test_worker_groups_and_ranges():
    for n, world in ((2, 2), (4, 2), (5, 3), (8, 8)):
        groups = WS.worker_groups(n, world)
        assert [g.first_worker for g in groups] == sorted(g.first_worker for g in groups)
        assert sum(g.count for g in groups) == n and all(g.count >= 1 for g in groups)
        assert all(groups[i].first_worker + groups[i].count == groups[i + 1].first_worker for i in range(world - 1))
    with pytest.raises(ValueError):
        WS.worker_groups(1, 2)


@pytest.mark.parametrize("case,n,world", [("adamw-bf16-rsignpm", 4, 2), ("sgdm-rsign0", 2, 2),
                                          ("adamw-bf16-rsignpm", 3, 3)],
                         ids=["adamw-n4-two-ranks", "sgdm-one-worker-per-rank", "adamw-three-ranks"])
def test_worker_sharded_rounds_equal_one_process(case, n, world):
    tau = 2
    port = _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, case, n, tau, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = sorted((q.get(timeout=300) for _ in range(world)), key=lambda o: o[0])
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    hp = CASES[case]
    whole = O.OracleRun(MODEL, n, tau, hp, with_stats=True)
    want_stats = []
    for _ in range(2):
        whole.run_round()
        want_stats.append(whole.last_stats)

    def bits(a):
        return np.ascontiguousarray(a, dtype=np.float32).view(np.uint32)

    groups = WS.worker_groups(n, world)
    m = np.zeros_like(whole.m)
    for rank, x, X, om, ov, first, m_shard, stats in out:
        g = groups[rank]
        assert np.array_equal(bits(x), bits(whole.x)), rank
        assert np.array_equal(bits(X), bits(np.stack(whole.X[g.first_worker:g.first_worker + g.count]))), rank
        assert np.array_equal(bits(om), bits(np.stack(whole.opt_m[g.first_worker:g.first_worker + g.count]))), rank
        if ov is not None:
            assert np.array_equal(bits(ov), bits(np.stack(whole.opt_v[g.first_worker:g.first_worker + g.count])))
        m[first:first + m_shard.size] = m_shard
        for t in range(2):
            for got, want in zip(stats[t], want_stats[t]):
                for k in S.STAT_COUNTS:
                    assert got[k] == want[k], (rank, t, k)
                for k in S.STAT_SUMS:
                    assert got[k] == pytest.approx(want[k], rel=1e-12, abs=0.0), (rank, t, k)
    assert np.array_equal(bits(m), bits(whole.m))     # the owners' momentum ranges make up m
