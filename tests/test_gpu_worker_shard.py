"""Worker-sharded rounds with the library as every rank's compute (paper_2411_17866_gb300/worker_shard.py).

Each gloo rank holds a group of the n workers in a library handle on the GPU (dsm_set_first_worker places
them among the n), runs their local steps there, and computes the global step of the parameter range it
owns with dsm_global_step_noalloc; dsm_end_round restarts the workers from the gathered model.  The ranks
are processes that share one GPU: none of their kernels waits on another rank, all exchanges are gloo
collectives on host tensors.  After two rounds every rank's x, its workers' models and base-optimizer
states, the owners' momentum ranges and the all-reduced statistics must equal the one-process oracle:
states bit for bit, counts exactly.  The two calls the backend adds are checked on their own first.
"""
import dataclasses
import os
import socket
import traceback

import numpy as np
import pytest

torch = pytest.importorskip("torch")
import torch.multiprocessing as mp  # noqa: E402

import workloads as W  # noqa: E402
from oracle import dsm_oracle as O  # noqa: E402
from paper_2411_17866_gb300 import shard as S  # noqa: E402
from paper_2411_17866_gb300 import worker_shard as WS  # noqa: E402

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
MODEL = (W.Tensor("a", 7, W.KIND_WEIGHT, 1e-2), W.Tensor("b", 2049, W.KIND_WEIGHT, 1e-3),
         W.Tensor("c", 8, W.KIND_BIAS, 1e-3, wd=0), W.Tensor("d", 5000, W.KIND_LN_W, 1e-3),
         W.Tensor("e", 4096, W.KIND_WEIGHT, 1e-2), W.Tensor("f", 333, W.KIND_LN_B, 1e-4))
CASES = {
    "adamw-bf16-rsignpm": dataclasses.replace(W.HParams(), sign_mode=W.RSIGN_PM, rsign_B=0.5, grad_dtype=W.BF16,
                                              seed=5),
    "adamw-fused-sign": dataclasses.replace(W.HParams(), flags=W.FLAG_FUSED_ROUND, seed=9),
    "sgdm-rsign0": dataclasses.replace(W.SGDM_HP, seed=2),
    "adamw-reset-local": dataclasses.replace(W.HParams(), flags=W.FLAG_RESET_LOCAL_STATE, seed=4),
    "adamw-slowmo": dataclasses.replace(W.HParams(), global_mode=W.GLOBAL_SLOWMO, seed=7),
}


def bits(a):
    return np.ascontiguousarray(a, dtype=np.float32).view(np.uint32)


@pytest.fixture(scope="module")
def dsm():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2411_17866_gb300 import dsm as D
    D.load_library()
    return D


def test_first_worker_draws_those_workers_gradients(dsm):
    """dsm_set_first_worker: the handle's worker i draws the synthetic gradient of worker first_worker + i."""
    for case, first in (("adamw-bf16-rsignpm", 3), ("sgdm-rsign0", 1)):
        hp = CASES[case]
        run = dsm.DistributedSignMomentum(MODEL, 2, 1, hp)
        run.set_first_worker(first)
        run.fill_synthetic_grads(5)
        ref = O.OracleRun(MODEL, 1, 1, hp)
        for i in range(2):
            want = O.synthetic_grad(ref.elems, ref.scale, hp.seed, 5, first + i, hp.grad_dtype)
            got = run.read(dsm.BUF_GRAD, i).float().numpy()
            assert np.array_equal(bits(got), bits(want)), (case, i)
        run.close()


@pytest.mark.parametrize("case", ["adamw-bf16-rsignpm", "adamw-fused-sign", "sgdm-rsign0", "adamw-reset-local"])
def test_end_round_restarts_from_the_given_model(dsm, case):
    """dsm_end_round after the local steps leaves the handle where a handle that ran the global step itself
    is (x, replicas, base-optimizer states, round counter), and the next round's local steps agree."""
    hp = CASES[case]
    n, tau = 3, 2
    a = dsm.DistributedSignMomentum(MODEL, n, tau, hp)
    b = dsm.DistributedSignMomentum(MODEL, n, tau, hp)
    a.synthetic_round()
    for k in range(tau):
        b.fill_synthetic_grads(k)
        b.local_step()
    c = dsm.DistributedSignMomentum(MODEL, n, tau, hp)
    c.fill_synthetic_grads(0)
    c.local_step()
    with pytest.raises(dsm.DsmError) as e:   # only once the round's local steps are done
        c.end_round(a.read(dsm.BUF_X))
    assert e.value.code == dsm.DSM_ESTATE
    c.close()
    b.end_round(a.read(dsm.BUF_X))
    assert b.info().round == a.info().round == 1 and b.info().local_steps == 0
    bufs = [dsm.BUF_REPLICA, dsm.BUF_OPT_M] + ([dsm.BUF_OPT_V] if hp.base == W.BASE_ADAMW else [])
    assert np.array_equal(bits(b.read(dsm.BUF_X).numpy()), bits(a.read(dsm.BUF_X).numpy()))
    for which in bufs:
        for i in range(n):
            assert np.array_equal(bits(b.read(which, i).numpy()), bits(a.read(which, i).numpy())), (which, i)
    for run in (a, b):
        for k in range(tau):
            run.fill_synthetic_grads(tau + k)
            run.local_step()
    for which in bufs:
        for i in range(n):
            assert np.array_equal(bits(b.read(which, i).numpy()), bits(a.read(which, i).numpy())), (which, i)
    a.close()
    b.close()


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, case, n, tau, q):
    import sys
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import torch.distributed as dist
    from paper_2411_17866_gb300 import dsm as D
    try:
        dist.init_process_group("gloo", rank=rank, world_size=world)
        try:
            hp = CASES[case]
            groups = WS.worker_groups(n, world)
            shard = S.shard_layout(MODEL, world, rank)
            backend = WS.LibraryWorkers(MODEL, n, tau, hp, groups[rank], shard, device="cuda:0")
            driver = WS.WorkerShardedRound(MODEL, n, backend)
            stats = [driver.run_round(with_stats=True) for _ in range(2)]
            run = backend.run
            X = np.stack([run.read(D.BUF_REPLICA, i).numpy() for i in range(run.n)])
            om = np.stack([run.read(D.BUF_OPT_M, i).numpy() for i in range(run.n)])
            ov = np.stack([run.read(D.BUF_OPT_V, i).numpy() for i in range(run.n)]) if hp.base == W.BASE_ADAMW \
                else None
            q.put((rank, run.read(D.BUF_X).numpy(), X, om, ov, shard.first_element, backend.momentum().numpy(),
                   stats))
            run.close()
        finally:
            dist.destroy_process_group()
    except Exception:
        q.put((rank, "error", traceback.format_exc()))


@pytest.mark.parametrize("case,n,world", [("adamw-bf16-rsignpm", 4, 2), ("sgdm-rsign0", 2, 2),
                                          ("adamw-fused-sign", 3, 3), ("adamw-slowmo", 4, 2)],
                         ids=["adamw-n4-two-ranks", "sgdm-one-worker-per-rank", "fused-flag-three-ranks",
                              "slowmo-two-ranks"])
def test_worker_sharded_rounds_on_the_gpu_equal_one_process(dsm, case, n, world):
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
    errors = [o[2] for o in out if isinstance(o[1], str)]
    assert not errors, errors[0]
    assert all(p.exitcode == 0 for p in procs)
    hp = CASES[case]
    whole = O.OracleRun(MODEL, n, tau, hp, with_stats=True)
    want_stats = []
    for _ in range(2):
        whole.run_round()
        want_stats.append(whole.last_stats)
    groups = WS.worker_groups(n, world)
    m = np.zeros_like(whole.m)
    for rank, x, X, om, ov, first, m_shard, stats in out:
        g = groups[rank]
        sl = slice(g.first_worker, g.first_worker + g.count)
        assert np.array_equal(bits(x), bits(whole.x)), rank
        assert np.array_equal(bits(X), bits(np.stack(whole.X[sl]))), rank
        assert np.array_equal(bits(om), bits(np.stack(whole.opt_m[sl]))), rank
        if ov is not None:
            assert np.array_equal(bits(ov), bits(np.stack(whole.opt_v[sl]))), rank
        m[first:first + m_shard.size] = m_shard
        for t in range(2):
            for got, want in zip(stats[t], want_stats[t]):
                for k in S.STAT_COUNTS:
                    assert got[k] == want[k], (rank, t, k)
                for k in S.STAT_SUMS:
                    assert got[k] == pytest.approx(want[k], rel=(n + 4) * 2.0 ** -24, abs=1e-30), (rank, t, k)
    assert np.array_equal(bits(m), bits(whole.m))     # the owners' momentum ranges make up m
