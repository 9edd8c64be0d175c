"""GPU kernels (through the C ABI) against the CPU oracle, element by element.

Tolerance: bit-exact.  The kernels evaluate the oracle's fp32 expression
trees one rounding at a time (no contraction), with the same worker order,
so x, m, every replica, every base-optimizer state and every gradient must
be identical bit for bit.  The statistics' sums are compared to a relative
(n + 4) * 2^-24 (derived in gpu_common.stats_rtol); their counts exactly.
"""
import dataclasses
import zlib

import numpy as np
import pytest

import workloads as W
from gpu_common import assert_bitexact, compare_state, compare_stats, sample_elements

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from oracle import dsm_oracle as O  # noqa: E402
from oracle.cxx_oracle import CxxOracleRun  # noqa: E402
from paper_2411_17866_gb300 import dsm  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    dsm.load_library()
    yield
    torch.cuda.empty_cache()


# tensors whose sizes leave ragged tails and unaligned starts, and an empty tensor
RAGGED = (W.Tensor("a", 7, W.KIND_WEIGHT, 1e-2), W.Tensor("b", 2049, W.KIND_WEIGHT, 1e-3),
          W.Tensor("c", 8, W.KIND_BIAS, 1e-3, wd=0), W.Tensor("d", 5000, W.KIND_LN_W, 1e-3),
          W.Tensor("e", 1, W.KIND_LN_B, 1e-3), W.Tensor("f", 0, W.KIND_WEIGHT, 1e-3),
          W.Tensor("g", 4096, W.KIND_WEIGHT, 1e-2), W.Tensor("h", 77, W.KIND_BIAS, 1e-4),
          W.Tensor("i", 65537, W.KIND_WEIGHT, 1e-3))
# a small GPT-2-shaped layout: every tensor a multiple of 64 elements (vector paths)
MINI = W.gpt2_layout(2, 64, 256)

ADAMW = W.HParams()
SGDM = W.SGDM_HP

CASES = [
    ("adamw-f32-n4-t3", ADAMW, 4, 3),
    ("adamw-bf16-n8-t2", dataclasses.replace(ADAMW, grad_dtype=W.BF16, seed=3), 8, 2),
    ("adamw-f32-n1-t1", ADAMW, 1, 1),
    ("adamw-f32-n3-t2", dataclasses.replace(ADAMW, seed=7), 3, 2),
    ("sgdm-rsign0-f32-n8-t2", SGDM, 8, 2),
    ("sgdm-rsignpm-bf16-n2-t3", dataclasses.replace(SGDM, sign_mode=W.RSIGN_PM, grad_dtype=W.BF16), 2, 3),
    ("sgd-plain-sign-n5-t1", dataclasses.replace(SGDM, mu=0.0, sign_mode=W.SIGN), 5, 1),
    ("adamw-rsignpm-n9-generic", dataclasses.replace(ADAMW, sign_mode=W.RSIGN_PM, rsign_B=1.0), 9, 2),
    ("sgdm-rsign0-n16-generic", dataclasses.replace(SGDM, seed=11), 16, 1),
    ("adamw-n6-t2", ADAMW, 6, 2),
    ("adamw-n7-t1", ADAMW, 7, 1),
]


@pytest.mark.parametrize("layout_name", ["ragged", "mini"])
@pytest.mark.parametrize("name,hp,n,tau", CASES, ids=[c[0] for c in CASES])
def test_rounds_bitexact(layout_name, name, hp, n, tau):
    tensors = RAGGED if layout_name == "ragged" else MINI
    run = dsm.DistributedSignMomentum(tensors, n, tau, hp)
    ora = O.OracleRun(tensors, n, tau, hp, with_stats=True)
    compare_state(run, ora)
    for t in range(2):
        base = t * tau
        for k in range(tau):
            run.fill_synthetic_grads(base + k)
            g = run.read(dsm.BUF_GRAD, n - 1)
            ora_g = O.synthetic_grad(ora.elems, ora.scale, hp.seed, base + k, n - 1, hp.grad_dtype)
            assert_bitexact(g.to(torch.float32).numpy(), ora_g, f"grad step {base + k}")
            run.local_step()
            ora.local_step()
        stats = run.global_step(with_stats=True)
        ora.global_step()
        compare_state(run, ora)
        compare_stats(stats, ora.last_stats, n)
    run.close()


VARIANTS = [
    ("slowmo-adamw-n4", dataclasses.replace(ADAMW, global_mode=W.GLOBAL_SLOWMO, g_b1=0.5, g_eta=0.8), 4, 2),
    ("signed-slowmo-sgdm-n3", dataclasses.replace(SGDM, sign_mode=W.SIGN, global_mode=W.GLOBAL_SIGNED_SLOWMO,
                                                  g_b1=0.5, g_b2=0.5), 3, 2),
    ("lookahead-adamw-n1", dataclasses.replace(ADAMW, global_mode=W.GLOBAL_LOOKAHEAD, g_b1=0.2, g_b2=0.2,
                                               g_wd=0.0, g_eta=1.0), 1, 3),
    ("lookahead-sgdm-n8", dataclasses.replace(SGDM, sign_mode=W.SIGN, global_mode=W.GLOBAL_LOOKAHEAD), 8, 1),
    ("global-adamw-bf16-n4", dataclasses.replace(ADAMW, grad_dtype=W.BF16, global_mode=W.GLOBAL_ADAMW), 4, 2),
    ("global-adamw-n9-generic", dataclasses.replace(SGDM, sign_mode=W.SIGN, global_mode=W.GLOBAL_ADAMW), 9, 1),
    ("global-adamw-sgdm-n8-t1", dataclasses.replace(SGDM, sign_mode=W.SIGN, global_mode=W.GLOBAL_ADAMW,
                                                     g_b1=0.8, g_b2=0.9), 8, 1),
    ("global-adamw-f32-n1-t3", dataclasses.replace(ADAMW, global_mode=W.GLOBAL_ADAMW, g_wd=0.0), 1, 3),
    ("global-adamw-bf16-n6-t2", dataclasses.replace(ADAMW, grad_dtype=W.BF16, global_mode=W.GLOBAL_ADAMW), 6, 2),
    ("slowmo-n16-generic", dataclasses.replace(SGDM, sign_mode=W.SIGN, global_mode=W.GLOBAL_SLOWMO), 16, 1),
]


@pytest.mark.parametrize("fused", [False, True], ids=["unfused", "fused"])
@pytest.mark.parametrize("layout_name", ["ragged", "mini"])
@pytest.mark.parametrize("name,hp,n,tau", VARIANTS, ids=[c[0] for c in VARIANTS])
def test_global_variants_bitexact(layout_name, name, hp, n, tau, fused):
    """The ablations' global steps (SlowMo, signed SlowMo, Lookahead, global AdamW), three rounds,
    in the unfused and the fused round (n > 8 falls back to unfused)."""
    tensors = RAGGED if layout_name == "ragged" else MINI
    hp = dataclasses.replace(hp, flags=W.FLAG_FUSED_ROUND if fused else 0)
    run = dsm.DistributedSignMomentum(tensors, n, tau, hp)
    ora = O.OracleRun(tensors, n, tau, hp, with_stats=True)
    for _ in range(3):
        stats = run.synthetic_round(with_stats=True)
        ora.run_round()
        compare_state(run, ora)
        compare_stats(stats, ora.last_stats, n)
    run.close()


FUSED = [
    ("adamw-f32-n4-t3", ADAMW, 4, 3),
    ("adamw-bf16-n8-t2", dataclasses.replace(ADAMW, grad_dtype=W.BF16), 8, 2),
    ("sgdm-rsign-n8-t1", SGDM, 8, 1),
    ("sgdm-rsignpm-n3-t2", dataclasses.replace(SGDM, sign_mode=W.RSIGN_PM, grad_dtype=W.BF16), 3, 2),
    ("adamw-n1-t1", ADAMW, 1, 1),
    ("adamw-n5-t2", ADAMW, 5, 2),
    # the split kernel (AdamW, 5 to 8 workers): odd and even worker counts, randomized signs, tau = 1
    # (every fused launch after the first starts the workers from x)
    ("adamw-f32-n6-t1-rsignpm", dataclasses.replace(ADAMW, sign_mode=W.RSIGN_PM, rsign_B=0.5, seed=4), 6, 1),
    ("adamw-bf16-n7-t3-rsign0", dataclasses.replace(ADAMW, grad_dtype=W.BF16, sign_mode=W.RSIGN_ZERO,
                                                     rsign_B=1.0), 7, 3),
    ("adamw-n9-deferred-reset", ADAMW, 9, 2),
    ("sgdm-rsign-n16-deferred-reset", SGDM, 16, 1),
    ("slowmo-unfused", dataclasses.replace(ADAMW, global_mode=W.GLOBAL_SLOWMO), 4, 2),
]


@pytest.mark.parametrize("layout_name", ["ragged", "mini"])
@pytest.mark.parametrize("name,hp,n,tau", FUSED, ids=[c[0] for c in FUSED])
def test_fused_round_bitexact(layout_name, name, hp, n, tau):
    """The fused round (last local step inside the global step, lazy reset; above 8 workers the lazy
    reset alone) gives the same state."""
    tensors = RAGGED if layout_name == "ragged" else MINI
    hp = dataclasses.replace(hp, flags=W.FLAG_FUSED_ROUND)
    run = dsm.DistributedSignMomentum(tensors, n, tau, hp)
    ora = O.OracleRun(tensors, n, tau, hp, with_stats=True)
    for _ in range(3):
        stats = run.synthetic_round(with_stats=True)
        ora.run_round()
        compare_state(run, ora)      # replicas read while their reset is pending return x
        compare_stats(stats, ora.last_stats, n)
    run.close()


def test_fused_round_pending_step_is_materialized():
    """Reading worker state while the last local step is deferred runs that step first."""
    tensors, n, tau = MINI, 4, 2
    hp = dataclasses.replace(ADAMW, flags=W.FLAG_FUSED_ROUND)
    run = dsm.DistributedSignMomentum(tensors, n, tau, hp)
    ora = O.OracleRun(tensors, n, tau, hp)
    for t in range(3):
        for k in range(tau):
            run.fill_synthetic_grads(t * tau + k)
            run.local_step()
            ora.local_step()
        if t == 1:   # deferred step: reading a replica runs it unfused, then the global step is unfused
            assert_bitexact(run.read(dsm.BUF_REPLICA, 2).numpy(), ora.X[2], "replica before global step")
        if t == 2:   # writing replicas while their reset is pending writes x into them first
            run.global_step()
            ora.global_step()
            run.write(dsm.BUF_REPLICA, torch.from_numpy(ora.X[1].copy()), worker=1)
            compare_state(run, ora)
            continue
        run.global_step()
        ora.global_step()
        compare_state(run, ora)
    run.close()


def test_caller_gradients_host_and_device():
    """dsm_load_grads: gradients written by the caller (pinned host and device)."""
    tensors, n, tau = MINI, 3, 2
    hp = ADAMW
    d = sum(t.numel for t in tensors)
    rng = np.random.default_rng(0)
    run = dsm.DistributedSignMomentum(tensors, n, tau, hp)
    ora = O.OracleRun(tensors, n, tau, hp)
    for k in range(tau):
        g = (rng.standard_normal((n, d)) * 1e-3).astype(np.float32)
        src = torch.from_numpy(g).pin_memory() if k == 0 else torch.from_numpy(g).cuda()
        run.load_grads(src)
        run.local_step()
        ora.local_step([g[i] for i in range(n)])
    run.global_step()
    ora.global_step()
    compare_state(run, ora)
    run.close()


def test_order_of_algorithm_1_is_enforced():
    run = dsm.DistributedSignMomentum(MINI, 2, 2, ADAMW)
    with pytest.raises(dsm.DsmError) as e:
        run.global_step()
    assert e.value.code == dsm.DSM_ESTATE
    run.fill_synthetic_grads(0)
    run.local_step()
    with pytest.raises(dsm.DsmError) as e:
        run.set_gamma(1e-3)
    assert e.value.code == dsm.DSM_ESTATE
    run.local_step()
    with pytest.raises(dsm.DsmError) as e:
        run.local_step()
    assert e.value.code == dsm.DSM_ESTATE
    run.global_step()
    with pytest.raises(dsm.DsmError) as e:
        run.read(dsm.BUF_REPLICA, worker=2)
    assert e.value.code == dsm.DSM_ERANGE
    with pytest.raises(dsm.DsmError) as e:
        run.read(dsm.BUF_X, offset=run.d, count=1)
    assert e.value.code == dsm.DSM_ERANGE
    run.close()


def test_gamma_schedule():
    """A different gamma_t each round (e.g. a cosine schedule) reaches the local and global steps."""
    tensors, n, tau = MINI, 2, 2
    run = dsm.DistributedSignMomentum(tensors, n, tau, ADAMW)
    ora = O.OracleRun(tensors, n, tau, ADAMW)
    for gamma in (6e-4, 3e-4, 1.5e-4):
        run.set_gamma(gamma)
        ora.gamma = gamma
        run.synthetic_round()
        ora.run_round()
    compare_state(run, ora)
    run.close()


def test_checkpoint_resume_bitexact():
    tensors, n, tau = MINI, 4, 2
    hp = dataclasses.replace(SGDM, sign_mode=W.RSIGN_ZERO)
    a = dsm.DistributedSignMomentum(tensors, n, tau, hp)
    a.synthetic_round()
    bufs = [(dsm.BUF_X, 0), (dsm.BUF_M, 0)] + [(b, i) for i in range(n) for b in (dsm.BUF_REPLICA, dsm.BUF_OPT_M)]
    saved = [(b, i, a.read(b, i).clone()) for b, i in bufs]
    b = dsm.DistributedSignMomentum(tensors, n, tau, hp, x0=torch.zeros(a.d))
    for which, i, v in saved:
        b.write(which, v, worker=i)
    dsm.dsm_set_round(b.h, 1)
    a.synthetic_round()
    b.synthetic_round()
    torch.cuda.synchronize()
    for which, i in bufs:
        assert torch.equal(a.read(which, i), b.read(which, i))
    a.close()
    b.close()


def test_deterministic_statistics():
    tensors, n, tau = MINI, 4, 2
    outs = []
    for _ in range(2):
        run = dsm.DistributedSignMomentum(tensors, n, tau, ADAMW)
        outs.append(run.synthetic_round(with_stats=True))
        run.close()
    assert outs[0] == outs[1]


def test_statistics_of_the_hand_built_global_step():
    """The hand-computed d = 8, n = 3 global step (tests/golden/stats_example_d8.json, deterministic sign)
    through the C ABI: one plain-SGD local step on zero gradients leaves every replica at x = 0, the
    replicas and m are then set to the example's values, and the global step must give the hand-computed
    x', m' and statistics exactly (every value is dyadic)."""
    import json
    import os
    from fractions import Fraction
    ex = json.load(open(os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "stats_example_d8.json")))
    hpj = ex["hparams"]
    fr = lambda v: float(Fraction(v))  # noqa: E731
    hp = W.HParams(base=W.BASE_SGDM, lr=fr(hpj["gamma"]), mu=0.0, wd=0.0, g_b1=fr(hpj["beta1"]),
                   g_b2=fr(hpj["beta2"]), g_eta=fr(hpj["eta"]), g_wd=fr(hpj["lambda"]), sign_mode=W.SIGN)
    tensors = (W.Tensor("t", 8, W.KIND_WEIGHT, 1.0),)
    vec = lambda vals: torch.tensor([fr(v) for v in vals], dtype=torch.float32)  # noqa: E731
    run = dsm.DistributedSignMomentum(tensors, hpj["n"], 1, hp, x0=vec(ex["x"]))
    run.load_grads(torch.zeros(hpj["n"], 8, dtype=torch.float32))
    run.local_step()
    for i, di in enumerate(ex["diffs"]["values"]):
        run.write(dsm.BUF_REPLICA, vec(ex["x"]) - vec(di), worker=i)
    run.write(dsm.BUF_M, vec(ex["m"]))
    st = run.global_step(with_stats=True)[0]
    torch.cuda.synchronize()
    want = ex["modes"]["sign"]
    sg = vec(want["sign"])
    assert torch.equal(run.read(dsm.BUF_X), -fr(hpj["eta"]) * fr(hpj["gamma"]) * sg)
    assert torch.equal(run.read(dsm.BUF_M), vec(ex["m_new"]))
    for key in ("delta_sq", "drift"):
        assert st[key] == fr(want["stats"][key]), key
    for key in ("zero_sign", "flips", "unanimous", "clamped"):
        assert st[key] == want["stats"][key], key
    run.close()


@pytest.mark.parametrize("fused", [False, True], ids=["unfused", "fused"])
def test_parameter_shards_of_one_model(fused):
    """One model cut into three parameter shards (paper_2411_17866_gb300/shard.py), each run by the
    library with its pieces as the layout and its first_element, one after another on this GPU: every shard
    equals the whole-model oracle on its range bit for bit over two rounds (randomized sign, bf16
    gradients), and the shards' per-piece statistics summed per tensor equal the whole-model statistics."""
    from paper_2411_17866_gb300 import shard as S
    model = RAGGED
    n, tau, world = 3, 2, 3
    hp = dataclasses.replace(ADAMW, sign_mode=W.RSIGN_PM, rsign_B=0.5, grad_dtype=W.BF16, seed=9,
                             flags=W.FLAG_FUSED_ROUND if fused else 0)
    whole = O.OracleRun(model, n, tau, hp, with_stats=True)
    whole_stats = []
    for _ in range(2):
        whole.run_round()
        whole_stats.append(whole.last_stats)
    per_round = [[], []]
    for r in range(world):
        sh = S.shard_layout(model, world, r)
        run = dsm.DistributedSignMomentum(sh.tensors, n, tau, hp, first_element=sh.first_element)
        ora = O.OracleRun(model, n, tau, hp, elems=np.arange(sh.first_element, sh.first_element + sh.count))
        for t in range(2):
            st = run.synthetic_round(with_stats=True)
            ora.run_round()
            compare_state(run, ora)
            per_round[t].append(S.stats_by_tensor(sh, st, len(model)))
        run.close()
    for t in range(2):
        compare_stats(S.reduce_stats(per_round[t]), whole_stats[t], n)


@pytest.mark.parametrize("first_element", [1 << 20, (1 << 35) + 8, (1 << 59) + 4096],
                         ids=["2^20", "2^35+8", "2^59+4096"])
def test_first_element_far_into_a_larger_model(first_element):
    """A layout placed far into a larger model: the 64-bit key offsets of the synthetic draws and the
    Philox counter's high word (first_element/4 >= 2^32) against the oracle with the same first_element."""
    hp = dataclasses.replace(SGDM, sign_mode=W.RSIGN_ZERO, rsign_B=1e-2, grad_dtype=W.BF16)
    for h in (hp, dataclasses.replace(ADAMW, flags=W.FLAG_FUSED_ROUND)):
        run = dsm.DistributedSignMomentum(RAGGED, 4, 2, h, first_element=first_element)
        ora = O.OracleRun(RAGGED, 4, 2, h, first_element=first_element, with_stats=True)
        for _ in range(2):
            st = run.synthetic_round(with_stats=True)
            ora.run_round()
            compare_state(run, ora)
            compare_stats(st, ora.last_stats, 4)
        run.close()


def test_x0_from_device_and_host():
    tensors, n, tau = MINI, 2, 1
    d = sum(t.numel for t in tensors)
    x0 = torch.linspace(-1, 1, d, dtype=torch.float32)
    for src in (x0, x0.cuda()):
        run = dsm.DistributedSignMomentum(tensors, n, tau, ADAMW, x0=src)
        ora = O.OracleRun(tensors, n, tau, ADAMW, x0=x0.numpy())
        compare_state(run, ora)
        run.synthetic_round()
        ora.run_round()
        compare_state(run, ora)
        run.close()


# The element-subset pin at full size: 10^7 random elements plus the first and last 4096 of every tensor.
FULL_SAMPLE, FULL_EDGE = 10_000_000, 4096
_FULL_ORACLE = {}


def _full_oracle(key):
    """The C++ oracle over the sampled elements of a full-size workload, through all of its rounds: x and m
    after every round and the final state (computed once per workload: the fused and the unfused round
    give the same results)."""
    if key not in _FULL_ORACLE:
        wl = W.WORKLOADS[key]
        elems = None if wl.d <= (1 << 20) else sample_elements(wl.tensors, FULL_SAMPLE, edge=FULL_EDGE)
        ora = CxxOracleRun(wl.tensors, wl.n, wl.tau, wl.hp, elems=elems, with_stats=elems is None)
        per_round = []
        for _ in range(wl.rounds):
            ora.run_round()
            per_round.append((ora.x.copy(), ora.m.copy(), ora.last_stats))
        _FULL_ORACLE[key] = (elems, ora, per_round)
    return _FULL_ORACLE[key]


FULL_CASES = [(key, fused) for key in W.WORKLOADS for fused in (False, True)]


@pytest.mark.parametrize("key,fused", FULL_CASES, ids=[f"{k}-{'fused' if f else 'unfused'}" for k, f in FULL_CASES])
def test_full_workloads_sampled(key, fused):
    """Each measured workload at full size through all of its rounds (5 for GPT-2 S and M, 3 for L, XL
    and the flat workload), in the launch sequence the benchmark uses, fused and unfused, against the C++
    oracle on sampled elements (10^7 random ones plus the first and last 4096 of every tensor; the whole
    model for the flat workload): x and m after every round, every replica and optimizer state after the
    last, bit for bit.  This reaches the round-keyed Philox draws at t > 0, AdamW's bias corrections at
    j > tau and the first local step from x after a deferred reset at full size."""
    wl = W.WORKLOADS[key]
    hp = dataclasses.replace(wl.hp, flags=W.FLAG_FUSED_ROUND if fused else 0)
    elems, ora, per_round = _full_oracle(key)
    run = dsm.DistributedSignMomentum(wl.tensors, wl.n, wl.tau, hp)
    sel = None if elems is None else torch.from_numpy(elems).cuda()
    buf = torch.empty(wl.d, dtype=torch.float32, device="cuda")

    def rd(which, i=0):
        run.read(which, i, out=buf)
        return (buf if sel is None else buf[sel]).cpu().numpy()

    for t, (x_t, m_t, stats_t) in enumerate(per_round):
        stats = run.synthetic_round(with_stats=True)
        assert_bitexact(rd(dsm.BUF_X), x_t, f"x after round {t}")
        assert_bitexact(rd(dsm.BUF_M), m_t, f"m after round {t}")
        if elems is None:
            compare_stats(stats, stats_t, wl.n)
        else:   # properties that hold at any size
            assert sum(s["unanimous"] for s in stats) <= wl.d
            assert all(s["delta_sq"] > 0 for s in stats)
    for i in range(wl.n):
        assert_bitexact(rd(dsm.BUF_REPLICA, i), ora.X[i], f"replica {i}")
        assert_bitexact(rd(dsm.BUF_OPT_M, i), ora.opt_m[i], f"opt_m {i}")
        if ora.opt_v is not None:
            assert_bitexact(rd(dsm.BUF_OPT_V, i), ora.opt_v[i], f"opt_v {i}")
    run.close()
    del run, buf
    torch.cuda.empty_cache()
    if fused:
        _FULL_ORACLE.pop(key, None)


@pytest.mark.parametrize("key", list(W.WORKLOADS))
def test_fp64_twin_within_stated_tolerance(key):
    """The GPU result against the float64 oracle on sampled elements (every 7th element of the flat
    workload): |x - x64| <= 1e-6 (1 + |x|); an element whose sign decision differs from the twin's is
    allowed only where |u| <= 1e-6 max|u|, and is counted."""
    wl = W.WORKLOADS[key]
    hp = dataclasses.replace(wl.hp, flags=W.FLAG_FUSED_ROUND)
    run = dsm.DistributedSignMomentum(wl.tensors, wl.n, wl.tau, hp)
    elems = np.arange(0, wl.d, 7) if wl.d <= (1 << 20) else sample_elements(wl.tensors, 5000, seed=1, edge=8)
    ora64 = O.OracleRun(wl.tensors, wl.n, wl.tau, hp, elems=elems, dtype=np.float64)
    sel = torch.from_numpy(elems).cuda()
    buf = torch.empty(wl.d, dtype=torch.float32, device="cuda")
    diverged = np.zeros(elems.size, dtype=bool)
    mismatches = 0
    for _ in range(min(wl.rounds, 2)):
        run.synthetic_round()
        ora64.run_round()
        u64 = ora64.last_inter["u"]
        run.read(dsm.BUF_X, out=buf)
        x = buf[sel].cpu().numpy().astype(np.float64)
        moved = np.abs(x - ora64.x) > 1e-6 * (1 + np.abs(ora64.x))
        near_zero = np.abs(u64) <= 1e-6 * np.max(np.abs(u64))
        assert np.all(near_zero[moved & ~diverged]), "a parameter left the tolerance away from u = 0"
        mismatches += int(np.sum(moved & ~diverged))
        diverged |= moved
    print(f"{key}: sign decisions that differ from the fp64 twin: {mismatches} of {elems.size}")
    run.close()
    del run
    torch.cuda.empty_cache()


DEGENERATE = [
    ("eta-zero", dataclasses.replace(ADAMW, g_eta=0.0), 3, 2),
    ("global-betas-one", dataclasses.replace(ADAMW, g_b1=1.0, g_b2=1.0), 2, 2),
    ("zero-global-decay-and-betas", dataclasses.replace(SGDM, sign_mode=W.SIGN, g_b1=0.0, g_b2=0.0, g_wd=0.0), 4, 1),
    ("rsign-huge-bound", dataclasses.replace(SGDM, rsign_B=1e30), 3, 1),
    ("rsign-tiny-bound", dataclasses.replace(SGDM, sign_mode=W.RSIGN_PM, rsign_B=1e-30), 3, 1),
    ("tiny-gamma", dataclasses.replace(ADAMW, lr=1e-8), 2, 3),
    ("large-seed-tau5", dataclasses.replace(ADAMW, seed=(1 << 63) + 5), 2, 5),
    ("max-workers-64", dataclasses.replace(SGDM, seed=3), 64, 1),
]


@pytest.mark.parametrize("name,hp,n,tau", DEGENERATE, ids=[c[0] for c in DEGENERATE])
def test_degenerate_cases_bitexact(name, hp, n, tau):
    """Degenerate settings of the method and the maximum worker count, against the oracle."""
    tensors = RAGGED
    run = dsm.DistributedSignMomentum(tensors, n, tau, hp)
    ora = O.OracleRun(tensors, n, tau, hp, with_stats=True)
    for _ in range(2):
        x_before = ora.x.copy()
        stats = run.synthetic_round(with_stats=True)
        ora.run_round()
        compare_state(run, ora)
        compare_stats(stats, ora.last_stats, n)
        if name == "eta-zero":
            assert np.array_equal(ora.x, x_before)
        if name == "rsign-tiny-bound":   # every nonzero u is above the bound: deterministic sign, all counted
            nonzero = int(np.count_nonzero(ora.last_inter["u"]))
            assert sum(s["clamped"] for s in stats) == nonzero
    run.close()


def test_zero_gradients():
    """All-zero gradients (scale 0): the workers only decay; Delta = lr * lambda * x for AdamW."""
    tensors = tuple(dataclasses.replace(t, grad_scale=0.0) for t in RAGGED)
    run = dsm.DistributedSignMomentum(tensors, 3, 2, ADAMW)
    ora = O.OracleRun(tensors, 3, 2, ADAMW, with_stats=True)
    run.synthetic_round()
    ora.run_round()
    compare_state(run, ora)
    run.close()


@pytest.mark.parametrize("grad_dtype", [W.F32, W.BF16], ids=["f32", "bf16"])
def test_gradient_scales_across_the_prescaled_limit(grad_dtype):
    """K1 multiplies by s*2^-24 when both s and 0.1*s are at least 2^-102 and by s otherwise; both forms
    must give the oracle's bits.  Scales on either side of the limit, a huge one and zero, every worker."""
    scales = [2.0 ** -102, 2.0 ** -98, 1e-35, 1e-30, 3e37, 0.0, 1e-3]
    tensors = tuple(W.Tensor(f"s{i}", numel, W.KIND_WEIGHT, sc)
                    for i, (sc, numel) in enumerate(zip(scales, [4096, 1031, 2048, 4100, 1024, 64, 3000])))
    n = 3
    hp = dataclasses.replace(ADAMW, grad_dtype=grad_dtype, seed=9)
    run = dsm.DistributedSignMomentum(tensors, n, 1, hp)
    ora = O.OracleRun(tensors, n, 1, hp)
    for step in (0, 5):
        run.fill_synthetic_grads(step)
        for w in range(n):
            g = run.read(dsm.BUF_GRAD, w).to(torch.float32).numpy()
            want = O.synthetic_grad(ora.elems, ora.scale, hp.seed, step, w, grad_dtype)
            assert_bitexact(g, want, f"grad step {step} worker {w}")
    run.close()


def test_guard_regions_detect_an_overrun():
    """A byte written past the end of the tensor table (a planted host-side write) is reported."""
    run = dsm.DistributedSignMomentum(MINI, 2, 1, ADAMW)
    assert run.check_guards() == 0
    first_guard = -(-len(MINI) * 48 // 256) * 256
    run.arena[first_guard + 7] = 0
    torch.cuda.synchronize()
    assert run.check_guards() == 1
    run.close()


@pytest.mark.parametrize("fused", [False, True], ids=["unfused", "fused"])
def test_many_rounds_stay_bitexact(fused):
    """Forty rounds with a learning-rate schedule: no drift between the GPU and the oracle."""
    tensors, n, tau = RAGGED, 3, 2
    hp = dataclasses.replace(ADAMW, flags=W.FLAG_FUSED_ROUND if fused else 0, sign_mode=W.SIGN)
    run = dsm.DistributedSignMomentum(tensors, n, tau, hp)
    ora = O.OracleRun(tensors, n, tau, hp, with_stats=True)
    for t in range(40):
        gamma = dsm.dsm_cosine_gamma(6e-4, 0.05, 10, 80, t * tau)
        run.set_gamma(gamma)
        ora.gamma = float(gamma)
        stats = run.synthetic_round(with_stats=True)
        ora.run_round()
        compare_stats(stats, ora.last_stats, n)
    compare_state(run, ora)
    run.close()


def test_injected_host_allocation_failure_on_device_arena(monkeypatch):
    """With a valid device arena, the injected host allocation failure is reported as DSM_ENOMEM."""
    monkeypatch.setenv("DSM_INJECT_HOST_ALLOC_FAILURE", "1")
    with pytest.raises(dsm.DsmError) as e:
        dsm.DistributedSignMomentum(MINI, 2, 1, ADAMW)
    assert e.value.code == dsm.DSM_ENOMEM


@pytest.mark.parametrize("fused", [False, True], ids=["unfused", "fused"])
def test_state_dict_round_trip(fused):
    """Checkpoint after a round, restore into a fresh handle, continue: identical to never stopping."""
    hp = dataclasses.replace(ADAMW, flags=W.FLAG_FUSED_ROUND if fused else 0, global_mode=W.GLOBAL_SIGN_MOMENTUM)
    a = dsm.DistributedSignMomentum(RAGGED, 3, 2, hp)
    a.set_gamma(5e-4)
    a.synthetic_round()
    st = a.state_dict()
    b = dsm.DistributedSignMomentum(RAGGED, 3, 2, hp, x0=torch.zeros(a.d))
    b.load_state_dict(st)
    for _ in range(2):
        a.synthetic_round()
        b.synthetic_round()
    torch.cuda.synchronize()
    for which, w in [(dsm.BUF_X, 0), (dsm.BUF_M, 0)] + [(dsm.BUF_OPT_V, i) for i in range(3)]:
        assert torch.equal(a.read(which, w), b.read(which, w))
    a.close()
    b.close()


RESET = [
    ("adamw-f32-n4-t3", ADAMW, 4, 3),
    ("adamw-bf16-n3-t1", dataclasses.replace(ADAMW, grad_dtype=W.BF16, seed=5), 3, 1),
    ("sgdm-rsign-n8-t2", SGDM, 8, 2),
    ("sgdm-bf16-n2-t1", dataclasses.replace(SGDM, grad_dtype=W.BF16, sign_mode=W.SIGN), 2, 1),
    ("adamw-n9-generic-t2", ADAMW, 9, 2),
    ("adamw-bf16-n8-t1", dataclasses.replace(ADAMW, grad_dtype=W.BF16), 8, 1),
    ("adamw-n7-t2", ADAMW, 7, 2),
    ("slowmo-adamw-n4-t2", dataclasses.replace(ADAMW, global_mode=W.GLOBAL_SLOWMO, g_b1=0.5, g_eta=0.8), 4, 2),
    ("global-adamw-n3-t2", dataclasses.replace(ADAMW, global_mode=W.GLOBAL_ADAMW), 3, 2),
]


@pytest.mark.parametrize("fused", [False, True], ids=["unfused", "fused"])
@pytest.mark.parametrize("layout_name", ["ragged", "mini"])
@pytest.mark.parametrize("name,hp,n,tau", RESET, ids=[c[0] for c in RESET])
def test_reset_local_state_bitexact(layout_name, name, hp, n, tau, fused):
    """Every round restarts each worker's base optimizer (zero state, AdamW count j = k + 1): three
    rounds against the oracle, the states read back mid-round (the restarted optimizer's values) and
    between rounds (zeros)."""
    tensors = RAGGED if layout_name == "ragged" else MINI
    flags = W.FLAG_RESET_LOCAL_STATE | (W.FLAG_FUSED_ROUND if fused else 0)
    hp = dataclasses.replace(hp, flags=flags)
    run = dsm.DistributedSignMomentum(tensors, n, tau, hp)
    ora = O.OracleRun(tensors, n, tau, hp, with_stats=True)
    for t in range(3):
        if t == 1:   # mid-round: the first local step restarted from zero state
            run.fill_synthetic_grads(t * tau)
            run.local_step()
            ora.local_step()
            compare_state(run, ora)
            for k in range(1, tau):
                run.fill_synthetic_grads(t * tau + k)
                run.local_step()
                ora.local_step()
            stats = run.global_step(with_stats=True)
            ora.global_step()
        else:
            stats = run.synthetic_round(with_stats=True)
            ora.run_round()
        compare_state(run, ora)   # states between rounds: zeros on both sides
        compare_stats(stats, ora.last_stats, n)
        assert all(not np.any(o) for o in ora.opt_m)
    run.close()


def test_reset_local_state_differs_from_persistent_state():
    """The flag changes the method (not only its execution): after two rounds the models differ."""
    tensors, n, tau = MINI, 2, 2
    xs = []
    for flags in (0, W.FLAG_RESET_LOCAL_STATE):
        run = dsm.DistributedSignMomentum(tensors, n, tau, dataclasses.replace(ADAMW, flags=flags))
        for _ in range(2):
            run.synthetic_round()
        xs.append(run.read(dsm.BUF_X))
        run.close()
    assert not torch.equal(xs[0], xs[1])


@pytest.mark.parametrize("fused", [False, True], ids=["unfused", "fused"])
def test_reset_local_state_checkpoint_and_partial_writes(fused):
    """With the restart pending: a partial write of a state buffer keeps the rest at zero, a checkpoint
    restores into a fresh handle, and both continue identically to the oracle."""
    tensors, n, tau = RAGGED, 3, 2
    flags = W.FLAG_RESET_LOCAL_STATE | (W.FLAG_FUSED_ROUND if fused else 0)
    hp = dataclasses.replace(ADAMW, flags=flags)
    a = dsm.DistributedSignMomentum(tensors, n, tau, hp)
    ora = O.OracleRun(tensors, n, tau, hp)
    a.synthetic_round()
    ora.run_round()
    st = a.state_dict()
    assert all(not torch.any(v) for v in st["opt_m"] + st["opt_v"])
    # a partial write into worker 1's first moment: the oracle gets the same values, the rest stays 0
    patch = torch.full((100,), 1e-4, dtype=torch.float32)
    a.write(dsm.BUF_OPT_M, patch, worker=1, offset=50)
    ora.opt_m[1][50:150] = patch.numpy()
    compare_state(a, ora)
    b = dsm.DistributedSignMomentum(tensors, n, tau, hp, x0=torch.zeros(a.d))
    b.load_state_dict(a.state_dict())
    for _ in range(2):
        a.synthetic_round()
        b.synthetic_round()
        ora.run_round()
    compare_state(a, ora)
    compare_state(b, ora)
    a.close()
    b.close()


HOST_GRADS = [
    ("adamw-f32-n3-t2-fused", dataclasses.replace(ADAMW, flags=W.FLAG_FUSED_ROUND), 3, 2),
    ("adamw-bf16-n8-t2", dataclasses.replace(ADAMW, grad_dtype=W.BF16), 8, 2),
    ("sgdm-n4-t1-fused", dataclasses.replace(SGDM, flags=W.FLAG_FUSED_ROUND), 4, 1),
    ("adamw-n9-generic-t2", ADAMW, 9, 2),
    ("adamw-n9-t2-deferred-reset", dataclasses.replace(ADAMW, flags=W.FLAG_FUSED_ROUND), 9, 2),
    ("reset-adamw-n4-t3-fused", dataclasses.replace(ADAMW, flags=W.FLAG_FUSED_ROUND | W.FLAG_RESET_LOCAL_STATE), 4, 3),
]


@pytest.mark.parametrize("chunk_bytes", ["default", "4096"])
@pytest.mark.parametrize("layout_name", ["ragged", "mini"])
@pytest.mark.parametrize("name,hp,n,tau", HOST_GRADS, ids=[c[0] for c in HOST_GRADS])
def test_host_gradient_steps_bitexact(layout_name, name, hp, n, tau, chunk_bytes, monkeypatch):
    """dsm_local_step_host_grads: gradients from pinned host memory, copied chunk by chunk on a second
    stream while the previous chunk is updated; three rounds against the oracle fed the same gradients.
    A 4096-byte chunk size cuts the model into many chunks, with boundaries inside tensors."""
    if chunk_bytes != "default":
        monkeypatch.setenv("DSM_HOST_GRAD_CHUNK_BYTES", chunk_bytes)
    tensors = RAGGED if layout_name == "ragged" else MINI
    d = sum(t.numel for t in tensors)
    rng = np.random.default_rng(zlib.crc32(name.encode()))
    run = dsm.DistributedSignMomentum(tensors, n, tau, hp)
    ora = O.OracleRun(tensors, n, tau, hp, with_stats=True)
    stream = torch.cuda.current_stream()
    copy_stream = torch.cuda.Stream()
    bf16 = hp.grad_dtype == W.BF16
    keep = []
    for t in range(3):
        for k in range(tau):
            g = torch.from_numpy((rng.standard_normal((n, d)) * 1e-3).astype(np.float32))
            if bf16:
                g = g.to(torch.bfloat16)
            src = g.pin_memory()
            keep.append(src)   # unchanged until the copies complete
            run.local_step_host_grads(src, stream, copy_stream)
            ora.local_step([g[i].to(torch.float32).numpy() for i in range(n)])
        stats = run.global_step(stream, with_stats=True)
        ora.global_step()
        compare_state(run, ora, grads=False)
        compare_stats(stats, ora.last_stats, n)
    run.close()


def test_host_gradient_steps_mix_with_device_fills():
    """Host-gradient steps interleaved with synthetic fills and plain local steps on the same handle."""
    tensors, n, tau = RAGGED, 3, 3
    hp = dataclasses.replace(ADAMW, flags=W.FLAG_FUSED_ROUND)
    d = sum(t.numel for t in tensors)
    run = dsm.DistributedSignMomentum(tensors, n, tau, hp)
    ora = O.OracleRun(tensors, n, tau, hp)
    copy_stream = torch.cuda.Stream()
    rng = np.random.default_rng(4)
    keep = []
    for t in range(2):
        for k in range(tau):
            if k == 1:
                run.fill_synthetic_grads(t * tau + k)
                run.local_step()
                ora.local_step()
            else:
                g = (rng.standard_normal((n, d)) * 1e-3).astype(np.float32)
                src = torch.from_numpy(g).pin_memory()
                keep.append(src)
                run.local_step_host_grads(src, copy_stream=copy_stream)
                ora.local_step([g[i] for i in range(n)])
        run.global_step()
        ora.global_step()
    compare_state(run, ora)
    with pytest.raises(ValueError):
        run.local_step_host_grads(torch.zeros((n, d + 1)))
    run.close()


SMALL = (W.Tensor("s9", 9, W.KIND_WEIGHT, 1e-2), W.Tensor("s1000", 1000, W.KIND_WEIGHT, 1e-3),
         W.Tensor("s1", 1, W.KIND_LN_W, 1e-3), W.Tensor("s8", 8, W.KIND_BIAS, 1e-3),
         W.Tensor("s1024", 1024, W.KIND_WEIGHT, 1e-3), W.Tensor("s1025", 1025, W.KIND_LN_B, 1e-4))


@pytest.mark.parametrize("fused", [False, True], ids=["unfused", "fused"])
@pytest.mark.parametrize("name,hp,n", [("adamw-n2", ADAMW, 2), ("sgdm-rsign-n5", SGDM, 5)], ids=["adamw-n2", "sgdm-rsign-n5"])
def test_small_tensors_tau4(name, hp, n, fused):
    """Tensors of 9, 1000, 1, 8, 1024 and 1025 elements (sub-tile, exactly one tile, one past a tile),
    four local steps per round, three rounds."""
    hp = dataclasses.replace(hp, flags=W.FLAG_FUSED_ROUND if fused else 0)
    run = dsm.DistributedSignMomentum(SMALL, n, 4, hp)
    ora = O.OracleRun(SMALL, n, 4, hp, with_stats=True)
    for _ in range(3):
        stats = run.synthetic_round(with_stats=True)
        ora.run_round()
        compare_state(run, ora)
        compare_stats(stats, ora.last_stats, n)
    run.close()


def test_two_handles_on_two_streams_are_independent():
    """Two handles (different base optimizers, sign modes and fused settings) whose rounds are issued
    alternately on two streams: each equals its own oracle bit for bit."""
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    hp_a = dataclasses.replace(ADAMW, flags=W.FLAG_FUSED_ROUND, seed=21)
    hp_b = dataclasses.replace(SGDM, seed=22)
    a = dsm.DistributedSignMomentum(RAGGED, 3, 2, hp_a)
    b = dsm.DistributedSignMomentum(MINI, 5, 3, hp_b)
    oa = O.OracleRun(RAGGED, 3, 2, hp_a)
    ob = O.OracleRun(MINI, 5, 3, hp_b)
    torch.cuda.synchronize()
    for t in range(2):
        for k in range(3):
            if k < 2:
                a.fill_synthetic_grads(t * 2 + k, s1)
                a.local_step(s1)
                oa.local_step()
            b.fill_synthetic_grads(t * 3 + k, s2)
            b.local_step(s2)
            ob.local_step()
        a.global_step(s1)
        b.global_step(s2)
        oa.global_step()
        ob.global_step()
    torch.cuda.synchronize()
    compare_state(a, oa)
    compare_state(b, ob)
    a.close()
    b.close()


@pytest.mark.parametrize("name,hp", [("adamw", ADAMW), ("sgdm-rsign", SGDM)], ids=["adamw", "sgdm-rsign"])
def test_non_finite_gradients_propagate_like_the_oracle(name, hp):
    """Gradients holding +inf, -inf and NaN at a few elements: the GPU state equals the oracle's, with
    NaN compared as NaN (the payload bits of a NaN are not fixed by IEEE 754) and every finite value
    bit for bit; the sign of a NaN argument is 0 on both sides."""
    tensors, n, tau = MINI, 3, 2
    d = sum(t.numel for t in tensors)
    run = dsm.DistributedSignMomentum(tensors, n, tau, hp)
    ora = O.OracleRun(tensors, n, tau, hp)
    rng = np.random.default_rng(5)
    for t in range(2):
        for k in range(tau):
            g = (rng.standard_normal((n, d)) * 1e-3).astype(np.float32)
            g[0, 10], g[1, 20], g[2, 30 + t] = np.inf, -np.inf, np.nan
            g[1, 40 + k] = np.float32(3e38)
            run.load_grads(torch.from_numpy(g).cuda())
            run.local_step()
            with np.errstate(all="ignore"):
                ora.local_step([g[i] for i in range(n)])
        run.global_step()
        with np.errstate(all="ignore"):
            ora.global_step()

    def same(got, want, what):
        got = np.asarray(got)
        nan_g, nan_w = np.isnan(got), np.isnan(want)
        assert np.array_equal(nan_g, nan_w), f"{what}: NaN positions differ"
        assert np.array_equal(got[~nan_g].view(np.uint32), np.asarray(want, np.float32)[~nan_w].view(np.uint32)), what
    same(run.read(dsm.BUF_X).numpy(), ora.x, "x")
    same(run.read(dsm.BUF_M).numpy(), ora.m, "m")
    for i in range(n):
        same(run.read(dsm.BUF_REPLICA, i).numpy(), ora.X[i], f"replica {i}")
        same(run.read(dsm.BUF_OPT_M, i).numpy(), ora.opt_m[i], f"opt_m {i}")
        if ora.opt_v is not None:
            same(run.read(dsm.BUF_OPT_V, i).numpy(), ora.opt_v[i], f"opt_v {i}")
    run.close()
