"""The C++ oracle (oracle/dsm_oracle.cpp) pinned, on CPU.

It is pinned to facts outside itself: the exact d = 8 worked examples
(Algorithm 1 evaluated by hand, statistics included), the published
known-answer vectors of SplitMix64 and Philox4x32-10, and the numpy oracle
(itself pinned by tests/oracle_pins.py and its mutation test), which it must
equal bit for bit on every buffer and exactly on every statistic, over the
configurations the workloads and the parity tests use.  Its OpenMP threads
must not change any result.
"""
import dataclasses
import json
import os
from fractions import Fraction

import numpy as np
import pytest

import workloads as W
from oracle import cxx_oracle as C
from oracle import dsm_oracle as O

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _load(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def _fr(vals):
    return np.array([float(Fraction(v)) for v in vals], dtype=np.float32)


def _bits(a):
    return np.ascontiguousarray(a, dtype=np.float32).view(np.uint32)


def test_known_answer_vectors():
    ka = _load("known_answers.json")
    seed = int(ka["splitmix64"]["seed"], 16)
    for j, want in enumerate(ka["splitmix64"]["outputs"], start=1):
        assert C.splitmix64_output(seed, j) == int(want, 16)
    for vec in ka["philox4x32_10"]["vectors"]:
        got = C.philox4x32_10([int(v, 16) for v in vec["ctr"]], [int(v, 16) for v in vec["key"]])
        assert got == [int(v, 16) for v in vec["out"]]


def test_generators_match_the_numpy_oracle():
    e = np.arange(0, 4099, dtype=np.int64)
    for seed, stream, idx in ((0, 0, 0), (7, 1, 3), (2 ** 40 + 5, 2, 0)):
        want = O.uniform24(seed, stream, idx, e)
        got = np.array([C.uniform24(seed, stream, idx, int(k)) for k in e], dtype=np.float32)
        assert np.array_equal(_bits(got), _bits(want))
    want = O.philox_uniform(e, seed=0x1234, t=9)
    got = np.array([C.philox_uniform(0x1234, 9, int(k)) for k in e], dtype=np.float32)
    assert np.array_equal(_bits(got), _bits(want))
    rng = np.random.default_rng(5)
    vals = np.concatenate([rng.integers(0, 2 ** 32, 20000, dtype=np.uint64).astype(np.uint32).view(np.float32),
                           np.array([1 + 2 ** -8, 1 + 3 * 2 ** -8, -(1 + 2 ** -8), np.inf, -np.inf, 0.0, -0.0],
                                    dtype=np.float32)])
    got = np.array([C.bf16_round(float(v)) for v in vals], dtype=np.float32)
    want = O.bf16_round(vals)
    ok = ~np.isnan(want)
    assert np.array_equal(_bits(got)[ok], _bits(want)[ok]) and np.all(np.isnan(got[~ok]))


def test_worked_example():
    """Algorithm 1 with plain-SGD local steps, d = 8, two rounds, evaluated by hand (dyadic values):
    Delta, u, the sign, x, m and all six statistics, exactly."""
    ex = _load("worked_example_d8.json")
    hpj = ex["hparams"]
    f = lambda k: float(Fraction(hpj[k]))  # noqa: E731
    hp = W.HParams(base=W.BASE_SGDM, lr=f("gamma"), mu=0.0, wd=0.0, g_b1=f("beta1"), g_b2=f("beta2"),
                   g_eta=f("eta"), g_wd=f("lambda"))
    run = C.CxxOracleRun(W.flat_layout(8, 1.0), hpj["n"], hpj["tau"], hp, x0=_fr(ex["x0"]), with_stats=True)
    for t, exp in enumerate(ex["rounds"]):
        run.run_round([[_fr(gi) for gi in gk] for gk in ex["grads"]["values"][t]])
        for key, got in (("delta", run.last_inter["delta"]), ("u", run.last_inter["u"]),
                         ("sign", run.last_inter["sg"]), ("x", run.x), ("m", run.m)):
            assert np.array_equal(got, _fr(exp[key])), (t, key)
        assert all(np.array_equal(row, run.x) for row in run.X)
        st, want = run.last_stats[0], exp["stats"]
        for key in ("delta_sq", "drift"):
            assert st[key] == float(Fraction(want[key])), (t, key)
        for key in ("zero_sign", "flips", "unanimous", "clamped"):
            assert st[key] == want[key], (t, key)


def test_stats_example():
    """The hand-built d = 8, n = 3 global step with chosen uniforms: every mode's applied sign, x', m' and
    statistics, exactly."""
    ex = _load("stats_example_d8.json")
    hpj = ex["hparams"]
    f = lambda k: float(Fraction(hpj[k]))  # noqa: E731
    for mode_name, mode in (("sign", W.SIGN), ("rand_sign_2", W.RSIGN_ZERO), ("rand_sign_1", W.RSIGN_PM)):
        hp = W.HParams(base=W.BASE_SGDM, lr=f("gamma"), mu=0.0, wd=0.0, g_b1=f("beta1"), g_b2=f("beta2"),
                       g_eta=f("eta"), g_wd=f("lambda"), sign_mode=mode, rsign_B=f("B"))
        run = C.CxxOracleRun(W.flat_layout(8, 1.0), hpj["n"], 1, hp, x0=_fr(ex["x"]), with_stats=True)
        run.m[:] = _fr(ex["m"])
        run.local_step([np.zeros(8, dtype=np.float32)] * hpj["n"])   # zero gradients: replicas stay at x
        for i, di in enumerate(ex["diffs"]["values"]):
            run.X[i] = _fr(ex["x"]) - _fr(di)
        run.global_step(r=_fr(ex["r"]))
        want = ex["modes"][mode_name]
        sg = _fr(want["sign"])
        assert np.array_equal(run.last_inter["delta"], _fr(ex["delta"])), mode_name
        assert np.array_equal(run.last_inter["u"], _fr(ex["u"])), mode_name
        assert np.array_equal(run.last_inter["sg"], sg), mode_name
        assert np.array_equal(run.m, _fr(ex["m_new"])), mode_name
        assert np.array_equal(run.x, (-f("eta") * f("gamma") * sg).astype(np.float32)), mode_name
        st = run.last_stats[0]
        for key in ("delta_sq", "drift"):
            assert st[key] == float(Fraction(want["stats"][key])), (mode_name, key)
        for key in ("zero_sign", "flips", "unanimous", "clamped"):
            assert st[key] == want["stats"][key], (mode_name, key)


RAGGED = (W.Tensor("a", 7, W.KIND_WEIGHT, 1e-2), W.Tensor("b", 2049, W.KIND_WEIGHT, 1e-3),
          W.Tensor("c", 8, W.KIND_BIAS, 1e-3, wd=0), W.Tensor("d", 5000, W.KIND_LN_W, 1e-3),
          W.Tensor("e", 1, W.KIND_LN_B, 1e-3), W.Tensor("f", 0, W.KIND_WEIGHT, 1e-3),
          W.Tensor("g", 4096, W.KIND_WEIGHT, 1e-2), W.Tensor("h", 77, W.KIND_BIAS, 1e-4))
ADAMW, SGDM = W.HParams(), W.SGDM_HP
CASES = [
    ("adamw-f32-n4-t3", ADAMW, 4, 3),
    ("adamw-bf16-n8-t2", dataclasses.replace(ADAMW, grad_dtype=W.BF16, seed=3), 8, 2),
    ("sgdm-rsign0-n8", SGDM, 8, 2),
    ("sgdm-rsignpm-bf16-n2", dataclasses.replace(SGDM, sign_mode=W.RSIGN_PM, grad_dtype=W.BF16), 2, 3),
    ("sgd-plain-n5", dataclasses.replace(SGDM, mu=0.0, sign_mode=W.SIGN), 5, 1),
    ("adamw-rsignpm-n9", dataclasses.replace(ADAMW, sign_mode=W.RSIGN_PM, rsign_B=1.0), 9, 2),
    ("slowmo", dataclasses.replace(ADAMW, global_mode=W.GLOBAL_SLOWMO, g_eta=0.5), 3, 2),
    ("signed-slowmo", dataclasses.replace(SGDM, global_mode=W.GLOBAL_SIGNED_SLOWMO, sign_mode=W.SIGN), 4, 2),
    ("lookahead", dataclasses.replace(ADAMW, global_mode=W.GLOBAL_LOOKAHEAD, g_eta=0.5), 2, 2),
    ("global-adamw", dataclasses.replace(ADAMW, global_mode=W.GLOBAL_ADAMW, g_eta=1e-3), 4, 2),
    ("reset-local-adamw", dataclasses.replace(ADAMW, flags=W.FLAG_RESET_LOCAL_STATE), 3, 2),
    ("reset-local-sgdm", dataclasses.replace(SGDM, flags=W.FLAG_RESET_LOCAL_STATE), 2, 3),
]


def _compare(c, o, where):
    assert np.array_equal(_bits(c.x), _bits(o.x)), (where, "x")
    assert np.array_equal(_bits(c.m), _bits(o.m)), (where, "m")
    for i in range(o.n):
        assert np.array_equal(_bits(c.X[i]), _bits(o.X[i])), (where, "replica", i)
        assert np.array_equal(_bits(c.opt_m[i]), _bits(o.opt_m[i])), (where, "opt_m", i)
        if o.opt_v is not None:
            assert np.array_equal(_bits(c.opt_v[i]), _bits(o.opt_v[i])), (where, "opt_v", i)
    if o.gv is not None:
        assert np.array_equal(_bits(c.gv), _bits(o.gv)), (where, "global v")


@pytest.mark.parametrize("name,hp,n,tau", CASES, ids=[c[0] for c in CASES])
def test_equals_numpy_oracle(name, hp, n, tau):
    """Three rounds with statistics (and a gamma change between rounds) on a ragged layout: every buffer
    bit for bit, every statistic exactly, Delta, u and the applied sign bit for bit."""
    o = O.OracleRun(RAGGED, n, tau, hp, with_stats=True)
    c = C.CxxOracleRun(RAGGED, n, tau, hp, with_stats=True)
    _compare(c, o, "init")
    for t in range(3):
        if t == 2:
            o.gamma = c.gamma = hp.lr * 0.5
        o.run_round()
        c.run_round()
        _compare(c, o, t)
        assert c.last_stats == o.last_stats, t
        for key in ("delta", "u", "sg"):
            assert np.array_equal(_bits(c.last_inter[key]), _bits(o.last_inter[key])), (t, key)


def test_subset_and_caller_gradients_equal_numpy_oracle():
    """Element subsets (sampled indices of a GPT-2-shaped layout) and caller-given gradients, including
    non-finite ones."""
    tensors = W.gpt2_layout(2, 64, 256)
    d = sum(t.numel for t in tensors)
    rng = np.random.default_rng(3)
    elems = np.unique(np.concatenate([rng.integers(0, d, 500), np.arange(0, 64), np.arange(d - 64, d)]))
    for hp in (dataclasses.replace(ADAMW, grad_dtype=W.BF16), SGDM):
        o = O.OracleRun(tensors, 4, 2, hp, elems=elems, with_stats=True)
        c = C.CxxOracleRun(tensors, 4, 2, hp, elems=elems, with_stats=True)
        for t in range(2):
            o.run_round()
            c.run_round()
            _compare(c, o, ("subset", t))
            assert c.last_stats == o.last_stats
    grads = rng.standard_normal((2, 3, elems.size)).astype(np.float32) * 1e-3
    grads[0, 1, :5] = [np.inf, -np.inf, np.nan, 3e38, -3e38]
    o = O.OracleRun(tensors, 3, 2, ADAMW, elems=elems, with_stats=True)
    c = C.CxxOracleRun(tensors, 3, 2, ADAMW, elems=elems, with_stats=True)
    o.run_round(grads)
    c.run_round(grads)
    for a, b in ((c.x, o.x), (c.m, o.m), (c.X, np.stack(o.X)), (c.opt_v, np.stack(o.opt_v))):
        a, b = np.asarray(a), np.asarray(b)
        same = (_bits(a) == _bits(b)) | (np.isnan(a) & np.isnan(b))
        assert same.all()


def test_threads_do_not_change_results():
    wl = W.WORKLOADS["gpt2s"]
    elems = np.arange(0, 200_000, dtype=np.int64)
    runs = [C.CxxOracleRun(wl.tensors, 2, 2, wl.hp, elems=elems, with_stats=True, threads=th) for th in (1, 0)]
    for r in runs:
        r.run_round()
    _compare(runs[0], runs[1], "threads")
    assert runs[0].last_stats == runs[1].last_stats


def test_outside_element_is_refused():
    with pytest.raises(ValueError):
        C.CxxOracleRun(W.flat_layout(10, 1.0), 2, 1, ADAMW, elems=np.array([0, 10]))


@pytest.mark.parametrize("first_element", [64, (1 << 35) + 8, (1 << 59) + 4096])
def test_first_element_equals_numpy_oracle(first_element):
    """A layout placed far into a larger model (64-bit draw indices, Philox counters above 2^32)."""
    hp = dataclasses.replace(SGDM, sign_mode=W.RSIGN_PM, grad_dtype=W.BF16)
    o = O.OracleRun(RAGGED, 3, 2, hp, with_stats=True, first_element=first_element)
    c = C.CxxOracleRun(RAGGED, 3, 2, hp, with_stats=True, first_element=first_element)
    _compare(c, o, "init")
    for t in range(2):
        o.run_round()
        c.run_round()
        _compare(c, o, t)
        assert c.last_stats == o.last_stats
