"""Checks that pin the CPU oracle to facts outside itself.

Each ``pin_*`` function takes the oracle module as its argument and raises
AssertionError when the oracle disagrees with the fact it checks.  The
tests in ``test_oracle_pins.py`` run them on the oracle; the mutation test
in ``test_oracle_mutants.py`` runs them on copies of the oracle with a
planted mistake and expects at least one of them to fail.
"""
from __future__ import annotations

import json
import os
from fractions import Fraction

import numpy as np

import workloads as W

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _load(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def _frac_array(vals, dt):
    return np.array([float(Fraction(v)) for v in vals], dtype=dt)


# ---------------------------------------------------------------------------
# Worked example: Algorithm 1 evaluated by hand in exact arithmetic
# ---------------------------------------------------------------------------

def pin_worked_example(o, dt=np.float32):
    ex = _load("worked_example_d8.json")
    hpj = ex["hparams"]
    hp = W.HParams(base=W.BASE_SGDM, lr=float(Fraction(hpj["gamma"])), mu=0.0, wd=0.0,
                   g_b1=float(Fraction(hpj["beta1"])), g_b2=float(Fraction(hpj["beta2"])),
                   g_eta=float(Fraction(hpj["eta"])), g_wd=float(Fraction(hpj["lambda"])))
    tensors = W.flat_layout(8, 1.0)
    x0 = _frac_array(ex["x0"], np.float32)
    run = o.OracleRun(tensors, hpj["n"], hpj["tau"], hp, x0=x0, dtype=dt, with_stats=True)
    for t, exp in enumerate(ex["rounds"]):
        grads = [[_frac_array(gi, np.float32) for gi in gk] for gk in ex["grads"]["values"][t]]
        run.run_round(grads)
        inter = run.last_inter
        for key, got in (("delta", inter["delta"]), ("u", inter["u"]), ("sign", inter["sg"]),
                         ("x", run.x), ("m", run.m)):
            want = _frac_array(exp[key], dt)
            assert np.array_equal(np.asarray(got, dtype=dt), want), (t, key, got, want)
        for Xi in run.X:
            assert np.array_equal(Xi, run.x)
        _check_stats(run.last_stats[0], exp["stats"], ("round", t))


def _check_stats(got, want, where):
    """Statistics against hand-computed values: dyadic sums exactly, counts exactly."""
    for key in ("delta_sq", "drift"):
        assert got[key] == float(Fraction(want[key])), (where, key, got[key], want[key])
    for key in ("zero_sign", "flips", "unanimous", "clamped"):
        assert got[key] == want[key], (where, key, got[key], want[key])


def pin_stats_example(o):
    """A hand-built global step (d = 8, n = 3, chosen uniforms r) whose statistics separate every count
    from a plausible mistake: unanimity over every worker (not any, and not skipping zero differences),
    flips of sign(u) against sign(Delta) (not of the applied randomized sign), zeros of the applied sign,
    clamping strictly above B; and the randomized signs' comparison r < p (strict)."""
    ex = _load("stats_example_d8.json")
    hpj = ex["hparams"]
    dt = np.float32
    x = _frac_array(ex["x"], dt)
    m = _frac_array(ex["m"], dt)
    X = [x - _frac_array(di, dt) for di in ex["diffs"]["values"]]
    r = _frac_array(ex["r"], dt)
    lam = np.full(8, float(Fraction(hpj["lambda"])), dtype=dt)
    B = float(Fraction(hpj["B"]))
    gamma, b1, b2, eta = (float(Fraction(hpj[k])) for k in ("gamma", "beta1", "beta2", "eta"))
    for mode_name, mode in (("sign", 0), ("rand_sign_2", 1), ("rand_sign_1", 2)):
        want = ex["modes"][mode_name]
        x_new, m_new, inter = o.global_step(x, m, X, gamma, b1, b2, eta, lam, mode, B, r, np.dtype(dt))
        for key, got in (("delta", inter["delta"]), ("u", inter["u"]), ("m_new", m_new)):
            assert np.array_equal(got, _frac_array(ex[key], dt)), (mode_name, key, got)
        sg = _frac_array(want["sign"], dt)
        assert np.array_equal(inter["sg"], sg), (mode_name, inter["sg"], sg)
        assert np.array_equal(x_new, (-float(Fraction(eta)) * float(Fraction(gamma)) * sg).astype(dt)), mode_name
        st = o.round_stats(inter, np.zeros(8, dtype=np.int64), 1, mode, B)
        _check_stats(st[0], want["stats"], mode_name)


# ---------------------------------------------------------------------------
# Published known-answer vectors of the two counter-based generators
# ---------------------------------------------------------------------------

def pin_splitmix64(o):
    ka = _load("known_answers.json")["splitmix64"]
    seed = np.array([int(ka["seed"], 16)], dtype=np.uint64)
    for j, want in enumerate(ka["outputs"], start=1):
        got = int(o.splitmix64_output(seed, np.array([j], dtype=np.uint64))[0])
        assert got == int(want, 16), (j, hex(got), want)


def pin_philox(o):
    for vec in _load("known_answers.json")["philox4x32_10"]["vectors"]:
        c = [np.array([int(v, 16)], dtype=np.uint64) for v in vec["ctr"]]
        k = [np.array([int(v, 16)], dtype=np.uint64) for v in vec["key"]]
        got = [int(w[0]) for w in o.philox4x32_10(*c, *k)]
        assert got == [int(v, 16) for v in vec["out"]], ([hex(g) for g in got], vec["out"])


def pin_philox_uniform_mapping(o):
    """r_e uses word e mod 4 of the block at counter floor(e/4), top 24 bits."""
    e = np.arange(0, 64, dtype=np.int64)
    r = o.philox_uniform(e, seed=0x1234, t=7)
    for ei in (0, 1, 2, 3, 17, 62):
        q = ei // 4
        words = o.philox4x32_10(np.array([q]), np.array([0]), np.array([0]), np.array([0]),
                                np.array([0x1234]), np.array([7]))
        w = int(words[ei % 4][0])
        assert r[ei] == np.float32((w >> 8) * 2.0 ** -24)


# ---------------------------------------------------------------------------
# bfloat16 rounding: the library routine (torch) rounds to nearest even
# ---------------------------------------------------------------------------

def pin_bf16(o):
    import torch
    rng = np.random.default_rng(1)
    bits = rng.integers(0, 2 ** 32, size=1 << 20, dtype=np.uint64).astype(np.uint32)
    # exact ties (low half 0x8000) with both parities of the kept bit, and near-ties
    ties = (rng.integers(0, 2 ** 16, size=4096, dtype=np.uint64).astype(np.uint32) << np.uint32(16))
    extra = np.concatenate([ties | np.uint32(0x8000), ties | np.uint32(0x7FFF), ties | np.uint32(0x8001),
                            np.array([0x7F7FFFFF, 0xFF7FFFFF, 0x7F7F8000, 0x00000001, 0x80008000,
                                      0x7F800000, 0x00000000, 0x80000000], dtype=np.uint32)])
    bits = np.concatenate([bits, extra])
    x = bits.view(np.float32)
    x = x[~np.isnan(x)]
    got = o.bf16_round(x)
    want = torch.from_numpy(x.copy()).to(torch.bfloat16).to(torch.float32).numpy()
    assert np.array_equal(got.view(np.uint32), want.view(np.uint32))


# ---------------------------------------------------------------------------
# Synthetic gradient / init generator: exactness and distribution
# ---------------------------------------------------------------------------

def pin_uniform24(o):
    e = np.arange(1 << 20, dtype=np.int64)
    for stream, idx in ((0, 0), (0, 5), (1, 3), (2, 0)):
        u = o.uniform24(11, stream, idx, e)
        k = u.astype(np.float64) * 2 ** 24
        assert np.all(k == np.floor(k)) and u.min() >= 0 and u.max() < 1
        # 256-bin chi-square, 255 dof: mean 255, sd ~22.6; 6 sd bound
        h = np.bincount((k.astype(np.int64) >> 16), minlength=256)
        exp = e.size / 256
        chi2 = float(((h - exp) ** 2 / exp).sum())
        assert chi2 < 255 + 6 * 22.6, chi2
    a = o.uniform24(11, 0, 3, e)
    b = o.uniform24(11, 1, 3, e)
    assert np.mean(a == b) < 1e-3          # the two streams are separated
    assert abs(np.corrcoef(a, b)[0, 1]) < 5e-3
    # the two draws taken from one 64-bit output are uncorrelated
    assert abs(np.corrcoef(a[0::2], a[1::2])[0, 1]) < 5e-3


def pin_hash_fields(o):
    """Elements 2q and 2q+1 take bits 63..40 and 39..16 of SplitMix64 output q+1 of the family's key."""
    seed, stream, idx = 7, 1, 5
    key = np.array([o.hash_key(seed, stream, idx)], dtype=np.uint64)
    e = np.array([0, 1, 2, 3, 1001], dtype=np.int64)
    h = o.hash24(seed, stream, idx, e)
    for ei, hi in zip(e.tolist(), h.tolist()):
        out = int(o.splitmix64_output(key, np.array([ei // 2 + 1], dtype=np.uint64))[0])
        want = (out >> 40) & 0xFFFFFF if ei % 2 == 0 else (out >> 16) & 0xFFFFFF
        assert hi == want, (ei, hi, want)
    # the family key is output 1 + stream*2^40 + idx of SplitMix64(seed)
    want_key = int(o.splitmix64_output(np.array([seed], dtype=np.uint64),
                                       np.array([1 + (stream << 40) + idx], dtype=np.uint64))[0])
    assert int(key[0]) == want_key


def pin_synthetic_grad(o):
    e = np.arange(50000, dtype=np.int64)
    s = np.full(e.shape, 1e-3, dtype=np.float32)
    g0 = o.synthetic_grad(e, s, 0, 3, 0, 0)
    g1 = o.synthetic_grad(e, s, 0, 3, 1, 0)
    h0 = o.synthetic_grad(e, s, 0, 4, 0, 0)
    bound = np.float32(1e-3) * 0.5 + np.float32(1e-4) * 0.5
    assert np.all(np.abs(g0) <= bound * (1 + 1e-6))
    # same step, different workers: only the worker term (0.1 s) differs
    assert np.all(np.abs(g0 - g1) <= np.float32(1e-4) * (1 + 1e-6))
    # same worker, different steps: the step term (s) differs
    assert np.mean(np.abs(g0 - h0)) > 2e-4
    assert abs(float(np.mean(g0))) < 1e-5
    gb = o.synthetic_grad(e, s, 0, 3, 0, 1)
    assert np.array_equal(gb, o.bf16_round(g0))


# ---------------------------------------------------------------------------
# Base optimizers against library routines and closed forms
# ---------------------------------------------------------------------------

def pin_adamw_vs_torch(o):
    import torch
    rng = np.random.default_rng(2)
    d = 4096
    x0 = rng.standard_normal(d)
    hp = dict(lr=6e-4, b1=0.9, b2=0.95, eps=1e-8, wd=0.1)
    p = torch.tensor(x0.copy(), dtype=torch.float64, requires_grad=True)
    # the oracle uses the fp32 values of the hyper-parameters
    opt = torch.optim.AdamW([p], lr=o.f32(hp["lr"]), betas=(o.f32(hp["b1"]), o.f32(hp["b2"])),
                            eps=o.f32(hp["eps"]), weight_decay=o.f32(hp["wd"]), foreach=False)
    x, m, v = x0.copy(), np.zeros(d), np.zeros(d)
    wd_e = np.full(d, o.f32(hp["wd"]))
    for j in range(1, 13):
        g = rng.standard_normal(d) * 10.0 ** rng.uniform(-4, 0)
        p.grad = torch.tensor(g, dtype=torch.float64)
        opt.step()
        x, m, v = o.adamw_step(x, m, v, g, j, hp["lr"], hp["b1"], hp["b2"], hp["eps"], wd_e,
                               np.dtype(np.float64))
        ref = p.detach().numpy()
        assert np.max(np.abs(x - ref)) <= 1e-12 * (1 + np.max(np.abs(ref))), j


def pin_adamw_constant_grad(o):
    """Constant g and no decay: mhat = g and vhat = g^2 at every step, so each step moves lr*g/(|g|+eps)."""
    g = np.array([1e-3, -2e-2, 5e-5, -1.0, 3.0], dtype=np.float64)
    x = np.zeros_like(g)
    m = np.zeros_like(g)
    v = np.zeros_like(g)
    lr, eps = o.f32(1e-3), o.f32(1e-8)
    for j in range(1, 31):
        x, m, v = o.adamw_step(x, m, v, g, j, 1e-3, 0.9, 0.95, 1e-8, np.zeros_like(g), np.dtype(np.float64))
        want = -j * lr * g / (np.abs(g) + eps)
        assert np.allclose(x, want, rtol=1e-12, atol=0), (j, x, want)


def pin_adamw_first_step_fp32(o):
    """j=1 from m=v=0: x' = x - lr (g/(|g|+eps) + wd x) within a few fp32 roundings."""
    rng = np.random.default_rng(3)
    g = (rng.standard_normal(1000) * 1e-3).astype(np.float32)
    x = rng.standard_normal(1000).astype(np.float32)
    wd = np.full(1000, np.float32(0.1), dtype=np.float32)
    xn, m, v = o.adamw_step(x, np.zeros_like(x), np.zeros_like(x), g, 1, 6e-4, 0.9, 0.95, 1e-8, wd,
                            np.dtype(np.float32))
    x64, g64 = x.astype(np.float64), g.astype(np.float64)
    want = x64 - o.f32(6e-4) * (g64 / (np.abs(g64) + o.f32(1e-8)) + o.f32(0.1) * x64)
    assert np.all(np.abs(xn - want) <= 4 * np.spacing(np.abs(want).astype(np.float32)))


def pin_sgdm_vs_torch(o):
    import torch
    rng = np.random.default_rng(4)
    d = 2048
    x0 = rng.standard_normal(d)
    p = torch.tensor(x0.copy(), dtype=torch.float64, requires_grad=True)
    opt = torch.optim.SGD([p], lr=o.f32(1e-2), momentum=o.f32(0.9), dampening=0.0, foreach=False)
    x, buf = x0.copy(), np.zeros(d)
    for _ in range(10):
        g = rng.standard_normal(d) * 1e-2
        p.grad = torch.tensor(g, dtype=torch.float64)
        opt.step()
        x, buf = o.sgdm_step(x, buf, g, 1e-2, 0.9, np.dtype(np.float64))
        ref = p.detach().numpy()
        assert np.max(np.abs(x - ref)) <= 1e-13 * (1 + np.max(np.abs(ref)))


def pin_sgd_plain_exact(o):
    """mu = 0 is plain SGD, Eq. (base-sgd): x - lr*g, bit for bit in fp32."""
    rng = np.random.default_rng(5)
    x = rng.standard_normal(1000).astype(np.float32)
    g = rng.standard_normal(1000).astype(np.float32)
    buf = rng.standard_normal(1000).astype(np.float32)   # stale buffer is ignored at mu = 0
    xn, b = o.sgdm_step(x, buf, g, 1e-2, 0.0, np.dtype(np.float32))
    assert np.array_equal(b, g)
    assert np.array_equal(xn, x - np.float32(o.f32(1e-2)) * g)


def pin_sgdm_constant_grad(o):
    """Constant g: buf_k = g (1 - mu^k)/(1 - mu)."""
    g = np.array([1.0, -0.5, 1e-3])
    buf = np.zeros(3)
    x = np.zeros(3)
    mu = o.f32(0.9)
    for k in range(1, 21):
        x, buf = o.sgdm_step(x, buf, g, 1e-2, 0.9, np.dtype(np.float64))
        assert np.allclose(buf, g * (1 - mu ** k) / (1 - mu), rtol=1e-13, atol=0)


# ---------------------------------------------------------------------------
# Global step: special cases named by the paper
# ---------------------------------------------------------------------------

def _lion_step(x, m, g, eta, b1, b2, lam):
    """One Lion step (Appendix A, Algorithm "Lion")."""
    u = b1 * m + (1 - b1) * g
    s = np.sign(u)
    return x - eta * (s + lam * x), b2 * m + (1 - b2) * g, u


def pin_lion(o):
    """n = 1, tau = 1, plain-SGD base: one round is one Lion step with lr eta*gamma on g."""
    rng = np.random.default_rng(6)
    d = 5000
    gamma, eta, b1, b2, lam = 2.0 ** -6, 0.5, 0.9, 0.99, 0.1
    hp = W.HParams(base=W.BASE_SGDM, lr=gamma, mu=0.0, g_b1=b1, g_b2=b2, g_eta=eta, g_wd=lam)
    x0 = rng.standard_normal(d)
    run = o.OracleRun(W.flat_layout(d, 1.0), 1, 1, hp, x0=x0, dtype=np.float64)
    xl, ml = x0.copy(), np.zeros(d)
    for t in range(4):
        g = rng.standard_normal(d).astype(np.float32).astype(np.float64)   # gradients are fp32 inputs
        run.run_round([[g]])
        xl, ml, ul = _lion_step(xl, ml, g, o.f32(eta) * o.f32(gamma), o.f32(b1), o.f32(b2), o.f32(lam))
        safe = np.abs(ul) > 1e-9
        assert np.all(np.abs(run.x - xl)[safe] <= 1e-12 * (1 + np.abs(xl[safe])))
        assert np.allclose(run.m, ml, rtol=1e-12, atol=1e-13)
        xl[~safe], ml[~safe] = run.x[~safe], run.m[~safe]


def pin_signsgd_momentum(o):
    """beta1 = beta2, lambda = 0, tau = 1: u_{t+1} = m_{t+1} and x' = x - eta gamma sign(m_{t+1}), Eq. (signmom)."""
    rng = np.random.default_rng(7)
    d, n = 3000, 3
    hp = W.HParams(base=W.BASE_SGDM, lr=1e-2, mu=0.0, g_b1=0.8, g_b2=0.8, g_eta=0.3, g_wd=0.0)
    run = o.OracleRun(W.flat_layout(d, 1.0), n, 1, hp, x0=rng.standard_normal(d).astype(np.float32))
    for t in range(3):
        x_old = run.x.copy()
        run.run_round([[rng.standard_normal(d).astype(np.float32) for _ in range(n)]])
        assert np.array_equal(run.last_inter["u"], run.m)
        eg = np.float32(o.f32(0.3) * o.f32(1e-2))
        assert np.array_equal(run.x, x_old - eg * (o.sign(run.m) + np.float32(0) * x_old))


def pin_identical_workers(o):
    """Identical workers: the average equals each worker's difference (exact for n = 1, 2, 4)."""
    rng = np.random.default_rng(8)
    d = 4000
    for n in (1, 2, 4):
        hp = W.HParams(base=W.BASE_ADAMW)
        run = o.OracleRun(W.flat_layout(d, 1e-3), n, 3, hp, x0=rng.standard_normal(d).astype(np.float32),
                          with_stats=True)
        for k in range(3):
            g = (rng.standard_normal(d) * 1e-3).astype(np.float32)
            run.local_step([g] * n)
        X0 = run.X[0].copy()
        x_before = run.x.copy()
        run.global_step()
        assert np.array_equal(run.last_inter["delta"], x_before - X0)
        st = run.last_stats[0]
        assert st["drift"] == 0.0 and st["unanimous"] == d


def pin_tau1_pseudo_gradient(o):
    """tau = 1, plain SGD, dyadic data: Delta = gamma * mean_i g_i exactly."""
    rng = np.random.default_rng(9)
    d, n = 1000, 4
    gamma = 2.0 ** -4
    hp = W.HParams(base=W.BASE_SGDM, lr=gamma, mu=0.0)
    x0 = (rng.integers(-64, 64, d) / 16.0).astype(np.float32)
    run = o.OracleRun(W.flat_layout(d, 1.0), n, 1, hp, x0=x0)
    g = [(rng.integers(-32, 32, d) / 8.0).astype(np.float32) for _ in range(n)]
    run.run_round([g])
    want = np.float32(gamma) * (np.sum(np.stack(g).astype(np.float64), axis=0) / n).astype(np.float32)
    assert np.array_equal(run.last_inter["delta"], want)


def pin_sign_range(o):
    rng = np.random.default_rng(10)
    u = rng.standard_normal(10000).astype(np.float32) * 1e-2
    u[:100] = 0.0
    u[100:110] = -0.0
    s = o.sign(u)
    assert set(np.unique(s).tolist()) <= {-1.0, 0.0, 1.0}
    assert np.all(s[:110] == 0) and np.all(s[110:] == np.sign(u[110:]))
    r = o.philox_uniform(np.arange(u.size), 0, 0)
    s2 = o.randomized_sign(u, np.float32(1e-2), r, 1)
    assert set(np.unique(s2).tolist()) <= {-1.0, 0.0, 1.0}
    s1 = o.randomized_sign(u, np.float32(1e-2), r, 2)
    assert np.all(s1[110:] != 0) and np.all(s1[:110] == 0)


def pin_lemma1(o):
    """Lemma 1: E[S_r(v)] = v/B for |v_j| <= B, and E||S_r(v) - v/B||^2 <= d; 10^7 draws."""
    B = np.float32(1e-2)
    v = (np.array([-1.0, -0.7, -0.3, -0.05, 0.0, 0.01, 0.2, 0.5, 0.9, 1.0]) * 1e-2).astype(np.float32)
    draws = 10 ** 6                      # per coordinate; 10^7 draws in total
    d = v.size
    for variant in (1, 2):
        e = np.arange(d * draws, dtype=np.int64)
        r = o.philox_uniform(e, seed=42, t=variant)
        vv = np.tile(v, draws)
        s = o.randomized_sign(vv, B, r, variant).astype(np.float64).reshape(draws, d)
        p = np.minimum(np.abs(v.astype(np.float64)) / np.float64(B), 1.0)
        mean_want = np.sign(v) * p
        var = (p - p ** 2) if variant == 1 else (1 - p ** 2)
        sigma = np.sqrt(np.maximum(var, 1e-12) / draws)
        assert np.all(np.abs(s.mean(axis=0) - mean_want) <= 5 * sigma + 1e-9), (variant, s.mean(axis=0), mean_want)
        sq = ((s - (v.astype(np.float64) / np.float64(B))) ** 2).sum(axis=1).mean()
        assert sq <= d
    # outside the bound p clamps to 1: the deterministic sign
    big = np.array([2e-2, -5e-2], dtype=np.float32)
    r = o.philox_uniform(np.arange(2), 0, 0)
    for variant in (1, 2):
        assert np.array_equal(o.randomized_sign(big, B, r, variant), np.sign(big))


def pin_stats(o):
    """Statistics against numpy reductions and invariants."""
    rng = np.random.default_rng(11)
    tensors = (W.Tensor("a", 300, W.KIND_WEIGHT, 1e-3), W.Tensor("b", 77, W.KIND_BIAS, 1e-4),
               W.Tensor("c", 1000, W.KIND_LN_W, 1e-4))
    hp = W.HParams(base=W.BASE_SGDM, lr=1e-2, mu=0.9, sign_mode=W.RSIGN_ZERO, rsign_B=2e-3)
    run = o.OracleRun(tensors, 3, 2, hp, with_stats=True)
    run.run_round()
    run.run_round()
    inter = run.last_inter
    D = inter["delta"].astype(np.float64)
    st = run.last_stats
    off = 0
    for T, t in enumerate(tensors):
        sl = slice(off, off + t.numel)
        off += t.numel
        assert np.isclose(st[T]["delta_sq"], np.dot(D[sl], D[sl]), rtol=1e-12, atol=0)
        dr = sum(np.sum((dd[sl].astype(np.float64) - D[sl]) ** 2) for dd in inter["diffs"])
        assert np.isclose(st[T]["drift"], dr, rtol=1e-12, atol=0)
        assert st[T]["zero_sign"] == int(np.sum(inter["sg"][sl] == 0))
        assert st[T]["clamped"] == int(np.sum(np.abs(inter["u"][sl]) > np.float32(2e-3)))
        assert 0 <= st[T]["unanimous"] <= t.numel and 0 <= st[T]["flips"] <= t.numel
    # with B at the median of the first round's |u| over the whole model (the first round's
    # u does not depend on B), half of the elements are clamped
    run0 = o.OracleRun(tensors, 3, 2, hp)
    run0.run_round()
    u_all = np.abs(run0.last_inter["u"].astype(np.float64))
    med = float(np.float32(np.sort(u_all)[u_all.size // 2]))
    hp_med = W.HParams(base=W.BASE_SGDM, lr=1e-2, mu=0.9, sign_mode=W.RSIGN_ZERO, rsign_B=med)
    runm = o.OracleRun(tensors, 3, 2, hp_med, with_stats=True)
    runm.run_round()
    assert np.array_equal(runm.last_inter["u"], run0.last_inter["u"])
    n_clamped = sum(s["clamped"] for s in runm.last_stats)
    assert abs(n_clamped - u_all.size / 2) <= 1 + int(np.sum(u_all == med))
    # first round from m = 0: u = c1*Delta with c1 > 0, so no flips
    run1 = o.OracleRun(tensors, 3, 2, hp, with_stats=True)
    run1.run_round()
    assert all(s["flips"] == 0 for s in run1.last_stats)


def pin_subset_mode(o):
    """Element-subset mode computes the same values as the full run."""
    tensors = (W.Tensor("a", 1000, W.KIND_WEIGHT, 1e-3), W.Tensor("b", 33, W.KIND_LN_W, 1e-4),
               W.Tensor("c", 500, W.KIND_BIAS, 1e-4))
    for hp in (W.HParams(grad_dtype=W.BF16),
               W.HParams(base=W.BASE_SGDM, lr=1e-2, sign_mode=W.RSIGN_PM, rsign_B=1e-3)):
        full = o.OracleRun(tensors, 2, 3, hp)
        sub_e = np.array([0, 5, 999, 1000, 1032, 1033, 1500, 1532])
        sub = o.OracleRun(tensors, 2, 3, hp, elems=sub_e)
        for _ in range(2):
            full.run_round()
            sub.run_round()
        assert np.array_equal(full.x[sub_e], sub.x)
        assert np.array_equal(full.m[sub_e], sub.m)
        assert np.array_equal(full.opt_m[1][sub_e], sub.opt_m[1])


def pin_fp32_vs_fp64(o):
    """The fp32 iteration stays within 1e-6 (1 + |x|) of the fp64 twin; sign flips only near u = 0."""
    tensors = W.flat_layout(20000, 1e-2)
    for hp in (W.HParams(), W.HParams(base=W.BASE_SGDM, lr=1e-2, mu=0.9)):
        a = o.OracleRun(tensors, 4, 4, hp, dtype=np.float32)
        b = o.OracleRun(tensors, 4, 4, hp, dtype=np.float64)
        diverged = np.zeros(20000, dtype=bool)
        c2 = (1 - o.f32(hp.g_b2)) / o.f32(hp.lr)
        for t in range(3):
            a.run_round()
            b.run_round()
            ua, ub = a.last_inter["u"], b.last_inter["u"]
            mism = o.sign(ua) != o.sign(ub)
            assert np.all(np.abs(ub[mism]) <= 1e-6 * np.max(np.abs(ub)))
            diverged |= mism
            # elements whose sign decisions always agreed agree to the stated tolerance
            ok = ~diverged
            assert np.all(np.abs(a.x - b.x)[ok] <= 1e-6 * (1 + np.abs(b.x[ok])))
            # m inherits the rounding of the fp32 worker models, about one ulp of x per local
            # step, scaled by (1-beta2)/gamma: the bound accumulates over rounds
            ulp_x = float(np.spacing(np.float32(np.max(np.abs(b.x)))))
            tol_m = (t + 1) * c2 * 4 * ulp_x + 1e-6 * np.abs(b.m[ok])
            assert np.all(np.abs(a.m - b.m)[ok] <= tol_m)


# ---------------------------------------------------------------------------
# Global-step variants of the ablations (Sec. 5) against textbook special cases
# ---------------------------------------------------------------------------

def _one_worker_sgd_rounds(o, hp, rounds, rng, d=3000):
    """n = 1, tau = 1, plain-SGD local step: the pseudo-gradient (x - x_1)/gamma is the gradient itself
    (up to the rounding of x - gamma g).  Returns the run, the initial model and the gradients used."""
    x0 = rng.standard_normal(d)
    run = o.OracleRun(W.flat_layout(d, 1.0), 1, 1, hp, x0=x0, dtype=np.float64)
    gs = [rng.standard_normal(d).astype(np.float32).astype(np.float64) for _ in range(rounds)]
    return run, x0, gs


def pin_slowmo_heavy_ball(o):
    """SlowMo with one worker and one plain-SGD step is heavy-ball momentum on g with lr alpha*gamma
    (torch.optim.SGD(momentum=beta))."""
    import torch
    rng = np.random.default_rng(12)
    gamma, beta, alpha = 2.0 ** -4, 0.7, 0.5
    hp = W.HParams(base=W.BASE_SGDM, lr=gamma, mu=0.0, g_b1=beta, g_eta=alpha, global_mode=W.GLOBAL_SLOWMO)
    run, x0, gs = _one_worker_sgd_rounds(o, hp, 5, rng)
    p = torch.tensor(x0.copy(), dtype=torch.float64, requires_grad=True)
    opt = torch.optim.SGD([p], lr=o.f32(alpha) * o.f32(gamma), momentum=o.f32(beta), dampening=0.0, foreach=False)
    for g in gs:
        run.run_round([[g]])
        p.grad = torch.tensor(g)
        opt.step()
        assert np.allclose(run.x, p.detach().numpy(), rtol=1e-12, atol=1e-13)


def pin_lookahead_slow_weights(o):
    """Lookahead with beta1 = beta2 = 0 is Zhang et al.'s slow-weight update x' = x + eta (xbar - x);
    with eta = 1 it is plain model averaging (local SGD)."""
    rng = np.random.default_rng(13)
    d, n = 2000, 3
    for eta in (0.5, 1.0):
        hp = W.HParams(base=W.BASE_SGDM, lr=2.0 ** -5, mu=0.0, g_b1=0.0, g_b2=0.0, g_eta=eta,
                       global_mode=W.GLOBAL_LOOKAHEAD)
        run = o.OracleRun(W.flat_layout(d, 1.0), n, 2, hp, x0=rng.standard_normal(d), dtype=np.float64)
        for _ in range(2):
            for k in range(2):
                run.local_step([rng.standard_normal(d).astype(np.float32) for _ in range(n)])
            xbar = np.mean(np.stack(run.X), axis=0)
            x = run.x.copy()
            run.global_step()
            assert np.allclose(run.x, x + o.f32(eta) * (xbar - x), rtol=1e-12, atol=1e-14)


def pin_signed_slowmo_signsgd(o):
    """Signed SlowMo with beta1 = 0 is signSGD on the averaged pseudo-gradient: x' = x - eta sign(x - xbar)."""
    rng = np.random.default_rng(14)
    d, n = 2000, 2
    hp = W.HParams(base=W.BASE_SGDM, lr=2.0 ** -5, mu=0.0, g_b1=0.0, g_b2=0.9, g_eta=0.25,
                   global_mode=W.GLOBAL_SIGNED_SLOWMO)
    run = o.OracleRun(W.flat_layout(d, 1.0), n, 1, hp, x0=rng.standard_normal(d), dtype=np.float64)
    for _ in range(3):
        run.local_step([rng.standard_normal(d).astype(np.float32) for _ in range(n)])
        xbar = np.mean(np.stack(run.X), axis=0)
        x = run.x.copy()
        run.global_step()
        assert np.allclose(run.x, x - 0.25 * np.sign(x - xbar), rtol=1e-14, atol=1e-14)


def pin_global_adamw_vs_torch(o):
    """Global AdamW with one worker and one plain-SGD step is AdamW on g with lr eta (torch.optim.AdamW)."""
    import torch
    rng = np.random.default_rng(15)
    gamma, eta = 2.0 ** -4, 1e-2
    hp = W.HParams(base=W.BASE_SGDM, lr=gamma, mu=0.0, g_b1=0.9, g_b2=0.95, g_eps=1e-8, g_eta=eta, g_wd=0.1,
                   global_mode=W.GLOBAL_ADAMW)
    run, x0, gs = _one_worker_sgd_rounds(o, hp, 6, rng)
    p = torch.tensor(x0.copy(), dtype=torch.float64, requires_grad=True)
    opt = torch.optim.AdamW([p], lr=o.f32(eta), betas=(o.f32(0.9), o.f32(0.95)), eps=o.f32(1e-8),
                            weight_decay=o.f32(0.1), foreach=False)
    for g in gs:
        run.run_round([[g]])
        p.grad = torch.tensor(g)
        opt.step()
        assert np.allclose(run.x, p.detach().numpy(), rtol=1e-10, atol=1e-12)


def pin_local_state_across_rounds(o):
    """Algorithm 1 synchronises only the model.  By default a worker's AdamW keeps its moments and its
    step count across rounds: one torch.optim.AdamW per worker for the whole run.  With
    FLAG_RESET_LOCAL_STATE every round starts a new torch.optim.AdamW per worker.  Between rounds the
    oracle's global step (itself pinned by the worked example) averages and synchronises."""
    import torch
    rng = np.random.default_rng(21)
    d, n, tau, rounds = 512, 3, 3, 3
    finals = []
    for flags in (0, W.FLAG_RESET_LOCAL_STATE):
        hp = W.HParams(flags=flags)
        x0 = rng.standard_normal(d).astype(np.float32)
        run = o.OracleRun(W.flat_layout(d, 1e-3), n, tau, hp, x0=x0, dtype=np.float64)
        x, m = x0.astype(np.float64), np.zeros(d)
        params = [torch.tensor(x.copy(), dtype=torch.float64, requires_grad=True) for _ in range(n)]

        def new_opt(p):
            return torch.optim.AdamW([p], lr=o.f32(hp.lr), betas=(o.f32(hp.b1), o.f32(hp.b2)),
                                     eps=o.f32(hp.eps), weight_decay=o.f32(hp.wd), foreach=False)

        opts = [new_opt(p) for p in params]
        for t in range(rounds):
            grads = [[(rng.standard_normal(d) * 1e-3).astype(np.float32) for _ in range(n)] for _ in range(tau)]
            if flags and t:
                opts = [new_opt(p) for p in params]
            for k in range(tau):
                for i in range(n):
                    params[i].grad = torch.tensor(grads[k][i].astype(np.float64))
                    opts[i].step()
            X = [p.detach().numpy().copy() for p in params]
            x, m, _ = o.global_step(x, m, X, hp.lr, hp.g_b1, hp.g_b2, hp.g_eta, np.full(d, o.f32(hp.g_wd)),
                                    0, hp.rsign_B, None, np.dtype(np.float64))
            with torch.no_grad():
                for p in params:
                    p.copy_(torch.from_numpy(x))
            run.run_round(grads)
            assert np.max(np.abs(run.x - x)) <= 1e-12 * (1 + np.max(np.abs(x))), (flags, t)
            assert np.max(np.abs(run.m - m)) <= 1e-9 * (1e-6 + np.max(np.abs(m))), (flags, t)
        finals.append(run.opt_m[0].copy())
    assert np.all(finals[1] == 0.0) and np.any(finals[0] != 0.0)


def pin_cosine_schedule(o):
    """Closed-form points of warm-up + cosine decay: P/W at step 0, P at the end of the warm-up,
    (P + F)/2 halfway through the decay, F at and after the last step; monotone decay."""
    P, r, W_, S = 6e-4, 0.05, 2000, 100000
    F = r * P
    assert np.isclose(o.cosine_gamma(P, r, W_, S, 0), P / W_, rtol=1e-15)
    assert np.isclose(o.cosine_gamma(P, r, W_, S, W_ - 1), P, rtol=1e-15)
    assert np.isclose(o.cosine_gamma(P, r, W_, S, W_), P, rtol=1e-15)
    assert np.isclose(o.cosine_gamma(P, r, W_, S, (W_ + S) // 2), (P + F) / 2, rtol=1e-12)
    assert np.isclose(o.cosine_gamma(P, r, W_, S, S), F, rtol=1e-15)
    assert np.isclose(o.cosine_gamma(P, r, W_, S, 10 * S), F, rtol=1e-15)
    vals = [o.cosine_gamma(P, r, W_, S, s) for s in range(W_, S + 1, 997)]
    assert all(a >= b for a, b in zip(vals, vals[1:]))


PINS = [pin_worked_example, pin_stats_example, pin_splitmix64, pin_philox, pin_philox_uniform_mapping, pin_bf16,
        pin_uniform24, pin_hash_fields, pin_synthetic_grad, pin_adamw_vs_torch, pin_adamw_constant_grad,
        pin_adamw_first_step_fp32, pin_sgdm_vs_torch, pin_sgd_plain_exact, pin_sgdm_constant_grad,
        pin_lion, pin_signsgd_momentum, pin_identical_workers, pin_tau1_pseudo_gradient,
        pin_sign_range, pin_lemma1, pin_stats, pin_subset_mode, pin_fp32_vs_fp64,
        pin_slowmo_heavy_ball, pin_lookahead_slow_weights, pin_signed_slowmo_signsgd, pin_global_adamw_vs_torch,
        pin_cosine_schedule, pin_local_state_across_rounds]
