"""CPU oracle for one global round of distributed sign momentum with local steps.

TEST INFRASTRUCTURE.  Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference arms of ``bench.py`` may import this module.  The
library (``paper_2411_17866_gb300``) never imports it, and it imports
nothing from the library: the two share no code.  Only the workload tables
in ``workloads.py`` (pure data) serve both.

What it computes (arXiv 2411.17866):

* Algorithm 1 (distributed sign momentum): tau local base-optimizer steps
  per worker, Eq. (local-steps); the average of the worker models (the
  all-reduce); the global update Eqs. (ut-update), (model-update) and
  (mom-update); and the reset of every worker to the new global model.
* Base optimizers of Appendix A: AdamW (Algorithm "AdamW") and Polyak's
  momentum (Algorithm "Polyak"), which is plain SGD, Eq. (base-sgd), at mu=0.
* The randomized sign operators of Sec. 4.1, Eqs. (rand-sign-1) and
  (rand-sign-2), driven by Philox4x32-10.
* Per-tensor round statistics (squared norm of the averaged pseudo-gradient,
  worker drift, sign counts), accumulated in float64 in element order.
* The global-step variants of the ablations (Sec. 5): SlowMo (Appendix A,
  Algorithm "SlowMo"), signed SlowMo and Lookahead (Sec. 5, ablation
  studies), and the global AdamW step (Appendix, Algorithm "global AdamW").
* Both readings of what Algorithm 1 leaves open about the base optimizer's
  state at a synchronisation: kept across rounds (the default), or restarted
  from zero every round (FLAG_RESET_LOCAL_STATE).

Precision.  The paper fixes no precision.  Every function is generic in the
float dtype: ``np.float32`` is the canonical mode whose expression trees the
CUDA path reproduces (one rounding per operation, no contraction), and
``np.float64`` is the high-precision twin used to measure fp32 rounding.
Hyper-parameters are the fp32 values in both modes.  Derived scalars
(bias corrections, (1-beta)/gamma, eta*gamma) are computed in float64 from
those fp32 values and rounded once to the working dtype.

Every step is elementwise, so the oracle can run on any subset of element
indices ("element-subset mode"); the full model is the subset of all
indices.

Parity pins: each function here is pinned by a test in
``tests/test_oracle_pins.py`` against something other than itself (the
exact worked example, closed forms, library routines, published test
vectors, invariants, Lemma 1).  The per-tensor statistics have no printed
values in the paper; they are pinned by hand-computed values of two d = 8
global steps (tests/golden/worked_example_d8.json, stats_example_d8.json),
by invariants and by numpy reductions.  The C++ oracle (dsm_oracle.cpp)
computes the same values bit for bit.
"""
from __future__ import annotations

import numpy as np

U64 = np.uint64
U32 = np.uint32
MASK32 = 0xFFFFFFFF
MASK64 = 0xFFFFFFFFFFFFFFFF

# ---------------------------------------------------------------------------
# Counter-based generators, each written from its published definition.
# ---------------------------------------------------------------------------

# SplitMix64 (Steele, Lea, Flood, "Fast splittable pseudorandom number
# generators", OOPSLA 2014): the generator's state advances by the odd
# constant GOLDEN_GAMMA and each output is the state passed through the
# 64-bit finaliser "variant 13" of Stafford's mixer study.
GOLDEN_GAMMA = 0x9E3779B97F4A7C15
_MIX_C1 = 0xBF58476D1CE4E5B9
_MIX_C2 = 0x94D049BB133111EB

STREAM_STEP = 0     # the step term of the synthetic gradient
STREAM_WORKER = 1   # the worker (heterogeneity) term
STREAM_INIT = 2     # the initial model x_{0,0}


def splitmix64_mix(z):
    """Stafford variant-13 finaliser on uint64 arrays (wrapping arithmetic)."""
    z = np.asarray(z, dtype=U64)
    z = (z ^ (z >> U64(30))) * U64(_MIX_C1)
    z = (z ^ (z >> U64(27))) * U64(_MIX_C2)
    return z ^ (z >> U64(31))


def splitmix64_output(state, j):
    """Output number j (j >= 1) of a SplitMix64 generator seeded with ``state``."""
    state = np.asarray(state, dtype=U64)
    j = np.asarray(j, dtype=U64)
    return splitmix64_mix(state + j * U64(GOLDEN_GAMMA))


def hash_key(seed: int, stream: int, idx: int):
    """Key of the draw family (seed, stream, idx): SplitMix64(seed) output 1 + stream*2^40 + idx."""
    j = (1 + (int(stream) << 40) + int(idx)) & MASK64
    return splitmix64_output(np.array([seed & MASK64], dtype=U64), np.array([j], dtype=U64))[0]


def hash24(seed: int, stream: int, idx: int, elems):
    """24-bit draw of element e from SplitMix64(key(seed, stream, idx)).

    Each 64-bit output serves two consecutive elements: output floor(e/2)+1
    gives bits 63..40 to the even element and bits 39..16 to the odd one.
    """
    key = hash_key(seed, stream, idx)
    e = np.asarray(elems, dtype=U64)
    h = splitmix64_output(np.full(e.shape, key, dtype=U64), (e >> U64(1)) + U64(1))
    shift = np.where((e & U64(1)) == 0, U64(40), U64(16))
    return (h >> shift) & U64(0xFFFFFF)


def uniform24(seed: int, stream: int, idx: int, elems) -> np.ndarray:
    """u = h * 2^-24 in [0, 1); exact in float32 because h < 2^24."""
    return hash24(seed, stream, idx, elems).astype(np.float32) * np.float32(2.0 ** -24)


def bf16_round(x) -> np.ndarray:
    """Round float32 to the nearest bfloat16, ties to even; returns float32 values.

    bfloat16 keeps the top 16 bits of the float32 encoding; round-to-nearest-
    even adds 0x7FFF plus the lowest kept bit before truncating.  NaN stays a
    (quiet) NaN.
    """
    x = np.asarray(x, dtype=np.float32)
    b = x.view(U32).astype(U64)
    kept_lsb = (b >> U64(16)) & U64(1)
    r = ((b + U64(0x7FFF) + kept_lsb) >> U64(16)) << U64(16)
    nan = np.isnan(x)
    r = np.where(nan, (b | U64(0x00400000)) & U64(0xFFFF0000), r)
    return (r & U64(MASK32)).astype(U32).view(np.float32)


def synthetic_grad(elems, scale, seed: int, step: int, worker: int, grad_dtype: int) -> np.ndarray:
    """Synthetic gradient standing in for the backward pass (float32).

    g = s*(u(seed, step, e) - 1/2) + s2*(u(seed, worker, e) - 1/2), with
    s2 = fp32(0.1f * s), evaluated left to right with one rounding per
    operation; bf16 gradients are the float32 value rounded to nearest even.
    """
    scale = np.asarray(scale, dtype=np.float32)
    s2 = (np.float32(0.1) * scale).astype(np.float32)
    half = np.float32(0.5)
    u_step = uniform24(seed, STREAM_STEP, step, elems)
    u_worker = uniform24(seed, STREAM_WORKER, worker, elems)
    a = scale * (u_step - half)
    b = s2 * (u_worker - half)
    g = (a + b).astype(np.float32)
    if grad_dtype == 1:
        g = bf16_round(g)
    return g


def init_x0(elems, kinds, seed: int) -> np.ndarray:
    """Initial global model x_{0,0} (the paper gives no initialisation).

    Weights: 0.02f * (2u - 1) with u = uniform24(seed, STREAM_INIT, 0, e);
    LayerNorm weights: 1; biases and LayerNorm biases: 0.
    """
    kinds = np.asarray(kinds)
    u = uniform24(seed, STREAM_INIT, 0, elems)
    w = np.float32(0.02) * (np.float32(2.0) * u - np.float32(1.0))
    x = np.zeros(u.shape, dtype=np.float32)
    x = np.where(kinds == 0, w, x)
    x = np.where(kinds == 2, np.float32(1.0), x)
    return x.astype(np.float32)


# Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as
# easy as 1, 2, 3", SC 2011): ten rounds of a two-multiplier S-box on a
# 4x32-bit counter, with a Weyl key schedule on the 2x32-bit key.
PHILOX_M0 = 0xD2511F53
PHILOX_M1 = 0xCD9E8D57
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85


def _mulhilo32(a: int, b):
    p = np.asarray(b, dtype=U64) * U64(a)
    return (p >> U64(32)) & U64(MASK32), p & U64(MASK32)


def philox4x32_10(c0, c1, c2, c3, k0, k1):
    """Philox4x32-10 block function on uint32 arrays; returns four uint32 arrays."""
    c = [np.asarray(v, dtype=U64) & U64(MASK32) for v in (c0, c1, c2, c3)]
    k0 = np.asarray(k0, dtype=U64) & U64(MASK32)
    k1 = np.asarray(k1, dtype=U64) & U64(MASK32)
    for r in range(10):
        if r > 0:
            k0 = (k0 + U64(PHILOX_W0)) & U64(MASK32)
            k1 = (k1 + U64(PHILOX_W1)) & U64(MASK32)
        hi0, lo0 = _mulhilo32(PHILOX_M0, c[0])
        hi1, lo1 = _mulhilo32(PHILOX_M1, c[2])
        c = [hi1 ^ c[1] ^ k0, lo1, hi0 ^ c[3] ^ k1, lo0]
    return tuple(v.astype(U32) for v in c)


def philox_uniform(elems, seed: int, t: int) -> np.ndarray:
    """r_e in [0, 1) for the randomized sign of round t.

    Key (seed mod 2^32, t); counter (floor(e/4) low word, high word, 0, 0);
    element e takes output word e mod 4 and keeps its top 24 bits:
    r = (word >> 8) * 2^-24, exact in float32.
    """
    e = np.asarray(elems, dtype=U64)
    q = e >> U64(2)
    words = philox4x32_10(q & U64(MASK32), q >> U64(32), np.zeros_like(q), np.zeros_like(q),
                          np.full(e.shape, seed & MASK32, dtype=U64),
                          np.full(e.shape, t & MASK32, dtype=U64))
    w = np.choose((e & U64(3)).astype(np.int64), words)
    return (w >> U32(8)).astype(np.float32) * np.float32(2.0 ** -24)


# ---------------------------------------------------------------------------
# Scalars
# ---------------------------------------------------------------------------

def f32(v) -> float:
    """The float32 value of a hyper-parameter, as a Python float (exact)."""
    return float(np.float32(v))


def beta_power(beta: float, j: int) -> float:
    """beta^j in float64 by j successive multiplications of the fp32 beta."""
    p = 1.0
    b = f32(beta)
    for _ in range(j):
        p *= b
    return p


def cosine_gamma(peak: float, final_ratio: float, warmup: int, total: int, step: int) -> float:
    """Learning rate at local step ``step`` of the paper's schedule (Sec. 5, implementations):
    linear warm-up over ``warmup`` steps to ``peak``, then a cosine decay to final_ratio * peak at
    ``total`` steps, constant after.  Algorithm 1's gamma_t of round t is the value at step t*tau."""
    final = final_ratio * peak
    if step < warmup:
        return peak * (step + 1) / warmup
    if step >= total:
        return final
    ratio = (step - warmup) / (total - warmup)
    return final + 0.5 * (1.0 + np.cos(np.pi * ratio)) * (peak - final)


# ---------------------------------------------------------------------------
# Base optimizers (Appendix A) as local steps, Eq. (local-steps)
# ---------------------------------------------------------------------------

def adamw_step(x, m, v, g, j: int, lr, b1, b2, eps, wd_e, dt):
    """One AdamW step (Appendix A, Algorithm "AdamW") at step count j >= 1.

    m <- b1 m + (1-b1) g;  v <- b2 v + (1-b2) g*g;
    mhat = m / (1 - b1^j);  vhat = v / (1 - b2^j);
    x <- x - lr (mhat / (sqrt(vhat) + eps) + wd x)
    ``wd_e`` is the per-element decay (wd for decayed tensors, else 0).
    Returns the new (x, m, v).
    """
    T = dt.type
    b1_, b2_ = T(f32(b1)), T(f32(b2))
    omb1, omb2 = T(1.0 - f32(b1)), T(1.0 - f32(b2))
    bc1 = T(1.0 - beta_power(b1, j))
    bc2 = T(1.0 - beta_power(b2, j))
    lr_, eps_ = T(f32(lr)), T(f32(eps))
    g = g.astype(dt)
    m = b1_ * m + omb1 * g
    v = b2_ * v + omb2 * (g * g)
    mhat = m / bc1
    vhat = v / bc2
    x = x - lr_ * (mhat / (np.sqrt(vhat) + eps_) + wd_e * x)
    return x, m, v


def sgdm_step(x, buf, g, lr, mu, dt):
    """One Polyak-momentum step (Appendix A, Algorithm "Polyak"): buf <- mu buf + g; x <- x - lr buf.

    mu = 0 gives plain SGD, Eq. (base-sgd).  Returns the new (x, buf).
    """
    T = dt.type
    buf = T(f32(mu)) * buf + g.astype(dt)
    x = x - T(f32(lr)) * buf
    return x, buf


# ---------------------------------------------------------------------------
# Global step of Algorithm 1
# ---------------------------------------------------------------------------

def sign(v):
    """sign(v) = (v > 0) - (v < 0): 0 at +-0 and at NaN (the paper leaves sign(0) undefined)."""
    v = np.asarray(v)
    return ((v > 0).astype(v.dtype) - (v < 0).astype(v.dtype))


def randomized_sign(u, B, r, variant: int):
    """Randomized sign S_r(u) with bound B and uniforms r (Sec. 4.1).

    p = min(|u|/B, 1).  Eq. (rand-sign-2) (variant 1): sign(u) if r < p else 0.
    Eq. (rand-sign-1) (variant 2): sign(u) if r < 1/2 + p/2 else -sign(u).
    Where |u| > B (outside the Lemma's assumption) p is clamped to 1.
    """
    dt = u.dtype.type
    s = sign(u)
    p = np.minimum(np.abs(u) / dt(B), dt(1.0))
    if variant == 1:
        return np.where(r < p, s, dt(0.0)).astype(u.dtype)
    if variant == 2:
        q = dt(0.5) + dt(0.5) * p
        return np.where(r < q, s, -s).astype(u.dtype)
    raise ValueError("variant must be 1 (rand-sign-2) or 2 (rand-sign-1)")


def global_step(x, m, X, gamma, b1, b2, eta, lam_e, sign_mode: int, B, r, dt):
    """Global sign-momentum step of Algorithm 1 on one set of elements.

    Delta = (1/n) sum_i (x - x_i), summed over i = 0..n-1 in order
        (the all-reduce average, written as the average of the worker
        differences: x - (1/n) sum_i x_i in exact arithmetic);
    u = b1 m + ((1-b1)/gamma) Delta                         Eq. (ut-update)
    x' = x - eta gamma (sign(u) + lam x)                   Eq. (model-update)
    m' = b2 m + ((1-b2)/gamma) Delta                        Eq. (mom-update)
    every worker replica <- x'                              (synchronise)
    ``sign_mode`` 0: deterministic sign; 1: Eq. (rand-sign-2); 2: Eq. (rand-sign-1)
    with uniforms ``r``.  Returns x', m' and a dict of per-element
    intermediates (Delta, u, the applied sign, the worker differences).
    """
    T = dt.type
    c1 = T((1.0 - f32(b1)) / f32(gamma))
    c2 = T((1.0 - f32(b2)) / f32(gamma))
    eg = T(f32(eta) * f32(gamma))
    delta, diffs = worker_average(x, X, dt)
    u = T(f32(b1)) * m + c1 * delta
    if sign_mode == 0:
        sg = sign(u)
    else:
        sg = randomized_sign(u, f32(B), r, sign_mode)
    x_new = x - eg * (sg + lam_e * x)
    m_new = T(f32(b2)) * m + c2 * delta
    return x_new, m_new, {"delta": delta, "u": u, "sg": sg, "diffs": diffs}


GLOBAL_SIGN_MOMENTUM = 0   # Algorithm 1
GLOBAL_SLOWMO = 1          # Appendix A, Algorithm "SlowMo"
GLOBAL_SIGNED_SLOWMO = 2   # Sec. 5, signed SlowMo
GLOBAL_LOOKAHEAD = 3       # Sec. 5, Lookahead (Eq. (model-update) replaced)
GLOBAL_ADAMW = 4           # Appendix, Algorithm "global AdamW"

FLAG_RESET_LOCAL_STATE = 2  # hp.flags bit: restart each worker's optimizer every round


def worker_average(x, X, dt):
    """Delta = (1/n) sum_i (x - x_i), summed over i = 0..n-1 in order (the all-reduce average)."""
    n = len(X)
    diffs = [x - X[i] for i in range(n)]
    acc = np.zeros_like(x)
    for i in range(n):
        acc = acc + diffs[i]
    return acc / dt.type(n), diffs


def global_step_slowmo(x, m, X, gamma, beta, alpha, dt):
    """SlowMo (Appendix A): exact averaging; u <- beta u + (1/gamma)(x - xbar); x <- x - alpha gamma u.

    ``m`` holds the slow momentum u.  Returns x', u', intermediates.
    """
    T = dt.type
    delta, diffs = worker_average(x, X, dt)
    inv_g = T(1.0 / f32(gamma))
    u = T(f32(beta)) * m + inv_g * delta
    x_new = x - T(f32(alpha) * f32(gamma)) * u
    return x_new, u, {"delta": delta, "u": u, "sg": sign(u), "diffs": diffs}


def global_step_signed_slowmo(x, m, X, gamma, b1, b2, eta, dt):
    """Signed SlowMo (Sec. 5): u = b1 m + ((1-b1)/gamma) sign(x - xbar); x' = x - eta gamma u;
    the momentum update, Eq. (mom-update), is kept: m' = b2 m + ((1-b2)/gamma)(x - xbar)."""
    T = dt.type
    delta, diffs = worker_average(x, X, dt)
    c1 = T((1.0 - f32(b1)) / f32(gamma))
    c2 = T((1.0 - f32(b2)) / f32(gamma))
    sd = sign(delta)
    u = T(f32(b1)) * m + c1 * sd
    x_new = x - T(f32(eta) * f32(gamma)) * u
    m_new = T(f32(b2)) * m + c2 * delta
    return x_new, m_new, {"delta": delta, "u": u, "sg": sd, "diffs": diffs}


def global_step_lookahead(x, m, X, gamma, b1, b2, eta, dt):
    """Lookahead (Sec. 5): Algorithm 1 with Eq. (model-update) replaced by x' = x - eta gamma u."""
    T = dt.type
    delta, diffs = worker_average(x, X, dt)
    c1 = T((1.0 - f32(b1)) / f32(gamma))
    c2 = T((1.0 - f32(b2)) / f32(gamma))
    u = T(f32(b1)) * m + c1 * delta
    x_new = x - T(f32(eta) * f32(gamma)) * u
    m_new = T(f32(b2)) * m + c2 * delta
    return x_new, m_new, {"delta": delta, "u": u, "sg": sign(u), "diffs": diffs}


def global_step_adamw(x, m, v, X, gamma, t: int, b1, b2, eps, eta, lam_e, dt):
    """Global AdamW with local steps (Appendix, Algorithm "global AdamW") at round t (0-based).

    g = (1/gamma)(x - xbar); m <- b1 m + (1-b1) g; v <- b2 v + (1-b2) g*g;
    mhat = m/(1 - b1^(t+1)); vhat = v/(1 - b2^(t+1));
    x' = x - eta (mhat/(sqrt(vhat) + eps) + lam x).
    """
    T = dt.type
    delta, diffs = worker_average(x, X, dt)
    g = T(1.0 / f32(gamma)) * delta
    m_new = T(f32(b1)) * m + T(1.0 - f32(b1)) * g
    v_new = T(f32(b2)) * v + T(1.0 - f32(b2)) * (g * g)
    mhat = m_new / T(1.0 - beta_power(b1, t + 1))
    vhat = v_new / T(1.0 - beta_power(b2, t + 1))
    x_new = x - T(f32(eta)) * (mhat / (np.sqrt(vhat) + T(f32(eps))) + lam_e * x)
    return x_new, m_new, v_new, {"delta": delta, "u": m_new, "sg": sign(m_new), "diffs": diffs}


def round_stats(inter, tensor_of, num_tensors: int, sign_mode: int, B) -> list:
    """Per-tensor statistics of one global step, accumulated in float64 in element order.

    delta_sq  = sum_e Delta_e^2
    drift     = sum_e sum_i ((x_e - x_i,e) - Delta_e)^2      (worker drift around the mean)
    zero_sign = #{applied sign = 0}
    flips     = #{sign(u_e) != sign(Delta_e)}  (momentum overrides the pseudo-gradient)
    unanimous = #{for all i: sign(x_e - x_i,e) = sign(Delta_e)}
    clamped   = #{|u_e| > B} in the randomized modes, else 0
    """
    delta = inter["delta"].astype(np.float64)
    u = inter["u"]
    sg = inter["sg"]
    diffs = [dd.astype(np.float64) for dd in inter["diffs"]]
    tensor_of = np.asarray(tensor_of)
    out = []
    sd = sign(inter["delta"])
    unanimous = np.ones(delta.shape, dtype=bool)
    for dd_, dd in zip(inter["diffs"], diffs):
        unanimous &= sign(dd_) == sd
    drift_e = np.zeros(delta.shape, dtype=np.float64)
    for dd in diffs:
        drift_e += (dd - delta) ** 2
    zero_e = sg == 0
    flip_e = sign(u) != sd
    clamp_e = (np.abs(u) > np.asarray(f32(B), dtype=u.dtype)) if sign_mode != 0 else np.zeros(delta.shape, bool)
    for T in range(num_tensors):
        sel = tensor_of == T
        # np.cumsum adds strictly left to right, i.e. in element order
        sq = delta[sel] ** 2
        dsq = float(np.cumsum(sq)[-1]) if sq.size else 0.0
        dr = float(np.cumsum(drift_e[sel])[-1]) if sq.size else 0.0
        out.append({
            "delta_sq": dsq,
            "drift": dr,
            "zero_sign": int(np.count_nonzero(zero_e[sel])),
            "flips": int(np.count_nonzero(flip_e[sel])),
            "unanimous": int(np.count_nonzero(unanimous[sel])),
            "clamped": int(np.count_nonzero(clamp_e[sel])),
        })
    return out


# ---------------------------------------------------------------------------
# Whole rounds
# ---------------------------------------------------------------------------

class OracleRun:
    """State of Algorithm 1 over a set of elements of one parameter layout.

    tensors: sequence with .numel, .kind, .grad_scale, .wd (see workloads.py)
    n, tau: workers and local steps per round; hp: hyper-parameters.
    elems: logical element indices to simulate (None = all of them).
    x0: initial model on those elements (None = the hash initialisation).
    dtype: np.float32 (canonical) or np.float64 (twin).
    first_element: the layout's first element within a larger model of
    which it is a contiguous part (a parameter shard); the synthetic draws
    and the randomized sign take element e as element first_element + e of
    that model.  0 for a whole model.

    Worker optimizer states persist across rounds and are never averaged;
    only the model is synchronised (Algorithm 1, last step).  AdamW's step
    count is j = t*tau + k + 1.  Algorithm 1 leaves the base optimizer's
    state at a synchronisation open; with hp.flags & FLAG_RESET_LOCAL_STATE
    every round instead restarts each worker's optimizer from scratch: its
    state is zero at the start of the round and j = k + 1.
    """

    def __init__(self, tensors, n, tau, hp, elems=None, x0=None, dtype=np.float32,
                 with_stats=False, first_element=0):
        self.tensors = list(tensors)
        self.n, self.tau, self.hp = int(n), int(tau), hp
        self.dt = np.dtype(dtype)
        numels = np.array([t.numel for t in self.tensors], dtype=np.int64)
        self.starts = np.concatenate([[0], np.cumsum(numels)[:-1]]).astype(np.int64)
        self.d = int(numels.sum())
        if elems is None:
            elems = np.arange(self.d, dtype=np.int64)
        self.elems = np.asarray(elems, dtype=np.int64)
        self.tensor_of = np.searchsorted(self.starts, self.elems, side="right") - 1
        # the elements' indices in the larger model that the layout is a part of: the generators and the
        # randomized sign's counter use them (first_element = 0 for a whole model)
        self.gidx = self.elems + np.int64(first_element)
        self.scale = np.array([t.grad_scale for t in self.tensors], dtype=np.float32)[self.tensor_of]
        kinds = np.array([t.kind for t in self.tensors])[self.tensor_of]
        wdflag = np.array([t.wd for t in self.tensors])[self.tensor_of] != 0
        T = self.dt.type
        self.wd_local = np.where(wdflag, T(f32(hp.wd)), T(0.0)).astype(self.dt)
        self.wd_global = np.where(wdflag, T(f32(hp.g_wd)), T(0.0)).astype(self.dt)
        if x0 is None:
            x0 = init_x0(self.gidx, kinds, hp.seed)
        self.x = np.asarray(x0).astype(self.dt)
        self.m = np.zeros_like(self.x)
        self.X = [self.x.copy() for _ in range(self.n)]
        self.opt_m = [np.zeros_like(self.x) for _ in range(self.n)]
        self.opt_v = [np.zeros_like(self.x) for _ in range(self.n)] if hp.base == 0 else None
        self.global_mode = getattr(hp, "global_mode", GLOBAL_SIGN_MOMENTUM)
        self.gv = np.zeros_like(self.x) if self.global_mode == GLOBAL_ADAMW else None
        self.reset_local = bool(getattr(hp, "flags", 0) & FLAG_RESET_LOCAL_STATE)
        self.t = 0
        self.k = 0
        self.gamma = hp.lr
        self.with_stats = with_stats
        self.last_stats = None
        self.last_inter = None

    def grads(self, step: int, worker: int) -> np.ndarray:
        return synthetic_grad(self.gidx, self.scale, self.hp.seed, step, worker, self.hp.grad_dtype)

    def local_step(self, grads=None):
        """Local step k of the current round for every worker, Eq. (local-steps)."""
        assert self.k < self.tau
        step = self.t * self.tau + self.k
        j = self.k + 1 if self.reset_local else step + 1
        hp = self.hp
        for i in range(self.n):
            g = self.grads(step, i) if grads is None else np.asarray(grads[i], dtype=np.float32)
            if hp.base == 0:
                self.X[i], self.opt_m[i], self.opt_v[i] = adamw_step(
                    self.X[i], self.opt_m[i], self.opt_v[i], g, j,
                    self.gamma, hp.b1, hp.b2, hp.eps, self.wd_local, self.dt)
            else:
                self.X[i], self.opt_m[i] = sgdm_step(self.X[i], self.opt_m[i], g, self.gamma, hp.mu, self.dt)
        self.k += 1

    def global_step(self):
        """All-reduce average, sign-momentum update and synchronisation (Algorithm 1)."""
        assert self.k == self.tau
        hp = self.hp
        mode = self.global_mode
        if mode == GLOBAL_SIGN_MOMENTUM:
            r = None
            if hp.sign_mode != 0:
                r = philox_uniform(self.gidx, hp.seed, self.t)
            x_new, m_new, inter = global_step(self.x, self.m, self.X, self.gamma, hp.g_b1, hp.g_b2,
                                              hp.g_eta, self.wd_global, hp.sign_mode, hp.rsign_B, r, self.dt)
        elif mode == GLOBAL_SLOWMO:
            x_new, m_new, inter = global_step_slowmo(self.x, self.m, self.X, self.gamma, hp.g_b1, hp.g_eta,
                                                     self.dt)
        elif mode == GLOBAL_SIGNED_SLOWMO:
            x_new, m_new, inter = global_step_signed_slowmo(self.x, self.m, self.X, self.gamma, hp.g_b1,
                                                            hp.g_b2, hp.g_eta, self.dt)
        elif mode == GLOBAL_LOOKAHEAD:
            x_new, m_new, inter = global_step_lookahead(self.x, self.m, self.X, self.gamma, hp.g_b1, hp.g_b2,
                                                        hp.g_eta, self.dt)
        elif mode == GLOBAL_ADAMW:
            x_new, m_new, self.gv, inter = global_step_adamw(self.x, self.m, self.gv, self.X, self.gamma, self.t,
                                                             hp.g_b1, hp.g_b2, hp.g_eps, hp.g_eta,
                                                             self.wd_global, self.dt)
        else:
            raise ValueError(f"global mode {mode} unknown")
        if self.with_stats:
            self.last_stats = round_stats(inter, self.tensor_of, len(self.tensors),
                                          hp.sign_mode if mode == GLOBAL_SIGN_MOMENTUM else 0, hp.rsign_B)
        self.last_inter = inter
        self.x, self.m = x_new, m_new
        self.X = [x_new.copy() for _ in range(self.n)]
        if self.reset_local:
            self.opt_m = [np.zeros_like(self.x) for _ in range(self.n)]
            if self.opt_v is not None:
                self.opt_v = [np.zeros_like(self.x) for _ in range(self.n)]
        self.t += 1
        self.k = 0

    def run_round(self, grads=None):
        """One global round; ``grads`` optionally gives grads[k][i] explicitly."""
        for k in range(self.tau):
            self.local_step(None if grads is None else grads[k])
        self.global_step()
