"""Helpers shared by the GPU parity tests."""
from __future__ import annotations

import numpy as np

from paper_2411_17866_gb300 import dsm

# Statistics.  Each element contributes Delta^2 (one fp32 rounding) and
# sum_i (d_i - Delta)^2 (per worker one rounding for the difference and one
# for the square, then n-1 roundings for the fp32 sum over workers); the
# kernel accumulates those terms with compensated (TwoSum) fp32 sums and fp64
# beyond, which adds nothing at this scale.  All terms are non-negative, so
# the relative error of a tensor's sum is below (n + 2) * 2^-24; the tests
# allow (n + 4) * 2^-24.  Counts are exact.
def stats_rtol(n: int) -> float:
    return (n + 4) * 2.0 ** -24


STATS_RTOL = stats_rtol(64)   # the largest n the library accepts


def bits(a) -> np.ndarray:
    a = np.ascontiguousarray(a)
    return a.view(np.uint16 if a.dtype.itemsize == 2 else np.uint32)


def assert_bitexact(got, want, what):
    got = np.asarray(got)
    want = np.asarray(want, dtype=got.dtype)
    if not np.array_equal(bits(got), bits(want)):
        bad = np.flatnonzero(bits(got) != bits(want))
        i = bad[0]
        raise AssertionError(f"{what}: {bad.size} of {got.size} elements differ; first at {i}: "
                             f"gpu {got[i]!r} oracle {want[i]!r}")


def compare_state(run, ora, elems=None, grads=True):
    """Every buffer of the GPU state against the oracle, bit for bit (optionally on a subset);
    also checks that no kernel wrote past the end of an arena buffer."""
    import torch
    assert run.check_guards() == 0, "an arena guard region was overwritten"
    sel = slice(None) if elems is None else elems

    def rd(which, w=0):
        t = run.read(which, w)
        if t.dtype == torch.bfloat16:
            t = t.to(torch.float32)
        return t.numpy()[sel]

    assert_bitexact(rd(dsm.BUF_X), ora.x, "x")
    assert_bitexact(rd(dsm.BUF_M), ora.m, "m")
    for i in range(ora.n):
        assert_bitexact(rd(dsm.BUF_REPLICA, i), ora.X[i], f"replica {i}")
        assert_bitexact(rd(dsm.BUF_OPT_M, i), ora.opt_m[i], f"opt_m {i}")
        if ora.opt_v is not None:
            assert_bitexact(rd(dsm.BUF_OPT_V, i), ora.opt_v[i], f"opt_v {i}")
    if getattr(ora, "gv", None) is not None:
        assert_bitexact(rd(dsm.BUF_GLOBAL_V), ora.gv, "global v")


def compare_stats(got, want, n=64):
    assert len(got) == len(want)
    rtol = stats_rtol(n)
    for T, (g, w) in enumerate(zip(got, want)):
        for key in ("zero_sign", "flips", "unanimous", "clamped"):
            assert g[key] == w[key], (T, key, g[key], w[key])
        for key in ("delta_sq", "drift"):
            assert abs(g[key] - w[key]) <= rtol * abs(w[key]), (T, key, g[key], w[key])


def sample_elements(tensors, count, seed=0, edge=64):
    """Sampled logical indices: the first and last `edge` elements of every tensor plus `count` random ones."""
    rng = np.random.default_rng(seed)
    starts = np.cumsum([0] + [t.numel for t in tensors])
    d = int(starts[-1])
    parts = [rng.integers(0, d, count)]
    for a, b in zip(starts[:-1], starts[1:]):
        if b > a:
            parts.append(np.arange(a, min(b, a + edge)))
            parts.append(np.arange(max(a, b - edge), b))
    v = np.sort(np.concatenate(parts).astype(np.int64))   # sorted, then duplicates dropped
    keep = np.ones(v.size, dtype=bool)
    keep[1:] = v[1:] != v[:-1]
    return v[keep]
