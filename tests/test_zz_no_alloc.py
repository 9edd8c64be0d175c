"""dsm_global_step_noalloc through the C ABI, against the oracle and against dsm_global_step.

The no-allocation entry point serves callers that cannot allocate device
memory themselves (a plugin inside a framework that owns all of HBM through
its own pool, or a loop that must not block in cudaMalloc/cudaFree).  It
runs the global step on the caller's own x, m and replica buffers and keeps
its tile table and per-tile statistics in the library's static scratch
array.  Its results must equal the oracle's global step and those of the
handle-based global step: bit for bit for x, m and the replicas, and to the
statistics tolerance of the other GPU tests.  Two calls in a row check that
a call is not disturbed by what the previous call left in the shared scratch
array, including a call on a small layout after one on a much larger layout.

This file is named so that pytest collects it last.
"""
import dataclasses

import numpy as np
import pytest

import workloads as W
from gpu_common import assert_bitexact, compare_stats, stats_rtol

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from oracle import dsm_oracle as O  # noqa: E402
from paper_2411_17866_gb300 import dsm  # noqa: E402

LAYOUT = (W.Tensor("a", 7, W.KIND_WEIGHT, 1e-2), W.Tensor("b", 4096, W.KIND_WEIGHT, 1e-3),
          W.Tensor("c", 0, W.KIND_BIAS, 1e-3), W.Tensor("d", 3001, W.KIND_LN_W, 1e-3, wd=0),
          W.Tensor("e", 65536, W.KIND_WEIGHT, 1e-3))
# many tiles and the generic (n > 8) global step: leaves large tables and many partials in the scratch array
LARGE = (W.Tensor("big0", 3 * (1 << 20) + 5, W.KIND_WEIGHT, 1e-3), W.Tensor("big1", 1 << 20, W.KIND_BIAS, 1e-4),
         W.Tensor("big2", 777, W.KIND_LN_W, 1e-4))

CASES = [("adamw-sign-n4", W.HParams(), 4, 2),
         ("sgdm-rsign-n3", dataclasses.replace(W.SGDM_HP, sign_mode=W.RSIGN_PM, rsign_B=1e-3), 3, 2),
         ("adamw-rsign0-n9", dataclasses.replace(W.HParams(), sign_mode=W.RSIGN_ZERO, rsign_B=1.0), 9, 1),
         # the ablation global steps that keep only x and m
         ("slowmo-n4", dataclasses.replace(W.HParams(), global_mode=W.GLOBAL_SLOWMO), 4, 2),
         ("signed-slowmo-sgdm-n5", dataclasses.replace(W.SGDM_HP, sign_mode=W.SIGN,
                                                       global_mode=W.GLOBAL_SIGNED_SLOWMO), 5, 1),
         ("lookahead-n9", dataclasses.replace(W.HParams(), global_mode=W.GLOBAL_LOOKAHEAD), 9, 1)]


def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")


def _caller_buffers(run, n):
    """The caller's own buffers: copies of x, m and the replicas before the global step."""
    d, stride = run.d, run.d_stride
    x = torch.empty(d, dtype=torch.float32, device="cuda")
    m = torch.empty(d, dtype=torch.float32, device="cuda")
    reps = torch.empty(n * stride, dtype=torch.float32, device="cuda")
    run.read(dsm.BUF_X, out=x)
    run.read(dsm.BUF_M, out=m)
    for i in range(n):
        run.read(dsm.BUF_REPLICA, i, out=reps[i * stride:i * stride + d])
    return x, m, reps


def _noalloc(tensors, n, hp, gamma, round_, x, m, reps, stride, stats=None, stats_is_device=False, first_element=0):
    dsm.dsm_global_step_noalloc(dsm.make_layout(tensors, first_element), n, dsm.make_hparams(hp), gamma, round_,
                                x.data_ptr(),
                                m.data_ptr(), reps.data_ptr(), stride,
                                stats if not stats_is_device else stats.data_ptr(), stats_is_device=stats_is_device)


def _assert_same_as_handle(run, n, x, m, reps):
    d, stride = run.d, run.d_stride
    assert torch.equal(x.cpu().view(torch.int32), run.read(dsm.BUF_X).view(torch.int32))
    assert torch.equal(m.cpu().view(torch.int32), run.read(dsm.BUF_M).view(torch.int32))
    for i in range(n):
        got = reps[i * stride:i * stride + d].cpu().view(torch.int32)
        assert torch.equal(got, run.read(dsm.BUF_REPLICA, i).view(torch.int32))


def _stats_close(a, b, n):
    for ta, tb in zip(a, b):
        for key in ("zero_sign", "flips", "unanimous", "clamped"):
            assert ta[key] == tb[key], key
        for key in ("delta_sq", "drift"):
            assert abs(ta[key] - tb[key]) <= stats_rtol(n) * abs(tb[key]), key


def _device_stats_rows(dev_stats, count):
    raw = dev_stats.cpu().numpy().view(np.uint64).reshape(count, 6)
    f = raw[:, :2].copy().view(np.float64)
    return [{"delta_sq": float(f[T, 0]), "drift": float(f[T, 1]), "zero_sign": int(raw[T, 2]),
             "flips": int(raw[T, 3]), "unanimous": int(raw[T, 4]), "clamped": int(raw[T, 5])} for T in range(count)]


@pytest.mark.parametrize("name,hp,n,tau", CASES, ids=[c[0] for c in CASES])
def test_noalloc_global_step_matches_handle_path(name, hp, n, tau):
    _need_gpu()
    run = dsm.DistributedSignMomentum(LAYOUT, n, tau, hp)
    stride = run.d_stride
    for call in range(2):                      # two calls in a row
        for k in range(tau):
            run.fill_synthetic_grads(call * tau + k)
            run.local_step()
        x, m, reps = _caller_buffers(run, n)
        x2, m2, reps2 = x.clone(), m.clone(), reps.clone()
        info = run.info()
        host_stats = (dsm.dsm_tensor_stats * len(LAYOUT))()
        _noalloc(LAYOUT, n, hp, info.gamma, info.round, x, m, reps, stride, host_stats)
        # the same call on copies of the inputs, statistics written to device memory instead
        dev_stats = torch.zeros(len(LAYOUT) * 6, dtype=torch.float64, device="cuda")
        _noalloc(LAYOUT, n, hp, info.gamma, info.round, x2, m2, reps2, stride, dev_stats, stats_is_device=True)
        want_stats = run.global_step(with_stats=True)
        torch.cuda.synchronize()
        _assert_same_as_handle(run, n, x, m, reps)
        _assert_same_as_handle(run, n, x2, m2, reps2)
        host_rows = [s.as_dict() for s in host_stats]
        _stats_close(host_rows, want_stats, n)
        assert _device_stats_rows(dev_stats, len(LAYOUT)) == host_rows   # field by field, bit for bit
    run.close()


@pytest.mark.parametrize("first_element", [0, (1 << 35) + 8], ids=["whole-model", "shard-at-2^35"])
@pytest.mark.parametrize("name,hp,n,tau", CASES, ids=[c[0] for c in CASES])
def test_noalloc_global_step_matches_oracle(name, hp, n, tau, first_element):
    """Two rounds: the oracle's local steps, then its state uploaded to the caller's buffers and the global
    step run by dsm_global_step_noalloc; x, m and every replica bit for bit, statistics to tolerance.  A layout
    placed far into a larger model moves the randomized sign's Philox counter."""
    _need_gpu()
    ora = O.OracleRun(LAYOUT, n, tau, hp, with_stats=True, first_element=first_element)
    d = ora.d
    stride = (d + 63) // 64 * 64
    for t in range(2):
        for _ in range(tau):
            ora.local_step()
        x = torch.from_numpy(ora.x.copy()).cuda()
        m = torch.from_numpy(ora.m.copy()).cuda()
        reps = torch.zeros(n * stride, dtype=torch.float32, device="cuda")
        for i in range(n):
            reps[i * stride:i * stride + d] = torch.from_numpy(ora.X[i])
        host_stats = (dsm.dsm_tensor_stats * len(LAYOUT))()
        _noalloc(LAYOUT, n, hp, ora.gamma, ora.t, x, m, reps, stride, host_stats, first_element=first_element)
        ora.global_step()
        torch.cuda.synchronize()
        assert_bitexact(x.cpu().numpy(), ora.x, f"x, round {t}")
        assert_bitexact(m.cpu().numpy(), ora.m, f"m, round {t}")
        r = reps.cpu().numpy()
        for i in range(n):
            assert_bitexact(r[i * stride:i * stride + d], ora.X[i], f"replica {i}, round {t}")
        compare_stats([s.as_dict() for s in host_stats], ora.last_stats, n)


def test_noalloc_small_layout_after_large_one():
    """A call on a small layout right after one on a much larger layout (more tensors' tables, more tiles,
    more partials, the generic n > 8 kernel) gives, bit for bit, what a fresh handle's global step gives."""
    _need_gpu()
    hp = dataclasses.replace(W.HParams(), sign_mode=W.RSIGN_ZERO, rsign_B=1e-2, seed=3)
    big = dsm.DistributedSignMomentum(LARGE, 9, 1, hp)
    big.fill_synthetic_grads(0)
    big.local_step()
    bx, bm, breps = _caller_buffers(big, 9)
    big_stats = (dsm.dsm_tensor_stats * len(LARGE))()
    _noalloc(LARGE, 9, hp, big.info().gamma, 0, bx, bm, breps, big.d_stride, big_stats)
    want_big = big.global_step(with_stats=True)
    torch.cuda.synchronize()
    _assert_same_as_handle(big, 9, bx, bm, breps)
    _stats_close([s.as_dict() for s in big_stats], want_big, 9)
    big.close()
    small = dsm.DistributedSignMomentum(LAYOUT, 4, 2, hp)   # a fresh handle
    for k in range(2):
        small.fill_synthetic_grads(k)
        small.local_step()
    x, m, reps = _caller_buffers(small, 4)
    small_stats = (dsm.dsm_tensor_stats * len(LAYOUT))()
    _noalloc(LAYOUT, 4, hp, small.info().gamma, 0, x, m, reps, small.d_stride, small_stats)
    want = small.global_step(with_stats=True)
    torch.cuda.synchronize()
    _assert_same_as_handle(small, 4, x, m, reps)
    _stats_close([s.as_dict() for s in small_stats], want, 4)
    small.close()


def test_noalloc_rejects_sizes_beyond_its_limit():
    _need_gpu()
    big = (W.Tensor("huge", (dsm_max_tiles() + 1) * 1024, W.KIND_WEIGHT, 1e-3),)
    x = torch.empty(16, dtype=torch.float32, device="cuda")
    with pytest.raises(dsm.DsmError) as e:
        dsm.dsm_global_step_noalloc(dsm.make_layout(big), 2, dsm.make_hparams(W.HParams()), 1e-3, 0,
                                    x.data_ptr(), x.data_ptr(), x.data_ptr(), (dsm_max_tiles() + 1) * 1024)
    assert e.value.code == dsm.DSM_ERANGE and "DSM_NOALLOC_MAX_TILES" in str(e.value)
    many = tuple(W.Tensor(f"t{i}", 8, W.KIND_BIAS, 1e-3) for i in range(4097))
    with pytest.raises(dsm.DsmError) as e:
        dsm.dsm_global_step_noalloc(dsm.make_layout(many), 2, dsm.make_hparams(W.HParams()), 1e-3, 0,
                                    x.data_ptr(), x.data_ptr(), x.data_ptr(), 4097 * 8)
    assert e.value.code == dsm.DSM_ERANGE


def test_noalloc_checks_every_buffer_and_the_tensor_list():
    """m, the replicas and device statistics must be device memory of the current device, as x must; the
    tensor list passes dsm_create's checks."""
    _need_gpu()
    tensors = (W.Tensor("a", 64, W.KIND_WEIGHT, 1e-3),)
    layout, chp = dsm.make_layout(tensors), dsm.make_hparams(W.HParams())
    dev = torch.zeros(4 * 64, dtype=torch.float32, device="cuda")
    host = torch.zeros(4 * 64, dtype=torch.float32)
    for args, what in (((dev, host, dev), "m"), ((dev, dev, host), "replicas")):
        with pytest.raises(dsm.DsmError) as e:
            dsm.dsm_global_step_noalloc(layout, 2, chp, 1e-3, 0, *(t.data_ptr() for t in args), 64)
        assert e.value.code in (dsm.DSM_EINVAL, dsm.DSM_ECUDA) and what in str(e.value)
    with pytest.raises(dsm.DsmError) as e:
        dsm.dsm_global_step_noalloc(layout, 2, chp, 1e-3, 0, dev.data_ptr(), dev.data_ptr(), dev.data_ptr(), 64,
                                    host.data_ptr(), stats_is_device=True)
    assert "stats" in str(e.value)
    bad = dsm.make_layout(tensors)
    bad._keep[0].reserved = 1
    with pytest.raises(dsm.DsmError) as e:
        dsm.dsm_global_step_noalloc(bad, 2, chp, 1e-3, 0, dev.data_ptr(), dev.data_ptr(), dev.data_ptr(), 64)
    assert e.value.code == dsm.DSM_EINVAL and "reserved" in str(e.value)


def dsm_max_tiles():
    return 524288


def test_noalloc_rejects_global_adamw_and_signed_variants_with_random_signs():
    """Global AdamW needs a second-moment buffer this entry point does not take; the randomized signs belong
    to Algorithm 1's global step only.  Both are refused before any work is enqueued."""
    _need_gpu()
    tensors = (W.Tensor("a", 64, W.KIND_WEIGHT, 1e-3),)
    dev = torch.zeros(4 * 64, dtype=torch.float32, device="cuda")
    for hp, what in ((dataclasses.replace(W.HParams(), global_mode=W.GLOBAL_ADAMW), "global AdamW"),
                     (dataclasses.replace(W.HParams(), global_mode=W.GLOBAL_SLOWMO, sign_mode=W.RSIGN_ZERO,
                                          rsign_B=1.0), "randomized signs")):
        with pytest.raises(dsm.DsmError) as e:
            dsm.dsm_global_step_noalloc(dsm.make_layout(tensors), 2, dsm.make_hparams(hp), 1e-3, 0,
                                        dev.data_ptr(), dev.data_ptr(), dev.data_ptr(), 64)
        assert e.value.code == dsm.DSM_EINVAL and what in str(e.value)
