"""dsm_global_step_noalloc against dsm_global_step, through the C ABI.

The no-allocation entry point serves callers that cannot allocate device
memory themselves (a plugin inside a framework that owns all of HBM through
its own pool, or a loop that must not block in cudaMalloc/cudaFree).  It
runs the global step on the caller's own x, m and replica buffers and keeps
its tile table and per-tile statistics in the library's static scratch
array.  Its results must equal those of the handle-based global step: bit
for bit for x, m and the replicas, and to the statistics tolerance of the
other GPU tests.  Two calls in a row check that a call is not disturbed by
what the previous call left in the shared scratch array.

This file is named so that pytest collects it last.
"""
import ctypes
import dataclasses

import pytest

import workloads as W
from gpu_common import stats_rtol

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2411_17866_gb300 import dsm  # noqa: E402

LAYOUT = (W.Tensor("a", 7, W.KIND_WEIGHT, 1e-2), W.Tensor("b", 4096, W.KIND_WEIGHT, 1e-3),
          W.Tensor("c", 0, W.KIND_BIAS, 1e-3), W.Tensor("d", 3001, W.KIND_LN_W, 1e-3, wd=0),
          W.Tensor("e", 65536, W.KIND_WEIGHT, 1e-3))

CASES = [("adamw-sign-n4", W.HParams(), 4, 2),
         ("sgdm-rsign-n3", dataclasses.replace(W.SGDM_HP, sign_mode=W.RSIGN_PM, rsign_B=1e-3), 3, 2),
         ("adamw-rsign0-n9", dataclasses.replace(W.HParams(), sign_mode=W.RSIGN_ZERO, rsign_B=1.0), 9, 1)]


def _stats_close(a, b, n):
    for ta, tb in zip(a, b):
        for key in ("zero_sign", "flips", "unanimous", "clamped"):
            assert ta[key] == tb[key], key
        for key in ("delta_sq", "drift"):
            assert abs(ta[key] - tb[key]) <= stats_rtol(n) * abs(tb[key]), key


@pytest.mark.parametrize("name,hp,n,tau", CASES, ids=[c[0] for c in CASES])
def test_noalloc_global_step_matches_handle_path(name, hp, n, tau):
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    run = dsm.DistributedSignMomentum(LAYOUT, n, tau, hp)
    d = run.d
    stride = run.d_stride
    layout = dsm.make_layout(LAYOUT)
    chp = dsm.make_hparams(hp)
    for call in range(2):                      # two calls in a row
        for k in range(tau):
            run.fill_synthetic_grads(call * tau + k)
            run.local_step()
        # the caller's own buffers: copies of x, m and the replicas before the global step
        x = torch.empty(d, dtype=torch.float32, device="cuda")
        m = torch.empty(d, dtype=torch.float32, device="cuda")
        reps = torch.empty(n * stride, dtype=torch.float32, device="cuda")
        run.read(dsm.BUF_X, out=x)
        run.read(dsm.BUF_M, out=m)
        for i in range(n):
            run.read(dsm.BUF_REPLICA, i, out=reps[i * stride:i * stride + d])
        gamma = run.info().gamma
        round_ = run.info().round
        host_stats = (dsm.dsm_tensor_stats * len(LAYOUT))()
        dsm.dsm_global_step_noalloc(layout, n, chp, gamma, round_, x.data_ptr(), m.data_ptr(), reps.data_ptr(),
                                    stride, host_stats)
        want_stats = run.global_step(with_stats=True)
        torch.cuda.synchronize()
        assert torch.equal(x.cpu().view(torch.int32), run.read(dsm.BUF_X).view(torch.int32))
        assert torch.equal(m.cpu().view(torch.int32), run.read(dsm.BUF_M).view(torch.int32))
        for i in range(n):
            got = reps[i * stride:i * stride + d].cpu().view(torch.int32)
            assert torch.equal(got, run.read(dsm.BUF_REPLICA, i).view(torch.int32))
        _stats_close([s.as_dict() for s in host_stats], want_stats, n)
        # statistics written to device memory instead
        if call == 1:
            dev_stats = torch.zeros(len(LAYOUT) * 6, dtype=torch.float64, device="cuda")
            x2, m2, r2 = x.clone(), m.clone(), reps.clone()
            dsm.dsm_global_step_noalloc(layout, n, chp, gamma, round_ + 1, x2.data_ptr(), m2.data_ptr(),
                                        r2.data_ptr(), stride, dev_stats.data_ptr(), stats_is_device=True)
            torch.cuda.synchronize()
            raw = dev_stats.cpu().numpy().view("u8").reshape(len(LAYOUT), 6)
            assert int(raw[4, 4]) <= LAYOUT[4].numel          # unanimous count of tensor e
    run.close()


def test_noalloc_rejects_sizes_beyond_its_limit():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
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


def dsm_max_tiles():
    return 524288
