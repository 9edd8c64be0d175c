"""The C-ABI library loads, exports every declared symbol, and checks its
arguments on the host (no GPU needed: every case fails before any CUDA call)."""
import ctypes
import os
import re

import pytest

import workloads as W
from paper_2411_17866_gb300 import dsm

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "dsm.h")


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(dsm_[a-z_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(dsm.LIB_PATH):
        from paper_2411_17866_gb300 import build
        build.build()
    return dsm.load_library()


def test_exports_every_declared_symbol(lib):
    names = declared_functions()
    assert len(names) >= 15
    for name in names:
        assert hasattr(lib, name), name
    assert set(names) == set(dsm._PROTOS), "binding and header disagree"


def test_struct_sizes_match_header_layout():
    assert ctypes.sizeof(dsm.dsm_tensor) == 24
    assert ctypes.sizeof(dsm.dsm_hparams) == 80
    assert ctypes.sizeof(dsm.dsm_tensor_stats) == 48
    assert ctypes.sizeof(dsm.dsm_layout) == 24
    assert dsm.dsm_layout.first_element.offset == 16


def test_first_element_must_be_a_multiple_of_4(lib):
    """A parameter shard starts at a multiple of 4 elements of the larger model (the synthetic draws come in
    pairs and the randomized sign's Philox blocks in fours)."""
    tensors = W.gpt2_layout(2, 64, 256)
    hp = dsm.make_hparams(W.HParams())
    assert dsm.dsm_state_bytes(dsm.make_layout(tensors, 1 << 20), 4, hp) > 0
    for bad in (2, 6, 1 << 61):
        with pytest.raises(dsm.DsmError) as e:
            dsm.dsm_state_bytes(dsm.make_layout(tensors, bad), 4, hp)
        assert "first_element" in str(e.value)


def _args(tensors=None, n=4, hp=None):
    tensors = tensors if tensors is not None else W.gpt2_layout(2, 64, 256)
    return dsm.make_layout(tensors), n, dsm.make_hparams(hp or W.HParams())


def test_state_bytes_covers_the_state(lib):
    lay, n, hp = _args()
    d = sum(t.numel for t in W.gpt2_layout(2, 64, 256))
    nb = dsm.dsm_state_bytes(lay, n, hp)
    # x, m, n replicas, n AdamW first and second moments, n fp32 gradients
    assert nb >= 4 * d * (2 + 4 * n)
    assert nb % 256 == 0
    # bf16 gradients take half the gradient bytes; SGD-momentum drops the second moment
    nb_bf16 = dsm.dsm_state_bytes(lay, n, dsm.make_hparams(W.HParams(grad_dtype=W.BF16)))
    nb_sgd = dsm.dsm_state_bytes(lay, n, dsm.make_hparams(W.SGDM_HP))
    assert nb - nb_bf16 >= 2 * d * n - 256 * 12
    assert nb - nb_sgd >= 4 * d * n - 256 * 12
    # grows with n
    assert dsm.dsm_state_bytes(lay, n + 1, hp) > nb


@pytest.mark.parametrize("bad,code", [
    (dict(n=0), dsm.DSM_EINVAL),
    (dict(n=65), dsm.DSM_ERANGE),
    (dict(hp=W.HParams(lr=0.0)), dsm.DSM_EINVAL),
    (dict(hp=W.HParams(lr=float("nan"))), dsm.DSM_EINVAL),
    (dict(hp=W.HParams(b1=1.0)), dsm.DSM_EINVAL),
    (dict(hp=W.HParams(b2=-0.1)), dsm.DSM_EINVAL),
    (dict(hp=W.HParams(eps=0.0)), dsm.DSM_EINVAL),
    (dict(hp=W.HParams(g_b1=1.5)), dsm.DSM_EINVAL),
    (dict(hp=W.HParams(g_eta=-1.0)), dsm.DSM_EINVAL),
    (dict(hp=W.HParams(sign_mode=3)), dsm.DSM_EINVAL),
    (dict(hp=W.HParams(sign_mode=W.RSIGN_ZERO, rsign_B=0.0)), dsm.DSM_EINVAL),
    (dict(hp=W.HParams(grad_dtype=2)), dsm.DSM_EINVAL),
    (dict(hp=W.HParams(flags=4)), dsm.DSM_EINVAL),
    (dict(hp=W.HParams(base=7)), dsm.DSM_EINVAL),
    (dict(hp=W.HParams(global_mode=5)), dsm.DSM_EINVAL),
    (dict(hp=W.HParams(global_mode=W.GLOBAL_SLOWMO, sign_mode=W.RSIGN_ZERO)), dsm.DSM_EINVAL),
    (dict(hp=W.HParams(global_mode=W.GLOBAL_ADAMW, g_b1=1.0)), dsm.DSM_EINVAL),
    (dict(hp=W.HParams(global_mode=W.GLOBAL_ADAMW, g_eps=0.0)), dsm.DSM_EINVAL),
    (dict(hp=W.SGDM_HP.__class__(**{**W.SGDM_HP.__dict__, "mu": 1.0})), dsm.DSM_EINVAL),
    (dict(tensors=()), dsm.DSM_EINVAL),
    (dict(tensors=(W.Tensor("z", 0, 0, 1.0),)), dsm.DSM_EINVAL),
    (dict(tensors=(W.Tensor("k", 8, 9, 1.0),)), dsm.DSM_EINVAL),
])
def test_invalid_arguments_are_rejected(lib, bad, code):
    lay, n, hp = _args(bad.get("tensors"), bad.get("n", 4), bad.get("hp"))
    assert lib.dsm_state_bytes(ctypes.byref(lay), n, ctypes.byref(hp)) == 0
    h = ctypes.c_void_p(1)
    rc = lib.dsm_create(ctypes.byref(lay), n, 2, ctypes.byref(hp), ctypes.c_void_p(1 << 20), 1 << 40, None, 0,
                        None, ctypes.byref(h))
    assert rc == code, dsm.last_error()
    assert h.value is None
    assert dsm.last_error()


def test_known_flags_are_accepted(lib):
    for flags in (W.FLAG_FUSED_ROUND, W.FLAG_RESET_LOCAL_STATE, W.FLAG_FUSED_ROUND | W.FLAG_RESET_LOCAL_STATE):
        lay, n, hp = _args(hp=W.HParams(flags=flags))
        assert dsm.dsm_state_bytes(lay, n, hp) > 0
    assert (dsm.FLAG_FUSED_ROUND, dsm.FLAG_RESET_LOCAL_STATE) == (W.FLAG_FUSED_ROUND, W.FLAG_RESET_LOCAL_STATE)


def test_arena_checks(lib):
    lay, n, hp = _args()
    need = dsm.dsm_state_bytes(lay, n, hp)
    h = ctypes.c_void_p()
    rc = lib.dsm_create(ctypes.byref(lay), n, 2, ctypes.byref(hp), ctypes.c_void_p((1 << 20) + 16), need, None, 0,
                        None, ctypes.byref(h))
    assert rc == dsm.DSM_EALIGN and "aligned" in dsm.last_error()
    rc = lib.dsm_create(ctypes.byref(lay), n, 2, ctypes.byref(hp), ctypes.c_void_p(1 << 20), need - 1, None, 0,
                        None, ctypes.byref(h))
    assert rc == dsm.DSM_ENOMEM
    rc = lib.dsm_create(ctypes.byref(lay), n, 0, ctypes.byref(hp), ctypes.c_void_p(1 << 20), need, None, 0,
                        None, ctypes.byref(h))
    assert rc == dsm.DSM_EINVAL and "tau" in dsm.last_error()
    rc = lib.dsm_create(ctypes.byref(lay), n, 2, ctypes.byref(hp), None, need, None, 0, None, ctypes.byref(h))
    assert rc == dsm.DSM_EINVAL
    rc = lib.dsm_create(ctypes.byref(lay), n, 2, ctypes.byref(hp), ctypes.c_void_p(1 << 20), need, None, 0,
                        None, None)
    assert rc == dsm.DSM_EINVAL


def test_null_handle_calls_fail_cleanly(lib):
    assert lib.dsm_local_step(None, None) == dsm.DSM_EINVAL
    assert lib.dsm_global_step(None, None, None, 0) == dsm.DSM_EINVAL
    assert lib.dsm_set_gamma(None, ctypes.c_float(1.0)) == dsm.DSM_EINVAL
    assert lib.dsm_fill_synthetic_grads(None, 0, None) == dsm.DSM_EINVAL
    assert lib.dsm_read_params(None, 0, 0, None, 0, 0, 0, None) == dsm.DSM_EINVAL
    assert lib.dsm_set_first_worker(None, 0) == dsm.DSM_EINVAL
    assert lib.dsm_end_round(None, None, 0, None) == dsm.DSM_EINVAL
    assert lib.dsm_destroy(None) == dsm.DSM_OK


def test_binding_fails_loudly_without_library(tmp_path, monkeypatch):
    monkeypatch.setattr(dsm, "_lib", None)
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        dsm.load_library(str(tmp_path / "missing.so"))


def test_cosine_schedule_matches_the_oracle(lib):
    """dsm_cosine_gamma against the oracle's schedule (itself pinned by closed-form points)."""
    import numpy as np
    from oracle import dsm_oracle as O
    P, r, W_, S = 6e-4, 0.05, 2000, 100000
    for step in list(range(0, 2100, 7)) + list(range(2000, 100001, 991)) + [100000, 100001, 10 ** 9]:
        want = np.float32(O.cosine_gamma(P, r, W_, S, step))
        got = np.float32(dsm.dsm_cosine_gamma(P, r, W_, S, step))
        assert abs(int(got.view(np.int32)) - int(want.view(np.int32))) <= 1, (step, got, want)
    for bad in [(0.0, r, W_, S, 0), (P, 1.5, W_, S, 0), (P, r, S + 1, S, 0), (P, r, 0, 0, 0)]:
        with pytest.raises(dsm.DsmError):
            dsm.dsm_cosine_gamma(*bad)


def test_host_memory_arena_is_refused(lib):
    """A host buffer as arena: DSM_EALIGN ('not device memory') with a GPU, DSM_ECUDA (the runtime's
    message) without one; never a crash."""
    lay, n, hp = _args()
    need = dsm.dsm_state_bytes(lay, n, hp)
    arena = ctypes.create_string_buffer(need + 256)
    ptr = (ctypes.addressof(arena) + 255) // 256 * 256
    h = ctypes.c_void_p()
    rc = lib.dsm_create(ctypes.byref(lay), n, 2, ctypes.byref(hp), ctypes.c_void_p(ptr), need, None, 0, None,
                        ctypes.byref(h))
    assert rc in (dsm.DSM_ECUDA, dsm.DSM_EALIGN)
    msg = dsm.last_error()
    assert ("device memory" in msg) if rc == dsm.DSM_EALIGN else ("cudaPointerGetAttributes" in msg)


def test_header_constants_match_the_python_side():
    """Every integer constant the header defines has the same value in the binding and, where the
    workload definitions use it, in workloads.py."""
    src = open(HEADER).read()
    defs = {m.group(1): int(m.group(2).rstrip("u"), 0)
            for m in re.finditer(r"#define\s+(DSM_[A-Z0-9_]+)\s+\(?(-?(?:0x[0-9A-Fa-f]+|\d+)u?)\)?", src)}
    assert len(defs) >= 30
    checked = 0
    for name, value in defs.items():
        if name.startswith("DSM_NOALLOC_"):
            continue
        short = name[len("DSM_"):]
        if name in ("DSM_OK", "DSM_EINVAL", "DSM_ENOMEM", "DSM_EALIGN", "DSM_ESTATE", "DSM_ECUDA", "DSM_ERANGE"):
            assert getattr(dsm, name) == value, name
            checked += 1
            continue
        assert hasattr(dsm, short), f"{name} has no counterpart in the binding"
        assert getattr(dsm, short) == value, name
        checked += 1
        if hasattr(W, short):
            assert getattr(W, short) == value, name
    assert checked == len([n for n in defs if not n.startswith("DSM_NOALLOC_")])
