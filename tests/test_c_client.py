"""The C ABI from plain C: include/dsm.h compiles as C99, a C client links
against libdsm.so (CPU), and on a GPU the client's rounds equal the oracle's
bit for bit (tests/c_client.c)."""
import os
import shutil
import subprocess

import numpy as np
import pytest

import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CUDA = os.environ.get("CUDA_HOME", "/usr/local/cuda")
PKG = os.path.join(ROOT, "paper_2411_17866_gb300")
SRC = os.path.join(ROOT, "tests", "c_client.c")

pytestmark = pytest.mark.skipif(shutil.which("gcc") is None, reason="no C compiler")


def _cuda_lib_dir():
    for d in ("lib64", "lib", os.path.join("targets", "sbsa-linux", "lib"), os.path.join("targets", "x86_64-linux", "lib")):
        if os.path.exists(os.path.join(CUDA, d, "libcudart.so")):
            return os.path.join(CUDA, d)
    pytest.skip("libcudart.so not found")


@pytest.fixture(scope="module")
def client(tmp_path_factory):
    from paper_2411_17866_gb300 import dsm
    if not os.path.exists(dsm.LIB_PATH):
        from paper_2411_17866_gb300 import build
        build.build()
    out = str(tmp_path_factory.mktemp("c_client") / "c_client")
    lib = _cuda_lib_dir()
    cmd = ["gcc", "-std=c99", "-Wall", "-Wextra", "-Werror", "-pedantic", "-O2", SRC, "-o", out,
           "-I" + os.path.join(ROOT, "include"), "-isystem", os.path.join(CUDA, "include"),
           "-L" + PKG, "-ldsm", "-Wl,-rpath," + PKG, "-L" + lib, "-lcudart", "-Wl,-rpath," + lib]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    return out


def test_header_is_c99():
    r = subprocess.run(["gcc", "-std=c99", "-Wall", "-Wextra", "-Werror", "-pedantic", "-fsyntax-only", "-x", "c",
                        os.path.join(ROOT, "include", "dsm.h")], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr


def test_client_links(client):
    assert os.access(client, os.X_OK)


def _oracle(kind, rounds):
    from oracle import dsm_oracle as O
    tensors = (W.Tensor("w", 5000, W.KIND_WEIGHT, 1e-2), W.Tensor("b", 77, W.KIND_BIAS, 1e-3),
               W.Tensor("ln", 2048, W.KIND_LN_W, 1e-3))
    if kind == "adamw":
        hp, n, tau = W.HParams(flags=W.FLAG_FUSED_ROUND), 3, 2
    else:
        hp, n, tau = W.HParams(base=W.BASE_SGDM, lr=1e-2, sign_mode=W.RSIGN_ZERO), 4, 3
    ora = O.OracleRun(tensors, n, tau, hp, with_stats=True)
    for _ in range(rounds):
        ora.run_round()
    return ora


@pytest.mark.gpu
@pytest.mark.parametrize("kind", ["adamw", "sgdm"])
def test_client_rounds_match_the_oracle(client, kind):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    rounds = 3
    r = subprocess.run([client, kind, str(rounds)], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr
    lines = r.stdout.split("\n")
    head = lines[0].split()
    d = int(head[1])
    assert int(head[3]) == rounds
    stats = [ln.split() for ln in lines[1:4]]
    x = np.array([int(v, 16) for v in lines[4:4 + d]], dtype=np.uint32).view(np.float32)
    ora = _oracle(kind, rounds)
    assert np.array_equal(x.view(np.uint32), ora.x.view(np.uint32))
    from gpu_common import stats_rtol
    for got, want in zip(stats, ora.last_stats):
        assert [int(v) for v in got[4:8]] == [want["zero_sign"], want["flips"], want["unanimous"], want["clamped"]]
        for v, key in ((float(got[2]), "delta_sq"), (float(got[3]), "drift")):
            assert abs(v - want[key]) <= stats_rtol(4) * abs(want[key])


def test_header_is_cxx11():
    if shutil.which("g++") is None:
        pytest.skip("no C++ compiler")
    r = subprocess.run(["g++", "-std=c++11", "-Wall", "-Wextra", "-Werror", "-pedantic", "-fsyntax-only", "-x", "c++",
                        os.path.join(ROOT, "include", "dsm.h")], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
