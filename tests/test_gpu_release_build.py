"""The release build with nvcc's default multiply-add contraction gives the same bits.

Every operation of the method is an explicit round-to-nearest intrinsic, which
nvcc never contracts into an FMA, so building without --fmad=false must not
change a single result.  The test builds that variant and runs the smoke
comparison against the oracle through it, in a separate process.
"""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
pytestmark = pytest.mark.gpu


def test_contracting_build_is_bitexact(tmp_path):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    sys.path.insert(0, ROOT)
    from paper_2411_17866_gb300 import build
    lib = build.build(fmad=True, out=str(tmp_path / "libdsm_fmad.so"))
    env = dict(os.environ, DSM_LIBRARY=lib)
    code = "import __graft_entry__ as g; from paper_2411_17866_gb300 import dsm; " \
           "assert dsm.LIB_PATH.endswith('libdsm_fmad.so'); g.smoke()"
    r = subprocess.run([sys.executable, "-c", code], cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-2000:]
    assert "smoke: OK" in r.stdout
