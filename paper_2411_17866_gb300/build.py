"""Builds libdsm.so, the C-ABI library, in-tree for sm_103a (GB300).

The translation units compile in parallel, then link into a shared
library next to this file.  No CMake; nvcc and the host compiler only.
"""
from __future__ import annotations

import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(ROOT, "_build")
LIB = os.path.join(PKG, "libdsm.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
# --fmad=false: no multiply-add contraction anywhere in the library (the
# kernels also spell every rounding with __f*_rn intrinsics); IEEE division
# and square root are nvcc's defaults and stay on.
NVCC_FLAGS = ["-O3", "-lineinfo", "--fmad=false", "-std=c++17", "-Xcompiler", "-fPIC",
              "-Xcompiler", "-ffp-contract=off", "-I" + INCLUDE, "-I" + CSRC]
SOURCES = ["dsm_kernels.cu", "dsm_local.cu", "dsm_fused.cu", "dsm_fused_sign.cu", "dsm_fused_variants.cu",
           "dsm_fused_adamw.cu", "dsm_api.cpp", "dsm_noalloc.cu"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libdsm.so")


def _run(cmd, verbose):
    if verbose:
        print(" ".join(cmd), flush=True)
    r = subprocess.run(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"build failed ({r.returncode}): {' '.join(cmd)}\n{r.stdout}")
    if verbose and r.stdout.strip():
        print(r.stdout)
    return r.stdout


def build(verbose: bool = False, fmad: bool = False, out: str = LIB) -> str:
    """Compile and link libdsm.so (to ``out``); returns its path.

    fmad=True builds with nvcc's default multiply-add contraction; the method's
    arithmetic is written with explicit round-to-nearest intrinsics, which are
    never contracted, so both builds give identical results (a GPU test checks).
    """
    objdir = os.path.join(BUILD, "fmad" if fmad else "nofmad")
    os.makedirs(objdir, exist_ok=True)
    os.makedirs(os.path.dirname(os.path.abspath(out)), exist_ok=True)
    nv = nvcc()
    flags = [f for f in NVCC_FLAGS if not (fmad and f == "--fmad=false")]
    objs = []
    cmds = []
    for src in SOURCES:
        obj = os.path.join(objdir, src + ".o")
        objs.append(obj)
        cmds.append([nv, *ARCH, *flags, "-c", os.path.join(CSRC, src), "-o", obj])
    with ThreadPoolExecutor(max_workers=len(cmds)) as ex:
        list(ex.map(lambda c: _run(c, verbose), cmds))
    tmp = out + ".tmp"
    _run([nv, *ARCH, "-shared", "-o", tmp, *objs, "-lcudart_static", "-lrt", "-ldl", "-lpthread"], verbose)
    os.replace(tmp, out)
    return out


if __name__ == "__main__":
    build(verbose="-v" in sys.argv)
    print(LIB)
