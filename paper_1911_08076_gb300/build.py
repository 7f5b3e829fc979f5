"""Build the C-ABI shared library libifq.so in-tree (nvcc for sm_103a + g++ for host code).

    python -m paper_1911_08076_gb300.build        # or build() from Python

The two translation units compile in parallel; the result is
paper_1911_08076_gb300/_build/libifq.so.
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
OUT = os.path.join(PKG, "_build")
LIB = os.path.join(OUT, "libifq.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def _nvcc() -> str:
    p = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(p):
        raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libifq.so")
    return p


def _sources():
    return [os.path.join(CSRC, f) for f in sorted(os.listdir(CSRC))] + [os.path.join(INCLUDE, "ifq.h")]


def _stale() -> bool:
    if not os.path.exists(LIB):
        return True
    t = os.path.getmtime(LIB)
    return any(os.path.getmtime(s) > t for s in _sources())


def build(force: bool = False, verbose: bool = False) -> str:
    if not force and not _stale():
        return LIB
    os.makedirs(OUT, exist_ok=True)
    nvcc = _nvcc()
    tag = f"{os.getpid()}"
    o_cu = os.path.join(OUT, f"ifq_api.{tag}.o")
    o_cpp = os.path.join(OUT, f"ifq_host.{tag}.o")
    cmds = [
        [nvcc, *ARCH, "-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-I", INCLUDE, "-I", CSRC,
         "-Xptxas", "-v" if verbose else "-O3", "-c", os.path.join(CSRC, "ifq_api.cu"), "-o", o_cu],
        ["g++", "-O2", "-std=c++17", "-fPIC", "-ffp-contract=off", "-fno-fast-math", "-I", INCLUDE, "-c",
         os.path.join(CSRC, "ifq_host.cpp"), "-o", o_cpp],
    ]

    def run(cmd):
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"build failed: {' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
        return r.stdout + r.stderr

    with ThreadPoolExecutor(2) as ex:
        logs = list(ex.map(run, cmds))
    tmp = LIB + f".{tag}.tmp"
    cudalib = os.path.join(os.path.dirname(os.path.dirname(nvcc)), "lib64")
    run([nvcc, *ARCH, "-shared", "-cudart", "shared", o_cu, o_cpp, "-Xlinker", f"-rpath={cudalib}", "-o", tmp])
    os.replace(tmp, LIB)
    for o in (o_cu, o_cpp):
        os.remove(o)
    if verbose:
        sys.stdout.write("".join(logs))
    return LIB


if __name__ == "__main__":
    print(build(force=True, verbose="-v" in sys.argv))
