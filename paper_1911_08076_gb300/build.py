"""Build the C-ABI shared library libifq.so in-tree (nvcc for sm_103a + g++ for host code).

    python -m paper_1911_08076_gb300.build        # or build() from Python

The two translation units compile in parallel; the result is
paper_1911_08076_gb300/_build/libifq.so.
"""
from __future__ import annotations

import os
import re
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


# The warp-specialised tensor-core kernels run at the 72-register cap of 864 threads per CTA; every
# instance must fit it without spilling to local memory (a build with spills is refused).
_GUARDED = ("conv_tc_kernel", "conv_stack_kernel")


def spilling_kernels(ptxas_log: str):
    """Entry points of the guarded kernels whose ptxas report shows spill stores or loads."""
    bad, cur = [], None
    for line in ptxas_log.splitlines():
        m = re.search(r"Compiling entry function '([^']+)'", line)
        if m:
            cur = m.group(1)
            continue
        m = re.search(r"(\d+) bytes spill stores, (\d+) bytes spill loads", line)
        if m and cur and any(g in cur for g in _GUARDED) and (int(m.group(1)) or int(m.group(2))):
            bad.append(cur)
    return bad


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
         "-Xptxas", "-v", "-c", os.path.join(CSRC, "ifq_api.cu"), "-o", o_cu],
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
    spilled = spilling_kernels(logs[0])
    if spilled:
        raise RuntimeError("tensor-core kernels spill registers to local memory: " + ", ".join(spilled))
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
