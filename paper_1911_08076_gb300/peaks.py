"""Build and run the peak-rate microbenchmark (csrc/peaks_main.cu) on cuda:0.

    python -m paper_1911_08076_gb300.peaks

Prints one JSON object with the measured rates of tcgen05 e4m3 MMA (N = 64,
128, 256), warp mma.sync (s8, e4m3, b1 and.popc) and CUDA-core popc.
"""
from __future__ import annotations

import os
import subprocess
import sys

from . import build as _build


def main() -> int:
    out = os.path.join(_build.OUT, "peaks_main")
    os.makedirs(_build.OUT, exist_ok=True)
    src = os.path.join(_build.CSRC, "peaks_main.cu")
    subprocess.check_call([_build._nvcc(), *_build.ARCH, "-O3", "-std=c++17", src, "-o", out])
    return subprocess.call([out])


if __name__ == "__main__":
    sys.exit(main())
