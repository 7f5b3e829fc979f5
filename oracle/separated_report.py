"""Separated vs integrated fixed-point conversion on the synthetic workloads (oracle only).

Analysis script, like the rest of oracle/: test infrastructure, not the product
path.  It is a data-free analogue of the paper's Table 2.  Table 2 measures
ImageNet accuracy; here, with calibrated synthetic parameters
(synth.draw_conv_params_calibrated), it counts how many 2-bit codes change:

* per layer: on the same input codes, the fraction of output codes of the separated
  conversion at Q_m = 2^m (Sec. 2.2) that differ from the float chain's;
* end to end: propagating each conversion through the whole stack (each layer takes
  its own previous outputs), the fraction of the last layer's outputs that differ.

The integrated conversion (Sec. 3.2) gives exactly the float chain's codes; that
is pinned exhaustively in tests/test_oracle.py, so its column is 0 by
construction.  A layer with accumulator output (FC7, detection) compares the
accumulators A, which the conversion does not touch, so it reports the codes of
its input instead.

    python -m oracle.separated_report [--images N]
"""
from __future__ import annotations

import argparse
import sys

import numpy as np

from oracle import oracle as O
from paper_1911_08076_gb300 import synth

MS = (8, 9, 10, 12)


def run(name: str, images: int):
    wl = synth.get(name, batch=images)
    rng = np.random.default_rng(wl.seed)
    params = [synth.draw_conv_params_calibrated(rng, l) if l.kind == "conv" else None for l in wl.layers]
    x = synth.draw_codes(rng, (images, wl.h, wl.w, wl.c))
    P = {i: O.Params.from_synth(c) for i, c in enumerate(params) if c is not None}
    sgn = {i: np.where(params[i].gamma < 0, -1, 1).astype(np.int8) for i in P}
    per_layer = {m: [] for m in MS}
    outs = {"float": {}}
    outs.update({m: {} for m in MS})
    last_codes = None
    for li, l in enumerate(wl.layers):
        for key in outs:
            src = x if l.src < 0 else outs[key][l.src]
            if l.kind == "pool":
                outs[key][li] = O.maxpool_codes(src, l.k, l.stride, l.pad, sgn[l.src] if l.signed else None)
                continue
            A = O.conv_acc(src, params[li].w, l.stride, l.pad)
            if l.out == "acc":
                outs[key][li] = src                       # the conversion only acts on coded layers
            elif key == "float":
                outs[key][li] = O.float_chain(A, P[li])
            else:
                outs[key][li] = O.separated_chain(A, P[li], key)
        if l.kind == "conv" and l.out != "acc":
            A = O.conv_acc(x if l.src < 0 else outs["float"][l.src], params[li].w, l.stride, l.pad)
            f = outs["float"][li]
            for m in MS:
                per_layer[m].append(float(np.mean(O.separated_chain(A, P[li], m) != f)))
            last_codes = li
    end = {m: float(np.mean(outs[m][last_codes] != outs["float"][last_codes])) for m in MS}
    return {m: float(np.mean(per_layer[m])) for m in MS}, {m: float(np.max(per_layer[m])) for m in MS}, end


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--images", type=int, default=2)
    ap.add_argument("--workloads", default="alexnet,resnet18,tinieryolo")
    a = ap.parse_args(argv)
    print("| workload | m | codes changed per layer (mean / max) | last coded layer, end to end |")
    print("|---|---:|---:|---:|")
    for name in a.workloads.split(","):
        mean, mx, end = run(name, a.images)
        for m in MS:
            print(f"| {name} | {m} | {100 * mean[m]:.3f} % / {100 * mx[m]:.3f} % | {100 * end[m]:.2f} % |")
        print(f"| {name} | integrated | 0 (exact) | 0 (exact) |")
        sys.stdout.flush()


if __name__ == "__main__":
    main()
