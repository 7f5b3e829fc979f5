"""Whole-stack parity helper for the GPU tests: a layer stack run through ifq_forward on the GPU,
compared output by output, image by image, with the CPU oracle (bit-exact codes and int32
accumulators)."""
import numpy as np
import torch

from oracle import oracle as O
from paper_1911_08076_gb300 import ifq, synth
from paper_1911_08076_gb300.stack import DeviceStack


def compare_stack_with_oracle(wl, x, params):
    """Run the whole stack on the GPU through ifq_forward and compare every output of every layer,
    for every image of the batch, with the oracle (which checks its own integer chain against the
    float chain on the way)."""
    st = DeviceStack(wl, params)
    xd = st.input_buffer()
    xd.copy_(torch.from_numpy(synth.pack_codes(x, 8 if wl.in_bits == 8 else wl.kbits)))
    st.forward(xd)
    torch.cuda.synchronize()
    assert ifq.ifq_device_status() == ifq.IFQ_OK
    ref = O.forward(wl, x, params)
    for li, l in enumerate(wl.layers):
        out = st.output(li)
        r = ref[li]
        if l.kind == "conv" and l.out == "both":
            assert (synth.unpack_codes(out["codes"], l.cout, wl.kbits) == r["codes"]).all(), l.name
            assert (out["acc"] == r["acc"]).all(), l.name
        elif l.kind == "fixed" or (l.kind == "conv" and l.out == "acc"):
            assert (out["acc"] == r).all(), l.name
        else:
            c = l.cout if l.kind == "conv" else l.c
            got = synth.unpack_codes(out["codes"], c, wl.kbits)
            if not (got == r).all():
                bad = np.argwhere(got != r)
                raise AssertionError(f"{wl.name} layer {l.name}: {len(bad)} codes differ, first at {bad[:4].tolist()}")
    st.release()
