"""ifq_forward_noalloc, the allocation-free form of ifq_forward (collected last on purpose).

Its persistent launch keeps completion counters in a file-scope device array
instead of a caller's workspace, so the checks here are that two calls in a
row give exactly what ifq_forward gives (the counters are re-zeroed on every
call), both for a stack that takes the persistent launch (checked with
ifq_last_forward_mode: the one persistent launch is what ran) and for one that
runs layer by layer, and that a stack needing more
counters than the array holds is refused before anything runs.
"""
import numpy as np
import pytest
import torch

from paper_1911_08076_gb300 import ifq, synth
from paper_1911_08076_gb300.stack import DeviceStack

DEV = "cuda"


def _outputs(st):
    return {li: {k: v.copy() for k, v in st.output(li).items()} for li in range(len(st.wl.layers))}


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["resnet18", "tinyyolo"])
def test_noalloc_forward_equals_forward_on_two_calls_in_a_row(name, monkeypatch):
    monkeypatch.setenv("IFQ_STACK", "1")
    wl = synth.get(name, batch=4)
    x, params = synth.draw_workload(wl)
    st = DeviceStack(wl, params)
    persistent = st.ws_bytes > 0          # resnet18: conv-only stack; tinyyolo has pooling layers
    assert persistent == (name == "resnet18")
    monkeypatch.delenv("IFQ_STACK")
    xd = torch.from_numpy(synth.pack_codes(x)).to(DEV)
    ifq.ifq_forward(st.layers, xd)        # reference: the default entry point, one launch per layer
    torch.cuda.synchronize()
    assert ifq.ifq_last_forward_mode() == ifq.IFQ_FORWARD_LAYERS
    ref = _outputs(st)
    for call in range(2):
        for t in list(st.y_codes.values()) + list(st.y_acc.values()):
            t.fill_(-1)                   # every output element must be written again
        ifq.ifq_forward_noalloc(st.layers, xd)
        torch.cuda.synchronize()
        assert ifq.ifq_device_status() == ifq.IFQ_OK, call
        # the persistent launch (the one that uses the device counter array) is what ran
        expect = ifq.IFQ_FORWARD_PERSISTENT if persistent else ifq.IFQ_FORWARD_LAYERS
        assert ifq.ifq_last_forward_mode() == expect, call
        got = _outputs(st)
        for li in ref:
            for k in ref[li]:
                assert np.array_equal(got[li][k], ref[li][k]), (call, wl.layers[li].name, k)


def test_noalloc_forward_refuses_stacks_beyond_its_counters():
    """A single 3x3 layer over 600 x 128 x 128 output pixels needs 76800 counters (one per 128 rows),
    more than the 65536 the array holds: refused with IFQ_EWORKSPACE before any launch (the
    buffers are never touched, so placeholder addresses do)."""
    fake = 1 << 20
    d = ifq.conv_desc(600, 128, 128, 64, 64, 3, 1, 1)
    L = ifq.Layer(kind=ifq.IFQ_LAYER_CONV, src=-1, conv=d, w_prep=fake, thr=fake, sign=fake, y_codes=fake)
    with pytest.raises(ifq.IfqError) as e:
        ifq.ifq_forward_noalloc([L], fake, stream=0)
    assert e.value.status == ifq.IFQ_EWORKSPACE
