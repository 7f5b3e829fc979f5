"""Host-side checks of the k-bit codes (k = 3, 4; Eq. (8) and Table 2's k columns), no GPU:
the storage format of the packed codes, descriptor refusals, chain checks of the code width,
and which kernel path a descriptor takes."""
import numpy as np
import pytest

from paper_1911_08076_gb300 import ifq, synth

FAKE = 1 << 20


def _status(fn, *a, **kw):
    with pytest.raises(ifq.IfqError) as e:
        fn(*a, **kw)
    return e.value.status


def test_storage_format_is_fields_of_2_or_4_bits():
    """k = 2: four 2-bit fields per byte; k = 3, 4: two 4-bit fields per byte, channel c in the
    field c % 2 of byte c // 2 (low nibble first), a 3-bit code in the low bits of its field."""
    codes = np.array([[1, 2, 3, 4, 15, 0, 7, 9]], np.uint8)
    assert synth.pack_codes(codes, 4).tolist() == [[0x21, 0x43, 0x0F, 0x97]]
    c3 = np.array([[1, 2, 3, 4, 7, 0, 5, 6]], np.uint8)
    assert synth.pack_codes(c3, 3).tolist() == [[0x21, 0x43, 0x07, 0x65]]
    c2 = np.array([[1, 2, 3, 0]], np.uint8)
    assert synth.pack_codes(c2, 2).tolist() == [[0b00111001]]
    rng = np.random.default_rng(0)
    for k in (2, 3, 4):
        x = rng.integers(0, 1 << k, (3, 5, 7, 24), dtype=np.uint8)
        p = synth.pack_codes(x, k)
        assert p.shape == (3, 5, 7, 24 * synth.field_bits(k) // 8)
        assert (synth.unpack_codes(p, kbits=k) == x).all()
        assert p.nbytes == ifq.ifq_codes_storage_bytes(3, 5, 7, 24, k)
    with pytest.raises(AssertionError):
        synth.pack_codes(np.full((1, 4), 8, np.uint8), 3)      # 8 is not a 3-bit code


def test_storage_bytes_refusals():
    assert ifq.ifq_codes_storage_bytes(2, 3, 3, 64, 0) == 2 * 9 * 16       # 0 means 2 bits
    assert _status(ifq.ifq_codes_storage_bytes, 1, 1, 1, 64, 5) == ifq.IFQ_EUNSUPPORTED
    assert _status(ifq.ifq_codes_storage_bytes, 1, 1, 1, 64, 1) == ifq.IFQ_EUNSUPPORTED
    assert _status(ifq.ifq_codes_storage_bytes, 1, 1, 1, 64, -1) == ifq.IFQ_EINVAL
    assert _status(ifq.ifq_codes_storage_bytes, 1, 1, 1, 62, 4) == ifq.IFQ_ESHAPE
    # the dense memory count of the paper's comparisons is a different number for k = 3
    assert ifq.ifq_codes_bytes(1, 1, 1, 64, 3) == 24
    assert ifq.ifq_codes_storage_bytes(1, 1, 1, 64, 3) == 32


def test_kbits_descriptor_refusals():
    for kb, st in ((5, ifq.IFQ_EUNSUPPORTED), (1, ifq.IFQ_EUNSUPPORTED), (-1, ifq.IFQ_EINVAL)):
        d = ifq.conv_desc(1, 8, 8, 64, 64, 3, 1, 1, kbits=kb)
        assert _status(ifq.ifq_weights_prep_bytes, d) == st
        assert _status(ifq.ifq_conv2bit, d, FAKE, FAKE, FAKE, FAKE, FAKE, stream=0) == st
        assert _status(ifq.ifq_maxpool2bit, ifq.pool_desc(1, 8, 8, 64, 2, 2, 0, kb), FAKE, None, FAKE,
                       stream=0) == st
    assert _status(ifq.ifq_pack_codes_kbits, FAKE, FAKE, 64, 6, stream=0) == ifq.IFQ_EUNSUPPORTED


def test_stack_rejects_a_code_width_change_along_the_chain():
    L0 = ifq.Layer(kind=ifq.IFQ_LAYER_CONV, src=-1, conv=ifq.conv_desc(1, 8, 8, 64, 32, 3, 1, 1, kbits=4),
                   w_prep=FAKE, thr=FAKE, sign=FAKE, y_codes=FAKE)
    L1 = ifq.Layer(kind=ifq.IFQ_LAYER_CONV, src=0, conv=ifq.conv_desc(1, 8, 8, 32, 32, 3, 1, 1, kbits=2),
                   w_prep=FAKE, thr=FAKE, sign=FAKE, y_codes=FAKE)
    assert _status(ifq.ifq_forward, [L0, L1], FAKE, stream=0) == ifq.IFQ_ESHAPE
    P1 = ifq.Layer(kind=ifq.IFQ_LAYER_POOL, src=0, pool=ifq.pool_desc(1, 8, 8, 32, 2, 2, 0, 3), y_codes=FAKE)
    assert _status(ifq.ifq_forward, [L0, P1], FAKE, stream=0) == ifq.IFQ_ESHAPE


def test_persistent_stack_is_2bit_only(monkeypatch):
    monkeypatch.setenv("IFQ_STACK", "1")
    for kb, eligible in ((2, True), (4, False)):
        layers = [ifq.Layer(kind=ifq.IFQ_LAYER_CONV, src=i - 1, conv=ifq.conv_desc(2, 16, 16, 64, 64, 3, 1, 1,
                                                                                     kbits=kb),
                            w_prep=FAKE, thr=FAKE, sign=FAKE, y_codes=FAKE) for i in range(2)]
        assert (ifq.ifq_forward_workspace_bytes(layers) > 0) == eligible


TC, BS = ifq.IFQ_PATH_TC, ifq.IFQ_PATH_BITSERIAL


@pytest.mark.parametrize("desc,kb,path", [
    ((8, 14, 14, 256, 256, 3, 1, 1), 4, TC),          # (2^4-1) K = 34560
    ((8, 6, 6, 256, 512, 6, 1, 0), 4, TC),            # FC6 as a conv, 15 * 9216 = 138240
    ((4, 1, 1, 13088, 64, 1, 1, 0), 4, TC),           # 15 * 13088 = 196320 (cin % 32 == 0: 16-byte granules)
    ((4, 1, 1, 13120, 64, 1, 1, 0), 4, BS),           # 15 * 13120 = 196800 > 196608
    ((4, 1, 1, 28064, 64, 1, 1, 0), 3, TC),           # 7 * 28064 = 196448
    ((4, 1, 1, 65536, 64, 1, 1, 0), 2, TC),           # 3 * 65536 = 196608
    ((2, 9, 9, 12, 16, 3, 1, 1), 4, BS),              # 4-bit fields need cin % 8 == 0 on the tensor cores
    ((2, 9, 9, 12, 16, 3, 1, 1), 2, TC),
    ((2, 9, 9, 40, 16, 3, 1, 1), 4, TC),              # 20 bytes a pixel: 4-byte granules
])
def test_conv_plan(desc, kb, path):
    d = ifq.conv_desc(*desc, out_mode=ifq.IFQ_OUT_BOTH, path=TC, kbits=kb)
    assert ifq.ifq_conv_plan(d) == path
    d.path = BS
    assert ifq.ifq_conv_plan(d) == BS


def test_conv_plan_refuses_a_fused_pool_off_the_tensor_cores():
    assert ifq.ifq_conv_plan(ifq.conv_desc(2, 8, 8, 64, 64, 3, 1, 1, pool=2, kbits=4)) == TC
    d = ifq.conv_desc(2, 8, 8, 12, 64, 3, 1, 1, pool=2, kbits=4)
    assert _status(ifq.ifq_conv_plan, d) == ifq.IFQ_EUNSUPPORTED


def test_conv_plan_takes_the_narrow_bitserial_kernel_where_it_wins():
    """2-bit 3x3 stride-1 layers with cin * cout <= 128 run on the narrow bit-serial kernel unless
    the warp-MMA kernel takes them (8 input channels: IFQ-Tinier-YOLO's conv2, 8 -> 16); wider ones
    take the tensor cores (the window path where it applies)."""
    assert ifq.ifq_conv_plan(ifq.conv_desc(64, 208, 208, 8, 16, 3, 1, 1, pool=2)) == ifq.IFQ_PATH_WARP
    assert ifq.ifq_conv_plan(ifq.conv_desc(64, 208, 208, 4, 16, 3, 1, 1, pool=2)) == BS
    assert ifq.ifq_conv_plan(ifq.conv_desc(64, 208, 208, 16, 32, 3, 1, 1, pool=2)) == ifq.IFQ_PATH_WIN
    assert ifq.ifq_conv_plan(ifq.conv_desc(2, 16, 16, 8, 16, 3, 2, 1)) == TC      # stride 2
    assert ifq.ifq_conv_plan(ifq.conv_desc(2, 16, 16, 16, 32, 3, 1, 1, pool=2, path=BS)) == BS
    assert _status(ifq.ifq_conv_plan, ifq.conv_desc(2, 16, 16, 64, 64, 3, 1, 1, pool=2, path=BS)) == \
        ifq.IFQ_EUNSUPPORTED                                                          # no narrow form
