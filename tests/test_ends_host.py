"""Host-side checks of the network's two non-binary-input ends (no GPU): the first layer on 8-bit
image values and the separated fixed-point output of the detection conv (Sec. 2.2, Sec. 4.2)."""
import numpy as np
import pytest

from oracle import oracle as O
from paper_1911_08076_gb300 import ifq, synth

FAKE = 1 << 20
TC, BS, DI = ifq.IFQ_PATH_TC, ifq.IFQ_PATH_BITSERIAL, ifq.IFQ_PATH_DIRECT


def _status(fn, *a, **kw):
    with pytest.raises(ifq.IfqError) as e:
        fn(*a, **kw)
    return e.value.status


def test_8bit_input_plan_and_refusals():
    d = ifq.conv_desc(2, 20, 20, 4, 8, 3, 1, 1, ifq.IFQ_OUT_BOTH, in_bits=8)
    assert ifq.ifq_conv_plan(d) == ifq.IFQ_PATH_WARP           # 3 x 3, few channels, no pool: warp MMAs
    d.path = TC
    assert ifq.ifq_conv_plan(d) == TC
    d.path = DI
    assert ifq.ifq_conv_plan(d) == DI
    assert ifq.ifq_conv_plan(ifq.conv_desc(2, 20, 20, 4, 8, 5, 1, 2, in_bits=8)) == DI      # 5 x 5: direct
    assert ifq.ifq_conv_plan(ifq.conv_desc(2, 20, 20, 4, 8, 3, 1, 1, pool=2, in_bits=8)) == DI
    assert ifq.ifq_conv_plan(ifq.conv_desc(2, 20, 20, 4, 64, 3, 1, 1, in_bits=8)) == TC      # cout > 32
    assert ifq.ifq_conv_plan(ifq.conv_desc(2, 20, 20, 32, 8, 3, 1, 1, in_bits=8)) == TC      # K = 288 > 257
    assert ifq.ifq_conv_plan(ifq.conv_desc(2, 20, 20, 64, 64, 3, 1, 1, path=DI)) == TC      # 2-bit codes
    assert _status(ifq.ifq_conv_plan, ifq.conv_desc(2, 20, 20, 4, 8, 3, 1, 1, path=BS, in_bits=8)) == \
        ifq.IFQ_EUNSUPPORTED                                   # no bit-serial path for 8-bit values
    assert _status(ifq.ifq_conv_plan, ifq.conv_desc(1, 9, 9, 88, 8, 3, 1, 1, in_bits=8)) == \
        ifq.IFQ_EUNSUPPORTED                                   # 255 * 792 > 196608
    assert ifq.ifq_conv_plan(ifq.conv_desc(1, 9, 9, 84, 8, 3, 1, 1, in_bits=8)) == TC   # 255 * 756, K > 257
    assert _status(ifq.ifq_weights_prep_bytes, ifq.conv_desc(1, 9, 9, 4, 8, 3, in_bits=5)) == ifq.IFQ_EUNSUPPORTED
    assert _status(ifq.ifq_weights_prep_bytes, ifq.conv_desc(1, 9, 9, 4, 8, 3, in_bits=-1)) == ifq.IFQ_EINVAL
    assert ifq.ifq_weights_prep_bytes(ifq.conv_desc(1, 9, 9, 4, 8, 3, in_bits=2)) > 0   # = kbits: plain codes


def test_stack_checks_for_the_ends():
    c0 = ifq.Layer(kind=ifq.IFQ_LAYER_CONV, src=-1, conv=ifq.conv_desc(1, 8, 8, 64, 32, 3, 1, 1), w_prep=FAKE,
                   thr=FAKE, sign=FAKE, y_codes=FAKE)
    # a layer on 8-bit values reads only the stack input
    c8 = ifq.Layer(kind=ifq.IFQ_LAYER_CONV, src=0, conv=ifq.conv_desc(1, 8, 8, 32, 32, 3, 1, 1, in_bits=8),
                   w_prep=FAKE, thr=FAKE, sign=FAKE, y_codes=FAKE)
    assert _status(ifq.ifq_forward, [c0, c8], FAKE, stream=0) == ifq.IFQ_ESHAPE
    # a fixed-point output needs a conv that writes accumulators
    fx = ifq.Layer(kind=ifq.IFQ_LAYER_FIXED, src=0, fixed=ifq.FixedDesc(14), fx_mul=FAKE, fx_add=FAKE, y_acc=FAKE)
    assert _status(ifq.ifq_forward, [c0, fx], FAKE, stream=0) == ifq.IFQ_ESHAPE
    p1 = ifq.Layer(kind=ifq.IFQ_LAYER_POOL, src=0, pool=ifq.pool_desc(1, 8, 8, 32, 2, 2), y_codes=FAKE)
    fx2 = ifq.Layer(kind=ifq.IFQ_LAYER_FIXED, src=1, fixed=ifq.FixedDesc(14), fx_mul=FAKE, fx_add=FAKE, y_acc=FAKE)
    assert _status(ifq.ifq_forward, [c0, p1, fx2], FAKE, stream=0) == ifq.IFQ_EINVAL
    fx3 = ifq.Layer(kind=ifq.IFQ_LAYER_FIXED, src=-1, fixed=ifq.FixedDesc(14), fx_mul=FAKE, fx_add=FAKE, y_acc=FAKE)
    assert _status(ifq.ifq_forward, [fx3], FAKE, stream=0) == ifq.IFQ_EINVAL
    ca = ifq.Layer(kind=ifq.IFQ_LAYER_CONV, src=-1,
                   conv=ifq.conv_desc(1, 8, 8, 64, 32, 3, 1, 1, out_mode=ifq.IFQ_OUT_ACC), w_prep=FAKE, y_acc=FAKE)
    fx4 = ifq.Layer(kind=ifq.IFQ_LAYER_FIXED, src=0, fixed=ifq.FixedDesc(25), fx_mul=FAKE, fx_add=FAKE, y_acc=FAKE)
    assert _status(ifq.ifq_forward, [ca, fx4], FAKE, stream=0) == ifq.IFQ_EINVAL       # m beyond 24


@pytest.mark.parametrize("m", [9, 14, 24])
def test_output_fold_equals_the_oracle(m):
    """ifq_fold_output_separated's (mul, add), applied as floor((mul A + add) / 2^m) in exact Python
    integers, equals the oracle's element-by-element separated output on every A."""
    rng = np.random.default_rng(m)
    cout = 30
    alpha = rng.uniform(0.001, 0.2, cout).astype(np.float32)
    bias = rng.normal(0, 1, cout).astype(np.float32)
    mul, add = ifq.ifq_fold_output_separated(m, alpha, synth.STEP, bias)
    A = rng.integers(-40000, 40000, (64, cout)).astype(np.int32)
    host = np.array([[max(min((int(mul[n]) * int(a) + int(add[n])) >> m, 2 ** 31 - 1), -2 ** 31)
                      for n, a in enumerate(row)] for row in A], dtype=np.int64)
    p = O.Params(alpha.astype(np.float64), np.ones(cout), np.zeros(cout), np.zeros(cout), np.ones(cout),
                 bias.astype(np.float64), synth.STEP, 0.5, -0.25, 0.0)
    assert (host == O.fixed_output(A, p, m)).all()


def test_output_fold_and_kernel_refusals():
    one = np.ones(3, np.float32)
    for m, al in ((0, one), (25, one), (14, one * 0), (14, one * np.nan)):
        assert _status(ifq.ifq_fold_output_separated, m, al) == ifq.IFQ_EINVAL
    assert _status(ifq.ifq_fixed_output, FAKE, -1, 30, FAKE, FAKE, 14, FAKE, stream=0) == ifq.IFQ_EINVAL
    assert _status(ifq.ifq_fixed_output, FAKE, 8, 30, FAKE, FAKE, 25, FAKE, stream=0) == ifq.IFQ_EINVAL
    assert _status(ifq.ifq_fixed_output, FAKE, 8, 30, FAKE + 4, FAKE, 14, FAKE, stream=0) == ifq.IFQ_EALIGN
    assert _status(ifq.ifq_fixed_output, FAKE, 1 << 26, 64, FAKE, FAKE, 14, FAKE, stream=0) == ifq.IFQ_ERANGE


def test_tinier_yolo_full_layer_table():
    """IFQ-Tinier-YOLO (Sec. 4.2): every conv binary, the first on the 8-bit image, half the Tiny-YOLO
    widths, a 1x1 third-to-last conv, the detection conv's accumulators converted at m = 14."""
    wl = synth.get("tinieryolo_full")
    convs = [l for l in wl.layers if l.kind == "conv"]
    assert convs[0].in_bits == 8 and all(l.in_bits == 0 for l in convs[1:])
    assert [l.cout for l in convs] == [8, 16, 32, 64, 128, 256, 512, 512, 30]
    assert convs[-3].k == 1 and convs[-1].out == "acc"
    assert wl.layers[-1].kind == "fixed" and wl.layers[-1].m == 14 and wl.layers[-1].src == len(wl.layers) - 2
    x, params = synth.draw_workload(wl, batch=2)
    assert x.shape == (2, 416, 416, 4) and x[..., 3].max() == 0 and x[..., :3].max() > 200
    assert params[0].delta_in == synth.PIXEL_STEP


def test_empty_batch_is_a_validated_no_op():
    """n = 0: shapes as usual, arguments still checked, nothing launched (so this runs without a GPU)."""
    d = ifq.conv_desc(0, 14, 14, 64, 64, 3, 1, 1, ifq.IFQ_OUT_BOTH)
    assert ifq.ifq_conv_out_shape(d) == (14, 14)
    ifq.ifq_conv2bit(d, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, stream=0)
    assert _status(ifq.ifq_conv2bit, d, None, FAKE, FAKE, FAKE, FAKE, FAKE, stream=0) == ifq.IFQ_EINVAL
    assert _status(ifq.ifq_conv2bit, d, FAKE + 4, FAKE, FAKE, FAKE, FAKE, FAKE, stream=0) == ifq.IFQ_EALIGN
    ifq.ifq_conv2bit(ifq.conv_desc(0, 16, 16, 64, 64, 3, 1, 1, pool=2), FAKE, FAKE, FAKE, FAKE, FAKE, stream=0)
    ifq.ifq_conv2bit(ifq.conv_desc(0, 16, 16, 4, 8, 3, 1, 1, in_bits=8), FAKE, FAKE, FAKE, FAKE, FAKE, stream=0)
    p = ifq.pool_desc(0, 8, 8, 64, 2, 2)
    assert ifq.ifq_pool_out_shape(p) == (4, 4)
    ifq.ifq_maxpool2bit(p, FAKE, None, FAKE, stream=0)
    layers = [ifq.Layer(kind=ifq.IFQ_LAYER_CONV, src=i - 1, conv=ifq.conv_desc(0, 8, 8, 64, 64, 3, 1, 1),
                        w_prep=FAKE, thr=FAKE, sign=FAKE, y_codes=FAKE) for i in range(3)]
    ifq.ifq_forward(layers, FAKE, stream=0)
    ifq.ifq_forward_noalloc(layers, FAKE, stream=0)
    assert _status(ifq.ifq_conv_out_shape, ifq.conv_desc(-1, 8, 8, 64, 64, 3)) == ifq.IFQ_ESHAPE


def test_wait_selftest_refuses_bad_limits():
    assert _status(ifq.ifq_wait_selftest, 0, stream=0) == ifq.IFQ_EINVAL
    assert _status(ifq.ifq_wait_selftest, 2000000, stream=0) == ifq.IFQ_EINVAL


def test_synthetic_draws_follow_the_stated_recipe():
    """The benchmark inputs follow the recipe of the design notes (all workloads seeded): codes
    uniform on {0..2^k-1}, filters uniform +-1, alpha ~ U(0.5, 1.5), gamma ~ N(1, 0.3), beta ~
    N(0, 0.5), mean ~ N(0, 2), var ~ U(0.5, 2); the seed is 1911_08076 + the workload index, so two
    draws are identical.  N(1, 0.3) puts 0.04 % of the channels at a negative BN scale (the parity
    tests draw their own parameters with many more)."""
    from paper_1911_08076_gb300 import synth
    wl = synth.get("resnet18")
    assert wl.seed == synth.SEED_BASE + wl.index
    x, params = synth.draw_workload(wl)
    x2, params2 = synth.draw_workload(wl)
    assert np.array_equal(x, x2) and np.array_equal(params[0].w, params2[0].w)
    counts = np.bincount(x.ravel(), minlength=4) / x.size
    assert np.allclose(counts, 0.25, atol=0.002)
    convs = [p for l, p in zip(wl.layers, params) if l.kind == "conv"]
    w = np.concatenate([p.w.ravel() for p in convs])
    assert set(np.unique(w)) == {-1, 1} and abs(w.mean()) < 0.002
    cat = lambda f: np.concatenate([getattr(p, f) for p in convs]).astype(np.float64)
    alpha, gamma, beta, mean, var = map(cat, ("alpha", "gamma", "beta", "mean", "var"))
    assert alpha.min() >= 0.5 and alpha.max() <= 1.5 and abs(alpha.mean() - 1.0) < 0.03
    assert abs(gamma.mean() - 1.0) < 0.03 and abs(gamma.std() - 0.3) < 0.02
    assert (gamma < 0).mean() < 0.002                 # P(N(1, 0.3) < 0) = 0.0004
    assert abs(beta.std() - 0.5) < 0.03 and abs(mean.std() - 2.0) < 0.1
    assert var.min() >= 0.5 and var.max() <= 2.0
