"""Host-side checks of the C ABI (no GPU): exported symbols, the product fold
against the oracle fold, synchronous argument errors, shapes and packed sizes."""
import ctypes
import re

import numpy as np
import pytest

from oracle import oracle as O
from paper_1911_08076_gb300 import ifq, synth

HEADER = __import__("os").path.join(__import__("os").path.dirname(__file__), "..", "include", "ifq.h")


def test_library_exports_every_declared_symbol():
    src = open(HEADER).read()
    declared = set(re.findall(r"^(?:int|const char\*)\s+(ifq_\w+)\(", src, re.M))
    assert declared, "no declarations parsed"
    L = ctypes.CDLL(ifq.lib_path()) if ifq.lib() else None
    missing = [n for n in sorted(declared) if not hasattr(L, n)]
    assert not missing, missing
    assert declared == set(ifq.EXPORTS), declared ^ set(ifq.EXPORTS)


def _fold_both(K, alpha, gamma, beta, mean, var, bias=None, eps=synth.EPS, kbits=2, delta=0.5, qb=0.5, qo=-0.25):
    T1, s1 = ifq.ifq_fold_layer(K, alpha, gamma, beta, mean, var, delta, bias, eps, qb, qo, kbits)
    f = lambda a: None if a is None else np.asarray(a, np.float32).astype(np.float64)
    p = O.Params(f(alpha), f(gamma), f(beta), f(mean), f(var), f(bias), delta, qb, qo, float(np.float32(eps)), kbits)
    T2, s2 = O.fold(p, K)
    return T1, s1, T2, s2


@pytest.mark.parametrize("seed", range(6))
def test_product_fold_equals_oracle_fold(seed):
    rng = np.random.default_rng(seed)
    n = 4096
    K = int(rng.choice([9, 72, 576, 2304, 9216]))
    gamma = rng.normal(0.5, 1.0, n)
    gamma[:16] = 0.0
    T1, s1, T2, s2 = _fold_both(K, rng.uniform(1e-3, 3, n), gamma, rng.normal(0, 1, n), rng.normal(0, 5, n),
                                rng.uniform(1e-3, 4, n), rng.normal(0, 2, n) if seed % 2 else None,
                                kbits=1 + seed % 4)
    assert (T1 == T2).all() and (s1 == s2).all()


@pytest.mark.parametrize("wl_name", list(synth.WORKLOADS))
def test_product_fold_equals_oracle_fold_on_workloads(wl_name):
    wl = synth.get(wl_name)
    rng = np.random.default_rng(wl.seed)
    for l in wl.layers:
        if l.kind != "conv":
            continue
        p = synth.draw_conv_params(rng, l)
        T1, s1, T2, s2 = _fold_both(l.k * l.k * l.cin, p.alpha, p.gamma, p.beta, p.mean, p.var)
        assert (T1 == T2).all() and (s1 == s2).all()


def test_fold_rejects_invalid_parameters():
    ok = dict(alpha=[1.0], gamma=[1.0], beta=[0.0], mean=[0.0], var=[1.0])
    for key, bad in (("alpha", [0.0]), ("alpha", [-1.0]), ("var", [-1.0]), ("gamma", [np.nan]), ("mean", [np.inf])):
        args = dict(ok, **{key: bad})
        with pytest.raises(ifq.IfqError) as e:
            ifq.ifq_fold_layer(9, **args)
        assert e.value.status == ifq.IFQ_EINVAL
    with pytest.raises(ifq.IfqError):
        ifq.ifq_fold_layer(9, **ok, q_base=0.0)
    with pytest.raises(ifq.IfqError):
        ifq.ifq_fold_layer(9, **ok, delta_in=-0.5)
    with pytest.raises(ifq.IfqError):
        ifq.ifq_fold_layer(0, **ok)


def test_feature_map_memory_numbers_of_the_paper():
    """Table 4 / Sec. 4.1.3: conv1 output 55x55x96; k=2 -> 0.6 Mbit, k=4 -> 1.1 Mbit; Lin et al.
    112x112x96 at 9 / 10 bits -> 10.8 / 12.0 Mbit; 18x and 10.9x savings."""
    mb = lambda b: b * 8 / 1e6
    k2 = mb(ifq.ifq_codes_bytes(1, 55, 55, 96, 2))
    k4 = mb(ifq.ifq_codes_bytes(1, 55, 55, 96, 4))
    lin9 = mb(ifq.ifq_codes_bytes(1, 112, 112, 96, 9))
    lin10 = mb(ifq.ifq_codes_bytes(1, 112, 112, 96, 10))
    assert round(k2, 1) == 0.6 and int(k4 * 10) / 10 == 1.1
    assert round(lin9, 1) == 10.8 and round(lin10, 1) == 12.0
    assert int(lin9 / k2) == 18
    assert round(round(lin10, 1) / int(k4 * 10) * 10, 1) == 10.9
    assert ifq.ifq_codes_bytes(1, 55, 55, 96, 2) == 72600


@pytest.mark.parametrize("shape", [(1, 9, 9, 8, 4, 3, 1, 1), (2, 27, 27, 96, 256, 5, 1, 2), (1, 56, 56, 64, 128, 1, 2, 0),
                                   (3, 6, 6, 256, 4096, 6, 1, 0), (1, 14, 14, 256, 512, 3, 2, 1)])
def test_conv_out_shape_matches_oracle(shape):
    n, h, w, cin, cout, k, s, p = shape
    assert ifq.ifq_conv_out_shape(ifq.conv_desc(n, h, w, cin, cout, k, s, p)) == (O.conv_out(h, k, s, p),
                                                                                 O.conv_out(w, k, s, p))


@pytest.mark.parametrize("shape", [(1, 27, 27, 256, 3, 2, 0), (1, 13, 13, 512, 2, 1, 1), (2, 208, 208, 32, 2, 2, 0)])
def test_pool_out_shape_matches_oracle(shape):
    n, h, w, c, k, s, p = shape
    assert ifq.ifq_pool_out_shape(ifq.PoolDesc(n, h, w, c, k, s, p)) == (O.pool_out(h, k, s, p),
                                                                          O.pool_out(w, k, s, p))


def test_argument_errors_are_synchronous():
    """Bad descriptors and pointers are rejected before any launch (works without a GPU)."""
    good = dict(n=1, h=8, w=8, cin=64, cout=64, k=3, stride=1, pad=1)
    fake = 1 << 20  # never dereferenced: validation fails first

    def conv(status, x=fake, w=fake, thr=fake, sign=fake, yc=fake, ya=None, **kw):
        d = ifq.conv_desc(**dict(good, **kw))
        with pytest.raises(ifq.IfqError) as e:
            ifq.ifq_conv2bit(d, x, w, thr, sign, yc, ya, stream=0)
        assert e.value.status == status, e.value

    conv(ifq.IFQ_ESHAPE, cin=62)
    conv(ifq.IFQ_ESHAPE, cout=30)                       # codes need cout % 4 == 0
    conv(ifq.IFQ_ESHAPE, k=11)                          # window larger than padded input
    conv(ifq.IFQ_EINVAL, out_mode=7)
    conv(ifq.IFQ_EINVAL, path=9)
    conv(ifq.IFQ_ERANGE, cin=8192, k=3)                 # K = 73728 > 65536
    conv(ifq.IFQ_EINVAL, x=None)
    conv(ifq.IFQ_EINVAL, yc=None)
    conv(ifq.IFQ_EINVAL, thr=None)
    conv(ifq.IFQ_EINVAL, out_mode=ifq.IFQ_OUT_ACC, ya=None)
    conv(ifq.IFQ_EALIGN, x=fake + 4)
    conv(ifq.IFQ_EALIGN, yc=fake + 8)
    pd = ifq.PoolDesc(1, 8, 8, 64, 2, 2, 2)             # pad >= k
    with pytest.raises(ifq.IfqError) as e:
        ifq.ifq_maxpool2bit(pd, fake, None, fake, stream=0)
    assert e.value.status == ifq.IFQ_ESHAPE
    with pytest.raises(ifq.IfqError) as e:
        ifq.ifq_maxpool2bit(ifq.PoolDesc(1, 8, 8, 66, 2, 2, 0), fake, None, fake, stream=0)
    assert e.value.status == ifq.IFQ_ESHAPE


def test_stack_validation_rejects_broken_chains():
    fake = 1 << 20
    L0 = ifq.Layer(kind=ifq.IFQ_LAYER_CONV, src=-1, conv=ifq.conv_desc(1, 8, 8, 64, 32, 3, 1, 1), w_prep=fake,
                   thr=fake, sign=fake, y_codes=fake)
    # next layer claims 16 input channels but layer 0 produces 32
    L1 = ifq.Layer(kind=ifq.IFQ_LAYER_CONV, src=0, conv=ifq.conv_desc(1, 8, 8, 16, 32, 3, 1, 1), w_prep=fake,
                   thr=fake, sign=fake, y_codes=fake)
    with pytest.raises(ifq.IfqError) as e:
        ifq.ifq_forward([L0, L1], fake, stream=0)
    assert e.value.status == ifq.IFQ_ESHAPE
    L2 = ifq.Layer(kind=ifq.IFQ_LAYER_POOL, src=3, pool=ifq.PoolDesc(1, 8, 8, 32, 2, 2, 0), y_codes=fake)
    with pytest.raises(ifq.IfqError) as e:
        ifq.ifq_forward([L0, L2], fake, stream=0)
    assert e.value.status == ifq.IFQ_EINVAL
    # a layer that only writes accumulators cannot feed another layer
    L3 = ifq.Layer(kind=ifq.IFQ_LAYER_CONV, src=-1,
                   conv=ifq.conv_desc(1, 8, 8, 64, 32, 3, 1, 1, out_mode=ifq.IFQ_OUT_ACC), w_prep=fake, y_acc=fake)
    L4 = ifq.Layer(kind=ifq.IFQ_LAYER_POOL, src=0, pool=ifq.PoolDesc(1, 8, 8, 32, 2, 2, 0), y_codes=fake)
    with pytest.raises(ifq.IfqError) as e:
        ifq.ifq_forward([L3, L4], fake, stream=0)
    assert e.value.status == ifq.IFQ_ESHAPE


def test_forward_workspace_is_counters_only_for_the_persistent_launch(monkeypatch):
    """ifq_forward_workspace_bytes: 0 for the default per-layer launches; with IFQ_STACK=1, one
    4-byte completion counter per 128-output-row block of every layer, rounded up to 256 bytes."""
    fake = 1 << 20
    descs = [ifq.conv_desc(3, 20, 20, 64, 64, 3, 1, 1), ifq.conv_desc(3, 20, 20, 64, 128, 3, 2, 1),
             ifq.conv_desc(3, 10, 10, 128, 128, 1, 1, 0)]
    layers = [ifq.Layer(kind=ifq.IFQ_LAYER_CONV, src=i - 1, conv=d, w_prep=fake, thr=fake, sign=fake, y_codes=fake)
              for i, d in enumerate(descs)]
    monkeypatch.delenv("IFQ_STACK", raising=False)
    assert ifq.ifq_forward_workspace_bytes(layers) == 0
    monkeypatch.setenv("IFQ_STACK", "1")
    rows = [3 * 20 * 20, 3 * 10 * 10, 3 * 10 * 10]
    blocks = sum((m + 127) // 128 for m in rows)
    assert ifq.ifq_forward_workspace_bytes(layers) == (4 * blocks + 255) // 256 * 256
    # a pooling layer keeps the stack on per-layer launches
    pool = ifq.Layer(kind=ifq.IFQ_LAYER_POOL, src=2, pool=ifq.PoolDesc(3, 10, 10, 128, 2, 2, 0), y_codes=fake)
    assert ifq.ifq_forward_workspace_bytes(layers + [pool]) == 0


def test_fused_pool_shapes_and_refusals():
    """pool = p in {2, 4}: the output shape is the convolution's divided by p; other windows,
    sizes not divisible by p, and accumulator outputs are refused before any launch."""
    d = ifq.conv_desc(2, 16, 12, 64, 64, 3, 1, 1, pool=2)
    assert ifq.ifq_conv_out_shape(d) == (8, 6)
    assert ifq.ifq_conv_out_shape(ifq.conv_desc(1, 16, 16, 64, 64, 3, 1, 1, pool=4)) == (4, 4)
    assert ifq.ifq_conv_out_shape(ifq.conv_desc(1, 16, 16, 64, 64, 3, 1, 1, pool=1)) == (16, 16)

    def status(**kw):
        args = dict(n=1, h=16, w=16, cin=64, cout=64, k=3, stride=1, pad=1)
        args.update(kw)
        with pytest.raises(ifq.IfqError) as e:
            ifq.ifq_conv_out_shape(ifq.conv_desc(**args))
        return e.value.status

    assert status(h=13, pool=2) == ifq.IFQ_ESHAPE        # 13 rows do not split into 2x2 windows
    assert status(pool=3) == ifq.IFQ_EUNSUPPORTED
    fake = 1 << 20
    d = ifq.conv_desc(1, 16, 16, 64, 64, 3, 1, 1, out_mode=ifq.IFQ_OUT_BOTH, pool=2)
    with pytest.raises(ifq.IfqError) as e:
        ifq.ifq_conv2bit(d, fake, fake, fake, fake, fake, fake, stream=0)
    assert e.value.status == ifq.IFQ_EUNSUPPORTED        # pooled accumulators are not an output


@pytest.mark.parametrize("m", [6, 8, 10, 12, 16])
def test_separated_fold_matches_oracle_chain_everywhere(m):
    """ifq_fold_layer_separated solves the separated conversion's inequalities for integer
    thresholds; on every achievable accumulator A in [-3K, 3K] its codes equal the oracle's
    element-by-element evaluation of the separated chain (Sec. 2.2), for calibrated parameters with
    both BN-scale signs."""
    rng = np.random.default_rng(100 + m)
    layer = synth.Conv("x", 64, 40, 3, 1, 1, 8, 8, 8, 8, -1)
    cp = synth.draw_conv_params_calibrated(rng, layer)
    cp.gamma[1::4] *= -1
    cp.gamma[3] = 0.0
    K = 9 * 64
    T, s = ifq.ifq_fold_layer_separated(K, m, cp.alpha, cp.gamma, cp.beta, cp.mean, cp.var, synth.STEP, None,
                                        synth.EPS)
    p = O.Params.from_synth(cp)
    A = np.arange(-3 * K, 3 * K + 1, dtype=np.int32)[:, None].repeat(40, 1)
    assert (O.int_chain(A, T, s) == O.separated_chain(A, p, m)).all()


def test_separated_fold_refusals():
    one = np.ones(4, np.float32)
    with pytest.raises(ifq.IfqError):
        ifq.ifq_fold_layer_separated(64, 21, one, one, one * 0, one * 0, one)      # m beyond 20
    with pytest.raises(ifq.IfqError):                                                # sigma floors to 0
        ifq.ifq_fold_layer_separated(64, 4, one, one * 1e4, one * 0, one * 0, one)


def test_build_refuses_spilling_tensor_core_kernels():
    """build() rejects a library in which a warp-specialised tensor-core kernel spills registers to
    local memory; other kernels may spill."""
    from paper_1911_08076_gb300 import build as B
    log = """ptxas info    : Compiling entry function '_ZN3ifq14conv_tc_kernelILi128ELi16ELi2ELi2ELi1EEEv' for 'sm_103a'
ptxas info    : Function properties for _ZN3ifq14conv_tc_kernelILi128ELi16ELi2ELi2ELi1EEEv
    24 bytes stack frame, 24 bytes spill stores, 68 bytes spill loads
ptxas info    : Compiling entry function '_ZN3ifq26maxpool_codes_bytes_kernelILi4EEEvNS_8PoolArgsE' for 'sm_103a'
    8 bytes stack frame, 8 bytes spill stores, 8 bytes spill loads
ptxas info    : Compiling entry function '_ZN3ifq17conv_stack_kernelENS_11StackParamsE' for 'sm_103a'
    16 bytes stack frame, 0 bytes spill stores, 0 bytes spill loads
ptxas info    : Compiling entry function '_ZN3ifq14conv_tc_kernelILi64ELi16ELi2ELi2ELi1EEEv' for 'sm_103a'
    0 bytes stack frame, 0 bytes spill stores, 4 bytes spill loads
"""
    assert B.spilling_kernels(log) == ["_ZN3ifq14conv_tc_kernelILi128ELi16ELi2ELi2ELi1EEEv",
                                       "_ZN3ifq14conv_tc_kernelILi64ELi16ELi2ELi2ELi1EEEv"]
    assert B.spilling_kernels("") == []


def test_graph_with_copies_validates_the_stack_before_any_capture():
    """ifq_graph_create_io checks the stack (and a missing output handle) on the host first, like
    ifq_graph_create (works without a GPU)."""
    fake = 1 << 20
    L0 = ifq.Layer(kind=ifq.IFQ_LAYER_CONV, src=-1, conv=ifq.conv_desc(1, 8, 8, 64, 32, 3, 1, 1), w_prep=fake,
                   thr=fake, sign=fake, y_codes=fake)
    L1 = ifq.Layer(kind=ifq.IFQ_LAYER_CONV, src=0, conv=ifq.conv_desc(1, 8, 8, 16, 32, 3, 1, 1), w_prep=fake,
                   thr=fake, sign=fake, y_codes=fake)
    with pytest.raises(ifq.IfqError) as e:   # layer 1 reads 16 channels, layer 0 writes 32
        ifq.ifq_graph_create_io([L0, L1], fake, None, 0, fake, 1024, [None, fake], None, stream=0)
    assert e.value.status == ifq.IFQ_ESHAPE
    with pytest.raises(ifq.IfqError) as e:   # no input buffer
        ifq.ifq_graph_create_io([L0], None, None, 0, fake, 1024, None, None, stream=0)
    assert e.value.status == ifq.IFQ_EINVAL
    arr = (ifq.Layer * 1)(L0)
    assert ifq.lib().ifq_graph_create_io(arr, 1, fake, None, 0, None, 0, None, None, None, None) == ifq.IFQ_EINVAL


def test_last_forward_mode_before_any_forward_is_einval():
    """A host thread that has made no forward call has no launch mode to report."""
    import threading
    out = {}

    def probe():
        try:
            ifq.ifq_last_forward_mode()
        except ifq.IfqError as e:
            out["status"] = e.status

    t = threading.Thread(target=probe)
    t.start()
    t.join()
    assert out.get("status") == ifq.IFQ_EINVAL


def test_tensor_core_path_filter_size_limit():
    """The tensor-core paths take filters of up to 15 x 15 (a row's valid filter rows and columns sit
    in one 32-bit mask, 15 bits each, so a granule's tap test is one AND and one compare); larger
    filters take the bit-serial path."""
    plan = lambda *a, **k: ifq.ifq_conv_plan(ifq.conv_desc(*a, **k))
    assert plan(1, 24, 24, 64, 64, 15, 1, 7) == ifq.IFQ_PATH_TC
    assert plan(1, 24, 24, 64, 64, 17, 1, 8) == ifq.IFQ_PATH_BITSERIAL
    assert plan(1, 24, 24, 64, 64, 17, 1, 8, path=ifq.IFQ_PATH_TC) == ifq.IFQ_PATH_BITSERIAL


def test_window_path_plan():
    """The window path applies to stride-1 k x k 'same' layers on 2-bit codes with cin 16 or a
    multiple of 32, cout 32, 64 or a multiple of 128, whose resident filter block and buffers fit
    one CTA's shared memory, and is the default for those with a fused 2 x 2 pool and cin <= 64;
    everything else keeps its previous path, and IFQ_WIN=0 turns it off."""
    WIN, TC = ifq.IFQ_PATH_WIN, ifq.IFQ_PATH_TC
    plan = lambda *a, **k: ifq.ifq_conv_plan(ifq.conv_desc(*a, **k))
    assert plan(64, 208, 208, 16, 32, 3, 1, 1, pool=2) == WIN       # Tiny-YOLO conv2, fused pool
    assert plan(64, 104, 104, 32, 64, 3, 1, 1, pool=2) == WIN       # Tiny-YOLO conv3
    assert plan(64, 52, 52, 64, 128, 3, 1, 1, pool=2) == WIN        # Tiny-YOLO conv4
    assert plan(32, 56, 56, 64, 64, 3, 1, 1) == TC                   # no pool: the other kernel is faster
    assert plan(32, 56, 56, 64, 64, 3, 1, 1, path=WIN) == WIN        # ... but the window path applies
    assert plan(64, 26, 26, 128, 256, 3, 1, 1, pool=2) == TC         # 128 input channels: likewise
    assert plan(1, 16, 16, 64, 64, 3, 1, 1, out_mode=ifq.IFQ_OUT_BOTH, path=WIN) == WIN
    assert plan(32, 56, 56, 64, 128, 3, 2, 1) == TC                  # stride 2
    assert plan(256, 56, 56, 256, 256, 3, 1, 1) == TC                # filter block too large
    assert plan(64, 13, 13, 1024, 30, 1, 1, 0, out_mode=ifq.IFQ_OUT_ACC) == TC   # cout 30
    assert plan(4, 20, 20, 48, 64, 3, 1, 1) == TC                    # cin 48
    assert plan(4, 20, 20, 64, 96, 3, 1, 1) == TC                    # cout 96
    assert plan(2, 10, 10, 16, 32, 3, 1, 1) == TC                    # a row of 40 bytes: no bulk copy
    assert plan(4, 20, 20, 64, 64, 3, 1, 1, path=WIN) == WIN
    assert plan(4, 20, 20, 64, 64, 3, 2, 1, path=WIN) == TC          # not applicable: tensor cores
    import os
    old = os.environ.get("IFQ_WIN")
    os.environ["IFQ_WIN"] = "0"
    try:
        assert plan(64, 208, 208, 16, 32, 3, 1, 1, pool=2) == TC
    finally:
        if old is None:
            del os.environ["IFQ_WIN"]
        else:
            os.environ["IFQ_WIN"] = old


def test_warp_path_plan():
    """The warp-MMA path applies to 3 x 3 stride-1 layers with padding 1 on 2-bit codes with cin 8 or
    16 or on 8-bit values with cin 4, cout 8, 16 or 32, no pool or a 2 x 2 pool on even sizes; a
    request for it elsewhere takes the tensor-core path, and IFQ_WARP=0 turns it off."""
    WARP, TC = ifq.IFQ_PATH_WARP, ifq.IFQ_PATH_TC
    plan = lambda *a, **k: ifq.ifq_conv_plan(ifq.conv_desc(*a, **k))
    assert plan(64, 208, 208, 8, 16, 3, 1, 1, pool=2, path=WARP) == WARP
    assert plan(64, 416, 416, 4, 8, 3, 1, 1, pool=2, in_bits=8, path=WARP) == WARP
    assert plan(64, 208, 208, 16, 32, 3, 1, 1, pool=2, path=WARP) == WARP
    assert plan(2, 13, 17, 8, 8, 3, 1, 1, out_mode=ifq.IFQ_OUT_BOTH, path=WARP) == WARP
    # the default where it was measured faster: 8-channel codes, and 8-bit values without a pool
    assert plan(64, 208, 208, 8, 16, 3, 1, 1, pool=2) == WARP
    assert plan(64, 208, 208, 8, 16, 3, 1, 1) == WARP
    assert plan(64, 416, 416, 4, 8, 3, 1, 1, in_bits=8) == WARP
    assert plan(64, 416, 416, 4, 8, 3, 1, 1, pool=2, in_bits=8) == ifq.IFQ_PATH_DIRECT
    assert plan(64, 208, 208, 16, 32, 3, 1, 1, pool=2) == ifq.IFQ_PATH_WIN
    assert plan(2, 16, 16, 32, 64, 3, 1, 1, path=WARP) == TC          # cin 32
    assert plan(2, 16, 16, 16, 64, 3, 1, 1, path=WARP) == TC          # cout 64
    assert plan(2, 16, 16, 16, 24, 3, 1, 1, path=WARP) == TC          # cout 24
    assert plan(2, 16, 16, 16, 32, 3, 2, 1, path=WARP) == TC          # stride 2
    assert plan(2, 16, 16, 16, 32, 5, 1, 2, path=WARP) == TC          # 5 x 5
    assert plan(2, 16, 16, 16, 32, 3, 1, 0, path=WARP) == TC          # no padding
    assert plan(2, 16, 16, 4, 8, 3, 1, 1, path=WARP) == TC            # cin 4 on codes
    assert plan(2, 16, 16, 8, 16, 3, 1, 1, kbits=4, path=WARP) == TC  # 4-bit codes
    assert plan(2, 16, 16, 16, 32, 3, 1, 1, pool=4, path=WARP) == TC  # 4 x 4 pool
    import os
    old = os.environ.get("IFQ_WARP")
    os.environ["IFQ_WARP"] = "0"
    try:
        assert plan(64, 208, 208, 8, 16, 3, 1, 1, pool=2, path=WARP) == TC
    finally:
        if old is None:
            del os.environ["IFQ_WARP"]
        else:
            os.environ["IFQ_WARP"] = old
