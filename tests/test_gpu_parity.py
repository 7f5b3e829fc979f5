"""GPU parity: the CUDA path through the C ABI against the CPU oracle, bit-exact.

Every comparison is element by element on seeded inputs: int32 accumulators
(the integer core of Eq. (1)) and 2-bit codes (the thresholds of Eq. (7) after
the floor of Sec. 3.2).  The oracle's own fold and chains give the expected
values; the GPU gets thresholds from the library's host fold.
"""
import os

import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_1911_08076_gb300 import ifq, synth
from paper_1911_08076_gb300.stack import DeviceStack
from stack_parity import compare_stack_with_oracle

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]

DEV = "cuda"


def _params(rng, cout, K):
    """Float parameters scaled so that the accumulators of random data reach every code."""
    sd = np.sqrt(K * 3.5)
    return O.Params(rng.uniform(0.5, 1.5, cout) * 4.0 / sd, rng.normal(1.0, 0.6, cout), rng.normal(0, 0.5, cout),
                    rng.normal(0, 1.0, cout), rng.uniform(0.5, 2.0, cout), None, 0.5, 0.5, -0.25, synth.EPS)


def _fold_gpu(p, K):
    T, s = ifq.ifq_fold_layer(K, p.alpha, p.gamma, p.beta, p.mean, p.var, p.delta_in, p.bias, p.eps, p.q_base,
                              p.q_offset)
    return T, s


def _run_conv(x, w, T, s, stride, pad, out_mode, path, bn=None, pool=0):
    B, H, W, C = x.shape
    cout, k, _, _ = w.shape
    K = k * k * C
    d = ifq.conv_desc(B, H, W, C, cout, k, stride, pad, out_mode, path, pool=pool)
    xp = torch.from_numpy(synth.pack_codes(x)).to(DEV)
    bits = torch.from_numpy(synth.pack_signs(w).view(np.int32)).to(DEV)
    prep = torch.empty(ifq.ifq_weights_prep_bytes(d), dtype=torch.uint8, device=DEV)
    ifq.ifq_pack_weights(d, bits, prep)
    ho, wo = ifq.ifq_conv_out_shape(d)
    yc = ya = None
    if out_mode & ifq.IFQ_OUT_CODES:
        yc = torch.full((B, ho, wo, cout // 4), 0x5A, dtype=torch.uint8, device=DEV)
    if out_mode & ifq.IFQ_OUT_ACC:
        ya = torch.full((B, ho, wo, cout), -777777, dtype=torch.int32, device=DEV)
    thr = torch.from_numpy(T).to(DEV)
    sg = torch.from_numpy(s).to(DEV)
    old = os.environ.get("IFQ_TC_BN")
    if bn:
        os.environ["IFQ_TC_BN"] = str(bn)
    try:
        ifq.ifq_conv2bit(d, xp, prep, thr, sg, yc, ya)
    finally:
        if bn:
            if old is None:
                del os.environ["IFQ_TC_BN"]
            else:
                os.environ["IFQ_TC_BN"] = old
    torch.cuda.synchronize()
    assert ifq.ifq_device_status() == ifq.IFQ_OK
    codes = None if yc is None else synth.unpack_codes(yc.cpu().numpy(), cout)
    acc = None if ya is None else ya.cpu().numpy()
    return codes, acc


CONV_CASES = [
    # B, H, W, C, cout, k, stride, pad, out_mode
    (1, 16, 16, 64, 64, 3, 1, 1, 3),      # single 3x3 64->64 layer
    (2, 9, 7, 64, 96, 3, 2, 1, 3),        # ragged M, partial N tile
    (3, 11, 13, 128, 256, 3, 1, 1, 3),    # several M tiles with a ragged tail
    (2, 8, 8, 256, 320, 1, 1, 0, 3),      # 1x1, two N tiles
    (1, 27, 27, 96, 64, 5, 1, 2, 3),      # 5x5, cin % 64 != 0
    (2, 12, 12, 48, 32, 3, 1, 1, 3),
    (2, 10, 10, 16, 32, 3, 1, 1, 3),      # K = 144 (partial K stage)
    (2, 10, 10, 8, 16, 3, 1, 1, 3),       # narrow cin
    (1, 9, 9, 4, 8, 3, 1, 1, 3),
    (1, 7, 7, 12, 20, 3, 1, 1, 3),
    (4, 6, 6, 256, 512, 6, 1, 0, 3),      # FC-as-conv, K = 9216
    (3, 1, 1, 4096, 128, 1, 1, 0, 3),     # K = 4096, M = 3
    (2, 13, 13, 1024, 30, 1, 1, 0, 2),    # accumulators only, cout = 30
    (1, 14, 14, 256, 512, 3, 2, 1, 1),    # stride 2, codes only
    (1, 5, 5, 64, 64, 3, 1, 0, 1),        # no padding
    (2, 14, 14, 32, 64, 3, 1, 1, 3),      # 8-byte pixels: 8-byte gather granules
    (2, 15, 13, 160, 128, 3, 2, 1, 3),    # 40-byte pixels, stride 2, ragged M
]


@pytest.mark.parametrize("path", [ifq.IFQ_PATH_TC, ifq.IFQ_PATH_BITSERIAL], ids=["tc", "bitserial"])
@pytest.mark.parametrize("case", CONV_CASES, ids=[str(c) for c in CONV_CASES])
def test_conv_matches_oracle(case, path):
    B, H, W, C, cout, k, s, p, mode = case
    rng = np.random.default_rng(abs(hash(case)) % (2 ** 32))
    x = rng.integers(0, 4, (B, H, W, C), dtype=np.uint8)
    w = np.where(rng.integers(0, 2, (cout, k, k, C)) == 1, 1, -1).astype(np.int8)
    K = k * k * C
    prm = _params(rng, cout, K)
    T, sg = _fold_gpu(prm, K)
    codes, acc = _run_conv(x, w, T, sg, s, p, mode, path)
    A = O.conv_acc(x, w, s, p)
    if acc is not None:
        assert (acc == A).all(), f"accumulators differ at {np.argwhere(acc != A)[:5].tolist()}"
    if codes is not None:
        To, so = O.fold(prm, K)
        ref, _ = O.check_chains(A, prm, To, so)
        assert len(np.unique(ref)) >= 3
        assert (codes == ref).all(), f"codes differ at {np.argwhere(codes != ref)[:5].tolist()}"


POOL_FUSED_CASES = [
    # B, H, W, C, cout, k, stride, pad, p, bn
    (2, 16, 16, 64, 64, 3, 1, 1, 2, None),      # 64 pooled pixels, one tile
    (3, 22, 26, 64, 96, 3, 1, 1, 2, None),      # ragged last tile, partial channel tile
    (2, 20, 20, 16, 32, 3, 1, 1, 2, None),      # 4-byte granules
    (2, 12, 12, 8, 16, 3, 1, 1, 2, None),       # 1-byte granules
    (2, 16, 16, 128, 256, 3, 1, 1, 4, None),    # 4x4 windows, 16 lanes each
    (1, 28, 28, 64, 128, 3, 2, 1, 2, None),     # strided convolution, then the pool
    (2, 16, 16, 32, 64, 3, 1, 1, 2, None),      # 8-byte pixels (8-byte granules), then the pool
    (2, 16, 16, 64, 200, 3, 1, 1, 2, 32),       # every channel-tile width
    (2, 16, 16, 64, 200, 3, 1, 1, 2, 64),
    (2, 16, 16, 64, 200, 3, 1, 1, 2, 128),
]


@pytest.mark.parametrize("case", POOL_FUSED_CASES, ids=[str(c) for c in POOL_FUSED_CASES])
def test_fused_pool_matches_oracle(case):
    """Convolution with the fused p x p pool: the codes are those of the window maximum of the
    accumulators (Sec. 2.1, pool before BN and the quantizer), bit-exact, including channels with
    a negative BN scale (there the code is the window minimum)."""
    B, H, W, C, cout, k, s, p, pool, bn = case
    rng = np.random.default_rng(abs(hash(case)) % (2 ** 32))
    x = rng.integers(0, 4, (B, H, W, C), dtype=np.uint8)
    w = np.where(rng.integers(0, 2, (cout, k, k, C)) == 1, 1, -1).astype(np.int8)
    K = k * k * C
    prm = _params(rng, cout, K)
    prm.gamma[1::3] = -np.abs(prm.gamma[1::3])      # channels with a negative BN scale in every case
    T, sg = _fold_gpu(prm, K)
    assert (sg < 0).any() and (sg > 0).any()
    codes, _ = _run_conv(x, w, T, sg, s, p, ifq.IFQ_OUT_CODES, ifq.IFQ_PATH_TC, bn=bn, pool=pool)
    A = O.conv_acc(x, w, s, p)
    ref = O.int_chain(O.maxpool_acc(A, pool, pool, 0), *O.fold(prm, K))
    assert codes.shape == ref.shape
    assert (codes == ref).all(), f"codes differ at {np.argwhere(codes != ref)[:5].tolist()}"
    # and it equals the separate sign-aware pool on the unpooled codes
    full, _ = _run_conv(x, w, T, sg, s, p, ifq.IFQ_OUT_CODES, ifq.IFQ_PATH_TC, bn=bn)
    assert (codes == O.maxpool_codes(full, pool, pool, 0, sg)).all()


@pytest.mark.parametrize("bn", [32, 64, 128])
def test_tc_every_channel_tile(bn):
    rng = np.random.default_rng(bn)
    B, H, W, C, cout, k = 2, 12, 11, 64, 200, 3
    x = rng.integers(0, 4, (B, H, W, C), dtype=np.uint8)
    w = np.where(rng.integers(0, 2, (cout, k, k, C)) == 1, 1, -1).astype(np.int8)
    prm = _params(rng, cout, k * k * C)
    T, sg = _fold_gpu(prm, k * k * C)
    codes, acc = _run_conv(x, w, T, sg, 1, 1, 3, ifq.IFQ_PATH_TC, bn=bn)
    A = O.conv_acc(x, w, 1, 1)
    assert (acc == A).all()
    assert (codes == O.int_chain(A, *O.fold(prm, k * k * C))).all()


@pytest.mark.parametrize("K_case", [(3, 1024, 3, 0), (1, 10880, 1, 0)], ids=["K9216", "K10880"])
def test_tc_extreme_accumulators_are_exact(K_case):
    """All codes 3 with all +1 (or all -1) filters give |A| = 3K, the largest the path accepts."""
    H, C, k, p = K_case
    B = 130 if H == 1 else 2
    x = np.full((B, H, H, C), 3, np.uint8)
    w = np.ones((64, k, k, C), np.int8)
    w[1::2] = -1
    w[5, ..., ::3] = -1
    K = k * k * C
    prm = _params(np.random.default_rng(1), 64, K)
    T, sg = _fold_gpu(prm, K)
    codes, acc = _run_conv(x, w, T, sg, 1, p, 3, ifq.IFQ_PATH_TC)
    A = O.conv_acc(x, w, 1, p)
    assert abs(int(A[..., 0].max())) == 3 * K
    assert (acc == A).all()
    assert (codes == O.int_chain(A, *O.fold(prm, K))).all()


def test_auto_path_beyond_tc_range_is_exact():
    rng = np.random.default_rng(3)
    B, C, cout = 40, 11008, 32
    x = rng.integers(0, 4, (B, 1, 1, C), dtype=np.uint8)
    w = np.where(rng.integers(0, 2, (cout, 1, 1, C)) == 1, 1, -1).astype(np.int8)
    prm = _params(rng, cout, C)
    T, sg = _fold_gpu(prm, C)
    codes, acc = _run_conv(x, w, T, sg, 1, 0, 3, ifq.IFQ_PATH_AUTO)
    A = O.conv_acc(x, w, 1, 0)
    assert (acc == A).all()
    assert (codes == O.int_chain(A, *O.fold(prm, C))).all()


POOL_CASES = [
    # B, H, W, C, k, stride, pad, signed
    (2, 27, 27, 256, 3, 2, 0, True),
    (2, 13, 13, 256, 3, 2, 0, True),
    (2, 8, 8, 32, 2, 2, 0, True),
    (1, 13, 13, 512, 2, 1, 1, True),
    (2, 9, 9, 16, 2, 2, 0, False),
    (1, 7, 7, 8, 2, 2, 0, True),
    (1, 7, 5, 4, 3, 2, 1, True),
    (3, 208, 208, 32, 2, 2, 0, True),
    # 2x2 / stride 2 on 4- and 8-byte pixels: the row-pair kernel (16-byte row segments) ...
    (2, 16, 16, 16, 2, 2, 0, True),
    (1, 12, 20, 16, 2, 2, 0, True),
    (2, 11, 14, 32, 2, 2, 0, True),             # odd height: the last input row is unused
    (1, 9, 6, 32, 2, 2, 0, False),
    # ... and the general kernel where a row is not a whole number of 16-byte segments
    (2, 6, 10, 16, 2, 2, 0, True),
    (1, 8, 7, 32, 2, 2, 0, True),
]


@pytest.mark.parametrize("case", POOL_CASES, ids=[str(c) for c in POOL_CASES])
def test_maxpool_matches_oracle(case):
    B, H, W, C, k, s, p, signed = case
    rng = np.random.default_rng(sum(case[:7]))
    x = rng.integers(0, 4, (B, H, W, C), dtype=np.uint8)
    sign = np.where(rng.integers(0, 10, C) == 0, -1, 1).astype(np.int8)
    sign[0] = -1
    d = ifq.PoolDesc(B, H, W, C, k, s, p)
    ho, wo = ifq.ifq_pool_out_shape(d)
    y = torch.full((B, ho, wo, C // 4), 0xA5, dtype=torch.uint8, device=DEV)
    sg = torch.from_numpy(sign).to(DEV) if signed else None
    ifq.ifq_maxpool2bit(d, torch.from_numpy(synth.pack_codes(x)).to(DEV), sg, y)
    torch.cuda.synchronize()
    got = synth.unpack_codes(y.cpu().numpy())
    ref = O.maxpool_codes(x, k, s, p, sign if signed else None)
    assert (got == ref).all()


def test_pack_helpers_match_formats():
    rng = np.random.default_rng(9)
    c = rng.integers(0, 4, 4 * 1237, dtype=np.uint8)
    ct = torch.from_numpy(c).to(DEV)
    packed = torch.empty(c.size // 4, dtype=torch.uint8, device=DEV)
    ifq.ifq_pack_codes(ct, packed, c.size)
    assert (packed.cpu().numpy() == synth.pack_codes(c)).all()
    back = torch.empty_like(ct)
    ifq.ifq_unpack_codes(packed, back, c.size)
    assert (back.cpu().numpy() == c).all()
    w = np.where(rng.integers(0, 2, (37, 291)) == 1, 1, -1).astype(np.int8)
    bits = torch.empty((37, (291 + 31) // 32), dtype=torch.int32, device=DEV)
    ifq.ifq_pack_signs(torch.from_numpy(w).to(DEV), bits, 37, 291)
    assert (bits.cpu().numpy().view(np.uint32) == synth.pack_signs(w)).all()


# ----------------------------------------------------------------------------- whole workloads

# Every configuration at full size: the single PR1 layer, the ResNet-18 body b32, AlexNet conv2-FC7
# b128, Tiny-YOLO and Tinier-YOLO b64 (separate and fused pools; Tinier also end to end from 8-bit
# pixels to fixed-point detections), and the two roofline layers b256.
WORKLOADS = ["pr1", "resnet18", "alexnet", "tinyyolo", "tinyyolo_fused", "tinieryolo", "tinieryolo_fused",
             "tinieryolo_full_fused", "roofline3x3", "roofline1x1"]


@pytest.mark.parametrize("name", WORKLOADS)
def test_workload_matches_oracle(name):
    """Full-size workload on the GPU; the oracle recomputes every image through every layer."""
    wl = synth.get(name)
    x, params = synth.draw_workload(wl)
    compare_stack_with_oracle(wl, x, params)


@pytest.mark.parametrize("name", WORKLOADS)
def test_workload_with_negative_bn_scales_matches_oracle(name):
    """The same full-size workloads with about 10 % of channels drawn with a negative BN scale (the
    sign-flipped thresholds of Eq. (7) and the min-pool of those channels), every image."""
    wl = synth.get(name)
    x, params = synth.draw_workload(wl, neg_gamma=0.1)
    negs = sum(int((p.gamma < 0).sum()) for p in params if p is not None)
    chans = sum(p.gamma.shape[0] for p in params if p is not None)
    assert 0.05 * chans <= negs <= 0.2 * chans or chans < 100, (negs, chans)
    compare_stack_with_oracle(wl, x, params)


@pytest.mark.parametrize("persistent", ["0", "1"], ids=["per_layer", "persistent"])
def test_graph_replay_equals_forward(persistent, monkeypatch):
    monkeypatch.setenv("IFQ_STACK", persistent)
    wl = synth.get("resnet18", batch=3)
    x, params = synth.draw_workload(wl)
    st = DeviceStack(wl, params)
    assert (st.ws_bytes > 0) == (persistent == "1")
    xd = torch.from_numpy(synth.pack_codes(x)).to(DEV)
    st.forward(xd)
    torch.cuda.synchronize()
    direct = {li: {k: v.copy() for k, v in st.output(li).items()} for li in range(len(wl.layers))}
    for t in st.y_codes.values():
        t.fill_(0)
    stream = torch.cuda.Stream()
    st.capture(xd, stream)
    st.replay(stream)
    stream.synchronize()
    for li in range(len(wl.layers)):
        for k, v in st.output(li).items():
            assert (v == direct[li][k]).all()
    st.release()
    assert ifq.ifq_device_status() == ifq.IFQ_OK


def _stack_outputs(st):
    return {li: {k: v.copy() for k, v in st.output(li).items()} for li in range(len(st.wl.layers))}


@pytest.mark.parametrize("name", ["resnet18", "custom"])
def test_persistent_stack_kernel_equals_per_layer_launches(name, monkeypatch):
    """With IFQ_STACK=1 and its workspace, ifq_forward runs the whole conv stack as one persistent
    launch; without a workspace it launches layer by layer.  Both must give identical codes and
    accumulators, and the oracle must agree on sampled images."""
    monkeypatch.setenv("IFQ_STACK", "1")
    if name == "resnet18":
        wl = synth.get("resnet18", batch=6)
    else:
        L = [synth.Conv("a", 16, 48, 3, 1, 1, 11, 11, 11, 11, -1),
             synth.Conv("b", 48, 64, 1, 2, 0, 11, 11, 6, 6, 0),
             synth.Conv("c", 48, 96, 3, 2, 1, 11, 11, 6, 6, 0, "both"),      # second reader of layer 0
             synth.Conv("d", 96, 256, 3, 1, 1, 6, 6, 6, 6, 2),
             synth.Conv("e", 256, 30, 1, 1, 0, 6, 6, 6, 6, 3, "acc")]
        wl = synth.Workload("custom_stack", 7, 5, 11, 11, 16, L)
    x, params = synth.draw_workload(wl)
    st = DeviceStack(wl, params)
    assert st.ws_bytes > 0, "the stack should qualify for the persistent kernel"
    xd = torch.from_numpy(synth.pack_codes(x)).to(DEV)
    st.forward(xd)
    torch.cuda.synchronize()
    assert ifq.ifq_device_status() == ifq.IFQ_OK
    fused = _stack_outputs(st)
    for t in list(st.y_codes.values()) + list(st.y_acc.values()):
        t.zero_()
    ifq.ifq_forward(st.layers, xd)          # no workspace: one launch per layer
    torch.cuda.synchronize()
    per_layer = _stack_outputs(st)
    for li in fused:
        for k in fused[li]:
            assert (fused[li][k] == per_layer[li][k]).all(), (wl.layers[li].name, k)
    ref = O.forward(wl, x, params, images=[0, wl.batch - 1])
    for li, l in enumerate(wl.layers):
        out, r = fused[li], ref[li]
        if l.out == "both":
            assert (synth.unpack_codes(out["codes"][[0, -1]], l.cout) == r["codes"]).all()
            assert (out["acc"][[0, -1]] == r["acc"]).all()
        elif l.out == "acc":
            assert (out["acc"][[0, -1]] == r).all()
        else:
            assert (synth.unpack_codes(out["codes"][[0, -1]], l.cout) == r).all(), l.name


def test_stack_with_reused_output_buffer_runs_layer_by_layer(monkeypatch):
    """A stack whose third layer writes into the first layer's output buffer (ping-pong reuse)
    must not run as one persistent launch (layers there are ordered only after their source);
    ifq_forward falls back to one launch per layer and the results follow stream order."""
    monkeypatch.setenv("IFQ_STACK", "1")
    L = [synth.Conv("a", 16, 64, 3, 1, 1, 9, 9, 9, 9, -1),
         synth.Conv("b", 64, 64, 3, 1, 1, 9, 9, 9, 9, 0),
         synth.Conv("c", 64, 64, 3, 1, 1, 9, 9, 9, 9, 1)]
    wl = synth.Workload("pingpong", 3, 3, 9, 9, 16, L)
    x, params = synth.draw_workload(wl)
    st = DeviceStack(wl, params)
    st.layers[2].y_codes = st.layers[0].y_codes          # c overwrites a's codes after b has read them
    xd = torch.from_numpy(synth.pack_codes(x)).to(DEV)
    st.forward(xd)
    torch.cuda.synchronize()
    assert ifq.ifq_device_status() == ifq.IFQ_OK
    ref = O.forward(wl, x, params, images=[0, 1, 2])
    assert (synth.unpack_codes(st.y_codes[1].cpu().numpy(), 64) == ref[1]).all()
    assert (synth.unpack_codes(st.y_codes[0].cpu().numpy(), 64) == ref[2]).all()


@pytest.mark.parametrize("name", ["tinyyolo", "tinieryolo"])
def test_fused_pool_stack_equals_separate_pools(name):
    """The YOLO stacks with each conv + 2x2/s2 pool pair fused into one launch: every fused layer's
    pooled codes equal the separate sign-aware pool's output, every other layer is unchanged, and
    the oracle (pool on the accumulators) agrees on the first and last image."""
    base = synth.get(name, batch=3)
    fused = synth.fuse_pools(base)
    assert len(fused.layers) < len(base.layers)
    x, params = synth.draw_workload(base)
    xf, params_f = synth.draw_workload(fused)
    assert (x == xf).all()
    xd = torch.from_numpy(synth.pack_codes(x)).to(DEV)
    sb, sf = DeviceStack(base, params), DeviceStack(fused, params_f)
    sb.forward(xd)
    sf.forward(xd)
    torch.cuda.synchronize()
    assert ifq.ifq_device_status() == ifq.IFQ_OK
    # map each fused layer to the base layer whose output it must equal (the pool, when fused)
    bi = 0
    ref = O.forward(fused, x, params_f, images=[0, base.batch - 1])
    for fi, lf in enumerate(fused.layers):
        while base.layers[bi].name != lf.name:
            bi += 1
        target = bi + 1 if (lf.kind == "conv" and lf.pool > 1) else bi
        got, want = sf.output(fi), sb.output(target)
        for k in got:
            assert (got[k] == want[k]).all(), (lf.name, k)
        r = ref[fi]
        if lf.kind == "conv" and lf.out == "acc":
            assert (got["acc"][[0, -1]] == r).all()
        elif not (lf.kind == "conv" and lf.out == "both"):
            c = lf.cout if lf.kind == "conv" else lf.c
            assert (synth.unpack_codes(got["codes"][[0, -1]], c) == r).all(), lf.name


@pytest.mark.parametrize("m", [6, 8, 12])
def test_separated_conversion_on_the_kernel(m):
    """The separated fixed-point conversion (Sec. 2.2) is also a per-channel integer threshold test;
    with ifq_fold_layer_separated's thresholds the tensor-core kernel reproduces the oracle's
    element-by-element separated chain bit-exactly, and (with calibrated, small filter scales) it
    differs from the integrated codes while the integrated codes equal the float chain."""
    rng = np.random.default_rng(300 + m)
    B, H, W, C, cout, k = 2, 14, 14, 64, 96, 3
    layer = synth.Conv("x", C, cout, k, 1, 1, H, W, H, W, -1)
    cp = synth.draw_conv_params_calibrated(rng, layer)
    x = synth.draw_codes(rng, (B, H, W, C))
    K = k * k * C
    Ts, ss = ifq.ifq_fold_layer_separated(K, m, cp.alpha, cp.gamma, cp.beta, cp.mean, cp.var, synth.STEP, None,
                                          synth.EPS)
    codes, acc = _run_conv(x, cp.w, Ts, ss, 1, 1, ifq.IFQ_OUT_BOTH, ifq.IFQ_PATH_TC)
    A = O.conv_acc(x, cp.w, 1, 1)
    assert (acc == A).all()
    p = O.Params.from_synth(cp)
    sep = O.separated_chain(A, p, m)
    assert (codes == sep).all()
    integ, _ = O.check_chains(A, p, *O.fold(p, K))
    if m <= 8:
        assert (sep != integ).any()


# ----------------------------------------------------------------------------- edge cases

@pytest.mark.parametrize("path", [ifq.IFQ_PATH_TC, ifq.IFQ_PATH_BITSERIAL], ids=["tc", "bitserial"])
def test_maximum_output_channels(path):
    """cout = 65536, the largest the library accepts: 512 channel tiles of 128 on the tensor cores,
    1024 blocks of 64 channels on the bit-serial path."""
    rng = np.random.default_rng(65536)
    B, H, W, C, cout = 2, 8, 8, 64, 65536
    x = rng.integers(0, 4, (B, H, W, C), dtype=np.uint8)
    w = np.where(rng.integers(0, 2, (cout, 1, 1, C)) == 1, 1, -1).astype(np.int8)
    prm = _params(rng, cout, C)
    T, sg = _fold_gpu(prm, C)
    codes, acc = _run_conv(x, w, T, sg, 1, 0, ifq.IFQ_OUT_BOTH, path)
    A = O.conv_acc(x, w, 1, 0)
    assert (acc == A).all()
    assert (codes == O.int_chain(A, *O.fold(prm, C))).all()


@pytest.mark.parametrize("path", [ifq.IFQ_PATH_TC, ifq.IFQ_PATH_BITSERIAL], ids=["tc", "bitserial"])
def test_all_zero_input(path):
    """Codes all 0: every accumulator is 0 and every code is #{ i : 0 > T_i } of its channel."""
    rng = np.random.default_rng(0)
    B, H, W, C, cout = 2, 9, 9, 64, 96
    x = np.zeros((B, H, W, C), np.uint8)
    w = np.where(rng.integers(0, 2, (cout, 3, 3, C)) == 1, 1, -1).astype(np.int8)
    prm = _params(rng, cout, 9 * C)
    T, sg = _fold_gpu(prm, 9 * C)
    codes, acc = _run_conv(x, w, T, sg, 1, 1, ifq.IFQ_OUT_BOTH, path)
    assert (acc == 0).all()
    expect = (0 > T.astype(np.int64)).sum(axis=1)
    assert (codes == expect[None, None, None, :]).all()


def test_empty_batch_leaves_outputs_untouched():
    d = ifq.conv_desc(0, 14, 14, 64, 64, 3, 1, 1, ifq.IFQ_OUT_BOTH)
    buf = torch.full((4096,), 0x5A, dtype=torch.uint8, device=DEV)
    acc = torch.full((1024,), 7, dtype=torch.int32, device=DEV)
    prep = torch.empty(ifq.ifq_weights_prep_bytes(d), dtype=torch.uint8, device=DEV)
    thr = torch.zeros((64, 3), dtype=torch.int32, device=DEV)
    sg = torch.ones(64, dtype=torch.int8, device=DEV)
    ifq.ifq_conv2bit(d, buf, prep, thr, sg, buf, acc)
    ifq.ifq_maxpool2bit(ifq.pool_desc(0, 8, 8, 64, 2, 2), buf, sg, buf)
    torch.cuda.synchronize()
    assert ifq.ifq_device_status() == ifq.IFQ_OK
    assert (buf == 0x5A).all() and (acc == 7).all()


NARROW_CASES = [
    # B, H, W, C, cout, pool: the narrow bit-serial kernel (3x3, stride 1, pad 1)
    (2, 20, 20, 8, 16, 0),
    (2, 20, 20, 8, 16, 2),
    (3, 13, 11, 4, 8, 0),
    (2, 18, 14, 4, 12, 2),
    (2, 11, 9, 16, 32, 0),
    (2, 16, 16, 16, 32, 2),
    (1, 7, 9, 16, 4, 0),
]


@pytest.mark.parametrize("case", NARROW_CASES, ids=[str(c) for c in NARROW_CASES])
def test_narrow_bitserial_matches_oracle(case):
    """The narrow bit-serial kernel (interleaved-code popcounts, one thread per output or pooled
    pixel), bit-exact, with negative BN scales, alone and with the fused pool."""
    B, H, W, C, cout, pool = case
    rng = np.random.default_rng(abs(hash(case)) % (2 ** 32))
    x = rng.integers(0, 4, (B, H, W, C), dtype=np.uint8)
    w = np.where(rng.integers(0, 2, (cout, 3, 3, C)) == 1, 1, -1).astype(np.int8)
    K = 9 * C
    prm = _params(rng, cout, K)
    prm.gamma[1::3] = -np.abs(prm.gamma[1::3])
    T, sg = _fold_gpu(prm, K)
    mode = ifq.IFQ_OUT_CODES if pool else ifq.IFQ_OUT_BOTH
    assert ifq.ifq_conv_plan(ifq.conv_desc(B, H, W, C, cout, 3, 1, 1, mode, ifq.IFQ_PATH_BITSERIAL, pool=pool)) == \
        ifq.IFQ_PATH_BITSERIAL
    codes, acc = _run_conv(x, w, T, sg, 1, 1, mode, ifq.IFQ_PATH_BITSERIAL, pool=pool)
    A = O.conv_acc(x, w, 1, 1)
    if pool:
        ref = O.int_chain(O.maxpool_acc(A, pool, pool, 0), *O.fold(prm, K))
    else:
        assert (acc == A).all()
        ref = O.int_chain(A, *O.fold(prm, K))
    assert (codes == ref).all(), f"codes differ at {np.argwhere(codes != ref)[:5].tolist()}"


def test_copy_bytes_between_device_and_host():
    """ifq_copy_bytes: the SM copy between device memory and pinned host memory, and the
    cudaMemcpyAsync fallback for unaligned sizes and for pageable host memory."""
    rng = np.random.default_rng(16)
    src = torch.from_numpy(rng.integers(0, 256, 1 << 20, dtype=np.uint8)).pin_memory()
    dev = torch.empty(1 << 20, dtype=torch.uint8, device=DEV)
    ifq.ifq_copy_bytes(dev, src, 1 << 20)                          # pinned host -> device (SMs)
    back = torch.zeros(1 << 20, dtype=torch.uint8).pin_memory()
    ifq.ifq_copy_bytes(back, dev, 1 << 20)                         # device -> pinned host (SMs)
    torch.cuda.synchronize()
    assert torch.equal(back, src)
    odd = torch.zeros(1 << 20, dtype=torch.uint8).pin_memory()
    ifq.ifq_copy_bytes(odd, dev, 1000003)                          # size not a multiple of 16
    pageable = torch.zeros(1 << 20, dtype=torch.uint8)
    ifq.ifq_copy_bytes(pageable, dev, 1 << 20)                     # pageable host: cudaMemcpyAsync
    torch.cuda.synchronize()
    assert torch.equal(odd[:1000003], src[:1000003]) and (odd[1000003:] == 0).all()
    assert torch.equal(pageable, src)


def test_bounded_wait_reports_timeout_and_the_context_survives():
    """A wait that nothing completes runs out after its limit, sets IFQ_ETIMEOUT in the device status
    word (read and cleared by ifq_device_status) and returns; kernels run normally afterwards."""
    assert ifq.ifq_device_status() == ifq.IFQ_OK
    t0 = __import__("time").perf_counter()
    ifq.ifq_wait_selftest(20000)                      # 20 ms
    assert ifq.ifq_device_status() == ifq.IFQ_ETIMEOUT
    assert __import__("time").perf_counter() - t0 >= 0.019
    assert ifq.ifq_device_status() == ifq.IFQ_OK      # cleared by the read
    rng = np.random.default_rng(5)
    x = rng.integers(0, 4, (1, 8, 8, 64), dtype=np.uint8)
    w = np.where(rng.integers(0, 2, (64, 3, 3, 64)) == 1, 1, -1).astype(np.int8)
    prm = _params(rng, 64, 576)
    T, sg = _fold_gpu(prm, 576)
    codes, acc = _run_conv(x, w, T, sg, 1, 1, ifq.IFQ_OUT_BOTH, ifq.IFQ_PATH_TC)
    assert (acc == O.conv_acc(x, w, 1, 1)).all()


@pytest.mark.parametrize("name,batch", [("resnet18", 4), ("alexnet", 2), ("tinieryolo_full", 2)])
def test_graph_with_copies_serves_requests_end_to_end(name, batch):
    """ifq_graph_create_io: one graph launch copies the pinned host input in, runs the stack and copies
    every result out (the side branch's right after its layer).  The host results equal the device
    buffers and a plain forward's, and a new input written into the same host buffer gives the new
    results on the next launch (the copies are part of the graph)."""
    wl = synth.get(name, batch=batch)
    x, params = synth.draw_workload(wl, batch=batch)
    fb = 8 if wl.in_bits == 8 else wl.kbits
    st = DeviceStack(wl, params, batch=batch, device=DEV)
    ref = DeviceStack(wl, params, batch=batch, device=DEV)
    x_host = torch.from_numpy(synth.pack_codes(x, fb)).pin_memory()
    leaf_host = torch.zeros(st.leaf_block.shape, dtype=torch.uint8).pin_memory()
    xd = st.input_buffer()
    stream = torch.cuda.Stream()
    st.capture_io(xd, x_host, leaf_host, stream)
    rng = np.random.default_rng(3)
    for trial in range(2):
        if trial:   # a new request in the same pinned buffer
            x2 = rng.integers(0, 256 if wl.in_bits == 8 else 1 << wl.kbits, x.shape, dtype=np.uint8)
            if wl.in_bits == 8:
                x2[..., 3:] = 0
            x_host.copy_(torch.from_numpy(synth.pack_codes(x2, fb)))
        st.replay(stream)
        stream.synchronize()
        assert ifq.ifq_device_status() == ifq.IFQ_OK
        ref.forward(x_host.to(DEV))
        torch.cuda.synchronize()
        assert st.leaf_results_equal(leaf_host)
        assert st.leaf_results_equal(leaf_host, ref.leaf_block)
    st.release()


def test_graph_with_copies_rejects_bad_io():
    wl = synth.get("resnet18", batch=2)
    x, params = synth.draw_workload(wl, batch=2)
    st = DeviceStack(wl, params, batch=2, device=DEV)
    xd = st.input_buffer()
    x_host = torch.empty(xd.numel(), dtype=torch.uint8).pin_memory()
    with pytest.raises(ifq.IfqError) as e:   # one byte short of the stack's input
        ifq.ifq_graph_create_io(st.layers, xd, st.ws, st.ws_bytes, x_host, xd.numel() - 1)
    assert e.value.status == ifq.IFQ_ESHAPE
    acc_dst = [None] * len(st.layers)
    acc_dst[0] = torch.empty(16, dtype=torch.int32, device=DEV)   # layer 0 writes no accumulators
    with pytest.raises(ifq.IfqError) as e:
        ifq.ifq_graph_create_io(st.layers, xd, st.ws, st.ws_bytes, None, 0, None, acc_dst)
    assert e.value.status == ifq.IFQ_EINVAL
    with pytest.raises(ValueError):
        ifq.ifq_graph_create_io(st.layers, xd, st.ws, st.ws_bytes, None, 0, [None])


# ----------------------------------------------------------------------------- window path

WIN_CASES = [
    # B, H, W, C, cout, k, pool, out_mode
    (1, 4, 16, 16, 32, 3, 1, 3),          # smallest: one tile of 4 rows x 16 anchors, 4 rows stacked on M
    (2, 10, 12, 16, 32, 3, 1, 3),         # ragged band (10 rows in tiles of 4), N = 16 > w
    (2, 12, 20, 16, 32, 3, 2, 1),         # fused pool, row pairs across warps
    (2, 9, 14, 32, 64, 3, 1, 3),          # 2 planes, 2 rows stacked on M, odd height
    (3, 14, 18, 32, 64, 3, 2, 1),         # fused pool over warp pairs (sy, sy + 1)
    (2, 11, 11, 64, 128, 3, 1, 3),        # one output row per M row, several anchor rows per tile
    (2, 12, 14, 64, 128, 3, 2, 1),        # fused pool over anchor-row pairs (16-aligned pitch)
    (2, 9, 9, 64, 256, 3, 1, 3),          # two channel tiles
    (1, 16, 16, 64, 64, 3, 1, 3),         # the single PR1 layer shape
    (2, 8, 30, 32, 128, 5, 1, 3),         # 5 x 5, 7 anchor rows of 34 slots
    (2, 6, 10, 96, 64, 3, 1, 3),          # 6 planes
    (2, 7, 12, 128, 128, 1, 1, 3),        # 1 x 1
    (1, 6, 40, 16, 32, 7, 1, 1),          # 7 x 7
    (2, 26, 28, 16, 32, 3, 2, 1),         # H % 4 != 0 with the pool: the last band's rows past h
    (1, 3, 208, 16, 32, 3, 1, 1),         # a full Tiny-YOLO row (N = 208)
    (3, 20, 52, 32, 64, 3, 2, 1),         # 4 row bands side by side along N, fused pool
    (2, 13, 56, 64, 64, 3, 1, 3),         # 4 row bands of 2 rows along N (ResNet stage-1 width), ragged
]


@pytest.mark.parametrize("case", WIN_CASES, ids=[str(c) for c in WIN_CASES])
def test_window_path_matches_oracle(case):
    """The window kernel (input band in shared memory, one descriptor per tap, Toeplitz filter
    block resident) against the oracle, bit-exact: accumulators and codes, or the codes of the
    window maximum with the fused pool, with channels of negative BN scale in every case."""
    B, H, W, C, cout, k, pool, mode = case
    rng = np.random.default_rng(abs(hash(case)) % (2 ** 32))
    x = rng.integers(0, 4, (B, H, W, C), dtype=np.uint8)
    w = np.where(rng.integers(0, 2, (cout, k, k, C)) == 1, 1, -1).astype(np.int8)
    K = k * k * C
    prm = _params(rng, cout, K)
    prm.gamma[1::3] = -np.abs(prm.gamma[1::3])
    T, sg = _fold_gpu(prm, K)
    pad = (k - 1) // 2
    d = ifq.conv_desc(B, H, W, C, cout, k, 1, pad, mode, ifq.IFQ_PATH_WIN, pool=pool if pool > 1 else 0)
    assert ifq.ifq_conv_plan(d) == ifq.IFQ_PATH_WIN
    codes, acc = _run_conv(x, w, T, sg, 1, pad, mode, ifq.IFQ_PATH_WIN, pool=pool if pool > 1 else 0)
    A = O.conv_acc(x, w, 1, pad)
    if acc is not None:
        assert (acc == A).all(), f"accumulators differ at {np.argwhere(acc != A)[:5].tolist()}"
    To, so = O.fold(prm, K)
    ref = O.int_chain(O.maxpool_acc(A, pool, pool, 0) if pool > 1 else A, To, so)
    assert codes.shape == ref.shape
    assert (codes == ref).all(), f"codes differ at {np.argwhere(codes != ref)[:5].tolist()}"
