"""GPU parity of the split-K tensor-core kernel (clusters of two CTAs, each summing a range of
the K stages of Eq. (1), partial sums exchanged through distributed shared memory), bit-exact
against the CPU oracle: accumulators and codes (Eq. (7) thresholds), 2- and 4-bit codes, 8-bit
inputs, the fused pool, ragged tiles and uneven K ranges, and several tiles per cluster (the
receive slots reused).  The split is forced with IFQ_TC_KS = 2; the planner's own choice
(AlexNet's FC layers) is covered by the whole-workload tests."""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_1911_08076_gb300 import ifq, synth
from paper_1911_08076_gb300.stack import DeviceStack

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]

DEV = "cuda"
TC = ifq.IFQ_PATH_TC


def _params(rng, cout, K, kbits):
    """Float parameters scaled so that the accumulators of uniform k-bit codes reach every code."""
    n = 1 << kbits
    L = n - 1
    sd = np.sqrt(K * (n - 1) * (2 * n - 1) / 6.0)
    return O.Params(rng.uniform(0.5, 1.5, cout) * L / sd, rng.normal(1.0, 0.6, cout), rng.normal(0, 0.5, cout),
                    rng.normal(0, 1.0, cout), rng.uniform(0.5, 2.0, cout), None, 0.5, 0.5, -0.25, synth.EPS, kbits)


def _run(x, w, T, s, stride, pad, out_mode, kbits, pool, in8, monkeypatch):
    B, H, W, C = x.shape
    cout, k, _, _ = w.shape
    d = ifq.conv_desc(B, H, W, C, cout, k, stride, pad, out_mode, TC, pool=pool, kbits=kbits,
                      in_bits=8 if in8 else 0)
    assert ifq.ifq_conv_plan(d) == TC
    xp = torch.from_numpy(x if in8 else synth.pack_codes(x, kbits)).to(DEV)
    bits = torch.from_numpy(synth.pack_signs(w).view(np.int32)).to(DEV)
    prep = torch.empty(ifq.ifq_weights_prep_bytes(d), dtype=torch.uint8, device=DEV)
    ifq.ifq_pack_weights(d, bits, prep)
    ho, wo = ifq.ifq_conv_out_shape(d)
    fb = synth.field_bits(kbits)
    yc = ya = None
    if out_mode & ifq.IFQ_OUT_CODES:
        yc = torch.full((B, ho, wo, cout * fb // 8), 0x5A, dtype=torch.uint8, device=DEV)
    if out_mode & ifq.IFQ_OUT_ACC:
        ya = torch.full((B, ho, wo, cout), -777777, dtype=torch.int32, device=DEV)
    monkeypatch.setenv("IFQ_TC_KS", "2")
    ifq.ifq_conv2bit(d, xp, prep, torch.from_numpy(T).to(DEV), torch.from_numpy(s).to(DEV), yc, ya)
    torch.cuda.synchronize()
    assert ifq.ifq_device_status() == ifq.IFQ_OK
    codes = None if yc is None else synth.unpack_codes(yc.cpu().numpy(), cout, kbits)
    acc = None if ya is None else ya.cpu().numpy()
    return codes, acc


SPLIT_CASES = [
    # B, H, W, C, cout, k, stride, pad, kbits, pool (split: BN = 64, two CTAs per cluster)
    (2, 7, 7, 512, 512, 3, 1, 1, 2, 0),      # the deep ResNet-18 layer, 36 K stages
    (3, 14, 14, 320, 96, 3, 2, 1, 2, 0),     # 23 K stages (uneven ranges), ragged M, partial N tile
    (3, 14, 14, 320, 200, 3, 2, 1, 2, 0),    # cout = 200: the last tile's second block partly empty
    (8, 14, 14, 256, 512, 3, 1, 1, 2, 0),    # 104 tiles: clusters with two tiles (receive slots reused)
    (16, 14, 14, 256, 256, 3, 1, 1, 2, 0),   # 392 tiles
    (4, 6, 6, 256, 512, 6, 1, 0, 2, 0),      # FC-as-conv, K = 9216
    (1, 1, 1, 4096, 4096, 1, 1, 0, 2, 0),    # FC7-like: one output row, 32 K stages
    (2, 14, 14, 256, 256, 3, 1, 1, 2, 2),    # fused 2x2 pool
    (1, 16, 16, 256, 128, 3, 1, 1, 2, 4),    # fused 4x4 pool
    (2, 7, 7, 256, 512, 3, 1, 1, 4, 0),      # 4-bit codes
    (2, 14, 14, 128, 256, 3, 1, 1, 3, 0),    # 3-bit codes in 4-bit fields
    (2, 14, 14, 128, 256, 3, 1, 1, 4, 2),    # 4-bit codes, fused pool
]


@pytest.mark.parametrize("case", SPLIT_CASES, ids=[str(c) for c in SPLIT_CASES])
def test_split_k_matches_oracle(case, monkeypatch):
    B, H, W, C, cout, k, s, p, kbits, pool = case
    rng = np.random.default_rng(sum(case) + 17)
    x = rng.integers(0, 1 << kbits, (B, H, W, C), dtype=np.uint8)
    w = np.where(rng.integers(0, 2, (cout, k, k, C)) == 1, 1, -1).astype(np.int8)
    K = k * k * C
    prm = _params(rng, cout, K, kbits)
    T, sg = _fold(prm, K)
    mode = ifq.IFQ_OUT_CODES if pool else ifq.IFQ_OUT_BOTH
    codes, acc = _run(x, w, T, sg, s, p, mode, kbits, pool, False, monkeypatch)
    A = O.conv_acc(x, w, s, p)
    if pool:
        ref = O.int_chain(O.maxpool_acc(A, pool, pool, 0), *O.fold(prm, K))
    else:
        assert (acc == A).all()
        ref = O.int_chain(A, *O.fold(prm, K))
    assert (codes == ref).all()


def _fold(p, K):
    return ifq.ifq_fold_layer(K, p.alpha, p.gamma, p.beta, p.mean, p.var, p.delta_in, p.bias, p.eps, p.q_base,
                              p.q_offset, p.kbits)


def test_split_k_on_8bit_input(monkeypatch):
    """A first layer on 8-bit values (nibble pairs, K doubled) with the split."""
    rng = np.random.default_rng(5)
    B, H, W, C, cout = 2, 12, 12, 64, 256
    x = rng.integers(0, 256, (B, H, W, C), dtype=np.uint8)
    w = np.where(rng.integers(0, 2, (cout, 3, 3, C)) == 1, 1, -1).astype(np.int8)
    K = 9 * C
    K_fold = -(-255 * K // 3)
    sd = np.sqrt(K * 21717.0)                        # spread of A for uniform bytes and +-1 filters
    prm = O.Params(rng.uniform(0.5, 1.5, cout) * 3.0 / (sd * synth.PIXEL_STEP), rng.normal(1.0, 0.6, cout),
                   rng.normal(0, 0.5, cout), rng.normal(0, 1.0, cout), rng.uniform(0.5, 2.0, cout), None,
                   synth.PIXEL_STEP, 0.5, -0.25, synth.EPS)
    T, sg = _fold(prm, K_fold)
    codes, acc = _run(x, w, T, sg, 1, 1, ifq.IFQ_OUT_BOTH, 2, 0, True, monkeypatch)
    A = O.conv_acc(x, w, 1, 1)
    assert (acc == A).all()
    assert (codes == O.int_chain(A, *O.fold(prm, K_fold))).all()


def test_split_k_resnet18_stack_equals_unsplit(monkeypatch):
    """The whole ResNet-18 body (batch 8) with every eligible layer forced to split: every layer's
    codes equal the unsplit run's, and the oracle agrees on the first image of the last layer."""
    wl = synth.get("resnet18", batch=8)
    x, params = synth.draw_workload(wl, batch=8)
    xd = torch.from_numpy(synth.pack_codes(x)).to(DEV)
    monkeypatch.setenv("IFQ_TC_KS", "1")
    ref = DeviceStack(wl, params, batch=8, device=DEV)
    ref.forward(xd)
    monkeypatch.setenv("IFQ_TC_KS", "2")
    st = DeviceStack(wl, params, batch=8, device=DEV)
    st.forward(xd)
    torch.cuda.synchronize()
    assert ifq.ifq_device_status() == ifq.IFQ_OK
    for li in range(len(wl.layers)):
        assert torch.equal(st.y_codes[li], ref.y_codes[li]), wl.layers[li].name
    one = O.forward(wl, x[:1], params)
    last = len(wl.layers) - 1
    got = synth.unpack_codes(st.y_codes[last][:1].cpu().numpy(), wl.layers[last].cout)
    assert (got == one[last]).all()


BITS_CASES = [c for c in SPLIT_CASES if c[8] == 2]


@pytest.mark.parametrize("case", BITS_CASES, ids=[str(c) for c in BITS_CASES])
def test_split_k_with_filter_tiles_from_sign_bits(case, monkeypatch):
    """The split kernel whose filter tiles are expanded in shared memory from the sign bits (one
    bit per weight streamed instead of an e4m3 byte; IFQ_TC_BX = 2 forces it), bit-exact against the
    oracle, including K padded past the filter (C = 320: 2880 of 2944 positions) and partial channel
    tiles."""
    monkeypatch.setenv("IFQ_TC_BX", "2")
    test_split_k_matches_oracle(case, monkeypatch)


def test_fc_layers_with_sign_bit_filters_equal_e4m3_filter_tiles(monkeypatch):
    """AlexNet's FC6 and FC7 shapes (one 128-row tile): the run with filter tiles from sign bits
    (IFQ_TC_BX = 1) equals the run that loads e4m3 filter tiles, codes and accumulators."""
    rng = np.random.default_rng(6)
    for (B, H, C, cout, k, mode) in ((128, 6, 256, 4096, 6, ifq.IFQ_OUT_CODES), (128, 1, 4096, 4096, 1, ifq.IFQ_OUT_ACC)):
        x = rng.integers(0, 4, (B, H, H, C), dtype=np.uint8)
        w = np.where(rng.integers(0, 2, (cout, k, k, C)) == 1, 1, -1).astype(np.int8)
        prm = _params(rng, cout, k * k * C, 2)
        T, sg = _fold(prm, k * k * C)
        outs = []
        for bx in ("1", "0"):
            monkeypatch.setenv("IFQ_TC_BX", bx)
            monkeypatch.delenv("IFQ_TC_KS", raising=False)
            d = ifq.conv_desc(B, H, H, C, cout, k, 1, 0, mode, TC)
            xp = torch.from_numpy(synth.pack_codes(x)).to(DEV)
            bits = torch.from_numpy(synth.pack_signs(w).view(np.int32)).to(DEV)
            prep = torch.empty(ifq.ifq_weights_prep_bytes(d), dtype=torch.uint8, device=DEV)
            ifq.ifq_pack_weights(d, bits, prep)
            yc = torch.zeros((B, 1, 1, cout // 4), dtype=torch.uint8, device=DEV) if mode & 1 else None
            ya = torch.zeros((B, 1, 1, cout), dtype=torch.int32, device=DEV) if mode & 2 else None
            ifq.ifq_conv2bit(d, xp, prep, torch.from_numpy(T).to(DEV), torch.from_numpy(sg).to(DEV), yc, ya)
            torch.cuda.synchronize()
            assert ifq.ifq_device_status() == ifq.IFQ_OK
            outs.append((None if yc is None else yc.cpu(), None if ya is None else ya.cpu()))
        for a, b in zip(outs[0], outs[1]):
            if a is not None:
                assert torch.equal(a, b)
        A = O.conv_acc(x, w, 1, 0)
        if mode & 2:
            assert (outs[0][1].numpy() == A).all()
        else:
            assert (synth.unpack_codes(outs[0][0].numpy(), cout) == O.int_chain(A, *O.fold(prm, k * k * C))).all()
