"""GPU parity of the k-bit codes (k = 3, 4: Eq. (8), Table 2's k columns) through the C ABI,
bit-exact against the CPU oracle: the convolution on both kernel paths, the fused and the
separate pools, the packing helpers, the exactness of the tensor-core accumulation at the
largest admitted magnitude, and whole k-bit stacks."""
import numpy as np
import pytest
import torch
from stack_parity import compare_stack_with_oracle

from oracle import oracle as O
from paper_1911_08076_gb300 import ifq, synth
from paper_1911_08076_gb300.stack import DeviceStack

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]

DEV = "cuda"
TC, BS = ifq.IFQ_PATH_TC, ifq.IFQ_PATH_BITSERIAL


def _params(rng, cout, K, kbits):
    """Float parameters scaled so that the accumulators of uniform k-bit codes reach every code."""
    n = 1 << kbits
    L = n - 1
    sd = np.sqrt(K * (n - 1) * (2 * n - 1) / 6.0)      # spread of A for uniform codes and +-1 filters
    return O.Params(rng.uniform(0.5, 1.5, cout) * L / sd, rng.normal(1.0, 0.6, cout), rng.normal(0, 0.5, cout),
                    rng.normal(0, 1.0, cout), rng.uniform(0.5, 2.0, cout), None, 0.5, 0.5, -0.25, synth.EPS, kbits)


def _fold(p, K):
    return ifq.ifq_fold_layer(K, p.alpha, p.gamma, p.beta, p.mean, p.var, p.delta_in, p.bias, p.eps, p.q_base,
                              p.q_offset, p.kbits)


def _run_conv(x, w, T, s, stride, pad, out_mode, path, kbits, bn=None, pool=0, expect_path=None, monkeypatch=None):
    B, H, W, C = x.shape
    cout, k, _, _ = w.shape
    d = ifq.conv_desc(B, H, W, C, cout, k, stride, pad, out_mode, path, pool=pool, kbits=kbits)
    if expect_path is not None:
        assert ifq.ifq_conv_plan(d) == expect_path
    xp = torch.from_numpy(synth.pack_codes(x, kbits)).to(DEV)
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
    if bn:
        monkeypatch.setenv("IFQ_TC_BN", str(bn))
    ifq.ifq_conv2bit(d, xp, prep, torch.from_numpy(T).to(DEV), torch.from_numpy(s).to(DEV), yc, ya)
    torch.cuda.synchronize()
    assert ifq.ifq_device_status() == ifq.IFQ_OK
    codes = None if yc is None else synth.unpack_codes(yc.cpu().numpy(), cout, kbits)
    acc = None if ya is None else ya.cpu().numpy()
    return codes, acc


KCONV_CASES = [
    # B, H, W, C, cout, k, stride, pad
    (1, 16, 16, 64, 64, 3, 1, 1),
    (2, 9, 7, 64, 96, 3, 2, 1),          # ragged M, partial N tile
    (3, 11, 13, 128, 256, 3, 1, 1),      # several M tiles with a ragged tail
    (2, 8, 8, 256, 320, 1, 1, 0),        # 1x1, two N tiles
    (1, 27, 27, 96, 64, 5, 1, 2),        # 5x5, 48-byte pixels at 4-bit fields
    (2, 12, 12, 48, 32, 3, 1, 1),        # 24-byte pixels: 4-byte granules
    (2, 10, 10, 16, 32, 3, 1, 1),        # K = 144 (partial K stage), 8-byte pixels
    (2, 10, 10, 8, 16, 3, 1, 1),
    (1, 9, 9, 12, 20, 3, 1, 1),          # cin % 8 != 0: bit-serial only at 4-bit fields
    (4, 6, 6, 256, 512, 6, 1, 0),        # FC-as-conv, K = 9216
    (1, 14, 14, 256, 512, 3, 2, 1),      # stride 2
]


@pytest.mark.parametrize("kbits", [3, 4])
@pytest.mark.parametrize("path", [TC, BS], ids=["tc", "bitserial"])
@pytest.mark.parametrize("case", KCONV_CASES, ids=[str(c) for c in KCONV_CASES])
def test_kbit_conv_matches_oracle(case, path, kbits):
    B, H, W, C, cout, k, s, p = case
    rng = np.random.default_rng(abs(hash((case, kbits))) % (2 ** 32))
    x = rng.integers(0, 1 << kbits, (B, H, W, C), dtype=np.uint8)
    w = np.where(rng.integers(0, 2, (cout, k, k, C)) == 1, 1, -1).astype(np.int8)
    K = k * k * C
    prm = _params(rng, cout, K, kbits)
    T, sg = _fold(prm, K)
    expect = BS if (path == BS or C % 8 != 0) else TC
    codes, acc = _run_conv(x, w, T, sg, s, p, ifq.IFQ_OUT_BOTH, path, kbits, expect_path=expect)
    A = O.conv_acc(x, w, s, p)
    assert (acc == A).all(), f"accumulators differ at {np.argwhere(acc != A)[:5].tolist()}"
    To, so = O.fold(prm, K)
    ref, _ = O.check_chains(A, prm, To, so)
    assert len(np.unique(ref)) >= (1 << kbits) - 2
    assert (codes == ref).all(), f"codes differ at {np.argwhere(codes != ref)[:5].tolist()}"


@pytest.mark.parametrize("bn", [32, 64, 128])
def test_kbit_every_channel_tile(bn, monkeypatch):
    rng = np.random.default_rng(bn + 40)
    B, H, W, C, cout, k = 2, 12, 11, 64, 200, 3
    x = rng.integers(0, 16, (B, H, W, C), dtype=np.uint8)
    w = np.where(rng.integers(0, 2, (cout, k, k, C)) == 1, 1, -1).astype(np.int8)
    prm = _params(rng, cout, k * k * C, 4)
    T, sg = _fold(prm, k * k * C)
    codes, acc = _run_conv(x, w, T, sg, 1, 1, ifq.IFQ_OUT_BOTH, TC, 4, bn=bn, expect_path=TC,
                           monkeypatch=monkeypatch)
    A = O.conv_acc(x, w, 1, 1)
    assert (acc == A).all()
    assert (codes == O.int_chain(A, *O.fold(prm, k * k * C))).all()


KPOOL_FUSED_CASES = [
    # B, H, W, C, cout, k, stride, pad, p, kbits
    (2, 16, 16, 64, 64, 3, 1, 1, 2, 4),
    (3, 22, 26, 64, 96, 3, 1, 1, 2, 4),       # ragged last tile, partial channel tile
    (2, 20, 20, 16, 32, 3, 1, 1, 2, 4),       # 8-byte pixels
    (2, 16, 16, 128, 256, 3, 1, 1, 4, 4),     # 4x4 windows
    (1, 28, 28, 64, 128, 3, 2, 1, 2, 3),
    (2, 16, 16, 64, 200, 3, 1, 1, 2, 3),
]


@pytest.mark.parametrize("case", KPOOL_FUSED_CASES, ids=[str(c) for c in KPOOL_FUSED_CASES])
def test_kbit_fused_pool_matches_oracle(case):
    """k-bit codes of the window maximum of A (Sec. 2.1), bit-exact, with negative BN scales."""
    B, H, W, C, cout, k, s, p, pool, kbits = case
    rng = np.random.default_rng(abs(hash(case)) % (2 ** 32))
    x = rng.integers(0, 1 << kbits, (B, H, W, C), dtype=np.uint8)
    w = np.where(rng.integers(0, 2, (cout, k, k, C)) == 1, 1, -1).astype(np.int8)
    K = k * k * C
    prm = _params(rng, cout, K, kbits)
    prm.gamma[1::3] = -np.abs(prm.gamma[1::3])
    T, sg = _fold(prm, K)
    codes, _ = _run_conv(x, w, T, sg, s, p, ifq.IFQ_OUT_CODES, TC, kbits, pool=pool, expect_path=TC)
    A = O.conv_acc(x, w, s, p)
    ref = O.int_chain(O.maxpool_acc(A, pool, pool, 0), *O.fold(prm, K))
    assert codes.shape == ref.shape
    assert (codes == ref).all(), f"codes differ at {np.argwhere(codes != ref)[:5].tolist()}"


KPOOL_CASES = [
    # B, H, W, C, k, stride, pad, signed
    (2, 27, 27, 256, 3, 2, 0, True),       # 128-byte pixels: 16-byte words
    (2, 8, 8, 40, 2, 2, 0, True),          # 20-byte pixels: 4-byte words
    (1, 13, 13, 512, 2, 1, 1, True),
    (2, 9, 9, 16, 2, 2, 0, False),
    (1, 7, 5, 12, 3, 2, 1, True),          # 6-byte pixels: bytes
    (2, 8, 12, 8, 2, 2, 0, True),          # 4-byte pixels, 2x2 / 2: the row-pair kernel
    (1, 10, 14, 16, 2, 2, 0, True),        # 8-byte pixels, 2x2 / 2: the row-pair kernel
    (1, 9, 14, 8, 2, 2, 0, True),          # 4-byte pixels, rows of 56 bytes: the general kernel
]


@pytest.mark.parametrize("kbits", [3, 4])
@pytest.mark.parametrize("case", KPOOL_CASES, ids=[str(c) for c in KPOOL_CASES])
def test_kbit_maxpool_matches_oracle(case, kbits):
    B, H, W, C, k, s, p, signed = case
    rng = np.random.default_rng(sum(case[:7]) + kbits)
    x = rng.integers(0, 1 << kbits, (B, H, W, C), dtype=np.uint8)
    sign = np.where(rng.integers(0, 4, C) == 0, -1, 1).astype(np.int8)
    sign[0] = -1
    d = ifq.pool_desc(B, H, W, C, k, s, p, kbits)
    ho, wo = ifq.ifq_pool_out_shape(d)
    y = torch.full((B, ho, wo, C // 2), 0xA5, dtype=torch.uint8, device=DEV)
    sg = torch.from_numpy(sign).to(DEV) if signed else None
    ifq.ifq_maxpool2bit(d, torch.from_numpy(synth.pack_codes(x, kbits)).to(DEV), sg, y)
    torch.cuda.synchronize()
    got = synth.unpack_codes(y.cpu().numpy(), kbits=kbits)
    assert (got == O.maxpool_codes(x, k, s, p, sign if signed else None)).all()


@pytest.mark.parametrize("kbits", [2, 3, 4])
def test_kbit_pack_helpers_match_formats(kbits):
    rng = np.random.default_rng(kbits)
    c = rng.integers(0, 1 << kbits, 4 * 1237, dtype=np.uint8)
    ct = torch.from_numpy(c).to(DEV)
    nb = c.size * synth.field_bits(kbits) // 8
    packed = torch.empty(nb, dtype=torch.uint8, device=DEV)
    ifq.ifq_pack_codes_kbits(ct, packed, c.size, kbits)
    assert (packed.cpu().numpy() == synth.pack_codes(c, kbits)).all()
    back = torch.empty_like(ct)
    ifq.ifq_unpack_codes_kbits(packed, back, c.size, kbits)
    assert (back.cpu().numpy() == c).all()


@pytest.mark.parametrize("kbits,K", [(2, 65536), (3, 28064), (4, 13088)])
def test_tc_accumulation_exact_at_the_admitted_bound(kbits, K):
    """Accumulators near the largest magnitude the tensor-core path admits, (2^k - 1) K <= 196608,
    with small odd addends all along K (codes mostly 2^k - 1 with some 1s and 2s; rows of all +1,
    all -1, 95 % +1 and random signs): the fp32 accumulation in tensor memory must stay exact."""
    rng = np.random.default_rng(K)
    L = (1 << kbits) - 1
    B, cout = 160, 64
    x = rng.choice(np.array([1, 2, L - 1, L], np.uint8), size=(B, 1, 1, K), p=[0.05, 0.05, 0.1, 0.8])
    w = np.ones((cout, 1, 1, K), np.int8)
    w[1] = -1
    for r in range(2, 40):
        w[r, 0, 0, rng.random(K) < 0.05] = -1
    for r in range(40, 64):
        w[r, 0, 0, rng.random(K) < 0.5] = -1
    prm = _params(rng, cout, K, kbits)
    prm.alpha[:2] = prm.alpha[:2] / 100.0        # keep the largest rows' codes off the clamp
    T, sg = _fold(prm, K)
    codes, acc = _run_conv(x, w, T, sg, 1, 0, ifq.IFQ_OUT_BOTH, TC, kbits, expect_path=TC)
    A = x.reshape(B, K).astype(np.int64) @ w.reshape(cout, K).astype(np.int64).T
    assert np.abs(A).max() > 0.8 * L * K
    assert (acc.reshape(B, cout) == A).all(), f"{int((acc.reshape(B, cout) != A).sum())} accumulators differ"
    assert (codes.reshape(B, cout) == O.int_chain(A.astype(np.int32), *O.fold(prm, K))).all()


@pytest.mark.parametrize("name", ["alexnet_k3", "alexnet_k4", "resnet18_k4", "tinyyolo_fused_k4"])
def test_kbit_workload_matches_oracle(name):
    """Whole k-bit stacks at full size through ifq_forward; the oracle recomputes every image."""
    wl = synth.get(name)
    x, params = synth.draw_workload(wl)
    compare_stack_with_oracle(wl, x, params)
