"""GPU parity of the warp-MMA path (mma.sync e4m3 tiles of 16 pixels x 8 channels, accumulators and
the fused 2 x 2 pool in registers) through the C ABI, bit-exact against the CPU oracle: 3 x 3
stride-1 layers on 2-bit codes with 8 or 16 input channels and on 8-bit values with 4, for 8, 16
and 32 output channels, with and without the pool, ragged widths and heights, channels of negative
BN scale, and the extreme accumulators of the 8-bit layer."""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_1911_08076_gb300 import ifq, synth

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]

DEV = "cuda"
WARP = ifq.IFQ_PATH_WARP


def _params_codes(rng, cout, K):
    sd = np.sqrt(K * 3.5)
    return O.Params(rng.uniform(0.5, 1.5, cout) * 4.0 / sd, rng.normal(1.0, 0.6, cout), rng.normal(0, 0.5, cout),
                    rng.normal(0, 1.0, cout), rng.uniform(0.5, 2.0, cout), None, 0.5, 0.5, -0.25, synth.EPS)


def _params_pixels(rng, cout, K):
    sd = np.sqrt(K * 21717.0)                        # spread of A for uniform bytes and +-1 filters
    return O.Params(rng.uniform(0.5, 1.5, cout) * 3.0 / (sd * synth.PIXEL_STEP), rng.normal(1.0, 0.6, cout),
                    rng.normal(0, 0.5, cout), rng.normal(0, 1.0, cout), rng.uniform(0.5, 2.0, cout), None,
                    synth.PIXEL_STEP, 0.5, -0.25, synth.EPS)


def run_warp(x, w, prm, K_fold, pool, mode, in8, path=WARP):
    """One conv through ifq_conv2bit on the requested path; returns (codes, acc, path taken)."""
    B, H, W, C = x.shape
    cout = w.shape[0]
    d = ifq.conv_desc(B, H, W, C, cout, 3, 1, 1, mode, path, pool=pool, in_bits=8 if in8 else 0)
    taken = ifq.ifq_conv_plan(d)
    T, sg = ifq.ifq_fold_layer(K_fold, prm.alpha, prm.gamma, prm.beta, prm.mean, prm.var, prm.delta_in, None,
                               prm.eps, prm.q_base, prm.q_offset)
    bits = torch.from_numpy(synth.pack_signs(w).view(np.int32)).to(DEV)
    prep = torch.empty(ifq.ifq_weights_prep_bytes(d), dtype=torch.uint8, device=DEV)
    ifq.ifq_pack_weights(d, bits, prep)
    ho, wo = ifq.ifq_conv_out_shape(d)
    yc = ya = None
    if mode & ifq.IFQ_OUT_CODES:
        yc = torch.full((B, ho, wo, cout // 4), 0x5A, dtype=torch.uint8, device=DEV)
    if mode & ifq.IFQ_OUT_ACC:
        ya = torch.full((B, ho, wo, cout), -777777, dtype=torch.int32, device=DEV)
    xin = torch.from_numpy(x if in8 else synth.pack_codes(x)).to(DEV)
    ifq.ifq_conv2bit(d, xin, prep, torch.from_numpy(T).to(DEV), torch.from_numpy(sg).to(DEV), yc, ya)
    torch.cuda.synchronize()
    assert ifq.ifq_device_status() == ifq.IFQ_OK
    codes = None if yc is None else synth.unpack_codes(yc.cpu().numpy(), cout)
    acc = None if ya is None else ya.cpu().numpy()
    return codes, acc, taken


def check(x, w, prm, K_fold, pool, mode, in8):
    codes, acc, taken = run_warp(x, w, prm, K_fold, pool, mode, in8)
    assert taken == WARP
    A = O.conv_acc(x, w, 1, 1)
    if acc is not None:
        assert (acc == A).all(), f"accumulators differ at {np.argwhere(acc != A)[:5].tolist()}"
    To, so = O.fold(prm, K_fold)
    if codes is not None:
        ref = O.int_chain(O.maxpool_acc(A, 2, 2, 0) if pool == 2 else A, To, so)
        assert codes.shape == ref.shape
        assert (codes == ref).all(), f"codes differ at {np.argwhere(codes != ref)[:5].tolist()}"
    return A


CODE_CASES = [
    # B, H, W, C, cout, pool, out_mode
    (1, 2, 2, 8, 8, 2, 1),          # one pooled pixel: one strip, one row pair, mostly halo
    (2, 16, 16, 8, 16, 2, 1),       # one band, one strip
    (2, 34, 38, 8, 16, 2, 1),       # ragged: 3 bands (16 + 16 + 2 rows), 3 strips (the last 6 wide)
    (1, 208, 208, 8, 16, 2, 1),     # IFQ-Tinier-YOLO conv2 at full size (one image)
    (2, 20, 24, 16, 32, 2, 1),      # 16-byte pixels, two K steps per filter row
    (1, 208, 208, 16, 32, 2, 1),    # Tiny-YOLO conv2 / IFQ-Tinier-YOLO conv3 shape at 208
    (3, 52, 52, 16, 32, 2, 1),
    (2, 13, 17, 8, 8, 0, 3),        # no pool: odd height (the last row pair's second row dropped)
    (2, 9, 33, 16, 32, 0, 3),       # no pool, 3 strips with a 1-pixel tail
    (1, 18, 40, 16, 16, 0, 2),      # accumulators only
    (2, 30, 30, 8, 32, 0, 1),       # codes only, 4 channel tiles on 8-byte pixels
    (2, 6, 100, 16, 8, 2, 1),       # one channel tile on 16-byte pixels
]


@pytest.mark.parametrize("case", CODE_CASES, ids=[str(c) for c in CODE_CASES])
def test_warp_path_on_codes_matches_oracle(case):
    B, H, W, C, cout, pool, mode = case
    rng = np.random.default_rng(abs(hash(("warp",) + case)) % (2 ** 32))
    x = rng.integers(0, 4, (B, H, W, C), dtype=np.uint8)
    w = np.where(rng.integers(0, 2, (cout, 3, 3, C)) == 1, 1, -1).astype(np.int8)
    K = 9 * C
    prm = _params_codes(rng, cout, K)
    prm.gamma[1::3] = -np.abs(prm.gamma[1::3])       # a third of the channels with a negative BN scale
    check(x, w, prm, K, pool, mode, False)


PIXEL_CASES = [
    # B, H, W, cout, pool, out_mode
    (1, 2, 2, 8, 2, 1),
    (2, 20, 20, 8, 2, 1),
    (2, 34, 50, 8, 2, 1),           # ragged bands and strips
    (1, 416, 416, 8, 2, 1),         # IFQ-Tinier-YOLO conv1 at full size (one image)
    (2, 17, 19, 16, 0, 3),          # no pool, odd sizes, accumulators and codes
    (2, 18, 18, 32, 2, 1),
    (1, 11, 64, 8, 0, 2),
]


@pytest.mark.parametrize("case", PIXEL_CASES, ids=[str(c) for c in PIXEL_CASES])
def test_warp_path_on_8bit_values_matches_oracle(case):
    """The first layer on 8-bit values (RGB plus a zero channel): each value is its two 4-bit fields
    with weights +-1 and +-16 in the same MMA."""
    B, H, W, cout, pool, mode = case
    rng = np.random.default_rng(abs(hash(("warp8",) + case)) % (2 ** 32))
    x = rng.integers(0, 256, (B, H, W, 4), dtype=np.uint8)
    x[..., 3] = 0
    w = np.where(rng.integers(0, 2, (cout, 3, 3, 4)) == 1, 1, -1).astype(np.int8)
    K = 36
    prm = _params_pixels(rng, cout, K)
    prm.gamma[2::4] = -np.abs(prm.gamma[2::4])
    check(x, w, prm, -(-255 * K // 3), pool, mode, True)


@pytest.mark.parametrize("in8", [False, True], ids=["codes", "pixels"])
def test_warp_path_extreme_accumulators_are_exact(in8):
    """Every input at its maximum (code 3, or value 255 in all 4 channels) under all-(+1) and all-(-1)
    filters and alternating ones: |A| reaches 3 K = 432 on codes and 255 * 36 = 9180 on pixels."""
    C = 16 if not in8 else 4
    B, H, W, cout = 1, 6, 20, 16
    x = np.full((B, H, W, C), 255 if in8 else 3, dtype=np.uint8)
    w = np.ones((cout, 3, 3, C), dtype=np.int8)
    w[1::2] = -1
    w[2] = np.where((np.arange(9 * C).reshape(3, 3, C) % 2) == 0, 1, -1)
    K = 9 * C
    rng = np.random.default_rng(5)
    prm = _params_pixels(rng, cout, K) if in8 else _params_codes(rng, cout, K)
    A = check(x, w, prm, -(-255 * K // 3) if in8 else K, 0, ifq.IFQ_OUT_BOTH, in8)
    top = 255 * 36 if in8 else 3 * K
    assert A[0, 2, 2, 0] == top and A[0, 2, 2, 1] == -top


def test_warp_path_plan():
    """Where the warp-MMA path applies when requested; elsewhere a request for it takes the
    tensor-core path."""
    plan = lambda *a, **k: ifq.ifq_conv_plan(ifq.conv_desc(*a, **k))
    assert plan(64, 208, 208, 8, 16, 3, 1, 1, pool=2, path=WARP) == WARP
    assert plan(64, 416, 416, 4, 8, 3, 1, 1, pool=2, in_bits=8, path=WARP) == WARP
    assert plan(64, 208, 208, 16, 32, 3, 1, 1, pool=2, path=WARP) == WARP
    assert plan(2, 16, 16, 32, 64, 3, 1, 1, path=WARP) == ifq.IFQ_PATH_TC      # cin 32
    assert plan(2, 16, 16, 16, 64, 3, 1, 1, path=WARP) == ifq.IFQ_PATH_TC      # cout 64
    assert plan(2, 16, 16, 16, 32, 3, 2, 1, path=WARP) == ifq.IFQ_PATH_TC      # stride 2
