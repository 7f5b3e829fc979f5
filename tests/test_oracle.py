"""Pins of the CPU oracle against what the paper and the mathematics fix (no GPU).

* hand-worked cases of Eq. (1)-(3) and Eq. (7) + floor (tests/golden/hand_cases.json);
* the integrated conversion reproduces the float chain on the whole achievable
  accumulator range (Sec. 3.2 / Sec. 4.1.1: "identical outputs"), by brute force;
* the integer convolution against torch.nn.functional.conv2d in float64 (exact
  for these integers), plus invariants (parity, bounds, negation, padding);
* pooling on codes with channel signs equals quantize(max of Y^conv) (Sec. 2.1);
* a planted mistake in the fold is caught.
"""
import json
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import oracle as O
from paper_1911_08076_gb300 import synth

HERE = os.path.dirname(os.path.abspath(__file__))
GOLD = json.load(open(os.path.join(HERE, "golden", "hand_cases.json")))


def _params(c):
    return O.Params([c["alpha"]], [c["gamma"]], [c["beta"]], [c["mean"]], [c["var"]], [c["bias"]],
                    c["delta_in"], c["q_base"], c["q_offset"], c["eps"])


@pytest.mark.parametrize("case", GOLD["cases"], ids=[c["name"] for c in GOLD["cases"]])
def test_hand_case_float_chain(case):
    A = np.array(case["A"], dtype=np.int32).reshape(-1, 1)
    assert O.float_chain(A, _params(case)).ravel().tolist() == case["codes"]


@pytest.mark.parametrize("case", GOLD["cases"], ids=[c["name"] for c in GOLD["cases"]])
def test_hand_case_fold_and_int_chain(case):
    T, s = O.fold(_params(case), case["K"])
    assert T[0].tolist() == case["T"]
    assert int(s[0]) == case["sign"]
    A = np.array(case["A"], dtype=np.int32).reshape(-1, 1)
    assert O.int_chain(A, T, s).ravel().tolist() == case["codes"]


@pytest.mark.parametrize("case", [c for c in GOLD["cases"] if "x" in c], ids=lambda c: c["name"])
def test_hand_case_conv(case):
    x = np.array(case["x"], dtype=np.uint8).reshape(1, 1, 1, -1)
    w = np.array(case["w"], dtype=np.int8).reshape(1, 1, 1, -1)
    assert int(O.conv_acc(x, w, 1, 0).ravel()[0]) == case["A"][0]


def _bitserial_dot(x, w):
    """dot = sum_p 2^p * (2*popc(a_p & w+) - popc(a_p)) over bit planes a_p of the codes."""
    wp = (np.asarray(w) > 0).astype(np.int64)
    tot = 0
    for p in (0, 1):
        a = (np.asarray(x, dtype=np.int64) >> p) & 1
        tot += (1 << p) * (2 * int((a & wp).sum()) - int(a.sum()))
    return tot


def test_bitserial_identity():
    g = GOLD["bitserial"]
    assert _bitserial_dot(g["x"], g["w"]) == g["dot"]
    rng = np.random.default_rng(5)
    for n in (1, 7, 64, 576, 4608):
        x = rng.integers(0, 4, n)
        w = np.where(rng.integers(0, 2, n) == 1, 1, -1)
        assert _bitserial_dot(x, w) == int((x * w).sum())


# ----------------------------------------------------------------------------- brute force


def _random_params(rng, cout, kbits=2, bias=True, eps=1e-5, spread=1.0):
    step = 0.5
    return O.Params(rng.uniform(0.05, 2.0, cout), rng.normal(0.0, 1.0, cout) * spread, rng.normal(0, 0.5, cout),
                    rng.normal(0, 3.0, cout), rng.uniform(0.1, 3.0, cout),
                    rng.normal(0, 1.0, cout) if bias else None, 0.5, step, -step / 2, eps, kbits)


def _full_domain(p, K):
    amax = p.levels * K
    A = np.repeat(np.arange(-amax, amax + 1, dtype=np.int32)[:, None], p.cout, axis=1)
    T, s = O.fold(p, K)
    codes, ties = O.check_chains(A, p, T, s)
    return A, T, s, codes, ties


@pytest.mark.parametrize("kbits,K", [(1, 9), (2, 9), (2, 64), (2, 576), (3, 144), (4, 72)])
def test_fold_reproduces_float_chain_on_whole_range(kbits, K):
    rng = np.random.default_rng(100 + kbits * 1000 + K)
    # gamma ~ N(0,1) gives both signs; accumulator scale chosen so that every code occurs
    p = _random_params(rng, 48, kbits=kbits)
    p.alpha = p.alpha * (4.0 / np.sqrt(K))
    A, T, s, codes, ties = _full_domain(p, K)
    assert ties == 0
    assert codes.max() == p.levels and codes.min() == 0
    # monotone in A: non-decreasing for sign +1, non-increasing for sign -1
    d = np.diff(codes.astype(np.int16), axis=0)
    assert (d[:, s > 0] >= 0).all() and (d[:, s < 0] <= 0).all()


@pytest.mark.parametrize("wl_name", ["pr1", "resnet18", "alexnet", "tinyyolo", "tinieryolo", "roofline3x3",
                                     "roofline1x1"])
def test_fold_on_workload_parameters(wl_name):
    """Every conv layer of each workload, 24 sampled channels, every A in [-3K, 3K]."""
    wl = synth.get(wl_name)
    rng = np.random.default_rng(wl.seed)
    for li, layer in enumerate(wl.layers):
        if layer.kind != "conv":
            continue
        cp = synth.draw_conv_params(rng, layer)
        sel = np.random.default_rng(li).choice(layer.cout, min(24, layer.cout), replace=False)
        p = O.Params(cp.alpha[sel], cp.gamma[sel], cp.beta[sel], cp.mean[sel], cp.var[sel], None, cp.delta_in,
                     cp.q_base, cp.q_offset, cp.eps)
        _, T, s, codes, ties = _full_domain(p, layer.k * layer.k * layer.cin)
        assert ties == 0
        assert (np.diff(T, axis=1) >= 0).all()


@pytest.mark.parametrize("kbits", [2, 3, 4])
def test_kbit_fold_is_floor_of_compact_thresholds(kbits):
    """Eq. (8): with uniform levels thr_i = i*base + offset, the composed thresholds lie on one
    line, thr'_i = i*base' + offset' with base' = sigma*base/(alpha*delta) and
    offset' = (theta - b + sigma*(offset - beta))/(alpha*delta), sigma = sqrt(var + eps)/gamma
    (the BN shift beta moves the offset), and the integer thresholds are their floors
    (gamma > 0) or the floors of -thr'_i (gamma < 0, compared with -A).  The compact form is
    evaluated here from the inputs in 40-digit decimal arithmetic, independently of the oracle's
    per-threshold double arithmetic; values within 1e-9 of an integer (where double rounding may
    decide) are skipped and counted."""
    from decimal import Decimal, getcontext
    getcontext().prec = 40
    rng = np.random.default_rng(300 + kbits)
    K, cout = 576, 96
    p = _random_params(rng, cout, kbits=kbits)
    p.alpha = p.alpha * (4.0 / np.sqrt(K))
    T, s = O.fold(p, K)
    L, amax = p.levels, p.levels * K
    D = lambda v: Decimal(float(v))
    skipped = 0
    for n in range(cout):
        sigma = (D(p.var[n]) + D(p.eps)).sqrt() / D(p.gamma[n])
        ad = D(p.alpha[n]) * D(p.delta_in)
        base_c = sigma * D(p.q_base) / ad
        off_c = (D(p.mean[n]) - D(p.bias[n]) + sigma * (D(p.q_offset) - D(p.beta[n]))) / ad
        assert s[n] == (1 if p.gamma[n] > 0 else -1)
        for i in range(1, L + 1):
            t = i * base_c + off_c
            v = t if p.gamma[n] > 0 else -t
            fl = int(v.to_integral_value(rounding="ROUND_FLOOR"))
            if abs(v - v.to_integral_value(rounding="ROUND_HALF_EVEN")) < Decimal("1e-9") * (1 + abs(v)):
                skipped += 1
                continue
            assert T[n, i - 1] == min(max(fl, -amax - 1), amax), (n, i)
    assert skipped <= 2


def test_fold_invariants():
    rng = np.random.default_rng(7)
    K = 576
    p = _random_params(rng, 512, spread=2.0)
    p.gamma[:8] = 0.0
    p.alpha[8:16] = 1e-6          # thresholds far outside the range -> clamped
    T, s = O.fold(p, K)
    amax = 3 * K
    assert (np.diff(T, axis=1) >= 0).all(), "thresholds ascend (Q7: non-strict)"
    assert T.min() >= -amax - 1 and T.max() <= amax
    assert ((s == -1) == (p.gamma < 0)).all()
    A = np.repeat(np.arange(-amax, amax + 1, dtype=np.int32)[:, None], p.cout, axis=1)
    codes = O.int_chain(A, T, s)
    assert (codes[:, :8] == codes[0, :8]).all(), "gamma = 0 gives a constant code"
    O.check_chains(A, p, T, s)


def test_exact_ties_resolved_by_floor():
    """z lands exactly on thresholds for a grid of A; the floor of Sec. 3.2 gives the lower code."""
    K = 16
    p = O.Params([1.0, 1.0], [1.0, -1.0], [0.0, 0.0], [0.0, 0.0], [1.0, 1.0], None, 0.5, 0.5, 0.0, 0.0)
    A = np.repeat(np.arange(-3 * K, 3 * K + 1, dtype=np.int32)[:, None], 2, axis=1)
    T, s = O.fold(p, K)
    assert T.tolist() == [[1, 2, 3], [1, 2, 3]] and s.tolist() == [1, -1]
    ci = O.int_chain(A, T, s)
    cf = O.float_chain(A, p)
    assert (ci == cf).all()
    z = 0.5 * A[:, 0]
    expect = (z > 0.5).astype(int) + (z > 1.0) + (z > 1.5)
    assert (ci[:, 0] == expect).all()
    assert (ci[:, 1] == (-z > 0.5).astype(int) + (-z > 1.0) + (-z > 1.5)).all()


def test_planted_fold_mistake_is_caught():
    """Off-by-one thresholds (a ceil in place of the floor) must break the chain comparison."""
    rng = np.random.default_rng(11)
    K = 64
    p = _random_params(rng, 16)
    p.alpha = p.alpha * (4.0 / np.sqrt(K))
    amax = 3 * K
    A = np.repeat(np.arange(-amax, amax + 1, dtype=np.int32)[:, None], p.cout, axis=1)
    T, s = O.fold(p, K)
    with pytest.raises(O.ChainMismatch):
        O.check_chains(A, p, T + 1, s)
    with pytest.raises(O.ChainMismatch):
        O.check_chains(A, p, T, -s)


# ----------------------------------------------------------------------------- convolution

CONV_SHAPES = [
    # B, H, W, C, cout, k, stride, pad
    (2, 7, 5, 8, 6, 3, 1, 1),
    (1, 9, 9, 12, 5, 5, 2, 2),
    (3, 8, 6, 4, 7, 1, 2, 0),
    (2, 6, 6, 16, 9, 6, 1, 0),
    (1, 1, 1, 40, 3, 1, 1, 0),
    (2, 5, 11, 4, 4, 3, 2, 1),
]


def _torch_conv(x, w, stride, pad):
    xt = torch.from_numpy(x.astype(np.float64)).permute(0, 3, 1, 2)
    wt = torch.from_numpy(w.astype(np.float64)).permute(0, 3, 1, 2)
    return F.conv2d(xt, wt, stride=stride, padding=pad).permute(0, 2, 3, 1).numpy()


@pytest.mark.parametrize("shape", CONV_SHAPES)
def test_conv_acc_matches_torch_conv2d(shape):
    B, H, W, C, cout, k, s, p = shape
    rng = np.random.default_rng(sum(shape))
    x = rng.integers(0, 4, (B, H, W, C), dtype=np.uint8)
    w = np.where(rng.integers(0, 2, (cout, k, k, C)) == 1, 1, -1).astype(np.int8)
    A = O.conv_acc(x, w, s, p)
    ref = _torch_conv(x, w, s, p)
    assert A.shape == ref.shape
    assert (A == ref.astype(np.int64)).all()


@pytest.mark.parametrize("shape", CONV_SHAPES)
def test_conv_invariants(shape):
    B, H, W, C, cout, k, s, p = shape
    rng = np.random.default_rng(1 + sum(shape))
    x = rng.integers(0, 4, (B, H, W, C), dtype=np.uint8)
    w = np.where(rng.integers(0, 2, (cout, k, k, C)) == 1, 1, -1).astype(np.int8)
    A = O.conv_acc(x, w, s, p).astype(np.int64)
    S = _torch_conv(x, np.ones((1, k, k, C), np.int8), s, p)[..., 0].astype(np.int64)[..., None]
    K = k * k * C
    assert ((A - S) % 2 == 0).all(), "A = S - 2*(codes under -1 weights)"
    assert (np.abs(A) <= S).all() and (S <= 3 * K).all()
    assert (O.conv_acc(x, np.ones_like(w), s, p) == np.broadcast_to(S, A.shape)).all()
    assert (O.conv_acc(x, -w, s, p) == -A).all()
    xp = np.pad(x, ((0, 0), (p, p), (p, p), (0, 0)))
    assert (O.conv_acc(xp, w, s, 0) == A).all(), "zero padding = code 0"


# ----------------------------------------------------------------------------- pooling

POOLS = [(3, 2, 0, 27), (3, 2, 0, 13), (2, 2, 0, 8), (2, 1, 1, 13), (2, 2, 0, 7)]


def _torch_pool(v, k, s, pad):
    t = torch.from_numpy(v.astype(np.float64)).permute(0, 3, 1, 2)
    if pad:
        t = F.pad(t, (0, pad, 0, pad), value=float("-inf"))
    return F.max_pool2d(t, k, s).permute(0, 2, 3, 1).numpy()


@pytest.mark.parametrize("k,s,pad,h", POOLS)
def test_maxpool_matches_torch(k, s, pad, h):
    rng = np.random.default_rng(k * 100 + h)
    A = rng.integers(-500, 500, (2, h, h + 1, 6)).astype(np.int32)
    assert (O.maxpool_acc(A, k, s, pad) == _torch_pool(A, k, s, pad)).all()
    c = rng.integers(0, 4, (2, h, h + 1, 8)).astype(np.uint8)
    assert (O.maxpool_codes(c, k, s, pad) == _torch_pool(c, k, s, pad)).all()


@pytest.mark.parametrize("k,s,pad,h", POOLS)
def test_signed_code_pool_equals_quantized_acc_pool(k, s, pad, h):
    """Sec. 2.1 places the pool on Y^conv before BN and quantizer; with the channel sign the
    code pool gives the same result (the composed quantizer is monotone in A)."""
    rng = np.random.default_rng(3 + k + h)
    K = 144
    p = _random_params(rng, 32)
    p.alpha = p.alpha * (4.0 / np.sqrt(K))
    T, sg = O.fold(p, K)
    assert (sg < 0).any() and (sg > 0).any()
    A = rng.integers(-3 * K, 3 * K + 1, (2, h, h, 32)).astype(np.int32)
    lhs = O.int_chain(O.maxpool_acc(A, k, s, pad), T, sg)
    rhs = O.maxpool_codes(O.int_chain(A, T, sg), k, s, pad, sg)
    assert (lhs == rhs).all()
    lhs_f = O.float_chain(O.maxpool_acc(A, k, s, pad), p)
    assert (lhs_f == lhs).all()
    # without the sign, a plain max differs on flipped channels (the reason for the sign mask)
    plain = O.maxpool_codes(O.int_chain(A, T, sg), k, s, pad, None)
    assert not (plain[..., sg < 0] == lhs[..., sg < 0]).all()


# ----------------------------------------------------------------------------- stack driver


def test_forward_small_stack_matches_layerwise():
    wl = synth.get("alexnet", batch=2)
    rng = np.random.default_rng(0)
    # shrink to a cheap stack with the same structure: conv -> pool -> conv -> acc conv
    L = [synth.Conv("c1", 8, 16, 3, 1, 1, 9, 9, 9, 9, -1),
         synth.Pool("p1", 16, 3, 2, 0, 9, 9, 4, 4, 0),
         synth.Conv("c2", 16, 8, 3, 1, 1, 4, 4, 4, 4, 1, "both"),
         synth.Conv("c3", 8, 12, 4, 1, 0, 4, 4, 1, 1, 2, "acc")]
    wl = synth.Workload("tiny", 9, 3, 9, 9, 8, L)
    params = [synth.draw_conv_params(rng, l) if l.kind == "conv" else None for l in L]
    x = synth.draw_codes(rng, (3, 9, 9, 8))
    out = O.forward(wl, x, params)
    A0 = O.conv_acc(x, params[0].w, 1, 1)
    T0, s0 = O.fold(O.Params.from_synth(params[0]), 72)
    c0 = O.int_chain(A0, T0, s0)
    assert (out[0] == c0).all()
    p1 = O.maxpool_codes(c0, 3, 2, 0, s0)
    assert (out[1] == p1).all()
    A2 = O.conv_acc(p1, params[2].w, 1, 1)
    assert (out[2]["acc"] == A2).all()
    T2, s2 = O.fold(O.Params.from_synth(params[2]), 144)
    assert (out[2]["codes"] == O.int_chain(A2, T2, s2)).all()
    assert (out[3] == O.conv_acc(out[2]["codes"], params[3].w, 1, 0)).all()
    sub = O.forward(wl, x, params, images=[2])
    assert (sub[3] == out[3][2:3]).all()


# ----------------------------------------------------------------------------- formats


def test_code_and_sign_packing_formats():
    assert synth.pack_codes(np.array([1, 2, 3, 0], np.uint8)).tolist() == [0b00111001]
    rng = np.random.default_rng(1)
    c = rng.integers(0, 4, (3, 5, 7, 12), dtype=np.uint8)
    assert (synth.unpack_codes(synth.pack_codes(c)) == c).all()
    w = np.array([[1, -1, -1, 1] + [1] * 30], np.int8)
    words = synth.pack_signs(w)
    assert words.shape == (1, 2)
    assert int(words[0, 0]) == (0b1001 | (((1 << 28) - 1) << 4)) and int(words[0, 1]) == 0b11
    W = np.where(rng.integers(0, 2, (5, 3, 3, 20)) == 1, 1, -1).astype(np.int8)
    assert (synth.unpack_signs(synth.pack_signs(W), 180) == W.reshape(5, -1)).all()


# ---------------------------------------------------------------- separated conversion (Sec. 2.2)

def _sep_params(alpha, gamma, beta, mean, var, eps=0.0):
    c = len(alpha)
    return O.Params(np.array(alpha, float), np.array(gamma, float), np.array(beta, float), np.array(mean, float),
                    np.array(var, float), None, 0.5, 0.5, -0.25, eps)


def test_separated_equals_float_when_every_constant_is_exact():
    """alpha = 3/4, delta = 1/2, mean = 1/4, sigma = 1, beta = 0 and the levels 1/4, 3/4, 5/4 are all
    multiples of 1/16, so at Q = 16 no floor loses anything: the separated chain reproduces the float
    chain for every achievable accumulator."""
    p = _sep_params([0.75, 0.75], [1.0, -1.0], [0.0, 0.0], [0.25, 0.25], [1.0, 1.0])
    K = 64
    A = np.arange(-3 * K, 3 * K + 1, dtype=np.int32)[:, None].repeat(2, 1)
    fc = O.float_chain(A, p)
    assert (O.separated_chain(A, p, 4) == fc).all()


def test_separated_hand_case_floor_loss():
    """alpha = 0.3 at Q = 4 (m = 2): floor(1.2) = 1, so the separated conv scale is 1*2/16 = 0.125
    per unit of A instead of 0.3*0.5 = 0.15 (delta 0.5 -> d = 2; sigma = 1 -> 4; mean = beta = 0;
    levels 0.25/0.75/1.25 -> 1/3/5 quarters).  Float: z = 0.15 A; separated: Y = 0.125 A, and the
    strict comparisons give, for A = 0..10,
      float      0 0 1 1 1 1 2 2 2 3 3
      separated  0 0 0 1 1 1 1 2 2 2 2   (A = 2: 0.25 is not above 0.25; A = 10: 1.25 not above 1.25)"""
    p = _sep_params([0.3], [1.0], [0.0], [0.0], [1.0])
    A = np.arange(0, 11, dtype=np.int32)[:, None]
    fc = O.float_chain(A, p)
    assert fc[:, 0].tolist() == [0, 0, 1, 1, 1, 1, 2, 2, 2, 3, 3]
    assert O.separated_chain(A, p, 2)[:, 0].tolist() == [0, 0, 0, 1, 1, 1, 1, 2, 2, 2, 2]


def test_separated_converges_and_is_monotone():
    """Calibrated parameters: at m = 20 the separated codes equal the float chain's except within
    rounding distance of a level; at every m the codes are monotone in A (non-decreasing for a
    positive BN scale, non-increasing for a negative one)."""
    rng = np.random.default_rng(7)
    layer = synth.Conv("x", 64, 48, 3, 1, 1, 8, 8, 8, 8, -1)
    cp = synth.draw_conv_params_calibrated(rng, layer)
    cp.gamma[::5] *= -1
    p = O.Params.from_synth(cp)
    K = 576
    A = np.arange(-3 * K, 3 * K + 1, dtype=np.int32)[:, None].repeat(48, 1)
    fc, gap = O.float_chain(A, p, return_gap=True)
    s20 = O.separated_chain(A, p, 20)
    assert ((s20 != fc) <= (gap < 1e-4)).all()
    for m in (4, 8, 12):
        sc = O.separated_chain(A, p, m).astype(int)
        d = np.diff(sc, axis=0)
        up = p.gamma > 0
        assert (d[:, up] >= 0).all() and (d[:, ~up] <= 0).all()


# ----------------------------------------------------------------------------- non-quantized ends

def test_fixed_output_hand_case():
    """Separated fixed-point output (Sec. 2.2) by hand: alpha = 0.3, delta = 0.5, b = 0.1 at m = 4
    (Q = 16): a = floor(4.8) = 4, d = floor(8) = 8, bq = floor(25.6) = 25, y = floor((32 A + 25)/16):
    A = 10 -> floor(345/16) = 21; A = -3 -> floor(-71/16) = -5; A = 0 -> floor(25/16) = 1."""
    p = O.Params([0.3], [1.0], [0.0], [0.0], [1.0], [0.1], 0.5, 0.5, -0.25, 0.0)
    A = np.array([[10], [-3], [0]], np.int32)
    assert O.fixed_output(A, p, 4).ravel().tolist() == [21, -5, 1]


@pytest.mark.parametrize("m", [8, 14, 20])
def test_fixed_output_within_the_floor_error_of_the_float_value(m):
    """|y/Q - (alpha delta A + b)| is bounded by the three floors and the final one:
    (|A| (alpha + delta) Q + |A| + 1) / Q^2 + 1/Q, and the bound shrinks as 2^-m."""
    rng = np.random.default_rng(m)
    cout, Q = 30, 2.0 ** m
    p = O.Params(rng.uniform(0.01, 1.5, cout), np.ones(cout), np.zeros(cout), np.zeros(cout), np.ones(cout),
                 rng.normal(0, 1, cout), 0.5, 0.5, -0.25, 0.0)
    amax = min(3000, int(0.5 * 2.0 ** 31 / Q / 0.8))    # |alpha delta A + b| stays inside int32 / Q
    A = rng.integers(-amax, amax, (500, cout)).astype(np.int32)
    y = O.fixed_output(A, p, m).astype(np.float64) / Q
    ref = p.alpha * p.delta_in * A + p.bias
    bound = (np.abs(A) * (p.alpha + p.delta_in) * Q + np.abs(A) + 1) / Q ** 2 + 1 / Q
    assert (np.abs(y - ref) <= bound + 1e-12).all()
    assert np.abs(y - ref).max() < 4000 * 2.0 ** -m * 2
    # beyond the int32 range the output saturates
    big = np.full((1, cout), 2 ** 30, np.int32)
    assert (O.fixed_output(big, p, 24) == np.iinfo(np.int32).max).all()
    assert (O.fixed_output(-big, p, 24) == np.iinfo(np.int32).min).all()


def test_conv_on_8bit_values_matches_torch():
    """The integer core of the first (image) layer: 8-bit input values, +-1 filters."""
    rng = np.random.default_rng(8)
    x = rng.integers(0, 256, (2, 11, 9, 4), dtype=np.uint8)
    w = np.where(rng.integers(0, 2, (8, 3, 3, 4)) == 1, 1, -1).astype(np.int8)
    A = O.conv_acc(x, w, 1, 1)
    ref = F.conv2d(torch.from_numpy(x.astype(np.float64)).permute(0, 3, 1, 2),
                   torch.from_numpy(w.astype(np.float64)).permute(0, 3, 1, 2), padding=1).permute(0, 2, 3, 1)
    assert (A == ref.numpy().astype(np.int64)).all()
    assert np.abs(A).max() > 3 * 36          # beyond any 2-bit input's range


def test_fold_for_8bit_input_covers_the_whole_range():
    """A first layer on pixels (step 1/255): with K_fold = ceil(255 K / 3) the fold's clamp covers
    every |A| <= 255 K, and the integer chain equals the float chain on all of them."""
    rng = np.random.default_rng(255)
    layer = synth.Conv("c1", 4, 8, 3, 1, 1, 8, 8, 8, 8, -1, in_bits=8)
    K = 36
    assert O.fold_k(layer) == -(-255 * K // 3)
    p = _random_params(rng, 24)
    p.delta_in = 1.0 / 255.0
    p.alpha = p.alpha * (4.0 / np.sqrt(K)) * 20.0
    amax = 255 * K
    A = np.repeat(np.arange(-amax, amax + 1, dtype=np.int32)[:, None], p.cout, axis=1)
    T, s = O.fold(p, O.fold_k(layer))
    codes, ties = O.check_chains(A, p, T, s)
    assert ties == 0 and codes.min() == 0 and codes.max() == 3


@pytest.mark.parametrize("h,k,s,p,want", [
    (227, 11, 4, 0, 55),   # AlexNet conv1
    (56, 3, 2, 1, 28),     # a ResNet stride-2 3x3
    (56, 1, 2, 0, 28),     # its 1x1 shortcut
    (13, 3, 1, 1, 13),     # AlexNet conv3-5 ("same" 3x3)
    (27, 5, 1, 2, 27),     # AlexNet conv2
    (7, 3, 1, 0, 5),       # no padding
])
def test_conv_out_known_shapes(h, k, s, p, want):
    """Output size floor((h + 2p - k) / s) + 1 on the shapes of well-known networks."""
    assert O.conv_out(h, k, s, p) == want


@pytest.mark.parametrize("h,k,s,p,want", [
    (55, 3, 2, 0, 27),     # AlexNet pool1 (overlapping 3x3 / 2)
    (27, 3, 2, 0, 13),     # pool2
    (13, 3, 2, 0, 6),      # pool5
    (416, 2, 2, 0, 208),   # Tiny-YOLO 2x2 / 2
    (13, 2, 1, 1, 13),     # Tiny-YOLO's last pool: 2x2 / 1 with one padded cell at the right and bottom
])
def test_pool_out_known_shapes(h, k, s, p, want):
    """Pool output size with `p` padded cells at the bottom / right only (Darknet's 2x2 / 1 pool keeps
    13 x 13)."""
    assert O.pool_out(h, k, s, p) == want
