"""Seeded synthetic inputs and data formats shared by the CUDA path's callers and the oracle.

This module holds no arithmetic of the method (no convolution, no folding, no
thresholding).  It provides:

* the layer tables of the benchmark workloads, written out with literal shapes;
* seeded draws of k-bit input codes, +-1 filters and the float parameters that
  the integrated conversion folds (alpha, BN, quantizer step);
* the packed storage formats:
    - k-bit codes, NHWC, in f-bit fields along C (f = 2 for k = 2, f = 4 for
      k = 3 and 4), channel c in bits f*(c%(8/f)).. of byte c//(8/f);
    - sign bits of +-1 filters, one row per output channel over K = kh*kw*cin
      in (dy, dx, c) order, bit k%32 of 32-bit word k//32 set for +1, rows
      padded to whole words.

Shapes stand in for the paper's workloads: AlexNet conv2..FC7 (Table 1,
Sec. 4.1; the k = 3 and 4 networks of Table 2 as alexnet_k3 / alexnet_k4),
Tiny-YOLO / Tinier-YOLO backbones (Sec. 4.2) and a ResNet-18 stack; the
datasets and trained weights are not used.  Distributions: codes uniform on
{0..2^k-1}, weights uniform +-1, alpha ~ U(0.5, 1.5), gamma ~ N(1, 0.3),
beta ~ N(0, 0.5), mean ~ N(0, 2), var ~ U(0.5, 2), quantizer step 0.5,
bias 0, eps 1e-5, seed 1911_08076 + config index.  For the separated-conversion
study, draw_conv_params_calibrated gives trained-layer ranges instead (small
alpha, BN statistics matched to the layer's pre-BN spread).
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Dict, List, Optional

import numpy as np

SEED_BASE = 1911_08076
STEP = 0.5          # quantizer step of every layer (the paper's beta / beta')
EPS = float(np.float32(1e-5))   # BN epsilon as the float32 the C ABI receives


@dataclass
class Conv:
    """One quantized convolution (a quantized substructure, Sec. 3.1).

    `src` is the index of the layer whose output codes feed this one (-1 for
    the stack input).  `out` is "codes", "acc" (int32 accumulators, for a
    layer whose substructure is not quantized) or "both".  `pool` = p >= 2
    max-pools the accumulators over p x p windows with stride p before the
    thresholds (Sec. 2.1), so the codes are [b][ho/p][wo/p][cout].
    """
    name: str
    cin: int
    cout: int
    k: int
    stride: int
    pad: int
    h: int
    w: int
    ho: int
    wo: int
    src: int
    out: str = "codes"
    pool: int = 0
    in_bits: int = 0    # 8: the layer reads 8-bit input values (image pixels), not codes
    kind: str = field(default="conv", init=False)

    @property
    def out_h(self) -> int:
        return self.ho // self.pool if self.pool > 1 else self.ho

    @property
    def out_w(self) -> int:
        return self.wo // self.pool if self.pool > 1 else self.wo


@dataclass
class Pool:
    """Max pooling on the codes of layer `src`, with that layer's channel signs
    (`signed`) or as a plain max.  `pad` extra cells at bottom/right."""
    name: str
    c: int
    k: int
    stride: int
    pad: int
    h: int
    w: int
    ho: int
    wo: int
    src: int
    signed: bool = True
    kind: str = field(default="pool", init=False)


@dataclass
class Fixed:
    """Separated fixed-point output (Sec. 2.2, Q_m = 2^m) of the int32 accumulators of conv
    layer `src`: the non-quantized last substructure of a network (a YOLO detection conv)."""
    name: str
    src: int
    m: int
    kind: str = field(default="fixed", init=False)


@dataclass
class Workload:
    name: str
    index: int
    batch: int
    h: int
    w: int
    c: int
    layers: list
    kbits: int = 2      # code width k of every quantized layer's input and output codes
    in_bits: int = 0    # 8: the stack input is 8-bit values (an image), read by the first conv

    @property
    def seed(self) -> int:
        return SEED_BASE + self.index


def _c3(name, cin, cout, h, ho, src, stride=1, out="codes"):
    return Conv(name, cin, cout, 3, stride, 1, h, h, ho, ho, src, out)


def _c1(name, cin, cout, h, ho, src, stride=1, out="codes"):
    return Conv(name, cin, cout, 1, stride, 0, h, h, ho, ho, src, out)


def pr1() -> Workload:
    """Single 3x3 64->64 layer on a 16x16 map, batch 1, codes and accumulators out."""
    return Workload("pr1_conv3x3_64_16x16_b1", 0, 1, 16, 16, 64, [_c3("conv", 64, 64, 16, 16, -1, out="both")])


def resnet18(batch: int = 32) -> Workload:
    """ResNet-18 body: 16 3x3 convs and 3 1x1 stride-2 shortcuts (first conv and FC excluded).
    Each conv's codes feed the next conv; shortcut codes are produced, not added."""
    L = []
    L += [_c3("s1.b1.a", 64, 64, 56, 56, -1), _c3("s1.b1.b", 64, 64, 56, 56, 0),
          _c3("s1.b2.a", 64, 64, 56, 56, 1), _c3("s1.b2.b", 64, 64, 56, 56, 2)]
    prev = 3
    for cin, cout, h, ho in ((64, 128, 56, 28), (128, 256, 28, 14), (256, 512, 14, 7)):
        s = len(L)
        L += [_c3(f"c{cout}.b1.a", cin, cout, h, ho, prev, stride=2),
              _c1(f"c{cout}.b1.sc", cin, cout, h, ho, prev, stride=2),
              _c3(f"c{cout}.b1.b", cout, cout, ho, ho, s),
              _c3(f"c{cout}.b2.a", cout, cout, ho, ho, s + 2),
              _c3(f"c{cout}.b2.b", cout, cout, ho, ho, s + 3)]
        prev = s + 4
    return Workload(f"resnet18_body_b{batch}", 1, batch, 56, 56, 64, L)


def alexnet(batch: int = 128) -> Workload:
    """AlexNet conv2..FC7 (Table 1 substructures 2-6 plus FC7 of substructure 7, int32 out)."""
    L = [Conv("conv2", 96, 256, 5, 1, 2, 27, 27, 27, 27, -1),
         Pool("pool2", 256, 3, 2, 0, 27, 27, 13, 13, 0),
         _c3("conv3", 256, 384, 13, 13, 1),
         _c3("conv4", 384, 384, 13, 13, 2),
         _c3("conv5", 384, 256, 13, 13, 3),
         Pool("pool5", 256, 3, 2, 0, 13, 13, 6, 6, 4),
         Conv("fc6", 256, 4096, 6, 1, 0, 6, 6, 1, 1, 5),
         _c1("fc7", 4096, 4096, 1, 1, 6, out="acc")]
    return Workload(f"alexnet_conv2_fc7_b{batch}", 2, batch, 27, 27, 96, L)


def tiny_yolo(batch: int = 64, tinier: bool = False) -> Workload:
    """Tiny-YOLO backbone at 416 (first conv and its pool excluded: input is 208x208x16),
    2x2 pools on codes, 1x1 detection conv to 30 channels with int32 out.  The Tinier
    variant halves every width and makes the third-to-last conv 1x1 (Sec. 4.2)."""
    d = 2 if tinier else 1
    ch = [16 // d, 32 // d, 64 // d, 128 // d, 256 // d, 512 // d, 1024 // d, 1024 // d]
    L, h, src = [], 208, -1
    for i in range(4):                      # 208 -> 104 -> 52 -> 26 -> 13
        L.append(_c3(f"conv{i + 2}", ch[i], ch[i + 1], h, h, src))
        L.append(Pool(f"pool{i + 2}", ch[i + 1], 2, 2, 0, h, h, h // 2, h // 2, len(L) - 1))
        h //= 2
        src = len(L) - 1
    L.append(_c3("conv6", ch[4], ch[5], 13, 13, src))
    L.append(Pool("pool6", ch[5], 2, 1, 1, 13, 13, 13, 13, len(L) - 1))
    mk = _c1 if tinier else _c3             # Tinier: third-to-last conv is 1x1
    L.append(mk("conv7", ch[5], ch[6], 13, 13, len(L) - 1))
    L.append(_c3("conv8", ch[6], ch[7], 13, 13, len(L) - 1))
    L.append(_c1("det", ch[7], 30, 13, 13, len(L) - 1, out="acc"))
    name = ("tinier" if tinier else "tiny") + f"_yolo416_b{batch}"
    return Workload(name, 3, batch, 208, 208, ch[0], L)


def tinier_yolo_full(batch: int = 64) -> Workload:
    """IFQ-Tinier-YOLO end to end at 416 (Sec. 4.2): every conv binarized, the first one on the
    8-bit RGB image (padded to 4 channels, pixel step 1/255, the integrated conversion to 2-bit
    codes), the Tinier backbone, and the 1x1 detection conv (a non-quantized substructure) as
    int32 accumulators converted to fixed point by the separated method at m = 14."""
    body = tiny_yolo(batch, True)
    L = [Conv("conv1", 4, 8, 3, 1, 1, 416, 416, 416, 416, -1, in_bits=8),
         Pool("pool1", 8, 2, 2, 0, 416, 416, 208, 208, 0)]
    for l in body.layers:
        src = l.src + 2 if l.src >= 0 else 1
        if l.kind == "conv":
            L.append(Conv(l.name, l.cin, l.cout, l.k, l.stride, l.pad, l.h, l.w, l.ho, l.wo, src, l.out, l.pool))
        else:
            L.append(Pool(l.name, l.c, l.k, l.stride, l.pad, l.h, l.w, l.ho, l.wo, src, l.signed))
    L.append(Fixed("det_fixed", len(L) - 1, 14))
    return Workload(f"tinier_yolo_full416_b{batch}", 5, batch, 416, 416, 4, L, 2, 8)


def roofline(batch: int = 256, which: str = "3x3") -> Workload:
    """Large single layers: 3x3 256->256 at 56x56, or 1x1 512->512 at 28x28."""
    if which == "3x3":
        return Workload(f"roofline_conv3x3_256_56_b{batch}", 4, batch, 56, 56, 256,
                        [_c3("conv3x3", 256, 256, 56, 56, -1)])
    return Workload(f"roofline_conv1x1_512_28_b{batch}", 4, batch, 28, 28, 512,
                    [_c1("conv1x1", 512, 512, 28, 28, -1)])


def fuse_pools(wl: Workload) -> Workload:
    """The same stack with every convolution whose codes feed only a signed p x p / stride p pool
    (p in {2, 4}, no padding, sizes divisible by p) computing that pool itself (Sec. 2.1 order:
    pool on the accumulators, then BN and the quantizer).  Same index, so the same draws."""
    consumers = {}
    for i, l in enumerate(wl.layers):
        consumers.setdefault(l.src, []).append(i)
    fused_into = {}   # conv index -> pool index merged into it
    for i, l in enumerate(wl.layers):
        if l.kind != "pool" or l.src < 0:
            continue
        c = wl.layers[l.src]
        if (c.kind == "conv" and c.out == "codes" and c.pool <= 1 and l.signed and l.pad == 0 and
                l.k == l.stride and l.k in (2, 4) and c.ho % l.k == 0 and c.wo % l.k == 0 and
                consumers.get(l.src) == [i]):
            fused_into[l.src] = i
    dropped = set(fused_into.values())
    new_index, layers = {}, []
    for i, l in enumerate(wl.layers):
        if i in dropped:
            continue
        new_index[i] = len(layers)
        layers.append(l)
    for i in dropped:   # a dropped pool's consumers read the fused conv
        new_index[i] = new_index[wl.layers[i].src]
    out = []
    for i, l in enumerate(layers):
        src = -1 if l.src < 0 else new_index[l.src]
        if l.kind == "conv":
            old = [j for j, m in enumerate(wl.layers) if m is l][0]
            p = wl.layers[fused_into[old]].k if old in fused_into else l.pool
            out.append(Conv(l.name, l.cin, l.cout, l.k, l.stride, l.pad, l.h, l.w, l.ho, l.wo, src, l.out, p,
                            l.in_bits))
        elif l.kind == "fixed":
            out.append(Fixed(l.name, src, l.m))
        else:
            out.append(Pool(l.name, l.c, l.k, l.stride, l.pad, l.h, l.w, l.ho, l.wo, src, l.signed))
    return Workload(wl.name + "_fused", wl.index, wl.batch, wl.h, wl.w, wl.c, out, wl.kbits, wl.in_bits)


def with_kbits(wl: Workload, kbits: int) -> Workload:
    """The same stack with k-bit codes between layers (Table 2's k = 3, 4 columns; Eq. (8)).
    Same index, so the same filter and parameter draws."""
    return Workload(f"{wl.name}_k{kbits}", wl.index, wl.batch, wl.h, wl.w, wl.c, wl.layers, kbits, wl.in_bits)


WORKLOADS = {
    "pr1": pr1,
    "resnet18": resnet18,
    "alexnet": alexnet,
    "tinyyolo": lambda batch=64: tiny_yolo(batch, False),
    "tinieryolo": lambda batch=64: tiny_yolo(batch, True),
    "tinyyolo_fused": lambda batch=64: fuse_pools(tiny_yolo(batch, False)),
    "tinieryolo_fused": lambda batch=64: fuse_pools(tiny_yolo(batch, True)),
    "roofline3x3": lambda batch=256: roofline(batch, "3x3"),
    "roofline1x1": lambda batch=256: roofline(batch, "1x1"),
    "alexnet_k3": lambda batch=128: with_kbits(alexnet(batch), 3),
    "alexnet_k4": lambda batch=128: with_kbits(alexnet(batch), 4),
    "resnet18_k4": lambda batch=32: with_kbits(resnet18(batch), 4),
    "tinyyolo_fused_k4": lambda batch=64: with_kbits(fuse_pools(tiny_yolo(batch, False)), 4),
    "tinieryolo_full": tinier_yolo_full,
    "tinieryolo_full_fused": lambda batch=64: fuse_pools(tinier_yolo_full(batch)),
}


def get(name: str, batch: Optional[int] = None) -> Workload:
    f = WORKLOADS[name]
    return f() if batch is None else f(batch)


# ----------------------------------------------------------------------------- draws

@dataclass
class ConvParams:
    """Float parameters of one quantized substructure and its +-1 filter."""
    w: np.ndarray          # int8 [cout][k][k][cin], values +-1
    alpha: np.ndarray      # float32 [cout] > 0
    gamma: np.ndarray      # float32 [cout]
    beta: np.ndarray       # float32 [cout]
    mean: np.ndarray       # float32 [cout]
    var: np.ndarray        # float32 [cout] > 0
    bias: Optional[np.ndarray] = None
    delta_in: float = STEP
    q_base: float = STEP
    q_offset: float = -STEP / 2
    eps: float = EPS


def draw_conv_params(rng: np.random.Generator, layer: Conv) -> ConvParams:
    cout, k, cin = layer.cout, layer.k, layer.cin
    w = np.where(rng.integers(0, 2, size=(cout, k, k, cin), dtype=np.int8) == 1, 1, -1).astype(np.int8)
    alpha = rng.uniform(0.5, 1.5, cout).astype(np.float32)
    gamma = rng.normal(1.0, 0.3, cout).astype(np.float32)
    beta = rng.normal(0.0, 0.5, cout).astype(np.float32)
    mean = rng.normal(0.0, 2.0, cout).astype(np.float32)
    var = rng.uniform(0.5, 2.0, cout).astype(np.float32)
    return ConvParams(w, alpha, gamma, beta, mean, var)


def draw_conv_params_calibrated(rng: np.random.Generator, layer: Conv) -> ConvParams:
    """Parameters in the ranges of a trained HWGQ layer, for the separated-conversion study:
    small filter scales alpha ~ U(0.005, 0.05) (the paper's loss case is small alpha), and BN
    statistics of the layer's own pre-BN output y = alpha*STEP*A, whose spread for uniform codes
    and +-1 filters is alpha*STEP*sqrt(3.5 K): mean ~ N(0, 0.1 sd), var = sd^2 * U(0.8, 1.25),
    gamma ~ N(1, 0.3), beta ~ N(0, 0.5), so that the codes spread over every level."""
    cout, k, cin = layer.cout, layer.k, layer.cin
    w = np.where(rng.integers(0, 2, size=(cout, k, k, cin), dtype=np.int8) == 1, 1, -1).astype(np.int8)
    alpha = rng.uniform(0.005, 0.05, cout).astype(np.float32)
    sd = alpha.astype(np.float64) * STEP * np.sqrt(3.5 * k * k * cin)
    gamma = rng.normal(1.0, 0.3, cout).astype(np.float32)
    beta = rng.normal(0.0, 0.5, cout).astype(np.float32)
    mean = (rng.normal(0.0, 0.1, cout) * sd).astype(np.float32)
    var = (sd * sd * rng.uniform(0.8, 1.25, cout)).astype(np.float32)
    return ConvParams(w, alpha, gamma, beta, mean, var)


def draw_codes(rng: np.random.Generator, shape, kbits: int = 2) -> np.ndarray:
    return rng.integers(0, 1 << kbits, size=shape, dtype=np.uint8)


PIXEL_STEP = 1.0 / 255.0   # input step of a layer on 8-bit image values (pixels scaled to [0, 1])


NEG_GAMMA_SEED = 77   # offset of the generator that picks the channels whose BN scale is negated


def draw_workload(wl: Workload, batch: Optional[int] = None, neg_gamma: float = 0.0):
    """Input [B][H][W][C] (uint8: k-bit codes, or 8-bit pixels with a zero 4th channel for an image
    input) and per-layer ConvParams (None for pools and fixed-point outputs).

    neg_gamma > 0: after the standard draw, each channel's BN scale gamma is negated with that
    probability, picked by a second generator (seed + NEG_GAMMA_SEED), so every other value equals
    the standard draw's.  The configurations call for about 10 % of channels with a negative BN
    scale, which gamma ~ N(1, 0.3) alone gives only 0.04 % of the time."""
    rng = np.random.default_rng(wl.seed)
    params = [draw_conv_params(rng, l) if l.kind == "conv" else None for l in wl.layers]
    if neg_gamma > 0:
        flip = np.random.default_rng(wl.seed + NEG_GAMMA_SEED)
        for p in params:
            if p is not None:
                neg = flip.random(p.gamma.shape[0]) < neg_gamma
                p.gamma = np.where(neg, -np.abs(p.gamma), np.abs(p.gamma)).astype(np.float32)
    for l, p in zip(wl.layers, params):
        if l.kind == "conv" and l.in_bits == 8:
            p.delta_in = PIXEL_STEP
    b = wl.batch if batch is None else batch
    if wl.in_bits == 8:
        x = rng.integers(0, 256, size=(b, wl.h, wl.w, wl.c), dtype=np.uint8)
        x[..., 3:] = 0
    else:
        x = draw_codes(rng, (b, wl.h, wl.w, wl.c), wl.kbits)
    return x, params


# ----------------------------------------------------------------------------- formats

def field_bits(kbits: int) -> int:
    """Bits of the storage field of a k-bit code: 2 for k = 2, 4 for k = 3 and 4, 8 for 8-bit
    input values."""
    assert kbits in (2, 3, 4, 8), kbits
    return {2: 2, 3: 4, 4: 4, 8: 8}[kbits]


def pack_codes(codes: np.ndarray, kbits: int = 2) -> np.ndarray:
    """uint8 codes [..., C] (C % 4 == 0, values < 2^kbits) -> packed uint8 [..., C*f/8]."""
    f = field_bits(kbits)
    c = np.ascontiguousarray(codes, dtype=np.uint8)
    assert c.shape[-1] % 4 == 0
    if f == 8:
        return c.copy()
    assert c.size == 0 or int(c.max()) < (1 << kbits)
    per = 8 // f
    q = c.reshape(c.shape[:-1] + (c.shape[-1] // per, per))
    out = np.zeros(q.shape[:-1], dtype=np.uint8)
    for l in range(per):
        out |= (q[..., l] << (f * l)).astype(np.uint8)
    return out


def unpack_codes(packed: np.ndarray, c: Optional[int] = None, kbits: int = 2) -> np.ndarray:
    """packed uint8 [..., C*f/8] -> uint8 codes [..., C] (optionally cut to c channels)."""
    f = field_bits(kbits)
    per = 8 // f
    p = np.ascontiguousarray(packed, dtype=np.uint8)
    if f == 8:
        return p.copy() if c is None else p[..., :c].copy()
    out = np.stack([(p >> (f * l)) & ((1 << f) - 1) for l in range(per)], axis=-1)
    out = out.reshape(p.shape[:-1] + (p.shape[-1] * per,))
    return out if c is None else out[..., :c]


def sign_words_per_row(K: int) -> int:
    return (K + 31) // 32


def pack_signs(w: np.ndarray) -> np.ndarray:
    """int8 +-1 [cout][...] -> uint32 [cout][ceil(K/32)] sign bits (1 <-> +1), K in (dy, dx, c) order."""
    w2 = np.ascontiguousarray(w).reshape(w.shape[0], -1)
    cout, K = w2.shape
    nw = sign_words_per_row(K)
    bits = np.zeros((cout, nw * 32), dtype=np.uint64)
    bits[:, :K] = (w2 > 0)
    weights = (np.uint64(1) << np.arange(32, dtype=np.uint64))
    words = (bits.reshape(cout, nw, 32) * weights).sum(axis=-1)
    return words.astype(np.uint32)


def unpack_signs(words: np.ndarray, K: int) -> np.ndarray:
    """uint32 [cout][ceil(K/32)] -> int8 +-1 [cout][K]."""
    wd = np.ascontiguousarray(words, dtype=np.uint32)
    bits = (wd[:, :, None] >> np.arange(32, dtype=np.uint32)) & 1
    bits = bits.reshape(wd.shape[0], -1)[:, :K]
    return np.where(bits == 1, 1, -1).astype(np.int8)
