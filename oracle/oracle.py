"""Python face of the CPU oracle (``ifq_oracle.c``) for the IFQ-Net quantized substructure.

TEST INFRASTRUCTURE ONLY.  The test suite, the package smoke test and the
benchmark's CPU-baseline / reference leg are the only callers.  Nothing here
is shared with, or called by, the CUDA library, and it never calls the CUDA
library.

Each function is a thin ctypes call into the plain C oracle, which follows the
paper's equations in double precision (see the header of ``ifq_oracle.c``).
``forward`` runs a layer stack image by image, computing for every conv both
the float chain (Eq. (1)-(3)) and the integer chain on folded thresholds
(Eq. (7) + floor, Sec. 3.2), and checks that they agree (the claim of
Sec. 4.1.1 that integrated conversion gives identical outputs).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from concurrent.futures import ThreadPoolExecutor
from typing import Dict, List, Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ifq_oracle.c")
_LIB = os.path.join(_HERE, "_build", "liboracle.so")
_lock = threading.Lock()
_lib = None

# The oracle is compiled without FP contraction so that every double operation
# is rounded exactly as written.
CFLAGS = ["-O2", "-std=c99", "-fPIC", "-shared", "-ffp-contract=off", "-fno-fast-math"]


def build(force: bool = False) -> str:
    """Compile ifq_oracle.c into _build/liboracle.so (gcc); returns the path."""
    os.makedirs(os.path.dirname(_LIB), exist_ok=True)
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".{os.getpid()}.tmp"
        subprocess.check_call(["gcc", *CFLAGS, _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def lib():
    global _lib
    with _lock:
        if _lib is None:
            L = ctypes.CDLL(build())
            P = ctypes.c_void_p
            i, l, d = ctypes.c_int, ctypes.c_long, ctypes.c_double
            L.ifqo_float_chain.argtypes = [l, i, P, i, P, d, P, P, P, P, P, d, d, d, P, P]
            L.ifqo_fold.argtypes = [i, l, i, P, d, P, P, P, P, P, d, d, d, P, P]
            L.ifqo_int_chain.argtypes = [l, i, P, i, P, P, P]
            L.ifqo_conv_acc.argtypes = [i, i, i, i, i, i, i, i, i, P, P, P]
            L.ifqo_maxpool_acc.argtypes = [i, i, i, i, i, i, i, P, P]
            L.ifqo_maxpool_codes.argtypes = [i, i, i, i, i, i, i, P, P, P]
            L.ifqo_separated_chain.argtypes = [l, i, P, i, i, P, d, P, P, P, P, P, d, d, d, P]
            L.ifqo_fixed_output.argtypes = [l, i, P, i, P, d, P, P]
            for f in ("ifqo_float_chain", "ifqo_fold", "ifqo_int_chain", "ifqo_conv_acc",
                      "ifqo_maxpool_acc", "ifqo_maxpool_codes", "ifqo_separated_chain"):
                getattr(L, f).restype = ctypes.c_int
            _lib = L
    return _lib


def _p(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _f64(a) -> Optional[np.ndarray]:
    return None if a is None else np.ascontiguousarray(a, dtype=np.float64)


def _check(rc: int, what: str):
    if rc != 0:
        raise ValueError(f"oracle {what}: invalid arguments (rc={rc})")


class Params:
    """Per-channel float parameters of one quantized substructure (double precision)."""

    def __init__(self, alpha, gamma, beta, mean, var, bias=None, delta_in=0.5, q_base=0.5, q_offset=-0.25,
                 eps=1e-5, kbits=2):
        self.alpha, self.gamma, self.beta = _f64(alpha), _f64(gamma), _f64(beta)
        self.mean, self.var, self.bias = _f64(mean), _f64(var), _f64(bias)
        self.delta_in, self.q_base, self.q_offset, self.eps = float(delta_in), float(q_base), float(q_offset), float(eps)
        self.kbits = int(kbits)

    @property
    def levels(self) -> int:
        return (1 << self.kbits) - 1

    @property
    def cout(self) -> int:
        return self.alpha.shape[0]

    @classmethod
    def from_synth(cls, cp, kbits=2):
        return cls(cp.alpha, cp.gamma, cp.beta, cp.mean, cp.var, cp.bias, cp.delta_in, cp.q_base, cp.q_offset,
                   cp.eps, kbits)


def float_chain(A: np.ndarray, p: Params, return_gap: bool = False):
    """Codes of Eq. (1)-(3) for accumulators A [..., cout]; optionally min |z - thr_i|."""
    A2 = np.ascontiguousarray(A, dtype=np.int32).reshape(-1, p.cout)
    codes = np.empty(A2.shape, dtype=np.uint8)
    gap = np.empty(A2.shape, dtype=np.float64) if return_gap else None
    rc = lib().ifqo_float_chain(A2.shape[0], p.cout, _p(A2), p.levels, _p(p.alpha), p.delta_in, _p(p.bias),
                                _p(p.gamma), _p(p.beta), _p(p.mean), _p(p.var), p.eps, p.q_base, p.q_offset,
                                _p(codes), _p(gap))
    _check(rc, "float_chain")
    codes = codes.reshape(A.shape)
    return (codes, gap.reshape(A.shape)) if return_gap else codes


def fold(p: Params, K: int):
    """Eq. (7) thresholds with the floor of Sec. 3.2: (T [cout][L] int32, sign [cout] int8)."""
    T = np.empty((p.cout, p.levels), dtype=np.int32)
    s = np.empty(p.cout, dtype=np.int8)
    rc = lib().ifqo_fold(p.cout, int(K), p.levels, _p(p.alpha), p.delta_in, _p(p.bias), _p(p.gamma), _p(p.beta),
                         _p(p.mean), _p(p.var), p.eps, p.q_base, p.q_offset, _p(T), _p(s))
    _check(rc, "fold")
    return T, s


def int_chain(A: np.ndarray, T: np.ndarray, sign: np.ndarray) -> np.ndarray:
    """Codes of Eq. (7)/(8) on integer accumulators A [..., cout]."""
    cout, L = T.shape
    A2 = np.ascontiguousarray(A, dtype=np.int32).reshape(-1, cout)
    T2 = np.ascontiguousarray(T, dtype=np.int32)
    s2 = np.ascontiguousarray(sign, dtype=np.int8)
    codes = np.empty(A2.shape, dtype=np.uint8)
    _check(lib().ifqo_int_chain(A2.shape[0], cout, _p(A2), L, _p(T2), _p(s2), _p(codes)), "int_chain")
    return codes.reshape(A.shape)


def conv_out(h: int, k: int, stride: int, pad: int) -> int:
    return (h + 2 * pad - k) // stride + 1


def separated_chain(A: np.ndarray, p: "Params", m: int) -> np.ndarray:
    """Codes of the separated fixed-point conversion (Sec. 2.2) at Q_m = 2^m, exact integers."""
    cout = p.alpha.shape[0]
    A2 = np.ascontiguousarray(A, dtype=np.int32).reshape(-1, cout)
    codes = np.empty(A2.shape, dtype=np.uint8)
    _check(lib().ifqo_separated_chain(A2.shape[0], cout, _p(A2), p.levels, m, _p(p.alpha), p.delta_in,
                                      _p(p.bias) if p.bias is not None else None, _p(p.gamma), _p(p.beta),
                                      _p(p.mean), _p(p.var), p.eps, p.q_base, p.q_offset, _p(codes)),
           "separated_chain")
    return codes.reshape(A.shape)


def fixed_output(A: np.ndarray, p: "Params", m: int) -> np.ndarray:
    """Separated fixed-point output of a non-quantized substructure (Sec. 2.2) at Q_m = 2^m:
    floor((floor(alpha Q) floor(delta Q) A + floor(b Q^2)) / Q), int32 of A's shape."""
    cout = p.alpha.shape[0]
    A2 = np.ascontiguousarray(A, dtype=np.int32).reshape(-1, cout)
    out = np.empty(A2.shape, dtype=np.int32)
    _check(lib().ifqo_fixed_output(A2.shape[0], cout, _p(A2), m, _p(p.alpha), p.delta_in,
                                   _p(p.bias) if p.bias is not None else None, _p(out)), "fixed_output")
    return out.reshape(A.shape)


def fold_k(layer) -> int:
    """K of a layer's fold: its kh*kw*cin, or for a layer on 8-bit input values the K whose
    clamp range L*K covers every accumulator |A| <= 255*K (L = 3 for 2-bit output codes)."""
    K = layer.k * layer.k * layer.cin
    return -(-255 * K // 3) if getattr(layer, "in_bits", 0) == 8 else K


def conv_acc(x: np.ndarray, w: np.ndarray, stride: int, pad: int) -> np.ndarray:
    """Integer core of Eq. (1): x uint8 codes [B][H][W][C], w int8 +-1 [cout][kh][kw][C] -> int32 NHWC."""
    x = np.ascontiguousarray(x, dtype=np.uint8)
    w = np.ascontiguousarray(w, dtype=np.int8)
    B, H, W, C = x.shape
    cout, kh, kw, cin = w.shape
    assert cin == C
    ho, wo = conv_out(H, kh, stride, pad), conv_out(W, kw, stride, pad)
    A = np.empty((B, ho, wo, cout), dtype=np.int32)
    _check(lib().ifqo_conv_acc(B, H, W, C, cout, kh, kw, stride, pad, _p(x), _p(w), _p(A)), "conv_acc")
    return A


def pool_out(h: int, k: int, stride: int, pad: int) -> int:
    return (h + pad - k) // stride + 1


def maxpool_acc(A: np.ndarray, k: int, stride: int, pad: int) -> np.ndarray:
    """Max pooling on Y^conv (Sec. 2.1), int32 NHWC; `pad` empty cells at bottom/right."""
    A = np.ascontiguousarray(A, dtype=np.int32)
    B, H, W, C = A.shape
    out = np.empty((B, pool_out(H, k, stride, pad), pool_out(W, k, stride, pad), C), dtype=np.int32)
    _check(lib().ifqo_maxpool_acc(B, H, W, C, k, stride, pad, _p(A), _p(out)), "maxpool_acc")
    return out


def maxpool_codes(x: np.ndarray, k: int, stride: int, pad: int, sign: Optional[np.ndarray] = None) -> np.ndarray:
    """Pooling on codes: plain max (sign None) or per-channel max/min by sign."""
    x = np.ascontiguousarray(x, dtype=np.uint8)
    B, H, W, C = x.shape
    s = None if sign is None else np.ascontiguousarray(sign, dtype=np.int8)
    out = np.empty((B, pool_out(H, k, stride, pad), pool_out(W, k, stride, pad), C), dtype=np.uint8)
    _check(lib().ifqo_maxpool_codes(B, H, W, C, k, stride, pad, _p(x), _p(s), _p(out)), "maxpool_codes")
    return out


class ChainMismatch(AssertionError):
    pass


def check_chains(A: np.ndarray, p: Params, T: np.ndarray, sign: np.ndarray, tie_tol: float = 1e-9):
    """Integer-chain codes, after checking them against the float chain.

    Elements where the two differ are accepted only at a rounding tie of the
    float chain (min_i |z - thr_i| <= tie_tol * (1 + max|thr|)); there the
    integer chain with the floor of Sec. 3.2 is the paper's result.  Returns
    (codes, number of accepted ties)."""
    ci = int_chain(A, T, sign)
    cf, gap = float_chain(A, p, return_gap=True)
    diff = ci != cf
    if diff.any():
        scale = 1.0 + max(abs(p.q_offset + p.q_base), abs(p.q_offset + p.levels * p.q_base))
        bad = diff & (gap > tie_tol * scale)
        if bad.any():
            idx = np.argwhere(bad)[:5]
            raise ChainMismatch(f"float and integer chains differ away from ties at {idx.tolist()}")
    return ci, int(diff.sum())


def forward(workload, x: np.ndarray, params: Sequence, images: Optional[Sequence[int]] = None,
            threads: Optional[int] = None, check_float: bool = True) -> Dict[int, np.ndarray]:
    """Run a layer stack on the oracle for the given images.

    Returns {layer index: output} where output is uint8 codes [b][ho][wo][c]
    for code layers and pools, int32 accumulators for "acc" layers, and for
    "both" layers a dict {"codes": ..., "acc": ...}.  Images are independent,
    so they run on a thread pool (ctypes releases the GIL).
    """
    idx = list(range(x.shape[0])) if images is None else list(images)
    kbits = getattr(workload, "kbits", 2)   # code width of every quantized layer (Eq. (8): 2^k - 1 thresholds)
    folded = {}
    for li, layer in enumerate(workload.layers):
        if layer.kind == "conv":
            p = Params.from_synth(params[li], kbits)
            kf = fold_k(layer) if kbits == 2 else layer.k * layer.k * layer.cin
            folded[li] = (p, *fold(p, kf))

    def one(b):
        outs = {}
        for li, layer in enumerate(workload.layers):
            src = x[b:b + 1] if layer.src < 0 else outs[layer.src]
            if isinstance(src, dict):
                src = src["codes"]
            if layer.kind == "conv":
                p, T, s = folded[li]
                A = conv_acc(src, params[li].w, layer.stride, layer.pad)
                if getattr(layer, "pool", 0) > 1:   # pool on Y^conv, before BN and the quantizer (Sec. 2.1)
                    A = maxpool_acc(A, layer.pool, layer.pool, 0)
                if check_float:
                    codes, _ = check_chains(A, p, T, s)
                else:
                    codes = int_chain(A, T, s)
                outs[li] = {"codes": codes, "acc": A} if layer.out == "both" else (A if layer.out == "acc" else codes)
            elif layer.kind == "fixed":   # the separated fixed-point output of a conv's accumulators
                acc = outs[layer.src]["acc"] if isinstance(outs[layer.src], dict) else outs[layer.src]
                outs[li] = fixed_output(acc, folded[layer.src][0], layer.m)
            else:
                sgn = folded[layer.src][2] if layer.signed else None
                outs[li] = maxpool_codes(src, layer.k, layer.stride, layer.pad, sgn)
        return outs

    nthreads = threads or max(1, min(len(idx), len(os.sched_getaffinity(0))))
    with ThreadPoolExecutor(nthreads) as ex:
        per = list(ex.map(one, idx))
    result = {}
    for li, layer in enumerate(workload.layers):
        if layer.kind == "conv" and layer.out == "both":
            result[li] = {k: np.concatenate([o[li][k] for o in per]) for k in ("codes", "acc")}
        else:
            result[li] = np.concatenate([o[li] for o in per])
    return result
