"""Thin Python binding of the C ABI in include/ifq.h (argument marshalling only).

Every function has the name of the C entry point it calls.  Device buffers are
torch CUDA tensors (or raw integer addresses); host buffers of the fold are
numpy arrays.  A non-zero status raises IfqError.  There is no fallback: if
libifq.so is missing or cannot be loaded, every call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading
from typing import Optional, Sequence

import numpy as np

from . import build as _build

_lock = threading.Lock()
_lib = None

IFQ_OK, IFQ_EINVAL, IFQ_ESHAPE, IFQ_EALIGN, IFQ_ERANGE, IFQ_ECUDA, IFQ_ETIMEOUT, IFQ_EUNSUPPORTED, IFQ_EWORKSPACE = range(9)
IFQ_OUT_CODES, IFQ_OUT_ACC, IFQ_OUT_BOTH = 1, 2, 3
IFQ_PATH_AUTO, IFQ_PATH_TC, IFQ_PATH_BITSERIAL, IFQ_PATH_DIRECT, IFQ_PATH_WIN, IFQ_PATH_WARP = 0, 1, 2, 3, 4, 5
IFQ_LAYER_CONV, IFQ_LAYER_POOL, IFQ_LAYER_FIXED = 1, 2, 3
IFQ_FORWARD_LAYERS, IFQ_FORWARD_PERSISTENT = 1, 2


class IfqError(RuntimeError):
    def __init__(self, status: int, what: str):
        super().__init__(f"{what}: {ifq_status_str(status)} (status {status})")
        self.status = status


class ConvDesc(ctypes.Structure):
    _fields_ = [(f, ctypes.c_int) for f in
                ("n", "h", "w", "cin", "cout", "kh", "kw", "stride", "pad", "out_mode", "path", "pool", "kbits",
                 "in_bits")]


class PoolDesc(ctypes.Structure):
    _fields_ = [(f, ctypes.c_int) for f in ("n", "h", "w", "c", "k", "stride", "pad", "kbits")]


class FixedDesc(ctypes.Structure):
    _fields_ = [("m", ctypes.c_int)]


class Layer(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int), ("src", ctypes.c_int), ("conv", ConvDesc), ("pool", PoolDesc),
                ("w_prep", ctypes.c_void_p), ("thr", ctypes.c_void_p), ("sign", ctypes.c_void_p),
                ("y_codes", ctypes.c_void_p), ("y_acc", ctypes.c_void_p), ("fixed", FixedDesc),
                ("fx_mul", ctypes.c_void_p), ("fx_add", ctypes.c_void_p)]


_P = ctypes.c_void_p
_I = ctypes.c_int
_SZ = ctypes.c_size_t
_F = ctypes.c_float

_SIGS = {
    "ifq_status_str": ([_I], ctypes.c_char_p),
    "ifq_version": ([], _I),
    "ifq_fold_layer": ([_I, _I, _I, _P, _F, _P, _P, _P, _P, _P, _F, _F, _F, _P, _P], _I),
    "ifq_fold_layer_separated": ([_I, _I, _I, _I, _P, _F, _P, _P, _P, _P, _P, _F, _F, _F, _P, _P], _I),
    "ifq_fold_output_separated": ([_I, _I, _P, _F, _P, _P, _P], _I),
    "ifq_fixed_output": ([_P, _I, _I, _P, _P, _I, _P, _P], _I),
    "ifq_codes_bytes": ([_I, _I, _I, _I, _I, ctypes.POINTER(_SZ)], _I),
    "ifq_codes_storage_bytes": ([_I, _I, _I, _I, _I, ctypes.POINTER(_SZ)], _I),
    "ifq_conv_out_shape": ([ctypes.POINTER(ConvDesc), ctypes.POINTER(_I), ctypes.POINTER(_I)], _I),
    "ifq_weights_prep_bytes": ([ctypes.POINTER(ConvDesc), ctypes.POINTER(_SZ)], _I),
    "ifq_pack_weights": ([ctypes.POINTER(ConvDesc), _P, _P, _P], _I),
    "ifq_conv_plan": ([ctypes.POINTER(ConvDesc), ctypes.POINTER(_I)], _I),
    "ifq_conv_workspace_bytes": ([ctypes.POINTER(ConvDesc), ctypes.POINTER(_SZ)], _I),
    "ifq_conv2bit": ([ctypes.POINTER(ConvDesc), _P, _P, _P, _P, _P, _P, _P, _SZ, _P], _I),
    "ifq_pool_out_shape": ([ctypes.POINTER(PoolDesc), ctypes.POINTER(_I), ctypes.POINTER(_I)], _I),
    "ifq_maxpool2bit": ([ctypes.POINTER(PoolDesc), _P, _P, _P, _P], _I),
    "ifq_forward_workspace_bytes": ([ctypes.POINTER(Layer), _I, ctypes.POINTER(_SZ)], _I),
    "ifq_forward": ([ctypes.POINTER(Layer), _I, _P, _P, _SZ, _P], _I),
    "ifq_forward_noalloc": ([ctypes.POINTER(Layer), _I, _P, _P], _I),
    "ifq_last_forward_mode": ([ctypes.POINTER(_I)], _I),
    "ifq_graph_create": ([ctypes.POINTER(Layer), _I, _P, _P, _SZ, _P, ctypes.POINTER(_P)], _I),
    "ifq_graph_create_io": ([ctypes.POINTER(Layer), _I, _P, _P, _SZ, _P, _SZ, ctypes.POINTER(_P), ctypes.POINTER(_P),
                             _P, ctypes.POINTER(_P)], _I),
    "ifq_graph_launch": ([_P, _P], _I),
    "ifq_graph_destroy": ([_P], _I),
    "ifq_pack_codes": ([_P, _P, _SZ, _P], _I),
    "ifq_unpack_codes": ([_P, _P, _SZ, _P], _I),
    "ifq_pack_codes_kbits": ([_P, _P, _SZ, _I, _P], _I),
    "ifq_unpack_codes_kbits": ([_P, _P, _SZ, _I, _P], _I),
    "ifq_pack_signs": ([_P, _P, _I, _I, _P], _I),
    "ifq_copy_bytes": ([_P, _P, _SZ, _P], _I),
    "ifq_wait_selftest": ([_I, _P], _I),
    "ifq_device_status": ([_P, ctypes.POINTER(_I)], _I),
}

# Every symbol that include/ifq.h declares.
EXPORTS = tuple(_SIGS)


def lib_path() -> str:
    return _build.LIB


def lib(build_if_missing: bool = True):
    """The loaded libifq.so (built in-tree on first use if missing)."""
    global _lib
    with _lock:
        if _lib is None:
            try:  # let torch load its CUDA runtime first so one libcudart serves both
                import torch  # noqa: F401
            except Exception:
                pass
            path = _build.build() if build_if_missing else _build.LIB
            if not os.path.exists(path):
                raise RuntimeError(f"libifq.so not found at {path}; build it with paper_1911_08076_gb300.build")
            L = ctypes.CDLL(path)
            for name, (args, res) in _SIGS.items():
                f = getattr(L, name)
                f.argtypes = args
                f.restype = res
            _lib = L
    return _lib


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _ok(rc: int, what: str):
    if rc != IFQ_OK:
        raise IfqError(rc, what)


def ifq_status_str(status: int) -> str:
    return lib().ifq_status_str(int(status)).decode()


def ifq_version() -> int:
    return lib().ifq_version()


def ifq_fold_layer(K: int, alpha, gamma, beta, mean, var, delta_in: float = 0.5, bias=None, eps: float = 1e-5,
                   q_base: float = 0.5, q_offset: float = -0.25, kbits: int = 2):
    """Integrated fixed-point fold (host): returns (T int32 [cout][2^k-1], sign int8 [cout])."""
    f32 = lambda a: None if a is None else np.ascontiguousarray(a, dtype=np.float32)
    al, ga, be, mu, va, bi = map(f32, (alpha, gamma, beta, mean, var, bias))
    cout = al.shape[0]
    L = (1 << kbits) - 1
    T = np.empty((cout, L), np.int32)
    s = np.empty(cout, np.int8)
    _ok(lib().ifq_fold_layer(cout, int(K), kbits, _ptr(al), delta_in, _ptr(bi), _ptr(ga), _ptr(be), _ptr(mu),
                             _ptr(va), eps, q_base, q_offset, _ptr(T), _ptr(s)), "ifq_fold_layer")
    return T, s


def ifq_fold_layer_separated(K: int, m: int, alpha, gamma, beta, mean, var, delta_in: float = 0.5, bias=None,
                             eps: float = 1e-5, q_base: float = 0.5, q_offset: float = -0.25, kbits: int = 2):
    """Thresholds of the separated fixed-point conversion at Q = 2^m (host): (T, sign)."""
    f32 = lambda a: None if a is None else np.ascontiguousarray(a, dtype=np.float32)
    al, ga, be, mu, va, bi = map(f32, (alpha, gamma, beta, mean, var, bias))
    cout = al.shape[0]
    L = (1 << kbits) - 1
    T = np.empty((cout, L), np.int32)
    s = np.empty(cout, np.int8)
    _ok(lib().ifq_fold_layer_separated(cout, int(K), kbits, int(m), _ptr(al), delta_in, _ptr(bi), _ptr(ga), _ptr(be),
                                       _ptr(mu), _ptr(va), eps, q_base, q_offset, _ptr(T), _ptr(s)),
        "ifq_fold_layer_separated")
    return T, s


def ifq_fold_output_separated(m: int, alpha, delta_in: float = 0.5, bias=None):
    """Separated fixed-point conversion of a non-quantized conv output (host): (mul, add) int64 [cout]."""
    al = np.ascontiguousarray(alpha, dtype=np.float32)
    bi = None if bias is None else np.ascontiguousarray(bias, dtype=np.float32)
    mul = np.empty(al.shape[0], np.int64)
    add = np.empty(al.shape[0], np.int64)
    _ok(lib().ifq_fold_output_separated(al.shape[0], int(m), _ptr(al), delta_in, _ptr(bi), _ptr(mul), _ptr(add)),
        "ifq_fold_output_separated")
    return mul, add


def ifq_fixed_output(acc, rows: int, cout: int, mul, add, m: int, y, stream=None):
    _ok(lib().ifq_fixed_output(_ptr(acc), rows, cout, _ptr(mul), _ptr(add), m, _ptr(y), _stream(stream)),
        "ifq_fixed_output")


def ifq_codes_bytes(n: int, h: int, w: int, c: int, kbits: int = 2) -> int:
    out = _SZ()
    _ok(lib().ifq_codes_bytes(n, h, w, c, kbits, ctypes.byref(out)), "ifq_codes_bytes")
    return out.value


def ifq_codes_storage_bytes(n: int, h: int, w: int, c: int, kbits: int = 2) -> int:
    out = _SZ()
    _ok(lib().ifq_codes_storage_bytes(n, h, w, c, kbits, ctypes.byref(out)), "ifq_codes_storage_bytes")
    return out.value


def conv_desc(n, h, w, cin, cout, k, stride=1, pad=0, out_mode=IFQ_OUT_CODES, path=IFQ_PATH_AUTO, kw=None, pool=0,
              kbits=2, in_bits=0):
    return ConvDesc(n, h, w, cin, cout, k, k if kw is None else kw, stride, pad, out_mode, path, pool, kbits,
                    in_bits)


def pool_desc(n, h, w, c, k, stride, pad=0, kbits=2):
    return PoolDesc(n, h, w, c, k, stride, pad, kbits)


def ifq_conv_out_shape(d: ConvDesc):
    ho, wo = _I(), _I()
    _ok(lib().ifq_conv_out_shape(ctypes.byref(d), ctypes.byref(ho), ctypes.byref(wo)), "ifq_conv_out_shape")
    return ho.value, wo.value


def ifq_pool_out_shape(d: PoolDesc):
    ho, wo = _I(), _I()
    _ok(lib().ifq_pool_out_shape(ctypes.byref(d), ctypes.byref(ho), ctypes.byref(wo)), "ifq_pool_out_shape")
    return ho.value, wo.value


def ifq_conv_plan(d: ConvDesc) -> int:
    p = _I()
    _ok(lib().ifq_conv_plan(ctypes.byref(d), ctypes.byref(p)), "ifq_conv_plan")
    return p.value


def ifq_weights_prep_bytes(d: ConvDesc) -> int:
    out = _SZ()
    _ok(lib().ifq_weights_prep_bytes(ctypes.byref(d), ctypes.byref(out)), "ifq_weights_prep_bytes")
    return out.value


def ifq_pack_weights(d: ConvDesc, w_bits, w_prep, stream=None):
    _ok(lib().ifq_pack_weights(ctypes.byref(d), _ptr(w_bits), _ptr(w_prep), _stream(stream)), "ifq_pack_weights")


def ifq_conv_workspace_bytes(d: ConvDesc) -> int:
    out = _SZ()
    _ok(lib().ifq_conv_workspace_bytes(ctypes.byref(d), ctypes.byref(out)), "ifq_conv_workspace_bytes")
    return out.value


def ifq_conv2bit(d: ConvDesc, x, w_prep, thr, sign, y_codes=None, y_acc=None, ws=None, ws_bytes: int = 0,
                 stream=None):
    _ok(lib().ifq_conv2bit(ctypes.byref(d), _ptr(x), _ptr(w_prep), _ptr(thr), _ptr(sign), _ptr(y_codes),
                           _ptr(y_acc), _ptr(ws), ws_bytes, _stream(stream)), "ifq_conv2bit")


def ifq_maxpool2bit(d: PoolDesc, x, sign, y, stream=None):
    _ok(lib().ifq_maxpool2bit(ctypes.byref(d), _ptr(x), _ptr(sign), _ptr(y), _stream(stream)), "ifq_maxpool2bit")


def _layer_array(layers: Sequence[Layer]):
    arr = (Layer * len(layers))(*layers)
    return arr, len(layers)


def ifq_forward_workspace_bytes(layers: Sequence[Layer]) -> int:
    arr, n = _layer_array(layers)
    out = _SZ()
    _ok(lib().ifq_forward_workspace_bytes(arr, n, ctypes.byref(out)), "ifq_forward_workspace_bytes")
    return out.value


def ifq_forward(layers: Sequence[Layer], x, ws=None, ws_bytes: int = 0, stream=None):
    arr, n = _layer_array(layers)
    _ok(lib().ifq_forward(arr, n, _ptr(x), _ptr(ws), ws_bytes, _stream(stream)), "ifq_forward")


def ifq_forward_noalloc(layers: Sequence[Layer], x, stream=None):
    arr, n = _layer_array(layers)
    _ok(lib().ifq_forward_noalloc(arr, n, _ptr(x), _stream(stream)), "ifq_forward_noalloc")


def ifq_last_forward_mode() -> int:
    """IFQ_FORWARD_LAYERS or IFQ_FORWARD_PERSISTENT for this thread's last forward call."""
    m = ctypes.c_int(0)
    _ok(lib().ifq_last_forward_mode(ctypes.byref(m)), "ifq_last_forward_mode")
    return m.value


def ifq_graph_create(layers: Sequence[Layer], x, ws=None, ws_bytes: int = 0, stream=None) -> int:
    arr, n = _layer_array(layers)
    g = _P()
    _ok(lib().ifq_graph_create(arr, n, _ptr(x), _ptr(ws), ws_bytes, _stream(stream), ctypes.byref(g)),
        "ifq_graph_create")
    return g.value


def ifq_graph_create_io(layers: Sequence[Layer], x, ws=None, ws_bytes: int = 0, x_src=None, x_bytes: int = 0,
                        y_codes_dst: Optional[Sequence] = None, y_acc_dst: Optional[Sequence] = None,
                        stream=None) -> int:
    """ifq_graph_create with the input copy (x_src -> x, x_bytes) and per-layer result copies
    (y_codes_dst[i] / y_acc_dst[i]: a tensor, an address or None) inside the graph."""
    arr, n = _layer_array(layers)

    def dsts(seq):
        if seq is None:
            return None
        if len(seq) != n:
            raise ValueError("one destination (or None) per layer")
        return (_P * n)(*[_ptr(t) for t in seq])

    g = _P()
    _ok(lib().ifq_graph_create_io(arr, n, _ptr(x), _ptr(ws), ws_bytes, _ptr(x_src), x_bytes, dsts(y_codes_dst),
                                  dsts(y_acc_dst), _stream(stream), ctypes.byref(g)), "ifq_graph_create_io")
    return g.value


def ifq_graph_launch(g: int, stream=None):
    _ok(lib().ifq_graph_launch(g, _stream(stream)), "ifq_graph_launch")


def ifq_graph_destroy(g: int):
    _ok(lib().ifq_graph_destroy(g), "ifq_graph_destroy")


def ifq_pack_codes(codes, packed, n: int, stream=None):
    _ok(lib().ifq_pack_codes(_ptr(codes), _ptr(packed), n, _stream(stream)), "ifq_pack_codes")


def ifq_unpack_codes(packed, codes, n: int, stream=None):
    _ok(lib().ifq_unpack_codes(_ptr(packed), _ptr(codes), n, _stream(stream)), "ifq_unpack_codes")


def ifq_pack_codes_kbits(codes, packed, n: int, kbits: int, stream=None):
    _ok(lib().ifq_pack_codes_kbits(_ptr(codes), _ptr(packed), n, kbits, _stream(stream)), "ifq_pack_codes_kbits")


def ifq_unpack_codes_kbits(packed, codes, n: int, kbits: int, stream=None):
    _ok(lib().ifq_unpack_codes_kbits(_ptr(packed), _ptr(codes), n, kbits, _stream(stream)), "ifq_unpack_codes_kbits")


def ifq_pack_signs(w, bits, rows: int, K: int, stream=None):
    _ok(lib().ifq_pack_signs(_ptr(w), _ptr(bits), rows, K, _stream(stream)), "ifq_pack_signs")


def ifq_copy_bytes(dst, src, n: int, stream=None):
    _ok(lib().ifq_copy_bytes(_ptr(dst), _ptr(src), n, _stream(stream)), "ifq_copy_bytes")


def ifq_wait_selftest(limit_us: int, stream=None):
    _ok(lib().ifq_wait_selftest(int(limit_us), _stream(stream)), "ifq_wait_selftest")


def ifq_device_status(stream=None) -> int:
    s = _I()
    _ok(lib().ifq_device_status(_stream(stream), ctypes.byref(s)), "ifq_device_status")
    return s.value
