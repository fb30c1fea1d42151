"""Plain fp64 CPU oracle for DMS decode (arXiv 2506.05345, Sec. 3.1-3.2).

TEST INFRASTRUCTURE ONLY: the test suite, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference leg of ``bench.py`` are the only callers.  The product
library never imports this package, and this package never imports the product.

The arithmetic lives in ``dms_oracle.c`` (plain C, fp64, sequential sums); this
module compiles it with gcc on first use and wraps it with ctypes.

Functions (all take bf16 data as ``numpy.uint16`` bit patterns):
  alpha(logit_bits)                      Sec. 3.2 decision, [logit > 0]
  retained(logits, j, w, immediate)      Sec. 3.1 / Fig. 1b retained positions (Sec. 5
                                         immediate-eviction ablation when immediate)
  decode(q, k, v, logits, j, w, scale, immediate)  softmax attention over the retained set
  borrowed(q, G)                         App. B decision neuron: (logits, attention q)
  e4m3_to_double(code), e4m3_from_float(x)   fp8 E4M3FN value of a code / nearest code
  quantize_rows_e4m3(rows)               per-row fp32 scale and E4M3 codes of bf16 rows
  decode_fp8(q, kc, ks, vc, vs, logits, j, w, scale, immediate)
                                         the attention over the dequantised rows
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "dms_oracle.c")
_LIB = os.path.join(_HERE, "libdms_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no fast-math: sums stay in source order)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(
            ["gcc", "-O2", "-fno-fast-math", "-ffp-contract=off", "-std=c11",
             "-shared", "-fPIC", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            u16p = ctypes.POINTER(ctypes.c_uint16)
            i32p = ctypes.POINTER(ctypes.c_int32)
            f64p = ctypes.POINTER(ctypes.c_double)
            lib.dms_oracle_bf16_to_double.argtypes = [ctypes.c_uint16]
            lib.dms_oracle_bf16_to_double.restype = ctypes.c_double
            lib.dms_oracle_alpha.argtypes = [ctypes.c_uint16]
            lib.dms_oracle_alpha.restype = ctypes.c_int
            lib.dms_oracle_retained.argtypes = [u16p, ctypes.c_int64, ctypes.c_int64,
                                                ctypes.c_int64, i32p]
            lib.dms_oracle_retained.restype = ctypes.c_int64
            lib.dms_oracle_decode.argtypes = [u16p, ctypes.c_int32, ctypes.c_int32, u16p, u16p,
                                              ctypes.c_int64, u16p, ctypes.c_int64,
                                              ctypes.c_int64, ctypes.c_int64, ctypes.c_double,
                                              f64p]
            lib.dms_oracle_decode.restype = None
            lib.dms_oracle_retained_policy.argtypes = [u16p, ctypes.c_int64, ctypes.c_int64,
                                                       ctypes.c_int64, ctypes.c_int, i32p]
            lib.dms_oracle_retained_policy.restype = ctypes.c_int64
            lib.dms_oracle_decode_policy.argtypes = [u16p, ctypes.c_int32, ctypes.c_int32, u16p,
                                                     u16p, ctypes.c_int64, u16p, ctypes.c_int64,
                                                     ctypes.c_int64, ctypes.c_int64, ctypes.c_int,
                                                     ctypes.c_double, f64p]
            lib.dms_oracle_decode_policy.restype = None
            u8p = ctypes.POINTER(ctypes.c_uint8)
            f32p = ctypes.POINTER(ctypes.c_float)
            lib.dms_oracle_e4m3_to_double.argtypes = [ctypes.c_uint8]
            lib.dms_oracle_e4m3_to_double.restype = ctypes.c_double
            lib.dms_oracle_e4m3_from_float.argtypes = [ctypes.c_float]
            lib.dms_oracle_e4m3_from_float.restype = ctypes.c_uint8
            lib.dms_oracle_quantize_row_e4m3.argtypes = [u16p, ctypes.c_int32, u8p, f32p]
            lib.dms_oracle_quantize_row_e4m3.restype = None
            lib.dms_oracle_decode_kv64.argtypes = [u16p, ctypes.c_int32, ctypes.c_int32, f64p,
                                                   f64p, ctypes.c_int64, u16p, ctypes.c_int64,
                                                   ctypes.c_int64, ctypes.c_int64, ctypes.c_int,
                                                   ctypes.c_double, f64p]
            lib.dms_oracle_decode_kv64.restype = None
            _lib = lib
    return _lib


def _u16(a) -> np.ndarray:
    a = np.asarray(a)
    if a.dtype != np.uint16:
        raise TypeError("bf16 data must be passed as uint16 bit patterns")
    return a


def _ptr(a: np.ndarray, ctype):
    return a.ctypes.data_as(ctypes.POINTER(ctype))


def bf16_to_double(bits: int) -> float:
    return _load().dms_oracle_bf16_to_double(int(bits) & 0xFFFF)


def alpha(logit_bits: int) -> int:
    """Sec. 3.2: alpha_bin = round(sigmoid(logit)) read as [logit > 0]."""
    return int(_load().dms_oracle_alpha(int(logit_bits) & 0xFFFF))


def retained(logits, j: int, w: int, immediate: bool = False) -> np.ndarray:
    """Sorted positions retained by one KV head after appending position j.

    ``logits`` is a 1-D uint16 array (any stride) holding positions 0..j.
    ``immediate``: the eviction ablation of Sec. 5 (token i decided by alpha_{i+w}).
    """
    lg = _u16(logits)
    if lg.ndim != 1:
        raise ValueError("logits must be 1-D")
    if j >= lg.shape[0]:
        raise ValueError("j beyond the logits given")
    stride = lg.strides[0] // 2
    out = np.empty(max(j + 1, 1), dtype=np.int32)
    n = _load().dms_oracle_retained_policy(_ptr(lg, ctypes.c_uint16), stride, j, w,
                                           1 if immediate else 0, _ptr(out, ctypes.c_int32))
    return out[:n].copy()


def decode(q, k, v, logits, j: int, w: int, scale: float = 0.0,
           immediate: bool = False) -> np.ndarray:
    """Attention of G query heads over the retained set of their KV head at step j.

    q: [G, D] uint16; k, v: [T, D] uint16 (row-strided views allowed, rows 0..j);
    logits: [T] uint16.  Returns [G, D] float64.
    """
    q = np.ascontiguousarray(_u16(q))
    k = _u16(k)
    v = _u16(v)
    lg = _u16(logits)
    if q.ndim != 2 or k.ndim != 2 or v.ndim != 2 or lg.ndim != 1:
        raise ValueError("q, k, v must be 2-D and logits 1-D")
    G, D = q.shape
    if k.shape[1] != D or v.shape[1] != D:
        raise ValueError("head_dim mismatch")
    if k.strides[1] != 2 or v.strides[1] != 2:
        raise ValueError("k and v rows must be contiguous")
    if k.strides[0] != v.strides[0]:
        v = np.ascontiguousarray(v)
        k = np.ascontiguousarray(k)
    if j >= k.shape[0] or j >= lg.shape[0]:
        raise ValueError("j beyond the data given")
    out = np.zeros((G, D), dtype=np.float64)
    _load().dms_oracle_decode_policy(_ptr(q, ctypes.c_uint16), G, D, _ptr(k, ctypes.c_uint16),
                                     _ptr(v, ctypes.c_uint16), k.strides[0] // 2,
                                     _ptr(lg, ctypes.c_uint16), lg.strides[0] // 2, j, w,
                                     1 if immediate else 0, float(scale),
                                     _ptr(out, ctypes.c_double))
    return out


def borrowed(q, group: int):
    """App. B: the decision logit of each query group is element 0 of the group's first
    query head, and that element is set to 0 before the attention; the other query
    heads of the group are unchanged.

    q: bf16 bits (numpy.uint16) of shape [..., kv_heads * group, D].  Returns
    (logits [..., kv_heads], q_attention) with q_attention a copy of q whose element
    0 of heads 0, group, 2 * group, ... is +0.
    """
    q = _u16(q)
    if q.shape[-2] % group:
        raise ValueError("query heads are not a multiple of the group size")
    logits = q[..., ::group, 0].copy()
    q_att = q.copy()
    q_att[..., ::group, 0] = 0
    return logits, q_att


def e4m3_to_double(code: int) -> float:
    """Value of an fp8 E4M3FN code (NaN for S.1111.111)."""
    return _load().dms_oracle_e4m3_to_double(int(code) & 0xFF)


def e4m3_from_float(x: float) -> int:
    """Nearest E4M3FN code of the float32 value x: ties to even, magnitudes above 448
    saturated, NaN -> 0x7f."""
    return int(_load().dms_oracle_e4m3_from_float(float(np.float32(x))))


def quantize_rows_e4m3(rows):
    """Per-row quantisation of bf16 rows [..., D] (uint16 bits): returns (codes uint8
    [..., D], scales float32 [...]) with scale = fl32(amax / 448) and code =
    E4M3(fl32(x / scale)); zero rows get scale 0 and zero codes."""
    r = np.ascontiguousarray(_u16(rows))
    D = r.shape[-1]
    flat = r.reshape(-1, D)
    codes = np.zeros(flat.shape, dtype=np.uint8)
    scales = np.zeros(flat.shape[0], dtype=np.float32)
    lib = _load()
    for i in range(flat.shape[0]):
        row = np.ascontiguousarray(flat[i])
        sc = ctypes.c_float(0.0)
        lib.dms_oracle_quantize_row_e4m3(_ptr(row, ctypes.c_uint16), D,
                                         codes[i].ctypes.data_as(ctypes.POINTER(ctypes.c_uint8)),
                                         ctypes.byref(sc))
        scales[i] = sc.value
    return codes.reshape(r.shape), scales.reshape(r.shape[:-1])


_E4M3 = None


def _e4m3_table() -> np.ndarray:
    global _E4M3
    if _E4M3 is None:
        _E4M3 = np.array([e4m3_to_double(c) for c in range(256)], dtype=np.float64)
    return _E4M3


def dequantize_e4m3(codes, scales) -> np.ndarray:
    """codes [..., D] uint8, scales [...] -> fp64 rows code value * scale (exact)."""
    c = np.asarray(codes, dtype=np.uint8)
    return _e4m3_table()[c] * np.asarray(scales, dtype=np.float64)[..., None]


def decode_fp8(q, k_codes, k_scales, v_codes, v_scales, logits, j: int, w: int,
               scale: float = 0.0, immediate: bool = False) -> np.ndarray:
    """Attention of G query heads (q [G, D] bf16 bits) over the retained set at step j
    of a cache whose rows are E4M3 codes [T, D] with per-row scales [T]."""
    q = np.ascontiguousarray(_u16(q))
    lg = _u16(logits)
    kd = np.ascontiguousarray(dequantize_e4m3(k_codes, k_scales))
    vd = np.ascontiguousarray(dequantize_e4m3(v_codes, v_scales))
    G, D = q.shape
    if kd.shape != vd.shape or kd.shape[1] != D:
        raise ValueError("shape mismatch")
    if j >= kd.shape[0] or j >= lg.shape[0]:
        raise ValueError("j beyond the data given")
    out = np.zeros((G, D), dtype=np.float64)
    _load().dms_oracle_decode_kv64(_ptr(q, ctypes.c_uint16), G, D, _ptr(kd, ctypes.c_double),
                                   _ptr(vd, ctypes.c_double), D, _ptr(lg, ctypes.c_uint16),
                                   lg.strides[0] // 2, j, w, 1 if immediate else 0, float(scale),
                                   _ptr(out, ctypes.c_double))
    return out
