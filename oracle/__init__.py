"""Plain CPU oracle for group-wise few-bit weight quantization.

TEST INFRASTRUCTURE ONLY: the test suite, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package; the product path
(``paper_2607_08779_gb300``) never does, and the two share no code.

The arithmetic lives in ``sss_oracle.c`` (plain single-threaded C, built with
``-O2 -ffp-contract=off``, no fast-math).  This module only builds that file
with gcc, loads it with ctypes and marshals numpy arrays.  What each function
computes, with the passage of the paper it follows:

* ``quantize_group`` / ``quantize_group_gamma`` -- eq:quantizer with the grid
  of eq:absmax (unsigned symmetric), eq:signed_sym_quant + eq:sign_rule
  (signed symmetric) or eq:minmax (asymmetric), including the clipped-set
  counts of def:clipped-set.
* ``pack_group`` / ``unpack_group`` -- the canonical packed layout (the paper
  fixes only the Q2/Q4 block contents, Appendix "Formats and block layout").
* ``quantize`` -- all groups of a row-major [n, k] matrix.
* ``dequantize`` -- s*c (symmetric) or s*u + min (asymmetric), Appendix
  "Zero-point cost in quantized GEMM".
* ``matmul_f64`` / ``gemv`` -- the fp64 reference y = x W^T over the
  dequantised weights.
* ``f32_to_f16`` / ``f16_to_f32`` -- IEEE binary16 from its definition.
* ``quantize_act_q8`` / ``gemv_q8`` -- the dynamic Q8_0 (narrow-range 8-bit,
  blocks of 32) activation quantizer the paper pairs with the weight formats
  (Sec. 5 "Composition with PTQ methods", Appendix C "Algorithm details"),
  and the fp64 GEMV over dequantised weights and activations.

Every function of the oracle is pinned by ``tests/test_oracle_pins.py``
against the paper's theorems, closed forms and brute force; nothing in it is
"parity unpinned".
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

GRID_UNSIGNED_SYM = 0
GRID_SIGNED_SYM = 1
GRID_ASYM = 2
FLAG_NONFINITE = 1
FLAG_RANGE = 2

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "sss_oracle.c")
_HDR = os.path.join(_HERE, "sss_oracle.h")
_LIB = os.path.join(_HERE, "liboracle_sss.so")
_lock = threading.Lock()
_lib = None

CFLAGS = ["-O2", "-ffp-contract=off", "-fno-fast-math", "-std=c11", "-fPIC",
          "-shared", "-Wall", "-Wextra"]


def build(force: bool = False) -> str:
    """Compile sss_oracle.c into liboracle_sss.so (in-tree) with gcc."""
    newest = max(os.path.getmtime(_SRC), os.path.getmtime(_HDR))
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < newest:
        tmp = _LIB + f".tmp{os.getpid()}"
        cmd = ["gcc", *CFLAGS, "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
    return _LIB


class GroupInfo(ctypes.Structure):
    _fields_ = [
        ("s32", ctypes.c_float),
        ("alpha", ctypes.c_float),
        ("mx", ctypes.c_float),
        ("mn", ctypes.c_float),
        ("M", ctypes.c_float),
        ("gamma", ctypes.c_int32),
        ("s16", ctypes.c_uint16),
        ("m16", ctypes.c_uint16),
        ("n_self", ctypes.c_int32),
        ("n_other", ctypes.c_int32),
        ("flags", ctypes.c_int32),
    ]

    def as_dict(self) -> dict:
        return {name: getattr(self, name) for name, _ in self._fields_}


def _p(a):
    return ctypes.c_void_p(a.ctypes.data) if a is not None else ctypes.c_void_p(0)


def lib():
    global _lib
    with _lock:
        if _lib is None:
            _lib = ctypes.CDLL(build())
            L = _lib
            vp, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
            L.orc_f32_to_f16.argtypes = [ctypes.c_float]
            L.orc_f32_to_f16.restype = ctypes.c_uint16
            L.orc_f16_to_f32.argtypes = [ctypes.c_uint16]
            L.orc_f16_to_f32.restype = ctypes.c_float
            L.orc_quantize_group.argtypes = [vp, i32, i32, i32, vp, vp, vp,
                                             ctypes.POINTER(GroupInfo)]
            L.orc_quantize_group.restype = i32
            L.orc_quantize_group_gamma.argtypes = [vp, i32, i32, i32, vp, vp, vp,
                                                   ctypes.POINTER(GroupInfo)]
            L.orc_quantize_group_gamma.restype = i32
            L.orc_pack_group.argtypes = [vp, i32, i32, vp]
            L.orc_pack_group.restype = None
            L.orc_unpack_group.argtypes = [vp, i32, i32, vp]
            L.orc_unpack_group.restype = None
            L.orc_quantize.argtypes = [vp, i64, i64, i32, i32, i32, vp, vp, vp, vp]
            L.orc_quantize.restype = i32
            L.orc_dequantize.argtypes = [vp, vp, vp, i64, i64, i32, i32, i32, vp]
            L.orc_dequantize.restype = None
            L.orc_dequantize_rows.argtypes = [vp, vp, vp, i64, i64, i32, i32, i32,
                                              i64, i64, vp]
            L.orc_dequantize_rows.restype = None
            L.orc_matmul_f64.argtypes = [vp, vp, i64, i64, i64, vp]
            L.orc_matmul_f64.restype = None
            L.orc_gemv.argtypes = [vp, vp, vp, i64, i64, i32, i32, i32, vp, i64, vp]
            L.orc_gemv.restype = None
            L.orc_quantize_act_q8.argtypes = [vp, i64, i64, vp, vp]
            L.orc_quantize_act_q8.restype = i32
            L.orc_gemv_q8.argtypes = [vp, vp, vp, i64, i64, i32, i32, i32, vp, vp, i64, vp]
            L.orc_gemv_q8.restype = None
            L.orc_fwht_f32.argtypes = [vp, i32]
            L.orc_fwht_f32.restype = None
            L.orc_rotate_rows.argtypes = [vp, i64, i64, i32, vp]
            L.orc_rotate_rows.restype = None
            L.orc_rotate_cols.argtypes = [vp, i64, i64, i32, vp]
            L.orc_rotate_cols.restype = None
            L.orc_lsq_scale.argtypes = [vp, i32, i32, i32, i32, ctypes.c_float]
            L.orc_lsq_scale.restype = ctypes.c_float
            L.orc_lsq_quantize.argtypes = [vp, i64, i64, i32, i32, i32, i32, ctypes.c_float,
                                           vp, vp]
            L.orc_lsq_quantize.restype = i32
        return _lib


def _f32(a):
    return np.ascontiguousarray(a, dtype=np.float32)


# --------------------------------------------------------------------------
# scalar helpers
# --------------------------------------------------------------------------

def f32_to_f16(x: float) -> int:
    return int(lib().orc_f32_to_f16(float(x)))


def f16_to_f32(h: int) -> float:
    return float(lib().orc_f16_to_f32(int(h)))


# --------------------------------------------------------------------------
# one group
# --------------------------------------------------------------------------

def _group_call(fn, w, q, sel):
    w = _f32(w).ravel()
    g = w.size
    c_pre = np.zeros(g, np.int32)
    c = np.zeros(g, np.int32)
    u = np.zeros(g, np.uint8)
    info = GroupInfo()
    fn(_p(w), g, int(q), int(sel), _p(c_pre), _p(c), _p(u), ctypes.byref(info))
    return {"c_pre": c_pre, "c": c, "u": u, **info.as_dict()}


def quantize_group(w, q: int, grid: int) -> dict:
    """Quantize one group with the given grid; returns codes and group info."""
    return _group_call(lib().orc_quantize_group, w, q, grid)


def quantize_group_gamma(w, q: int, gamma: int) -> dict:
    """Symmetric quantizer Q(w; gamma*alpha, 0), alpha = ||w||_inf / 2^(q-1)."""
    return _group_call(lib().orc_quantize_group_gamma, w, q, gamma)


def pack_group(u, q: int) -> np.ndarray:
    u = np.ascontiguousarray(u, dtype=np.uint8)
    out = np.zeros(u.size * q // 8, np.uint8)
    lib().orc_pack_group(_p(u), u.size, int(q), _p(out))
    return out


def unpack_group(b, g: int, q: int) -> np.ndarray:
    b = np.ascontiguousarray(b, dtype=np.uint8)
    u = np.zeros(g, np.uint8)
    lib().orc_unpack_group(_p(b), int(g), int(q), _p(u))
    return u


# --------------------------------------------------------------------------
# whole matrices
# --------------------------------------------------------------------------

def codes_bytes(n: int, k: int, q: int) -> int:
    return n * k * q // 8


def quantize(W, q: int, g: int, grid: int, clip_counts: bool = False):
    """Quantize a row-major [n, k] fp32 matrix in groups of g along k.

    Returns (codes uint8 [n, k*q/8], scales uint16 [n, k/g] (fp16 bits),
    mins uint16 [n, k/g] or None, clip uint8 [n, k/g, 2] or None, flags)."""
    W = _f32(W)
    n, k = W.shape
    assert k % g == 0
    codes = np.zeros((n, k * q // 8), np.uint8)
    scales = np.zeros((n, k // g), np.uint16)
    mins = np.zeros((n, k // g), np.uint16) if grid == GRID_ASYM else None
    clip = np.zeros((n, k // g, 2), np.uint8) if clip_counts else None
    flags = lib().orc_quantize(_p(W), n, k, q, g, grid, _p(codes), _p(scales),
                               _p(mins), _p(clip))
    return codes, scales, mins, clip, int(flags)


def dequantize(codes, scales, mins, n: int, k: int, q: int, g: int, grid: int,
               rows=None) -> np.ndarray:
    """fp32 dequantised weights [n, k] (or only rows r0..r0+nr-1)."""
    codes = np.ascontiguousarray(codes, np.uint8)
    scales = np.ascontiguousarray(scales, np.uint16)
    mins = None if mins is None else np.ascontiguousarray(mins, np.uint16)
    if rows is None:
        out = np.zeros((n, k), np.float32)
        lib().orc_dequantize(_p(codes), _p(scales), _p(mins), n, k, q, g, grid,
                             _p(out))
    else:
        r0, nr = rows
        out = np.zeros((nr, k), np.float32)
        lib().orc_dequantize_rows(_p(codes), _p(scales), _p(mins), n, k, q, g,
                                  grid, r0, nr, _p(out))
    return out


def matmul_f64(What, x_bf16) -> np.ndarray:
    """y[b, j] = sum_k What[j, k] * x[b, k] in fp64; x given as bf16 bits."""
    What = _f32(What)
    x = np.ascontiguousarray(x_bf16, np.uint16)
    if x.ndim == 1:
        x = x[None, :]
    nb, k = x.shape
    n = What.shape[0]
    assert What.shape[1] == k
    y = np.zeros((nb, n), np.float64)
    lib().orc_matmul_f64(_p(What), _p(x), nb, n, k, _p(y))
    return y


def gemv(codes, scales, mins, n: int, k: int, q: int, g: int, grid: int,
         x_bf16) -> np.ndarray:
    """fp64 decode GEMV over the packed weights, y [nb, n]."""
    codes = np.ascontiguousarray(codes, np.uint8)
    scales = np.ascontiguousarray(scales, np.uint16)
    mins = None if mins is None else np.ascontiguousarray(mins, np.uint16)
    x = np.ascontiguousarray(x_bf16, np.uint16)
    if x.ndim == 1:
        x = x[None, :]
    nb = x.shape[0]
    y = np.zeros((nb, n), np.float64)
    lib().orc_gemv(_p(codes), _p(scales), _p(mins), n, k, q, g, grid, _p(x), nb,
                   _p(y))
    return y


def quantize_act_q8(x_bf16):
    """Q8_0 activations: per block of 32, d = fl32(max|x|/127), q = clip(RNE(x/d),
    -127, 127), stored fp16 d.  x as bf16 bits [nb, k] (k % 32 == 0).
    Returns (q int8 [nb, k], d uint16 [nb, k/32] fp16 bits, flags)."""
    x = np.ascontiguousarray(x_bf16, np.uint16)
    if x.ndim == 1:
        x = x[None, :]
    nb, k = x.shape
    assert k % 32 == 0
    q = np.zeros((nb, k), np.int8)
    d = np.zeros((nb, k // 32), np.uint16)
    flags = lib().orc_quantize_act_q8(_p(x), nb, k, _p(q), _p(d))
    return q, d, int(flags)


def gemv_q8(codes, scales, mins, n: int, k: int, q: int, g: int, grid: int,
            xq, xd) -> np.ndarray:
    """fp64 decode GEMV over the packed weights and Q8_0 activations
    (xq int8 [nb, k], xd fp16 bits [nb, k/32]); y [nb, n]."""
    codes = np.ascontiguousarray(codes, np.uint8)
    scales = np.ascontiguousarray(scales, np.uint16)
    mins = None if mins is None else np.ascontiguousarray(mins, np.uint16)
    xq = np.ascontiguousarray(xq, np.int8)
    xd = np.ascontiguousarray(xd, np.uint16)
    if xq.ndim == 1:
        xq, xd = xq[None, :], xd[None, :]
    nb = xq.shape[0]
    y = np.zeros((nb, n), np.float64)
    lib().orc_gemv_q8(_p(codes), _p(scales), _p(mins), n, k, q, g, grid, _p(xq), _p(xd),
                      nb, _p(y))
    return y


def fwht(x) -> np.ndarray:
    """Normalized Walsh-Hadamard transform of one fp32 vector (length a
    power of two): the fp32 fast transform, strides 1, 2, ..., b/2, then
    times fl32(1/sqrt(b))."""
    v = np.array(x, np.float32, copy=True)
    lib().orc_fwht_f32(_p(v), v.size)
    return v


def rotate(W, b: int, side: str = "rows") -> np.ndarray:
    """W [n, k] fp32 rotated by the normalized Hadamard of block size b on
    its input side (side="rows": every b-block of a row) or its output side
    (side="cols": every b-block of a column)."""
    W = np.ascontiguousarray(W, np.float32)
    n, k = W.shape
    out = np.empty_like(W)
    if side == "rows":
        assert k % b == 0
        lib().orc_rotate_rows(_p(W), n, k, b, _p(out))
    else:
        assert n % b == 0
        lib().orc_rotate_cols(_p(W), n, k, b, _p(out))
    return out


def lsq_scale(w, q: int, signed: bool, steps: int, lr: float) -> float:
    """The LSQ-refined fp32 scale of one group (see orc_lsq_scale)."""
    w = np.ascontiguousarray(w, np.float32)
    return float(np.float32(lib().orc_lsq_scale(_p(w), w.size, q, int(signed), steps, lr)))


def lsq_quantize(W, q: int, g: int, grid: int, steps: int, lr: float):
    """Symmetric-grid quantization with LSQ-refined scales: (codes, scales, flags)."""
    W = np.ascontiguousarray(W, np.float32)
    n, k = W.shape
    codes = np.zeros((n, k * q // 8), np.uint8)
    scales = np.zeros((n, k // g), np.uint16)
    flags = lib().orc_lsq_quantize(_p(W), n, k, q, g, grid, steps, np.float32(lr), _p(codes),
                                   _p(scales))
    return codes, scales, int(flags)
