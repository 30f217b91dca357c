"""Thin ctypes binding of the C ABI in include/sss.h.

Argument marshalling only: every step of the path runs in libsss.so's CUDA
kernels.  torch supplies device memory and streams.  There is no fallback:
if the library cannot be built or loaded, these functions raise.
"""
from __future__ import annotations

import ctypes
import os
import threading
from dataclasses import dataclass
from typing import Optional

from . import _build

GRID_UNSIGNED_SYM = 0
GRID_SIGNED_SYM = 1
GRID_ASYM = 2
GRIDS = {"unsigned": GRID_UNSIGNED_SYM, "signed": GRID_SIGNED_SYM, "asym": GRID_ASYM}

OUT_F32, OUT_F16, OUT_BF16 = 0, 1, 2
OP_GEMV, OP_GEMM = 0, 1

FLAG_NONFINITE = 0x1
FLAG_RANGE = 0x2
FLAG_TIMEOUT = 0x4

SSS_OK = 0
STATUS_NAMES = {0: "SSS_OK", 1: "SSS_E_ARG", 2: "SSS_E_UNSUPPORTED", 3: "SSS_E_ALIGN",
                4: "SSS_E_CUDA", 5: "SSS_E_WORKSPACE"}

EXPORTS = ("sss_codes_bytes", "sss_status_string", "sss_last_error", "sss_quantize",
           "sss_dequantize", "sss_gemv", "sss_gemv_multi", "sss_gemm", "sss_workspace_bytes",
           "sss_gemm_noalloc", "sss_gemm_noalloc_max_scratch_bytes", "sss_test_set_stall",
           "sss_gemm_multi", "sss_gemm_multi_workspace_bytes",
           "sss_gemm_q8", "sss_quantize_act_q8", "sss_sign_diagnostics", "sss_hadamard",
           "sss_quantize_rotated", "sss_quantize_lsq")

GEMV_PDL = 0x1
GEMV_WEIGHTS_READY = 0x2
GEMV_ACT_Q8 = 0x4

ROTATE_INPUT, ROTATE_OUTPUT = 0, 1

TEST_STALL_GEMV = 0x1
TEST_STALL_GEMV_BATCH = 0x2
TEST_STALL_GEMM = 0x4


class SssError(RuntimeError):
    def __init__(self, fn: str, status: int, detail: str = ""):
        self.status = status
        super().__init__(f"{fn} -> {STATUS_NAMES.get(status, status)}"
                         + (f" ({detail})" if detail else ""))


class QTensorDesc(ctypes.Structure):
    """Mirror of sss_qtensor_t."""
    _fields_ = [
        ("n", ctypes.c_int64),
        ("k", ctypes.c_int64),
        ("q", ctypes.c_int32),
        ("group", ctypes.c_int32),
        ("grid", ctypes.c_int32),
        ("reserved", ctypes.c_int32),
        ("codes", ctypes.c_void_p),
        ("scales", ctypes.c_void_p),
        ("mins", ctypes.c_void_p),
    ]


_lock = threading.Lock()
_lib = None


def library_path() -> str:
    return _build.LIB


def load(build_if_needed: bool = True):
    """Load libsss.so (building it with nvcc first if it is missing/stale)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if build_if_needed:
            _build.build()
        if not os.path.exists(_build.LIB):
            raise RuntimeError(f"CUDA library missing: {_build.LIB}")
        L = ctypes.CDLL(_build.LIB)
        vp, i32, i64, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
        P = ctypes.POINTER(QTensorDesc)
        L.sss_codes_bytes.argtypes = [i64, i64, i32]
        L.sss_codes_bytes.restype = sz
        L.sss_status_string.argtypes = [i32]
        L.sss_status_string.restype = ctypes.c_char_p
        L.sss_last_error.argtypes = []
        L.sss_last_error.restype = ctypes.c_char_p
        L.sss_quantize.argtypes = [vp, P, vp, vp, vp]
        L.sss_quantize.restype = i32
        L.sss_dequantize.argtypes = [P, vp, i32, vp]
        L.sss_dequantize.restype = i32
        L.sss_gemv.argtypes = [P, vp, i32, vp, vp, sz, vp, vp]
        L.sss_gemv.restype = i32
        L.sss_gemv_multi.argtypes = [ctypes.POINTER(P), ctypes.POINTER(vp), i32, vp,
                                     ctypes.c_uint32, vp, vp]
        L.sss_gemv_multi.restype = i32
        L.sss_gemm.argtypes = [P, vp, i64, vp, vp, sz, vp, vp]
        L.sss_gemm.restype = i32
        L.sss_gemm_multi.argtypes = [ctypes.POINTER(P), ctypes.POINTER(vp), i32, vp, i64, vp, sz,
                                     vp, vp]
        L.sss_gemm_multi.restype = i32
        L.sss_gemm_multi_workspace_bytes.argtypes = [ctypes.POINTER(P), i32, i64]
        L.sss_gemm_multi_workspace_bytes.restype = sz
        L.sss_workspace_bytes.argtypes = [P, i64, i32]
        L.sss_workspace_bytes.restype = sz
        L.sss_gemm_noalloc.argtypes = [P, vp, i64, vp, vp, vp]
        L.sss_gemm_noalloc.restype = i32
        L.sss_gemm_noalloc_max_scratch_bytes.argtypes = []
        L.sss_gemm_noalloc_max_scratch_bytes.restype = sz
        L.sss_gemm_q8.argtypes = [P, vp, i64, vp, vp, sz, vp, vp]
        L.sss_gemm_q8.restype = i32
        L.sss_quantize_act_q8.argtypes = [vp, i64, i64, vp, vp, vp, vp]
        L.sss_quantize_act_q8.restype = i32
        L.sss_sign_diagnostics.argtypes = [vp, i64, i64, i32, i32, vp, vp, vp, vp, vp]
        L.sss_sign_diagnostics.restype = i32
        L.sss_hadamard.argtypes = [vp, vp, i64, i64, i32, i32, vp]
        L.sss_hadamard.restype = i32
        L.sss_quantize_rotated.argtypes = [vp, i32, P, vp, vp, vp]
        L.sss_quantize_rotated.restype = i32
        L.sss_quantize_lsq.argtypes = [vp, P, i32, ctypes.c_float, vp, vp]
        L.sss_quantize_lsq.restype = i32
        L.sss_test_set_stall.argtypes = [ctypes.c_uint32]
        L.sss_test_set_stall.restype = None
        _lib = L
        return L


def _ptr(t) -> int:
    return 0 if t is None else int(t.data_ptr())


def _stream(stream) -> int:
    import torch

    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream)


def _check(fn: str, st: int):
    if st != SSS_OK:
        L = load(False)
        raise SssError(fn, st, L.sss_last_error().decode())


def _need(fn: str, name: str, t, dtype, numel=None, optional=False):
    """The C ABI takes bare device pointers: check here what a pointer cannot
    carry (its dtype, a dense layout, its element count) and raise
    SssError(SSS_E_ARG) before the call; _on_device checks the memory."""
    if t is None:
        if optional:
            return
        raise SssError(fn, 1, f"{name} is required")
    if t.dtype != dtype:
        raise SssError(fn, 1, f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise SssError(fn, 1, f"{name} must be contiguous")
    if numel is not None and t.numel() != numel:
        raise SssError(fn, 1, f"{name} holds {t.numel()} elements, expected {numel}")


def _on_device(fn: str, **tensors):
    """Every given tensor (None skipped) lives in CUDA device memory."""
    for name, t in tensors.items():
        if t is not None and not getattr(t, "is_cuda", False):
            raise SssError(fn, 1, f"{name} must be a CUDA tensor")


def _need_qtensor(fn: str, qt: "QTensor"):
    import torch

    ng = qt.k // qt.group if qt.group > 0 else 0
    _need(fn, "codes", qt.codes, torch.uint8, qt.n * qt.k * qt.q // 8)
    _need(fn, "scales", qt.scales, torch.int16, qt.n * ng)
    _need(fn, "mins", qt.mins, torch.int16, qt.n * ng, optional=qt.grid != GRID_ASYM)


def _need_status(fn: str, dev_status):
    import torch

    _need(fn, "dev_status", dev_status, torch.int32, optional=True)
    if dev_status is not None and dev_status.numel() < 1:
        raise SssError(fn, 1, "dev_status must hold one int32")


@dataclass
class QTensor:
    """A packed weight tensor: torch device buffers plus its shape metadata."""
    n: int
    k: int
    q: int
    group: int
    grid: int
    codes: "object"   # torch.uint8 [n, k*q/8]
    scales: "object"  # torch.int16 (fp16 bits) [n, k/group]
    mins: Optional["object"] = None  # torch.int16 [n, k/group] for ASYM

    def desc(self) -> QTensorDesc:
        return QTensorDesc(self.n, self.k, self.q, self.group, self.grid, 0,
                           _ptr(self.codes), _ptr(self.scales), _ptr(self.mins))

    @property
    def nbytes(self) -> int:
        b = self.codes.numel() + 2 * self.scales.numel()
        if self.mins is not None:
            b += 2 * self.mins.numel()
        return b


def empty_qtensor(n: int, k: int, q: int, group: int, grid: int, device="cuda") -> QTensor:
    import torch

    codes = torch.empty((n, k * q // 8), dtype=torch.uint8, device=device)
    scales = torch.empty((n, k // group), dtype=torch.int16, device=device)
    mins = (torch.empty((n, k // group), dtype=torch.int16, device=device)
            if grid == GRID_ASYM else None)
    return QTensor(n, k, q, group, grid, codes, scales, mins)


# ---------------------------------------------------------------------------
# entry points (same names as the C ABI)
# ---------------------------------------------------------------------------

def sss_codes_bytes(n: int, k: int, q: int) -> int:
    return int(load().sss_codes_bytes(n, k, q))


def sss_workspace_bytes(qt: QTensor, m_or_batch: int, op: int) -> int:
    d = qt.desc()
    return int(load().sss_workspace_bytes(ctypes.byref(d), m_or_batch, op))


def sss_status_string(status: int) -> str:
    return load().sss_status_string(status).decode()


def sss_quantize(w, q: int, group: int, grid: int, out: Optional[QTensor] = None,
                 clip_counts=None, dev_status=None, stream=None) -> QTensor:
    """Quantize fp32 weights w [n, k] (CUDA tensor) into a packed QTensor."""
    import torch

    n, k = w.shape
    _need("sss_quantize", "w", w, torch.float32)
    if out is None:
        out = empty_qtensor(n, k, q, group, grid, device=w.device)
    if (out.n, out.k, out.q, out.group, out.grid) != (n, k, q, group, grid):
        raise SssError("sss_quantize", 1, "out does not match w's shape, q, group and grid")
    _need_qtensor("sss_quantize", out)
    if clip_counts is not None and group > 0:
        _need("sss_quantize", "clip_counts", clip_counts, torch.uint8, n * (k // group) * 2)
    _need_status("sss_quantize", dev_status)
    _on_device("sss_quantize", w=w, codes=out.codes, scales=out.scales, mins=out.mins,
               clip_counts=clip_counts, dev_status=dev_status)
    d = out.desc()
    st = load().sss_quantize(_ptr(w), ctypes.byref(d), _ptr(clip_counts), _ptr(dev_status),
                             _stream(stream))
    _check("sss_quantize", st)
    return out


def sss_dequantize(qt: QTensor, out=None, out_dtype: int = OUT_F32, stream=None):
    import torch

    if out is None:
        dt = {OUT_F32: torch.float32, OUT_F16: torch.float16, OUT_BF16: torch.bfloat16}[out_dtype]
        out = torch.empty((qt.n, qt.k), dtype=dt, device=qt.codes.device)
    _need_qtensor("sss_dequantize", qt)
    want = {OUT_F32: torch.float32, OUT_F16: torch.float16, OUT_BF16: torch.bfloat16}.get(out_dtype)
    if want is not None:
        _need("sss_dequantize", "out", out, want, qt.n * qt.k)
    _on_device("sss_dequantize", codes=qt.codes, scales=qt.scales, mins=qt.mins, out=out)
    d = qt.desc()
    st = load().sss_dequantize(ctypes.byref(d), _ptr(out), out_dtype, _stream(stream))
    _check("sss_dequantize", st)
    return out


def sss_gemv(qt: QTensor, x, y=None, workspace=None, dev_status=None, stream=None):
    """y [batch, n] fp32 = x [batch, k] (bf16) @ dequant(qt)^T."""
    import torch

    batch = x.shape[0] if x.dim() == 2 else 1
    _need("sss_gemv", "x", x, torch.bfloat16, batch * qt.k)
    if y is None:
        y = torch.empty((batch, qt.n), dtype=torch.float32, device=x.device)
    _need("sss_gemv", "y", y, torch.float32, batch * qt.n)
    _need_qtensor("sss_gemv", qt)
    _need("sss_gemv", "workspace", workspace, torch.uint8, optional=True)
    _need_status("sss_gemv", dev_status)
    _on_device("sss_gemv", x=x, y=y, codes=qt.codes, scales=qt.scales, mins=qt.mins,
               workspace=workspace, dev_status=dev_status)
    d = qt.desc()
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    st = load().sss_gemv(ctypes.byref(d), _ptr(x), batch, _ptr(y), _ptr(workspace), ws_bytes,
                         _ptr(dev_status), _stream(stream))
    _check("sss_gemv", st)
    return y


def sss_gemv_multi(qts, x, ys=None, flags: int = 0, dev_status=None, stream=None):
    """y_j [n_j] fp32 = x [k] (bf16) @ dequant(qt_j)^T for 1..4 matrices sharing x."""
    import torch

    if ys is None:
        ys = [torch.empty((qt.n,), dtype=torch.float32, device=x.device) for qt in qts]
    if len(ys) != len(qts):
        raise SssError("sss_gemv_multi", 1, "one output per matrix")
    for qt, y in zip(qts, ys):
        _need("sss_gemv_multi", "x", x, torch.bfloat16, qt.k)
        _need("sss_gemv_multi", "y", y, torch.float32, qt.n)
        _need_qtensor("sss_gemv_multi", qt)
    _need_status("sss_gemv_multi", dev_status)
    _on_device("sss_gemv_multi", x=x, dev_status=dev_status)
    for qt, y in zip(qts, ys):
        _on_device("sss_gemv_multi", y=y, codes=qt.codes, scales=qt.scales, mins=qt.mins)
    descs = [qt.desc() for qt in qts]
    parr = (ctypes.POINTER(QTensorDesc) * len(qts))(*[ctypes.pointer(d) for d in descs])
    yarr = (ctypes.c_void_p * len(qts))(*[_ptr(y) for y in ys])
    st = load().sss_gemv_multi(parr, yarr, len(qts), _ptr(x), flags, _ptr(dev_status),
                               _stream(stream))
    _check("sss_gemv_multi", st)
    return ys


def _gemm(fn: str, qt: QTensor, x, y, workspace, dev_status, stream):
    import torch

    m = x.shape[0]
    _need(fn, "x", x, torch.bfloat16, m * qt.k)
    if y is None:
        y = torch.empty((m, qt.n), dtype=torch.float32, device=x.device)
    _need(fn, "y", y, torch.float32, m * qt.n)
    _need_qtensor(fn, qt)
    _need(fn, "workspace", workspace, torch.uint8, optional=True)
    _need_status(fn, dev_status)
    _on_device(fn, x=x, y=y, codes=qt.codes, scales=qt.scales, mins=qt.mins,
               workspace=workspace, dev_status=dev_status)
    d = qt.desc()
    if workspace is None:
        need = int(load().sss_workspace_bytes(ctypes.byref(d), m, OP_GEMM))
        if need > 0:
            workspace = torch.empty(need, dtype=torch.uint8, device=x.device)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    st = getattr(load(), fn)(ctypes.byref(d), _ptr(x), m, _ptr(y), _ptr(workspace), ws_bytes,
                             _ptr(dev_status), _stream(stream))
    _check(fn, st)
    return y


def sss_gemm(qt: QTensor, x, y=None, workspace=None, dev_status=None, stream=None):
    """Y [m, n] fp32 = X [m, k] (bf16) @ dequant(qt)^T on the tensor cores."""
    return _gemm("sss_gemm", qt, x, y, workspace, dev_status, stream)


def sss_gemm_multi_workspace_bytes(qts, m: int) -> int:
    """Workspace bytes for sss_gemm_multi over these tensors at m tokens."""
    descs = [qt.desc() for qt in qts]
    parr = (ctypes.POINTER(QTensorDesc) * len(qts))(*[ctypes.pointer(d) for d in descs])
    return int(load().sss_gemm_multi_workspace_bytes(parr, len(qts), m))


def sss_gemm_multi(qts, x, ys=None, workspace=None, dev_status=None, stream=None):
    """Y_j [m, n_j] fp32 = X [m, k] (bf16) @ dequant(qt_j)^T for 1..4 matrices
    sharing X, in one launch."""
    import torch

    fn = "sss_gemm_multi"
    m = x.shape[0]
    if ys is None:
        ys = [torch.empty((m, qt.n), dtype=torch.float32, device=x.device) for qt in qts]
    if len(ys) != len(qts):
        raise SssError(fn, 1, "one output per matrix")
    for qt, y in zip(qts, ys):
        _need(fn, "x", x, torch.bfloat16, m * qt.k)
        _need(fn, "y", y, torch.float32, m * qt.n)
        _need_qtensor(fn, qt)
        _on_device(fn, y=y, codes=qt.codes, scales=qt.scales, mins=qt.mins)
    _need(fn, "workspace", workspace, torch.uint8, optional=True)
    _need_status(fn, dev_status)
    _on_device(fn, x=x, workspace=workspace, dev_status=dev_status)
    if workspace is None:
        need = sss_gemm_multi_workspace_bytes(qts, m)
        if need > 0:
            workspace = torch.empty(need, dtype=torch.uint8, device=x.device)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    descs = [qt.desc() for qt in qts]
    parr = (ctypes.POINTER(QTensorDesc) * len(qts))(*[ctypes.pointer(d) for d in descs])
    yarr = (ctypes.c_void_p * len(qts))(*[_ptr(y) for y in ys])
    st = load().sss_gemm_multi(parr, yarr, len(qts), _ptr(x), m, _ptr(workspace), ws_bytes,
                               _ptr(dev_status), _stream(stream))
    _check(fn, st)
    return ys


def sss_gemm_q8(qt: QTensor, x, y=None, workspace=None, dev_status=None, stream=None):
    """sss_gemm with X quantized to Q8_0 (per token, per block of 32) first."""
    return _gemm("sss_gemm_q8", qt, x, y, workspace, dev_status, stream)


def sss_quantize_act_q8(x, q=None, d=None, dev_status=None, stream=None):
    """Q8_0 activations of bf16 x [rows, k]: int8 codes [rows, k] and fp16
    block scales [rows, k/32] (returned as int16 bit patterns)."""
    import torch

    rows, k = x.shape
    _need("sss_quantize_act_q8", "x", x, torch.bfloat16, rows * k)
    if q is None:
        q = torch.empty((rows, k), dtype=torch.int8, device=x.device)
    if d is None:
        d = torch.empty((rows, k // 32), dtype=torch.int16, device=x.device)
    _need("sss_quantize_act_q8", "q", q, torch.int8, rows * k)
    _need("sss_quantize_act_q8", "d", d, torch.int16, rows * (k // 32))
    _need_status("sss_quantize_act_q8", dev_status)
    _on_device("sss_quantize_act_q8", x=x, q=q, d=d, dev_status=dev_status)
    st = load().sss_quantize_act_q8(_ptr(x), rows, k, _ptr(q), _ptr(d), _ptr(dev_status),
                                    _stream(stream))
    _check("sss_quantize_act_q8", st)
    return q, d


def sss_gemm_noalloc(qt: QTensor, x, y, dev_status=None, stream=None):
    """sss_gemm with the library's static scratch instead of a workspace;
    `y` [m, n] fp32 must be given (the call allocates nothing)."""
    import torch

    m = x.shape[0]
    _need("sss_gemm_noalloc", "x", x, torch.bfloat16, m * qt.k)
    _need("sss_gemm_noalloc", "y", y, torch.float32, m * qt.n)
    _need_qtensor("sss_gemm_noalloc", qt)
    _need_status("sss_gemm_noalloc", dev_status)
    _on_device("sss_gemm_noalloc", x=x, y=y, codes=qt.codes, scales=qt.scales, mins=qt.mins,
               dev_status=dev_status)
    d = qt.desc()
    st = load().sss_gemm_noalloc(ctypes.byref(d), _ptr(x), x.shape[0], _ptr(y),
                                 _ptr(dev_status), _stream(stream))
    _check("sss_gemm_noalloc", st)
    return y


def sss_gemm_noalloc_max_scratch_bytes() -> int:
    return int(load().sss_gemm_noalloc_max_scratch_bytes())


def sss_test_set_stall(mask: int) -> None:
    """Test hook of the bounded waits (TEST_STALL_* bits; 0 restores normal
    launches): later GEMM launches leave one barrier one arrive short, so a
    wait runs out and the kernel raises FLAG_TIMEOUT.  The GEMV kernels have
    no waits; their bits have no effect."""
    load().sss_test_set_stall(int(mask))


def sss_sign_diagnostics(w, q: int, group: int, margin=None, gain=None, hist=None,
                         dev_status=None, stream=None):
    """Per-group cardinality margin (int16 [n, k/group]) and exact l2 gain
    (float64 [n, k/group]) of the signed absmax sign rule, and their
    histogram (int64 [2*group+1, 3], added to: row m + group, column g<0 /
    g==0 / g>0).  Returns (margin, gain, hist)."""
    import torch

    n, k = w.shape
    fn = "sss_sign_diagnostics"
    _need(fn, "w", w, torch.float32, n * k)
    ng = n * (k // group) if group > 0 else 0
    if margin is None:
        margin = torch.empty((n, k // group), dtype=torch.int16, device=w.device)
    if gain is None:
        gain = torch.empty((n, k // group), dtype=torch.float64, device=w.device)
    if hist is None:
        hist = torch.zeros((2 * group + 1, 3), dtype=torch.int64, device=w.device)
    _need(fn, "margin", margin, torch.int16, ng)
    _need(fn, "gain", gain, torch.float64, ng)
    _need(fn, "hist", hist, torch.int64, (2 * group + 1) * 3)
    _need_status(fn, dev_status)
    _on_device(fn, w=w, margin=margin, gain=gain, hist=hist, dev_status=dev_status)
    st = load().sss_sign_diagnostics(_ptr(w), n, k, q, group, _ptr(margin), _ptr(gain),
                                     _ptr(hist), _ptr(dev_status), _stream(stream))
    _check(fn, st)
    return margin, gain, hist


def sss_hadamard(w, block: int, side: int = ROTATE_INPUT, out=None, stream=None):
    """The normalized Hadamard rotation of fp32 w [n, k] (block b, input or
    output side) into out (new tensor if None; may be w itself)."""
    import torch

    n, k = w.shape
    _need("sss_hadamard", "w", w, torch.float32, n * k)
    if out is None:
        out = torch.empty_like(w)
    _need("sss_hadamard", "out", out, torch.float32, n * k)
    _on_device("sss_hadamard", w=w, out=out)
    st = load().sss_hadamard(_ptr(w), _ptr(out), n, k, block, side, _stream(stream))
    _check("sss_hadamard", st)
    return out


def sss_quantize_rotated(w, block: int, q: int, group: int, grid: int,
                         out: Optional["QTensor"] = None, clip_counts=None, dev_status=None,
                         stream=None) -> "QTensor":
    """sss_quantize of the input-side Hadamard rotation of w (block b), fused."""
    import torch

    n, k = w.shape
    fn = "sss_quantize_rotated"
    _need(fn, "w", w, torch.float32, n * k)
    if out is None:
        out = empty_qtensor(n, k, q, group, grid, device=w.device)
    _need_qtensor(fn, out)
    _need(fn, "clip_counts", clip_counts, torch.uint8, n * (k // group) * 2, optional=True)
    _need_status(fn, dev_status)
    _on_device(fn, w=w, codes=out.codes, scales=out.scales, mins=out.mins,
               clip_counts=clip_counts, dev_status=dev_status)
    d = out.desc()
    st = load().sss_quantize_rotated(_ptr(w), block, ctypes.byref(d), _ptr(clip_counts),
                                     _ptr(dev_status), _stream(stream))
    _check(fn, st)
    return out


def sss_quantize_lsq(w, q: int, group: int, grid: int, steps: int, lr: float,
                     out: Optional["QTensor"] = None, dev_status=None, stream=None) -> "QTensor":
    """Symmetric-grid quantization of fp32 w [n, k] with LSQ-refined scales."""
    import torch

    n, k = w.shape
    fn = "sss_quantize_lsq"
    _need(fn, "w", w, torch.float32, n * k)
    if out is None:
        out = empty_qtensor(n, k, q, group, grid, device=w.device)
    _need_qtensor(fn, out)
    _need_status(fn, dev_status)
    _on_device(fn, w=w, codes=out.codes, scales=out.scales, dev_status=dev_status)
    d = out.desc()
    st = load().sss_quantize_lsq(_ptr(w), ctypes.byref(d), int(steps), float(lr),
                                 _ptr(dev_status), _stream(stream))
    _check(fn, st)
    return out
