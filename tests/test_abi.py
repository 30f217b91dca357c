"""The C-ABI library builds, loads without a GPU, and exports every entry
point include/sss.h declares; host-side argument checks return the documented
status codes before any CUDA call (no compute calls here)."""
import ctypes
import os
import re

import pytest

from paper_2607_08779_gb300 import sss

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    names = []
    for h in sorted(os.listdir(os.path.join(ROOT, "include"))):
        if not h.endswith(".h"):
            continue
        text = open(os.path.join(ROOT, "include", h)).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        names += re.findall(r"\b(sss_[a-z0-9_]+)\s*\(", text)
    return sorted(set(names))


def test_library_builds_and_exports_every_declared_symbol():
    L = sss.load()
    decl = declared_functions()
    assert len(decl) >= 8
    for name in decl:
        assert hasattr(L, name), f"{name} declared in include/ but not exported"
    assert set(sss.EXPORTS) <= set(decl)


def test_pure_host_helpers():
    assert sss.sss_codes_bytes(4096, 4096, 4) == 4096 * 4096 // 2
    assert sss.sss_codes_bytes(4096, 4096, 3) == 4096 * 4096 * 3 // 8
    assert sss.sss_codes_bytes(-1, 4, 4) == 0
    assert sss.sss_status_string(0) == "SSS_OK"
    assert "ARG" in sss.sss_status_string(1)


def _desc(n=64, k=256, q=4, g=32, grid=1, codes=16, scales=16, mins=0):
    return sss.QTensorDesc(n, k, q, g, grid, 0, codes, scales, mins)


@pytest.mark.parametrize("kw,want", [
    (dict(q=5), 1), (dict(q=1), 1), (dict(g=48), 1), (dict(g=256), 1),
    (dict(grid=3), 1), (dict(k=100), 1), (dict(n=-1), 1), (dict(codes=0), 1),
    (dict(grid=2, mins=0), 1),
])
def test_quantize_rejects_bad_arguments(kw, want):
    L = sss.load()
    d = _desc(**kw)
    st = L.sss_quantize(ctypes.c_void_p(4096), ctypes.byref(d), None, None, None)
    assert st == want


def test_alignment_checks():
    L = sss.load()
    d = _desc()
    assert L.sss_quantize(ctypes.c_void_p(4100), ctypes.byref(d), None, None, None) == 3
    d2 = _desc(codes=24)
    assert L.sss_gemv(ctypes.byref(d2), ctypes.c_void_p(4096), 1, ctypes.c_void_p(4096),
                      None, 0, None, None) == 3


def test_gemv_gemm_argument_checks():
    L = sss.load()
    d = _desc()
    x = ctypes.c_void_p(4096)
    y = ctypes.c_void_p(8192)
    assert L.sss_gemv(ctypes.byref(d), x, 0, y, None, 0, None, None) == 1
    assert L.sss_gemv(ctypes.byref(d), x, 17, y, None, 0, None, None) == 1
    assert L.sss_gemv(ctypes.byref(d), None, 1, y, None, 0, None, None) == 1
    assert L.sss_gemm(ctypes.byref(d), x, -1, y, None, 0, None, None) == 1
    # empty problems are no-ops that touch nothing
    d0 = _desc(n=0)
    assert L.sss_gemv(ctypes.byref(d0), x, 1, y, None, 0, None, None) == 0
    assert L.sss_gemm(ctypes.byref(d), x, 0, y, None, 0, None, None) == 0
    assert L.sss_quantize(ctypes.c_void_p(4096), ctypes.byref(_desc(n=0)), None, None, None) == 0


def test_gemm_multi_argument_checks():
    L = sss.load()
    P = ctypes.POINTER(sss.QTensorDesc)

    def call(descs, ys, m=64, x=4096, ws=None, ws_bytes=0, count=None):
        parr = (P * max(len(descs), 1))(*[ctypes.pointer(d) for d in descs])
        yarr = (ctypes.c_void_p * max(len(ys), 1))(*ys)
        n = len(descs) if count is None else count
        return L.sss_gemm_multi(parr, yarr, n, ctypes.c_void_p(x), m, ws, ws_bytes, None, None)

    a, b = _desc(n=64), _desc(n=32)
    ys = [8192, 16384]
    assert call([a, b], ys, count=0) == 1
    assert call([a, b], ys, count=5) == 1
    assert call([a, _desc(k=512)], ys) == 1           # k differs
    assert call([a, _desc(q=2)], ys) == 1             # q differs
    assert call([a, _desc(grid=0)], ys) == 1          # grid differs
    assert call([a, _desc(n=30)], ys) == 2            # n % 4 != 0
    assert call([a, b], [8192, 16388]) == 3           # y not 16-byte aligned
    assert call([a, b], ys, x=4104) == 3              # x not 16-byte aligned
    assert call([a, b], ys, m=-1) == 1
    assert call([a, b], ys) == 5                      # no workspace for the fp16 X
    # empty calls touch nothing
    assert call([a, b], ys, m=0) == 0
    assert call([_desc(n=0), _desc(n=0)], [0, 0]) == 0
    # sizing: at least the fp16 copy of X; 0 for a bad call
    parr = (P * 2)(ctypes.pointer(a), ctypes.pointer(b))
    assert L.sss_gemm_multi_workspace_bytes(parr, 2, 64) >= 64 * 256 * 2
    assert L.sss_gemm_multi_workspace_bytes(parr, 0, 64) == 0
    assert L.sss_gemm_multi_workspace_bytes(parr, 2, -1) == 0


def test_gemm_workspace_follows_the_tile_plan():
    # The workspace holds the fp16 X, plus the split-K partial tiles when the
    # preferred plan splits K (the plan depends only on shapes and the SM
    # count; without a GPU the library assumes 148 SMs, which gives the same
    # plans here as the GB300's 152).
    L = sss.load()
    P = ctypes.POINTER(sss.QTensorDesc)
    m, k = 512, 4096
    x16 = m * k * 2

    def ws(*ns):
        ds = [_desc(n=n, k=k) for n in ns]
        parr = (P * len(ds))(*[ctypes.pointer(d) for d in ds])
        return L.sss_gemm_multi_workspace_bytes(parr, len(ds), m)

    # fused q/k/v: 48 row tiles; 256-token tiles make 96 CTAs in one wave,
    # 128-token ones would need two, so it runs unsplit
    assert ws(4096, 1024, 1024) == x16
    # k_proj alone: 32 CTAs of 128-token tiles, K split over the idle SMs
    assert ws(1024) > x16
    # the one-matrix helper agrees with the multi one
    d = _desc(n=1024, k=k)
    assert L.sss_workspace_bytes(ctypes.byref(d), m, sss.OP_GEMM) == ws(1024)


def test_binding_checks_what_a_pointer_cannot_carry():
    """The Python binding rejects tensors the C ABI would misread (wrong
    dtype, strided, wrong element count, host memory) with SSS_E_ARG before
    any call into the library."""
    torch = pytest.importorskip("torch")
    n, k = 16, 256
    qt = sss.empty_qtensor(n, k, 4, 32, sss.GRID_SIGNED_SYM, device="cpu")
    x = torch.zeros((2, k), dtype=torch.bfloat16)
    y = torch.zeros((2, n), dtype=torch.float32)
    cases = [
        (lambda: sss.sss_gemv(qt, x.float(), y=y), "bfloat16"),
        (lambda: sss.sss_gemv(qt, torch.zeros((k, 2), dtype=torch.bfloat16).t(), y=y),
         "contiguous"),
        (lambda: sss.sss_gemv(qt, torch.zeros((2, 128), dtype=torch.bfloat16), y=y),
         "elements"),
        (lambda: sss.sss_gemv(qt, x, y=torch.zeros((2, n + 1))), "elements"),
        (lambda: sss.sss_gemv(qt, x, y=y), "CUDA"),
        (lambda: sss.sss_gemv_multi([qt], x[0], ys=[y[0].double()]), "float32"),
        (lambda: sss.sss_gemm(qt, x, y=y.int()), "float32"),
        (lambda: sss.sss_quantize(torch.zeros((n, k), dtype=torch.float64), 4, 32,
                                  sss.GRID_SIGNED_SYM), "float32"),
        (lambda: sss.sss_quantize(torch.zeros((n, k)), 4, 32, sss.GRID_SIGNED_SYM,
                                  out=sss.empty_qtensor(n, k, 3, 32, sss.GRID_SIGNED_SYM,
                                                        device="cpu")), "out"),
        (lambda: sss.sss_dequantize(qt, out=torch.zeros((n, k), dtype=torch.float16)),
         "float32"),
        (lambda: sss.sss_gemm_noalloc(qt, x, y[:1]), "elements"),
    ]
    for call, what in cases:
        with pytest.raises(sss.SssError) as e:
            call()
        assert e.value.status == 1 and what in str(e.value), str(e.value)
    # a min-max tensor needs its mins
    asym = sss.empty_qtensor(n, k, 4, 32, sss.GRID_ASYM, device="cpu")
    asym.mins = None
    with pytest.raises(sss.SssError, match="mins"):
        sss.sss_gemv(asym, x, y=y)
