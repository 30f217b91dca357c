"""Parity of the CUDA quantizer with the CPU oracle: packed codes, fp16
scales, fp16 mins, clip counts and status bits must match bit for bit."""
import numpy as np
import pytest

import oracle
from paper_2607_08779_gb300 import inputs, sss

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from gpu_util import gpu_quantize  # noqa: E402

QS = (2, 3, 4)
GRIDS = (sss.GRID_UNSIGNED_SYM, sss.GRID_SIGNED_SYM, sss.GRID_ASYM)


def assert_same(W, q, g, grid, rows=None):
    qt, cc, st = gpu_quantize(W, q, g, grid)
    Wc = W if rows is None else W[rows]
    codes, scales, mins, clip, flags = oracle.quantize(Wc, q, g, grid, clip_counts=True)
    gc = qt.codes.cpu().numpy()
    gs = qt.scales.cpu().numpy().view(np.uint16)
    if rows is not None:
        gc, gs = gc[rows], gs[rows]
        cc = cc[rows]
    bad = None
    if flags & oracle.FLAG_NONFINITE:
        # groups holding NaN/Inf: placeholder codes/scale must match, the
        # stored minimum is unspecified
        bad = ~np.isfinite(Wc.reshape(-1, g)).all(axis=1)
    np.testing.assert_array_equal(gc, codes)
    np.testing.assert_array_equal(gs, scales)
    if grid == sss.GRID_ASYM:
        gm = qt.mins.cpu().numpy().view(np.uint16)
        if rows is not None:
            gm = gm[rows]
        if bad is not None:
            gm = gm.reshape(-1)[~bad]
            mins = mins.reshape(-1)[~bad]
        np.testing.assert_array_equal(gm, mins)
    np.testing.assert_array_equal(cc, clip)
    if rows is None:
        assert st == flags


@pytest.mark.parametrize("grid", GRIDS)
@pytest.mark.parametrize("q", QS)
@pytest.mark.parametrize("g", [32, 64, 128])
def test_quantize_small_ragged(q, g, grid):
    # 37 rows x 5 groups: the group count is not a multiple of any sweep width
    W = inputs.student_t_weights(37, 5 * g, 100 + q * 7 + g)
    assert_same(W, q, g, grid)


@pytest.mark.parametrize("grid", GRIDS)
@pytest.mark.parametrize("q", QS)
def test_quantize_4096_square(q, grid):
    """The 4096x4096 fp32 Student-t matrix at g=32 (the small benchmark case)."""
    W = inputs.student_t_weights(4096, 4096, 1, outliers=False)
    assert_same(W, q, 32, grid)


@pytest.mark.parametrize("q", QS)
def test_quantize_llama_gate_shape(q):
    W = inputs.student_t_weights(14336, 4096, inputs.weight_seed(2, 0, 4))
    assert_same(W, q, 32, sss.GRID_SIGNED_SYM)


@pytest.mark.parametrize("q,g", [(2, 32), (2, 128), (3, 32), (3, 128)])
def test_quantize_qwen_down_shape_sampled(q, g):
    """Qwen3-32B down_proj shape (5120 x 25600): all rows on the GPU, a
    random sample of rows checked against the oracle."""
    W = inputs.student_t_weights(5120, 25600, inputs.weight_seed(4, 0, 6))
    rows = np.sort(np.random.default_rng(q * g).choice(5120, 96, replace=False))
    assert_same(W, q, g, sss.GRID_SIGNED_SYM, rows=rows)


def special_groups(g):
    rng = np.random.default_rng(5)
    out = []
    base = inputs.student_t_weights(8, g, 9)
    out.append(np.zeros(g))                          # M = 0
    z = np.zeros(g); z[3] = -0.0; z[5] = 0.0; out.append(z)
    t = base[0].copy(); t[0] = 1.0; t[1] = -1.0; out.append(t * 0.5)  # sign tie
    lat = rng.integers(-16, 17, g) / 16.0; lat[0] = 1.0; out.append(lat)  # exact ties
    lat2 = rng.integers(-16, 17, g) / 16.0; lat2[1] = -1.0; out.append(lat2)
    for e in (-140, -130, -126, -100, -97, 97, 100, 120):
        out.append(base[1] * 2.0 ** e)              # subnormal / tiny / huge
    for j in (1, 2, 3, 4, 5):                        # M = j * 2^-149: alpha may round to 0
        t = np.zeros(g); t[2] = j * 2.0 ** -149; t[9] = -2.0 ** -149
        out.append(t)
        out.append(-t)
    out.append(np.full(g, 0.375))                    # constant group
    out.append(base[2] * 1e6)                        # fp16 scale overflow
    return np.stack(out).astype(np.float32)


@pytest.mark.parametrize("grid", GRIDS)
@pytest.mark.parametrize("q", QS)
@pytest.mark.parametrize("g", [32, 128])
def test_quantize_special_groups(q, g, grid):
    W = special_groups(g)
    assert_same(W, q, g, grid)


@pytest.mark.parametrize("grid", GRIDS)
def test_quantize_nonfinite_flag(grid):
    W = inputs.student_t_weights(4, 64, 3)
    W[1, 7] = np.nan
    W[2, 40] = np.inf
    assert_same(W, 4, 32, grid)
    _, _, st = gpu_quantize(W, 4, 32, grid)
    assert st & sss.FLAG_NONFINITE


def test_quantize_empty():
    w = torch.zeros((0, 64), device="cuda")
    qt = sss.sss_quantize(w, 4, 32, sss.GRID_SIGNED_SYM)
    torch.cuda.synchronize()
    assert qt.codes.numel() == 0


def test_quantize_is_deterministic():
    W = inputs.student_t_weights(256, 1024, 4)
    a, _, _ = gpu_quantize(W, 3, 32, sss.GRID_SIGNED_SYM)
    b, _, _ = gpu_quantize(W, 3, 32, sss.GRID_SIGNED_SYM)
    assert torch.equal(a.codes, b.codes) and torch.equal(a.scales, b.scales)


@pytest.mark.parametrize("grid", GRIDS)
@pytest.mark.parametrize("q", QS)
def test_dequantize_matches_oracle(q, grid):
    W = inputs.student_t_weights(48, 512, 12 + q)
    codes, scales, mins, _, _ = oracle.quantize(W, q, 32, grid)
    from gpu_util import qtensor_from_oracle
    qt = qtensor_from_oracle(codes, scales, mins, 48, 512, q, 32, grid)
    ref = oracle.dequantize(codes, scales, mins, 48, 512, q, 32, grid)
    got = sss.sss_dequantize(qt, out_dtype=sss.OUT_F32).cpu().numpy()
    np.testing.assert_array_equal(got.view(np.uint32), ref.view(np.uint32))
    got16 = sss.sss_dequantize(qt, out_dtype=sss.OUT_F16).cpu().numpy()
    np.testing.assert_array_equal(got16.view(np.uint16), ref.astype(np.float16).view(np.uint16))
    gotb = sss.sss_dequantize(qt, out_dtype=sss.OUT_BF16).cpu()
    refb = torch.from_numpy(ref).to(torch.bfloat16)
    assert torch.equal(gotb.view(torch.int16), refb.view(torch.int16))
