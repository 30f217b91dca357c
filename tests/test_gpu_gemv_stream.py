"""Parity of the streaming batch-1 GEMV (sss_gemv_multi and the batch-1
sss_gemv path) with the fp64 oracle, for single and fused multi-matrix
launches, with and without programmatic dependent launch."""
import numpy as np
import pytest

import oracle
from paper_2607_08779_gb300 import inputs, sss

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from gpu_util import REL_TOL, qtensor_from_oracle, rel_err_per_row, to_dev, x_bits  # noqa: E402

QS = (2, 3, 4)
GRIDS = (sss.GRID_UNSIGNED_SYM, sss.GRID_SIGNED_SYM, sss.GRID_ASYM)


def make(n, k, q, g, grid, seed):
    W = inputs.student_t_weights(n, k, seed)
    codes, scales, mins, _, _ = oracle.quantize(W, q, g, grid)
    return qtensor_from_oracle(codes, scales, mins, n, k, q, g, grid), (codes, scales, mins)


def check_multi(ns, k, q, g, grid, seed, flags=0):
    mats = [make(n, k, q, g, grid, seed + 31 * i) for i, n in enumerate(ns)]
    xb = x_bits(1, k, seed + 7)
    x = to_dev(xb[0].view(np.int16)).view(torch.bfloat16)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    ys = sss.sss_gemv_multi([m[0] for m in mats], x, flags=flags, dev_status=status)
    ys2 = sss.sss_gemv_multi([m[0] for m in mats], x, flags=flags)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    worst = 0.0
    for (qt, (codes, scales, mins)), y, y2, n in zip(mats, ys, ys2, ns):
        assert torch.equal(y, y2), "not deterministic"
        yref = oracle.gemv(codes, scales, mins, n, k, q, g, grid, xb)
        err = rel_err_per_row(y.cpu().numpy()[None, :], yref)
        assert err.max() <= REL_TOL, f"rel err {err.max():.3e}"
        worst = max(worst, float(err.max()))
    return worst


@pytest.mark.parametrize("grid", GRIDS)
@pytest.mark.parametrize("q", QS)
@pytest.mark.parametrize("g", [32, 64, 128])
def test_stream_single_ragged_rows(q, g, grid):
    # 100 rows: a ragged last tile; k = 2048 (8 units of 256 codes)
    check_multi([100], 2048, q, g, grid, q * 10 + g + grid)


@pytest.mark.parametrize("q", QS)
def test_stream_fused_three(q):
    """q/k/v-shaped fusion at reduced rows: three matrices, one x."""
    check_multi([512, 128, 128], 4096, q, 32, sss.GRID_SIGNED_SYM, 40 + q)


@pytest.mark.parametrize("flags", [0, sss.GEMV_PDL, sss.GEMV_PDL | sss.GEMV_WEIGHTS_READY])
def test_stream_flags(flags):
    check_multi([300, 77], 1024, 4, 32, sss.GRID_SIGNED_SYM, 9, flags=flags)


@pytest.mark.parametrize("grid", GRIDS)
def test_stream_llama_qkv_and_gate_up(grid):
    n_q, k = inputs.LLAMA3_8B_LAYER["q_proj"]
    check_multi([n_q, 1024, 1024], k, 4, 32, grid, 3)
    check_multi([14336, 14336], 4096, 4, 32, grid, 4)


@pytest.mark.parametrize("q", QS)
def test_stream_down_proj_long_k(q):
    n, k = inputs.LLAMA3_8B_LAYER["down_proj"]
    check_multi([n], k, q, 32, sss.GRID_SIGNED_SYM, 5 + q)


def test_stream_small_rows_many_tiles():
    check_multi([1, 17, 16, 33], 256, 4, 32, sss.GRID_SIGNED_SYM, 12)


def test_multi_fallback_shapes():
    """k not a multiple of 256: the multi entry falls back to per-matrix GEMVs."""
    check_multi([70, 9], 96, 4, 32, sss.GRID_ASYM, 13)
    check_multi([70], 1024 + 128, 3, 128, sss.GRID_SIGNED_SYM, 14)


def test_stream_precision_far_inside_gate():
    assert check_multi([2048], 4096, 4, 32, sss.GRID_SIGNED_SYM, 15) < 2e-5


def test_multi_rejects_mixed_shapes():
    a, _ = make(64, 256, 4, 32, sss.GRID_SIGNED_SYM, 1)
    b, _ = make(64, 512, 4, 32, sss.GRID_SIGNED_SYM, 2)
    x = torch.zeros(256, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(sss.SssError):
        sss.sss_gemv_multi([a, b], x)


@pytest.mark.parametrize("grid", GRIDS)
@pytest.mark.parametrize("q", QS)
@pytest.mark.parametrize("k,g", [(1280, 32), (2304, 128), (768, 64)])
def test_stream_k_not_multiple_of_1024(q, grid, k, g):
    """k a multiple of 256 only: units of the last stretch of a row."""
    check_multi([200, 48], k, q, g, grid, 60 + q + k)


@pytest.mark.parametrize("g", [32, 64, 128])
@pytest.mark.parametrize("grid", GRIDS)
def test_stream_ragged_jobs(g, grid):
    """Ragged tiles in every job of a fused launch, all group sizes."""
    check_multi([1000, 33, 7, 250], 3072, 4, g, grid, 70 + g + grid)
    check_multi([517], 1024, 3, g, grid, 71 + g + grid)
    check_multi([96, 1], 2048, 2, g, grid, 72 + g + grid)


def check_scaled_x(n, k, q, g, grid, seed, scale_of_chunk):
    """The GEMV with activations whose 32-element sub-chunks are scaled by
    scale_of_chunk(i) (powers of ten over many orders of magnitude, or all
    small): bf16 values the fp16 mma operand cannot hold unscaled."""
    qt, (codes, scales, mins) = make(n, k, q, g, grid, seed)
    x = inputs.bf16_bits_to_f32(x_bits(1, k, seed + 3))[0].astype(np.float64)
    x = x * np.repeat([scale_of_chunk(i) for i in range(k // 32)], 32)
    xb = inputs.f32_to_bf16_bits(x.astype(np.float32)[None, :])
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    y = sss.sss_gemv_multi([qt], to_dev(xb[0].view(np.int16)).view(torch.bfloat16),
                           dev_status=st)[0]
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    yref = oracle.gemv(codes, scales, mins, n, k, q, g, grid, xb)
    err = rel_err_per_row(y.cpu().numpy()[None, :], yref)
    assert err.max() <= REL_TOL, f"rel err {err.max():.3e}"
    return float(err.max())


@pytest.mark.parametrize("grid", GRIDS)
@pytest.mark.parametrize("q", QS)
@pytest.mark.parametrize("scale", [1e-4, 1e-6, 3e4])
def test_stream_small_and_large_activations(q, grid, scale):
    """Every element scaled alike: the result must not depend on where the
    activations sit in the fp16 range."""
    assert check_scaled_x(256, 2048, q, 32, grid, 80 + q, lambda i: scale) < 1e-4


@pytest.mark.parametrize("q", QS)
@pytest.mark.parametrize("g", [32, 128])
def test_stream_activation_scale_varies_per_chunk(q, g):
    """Sub-chunk magnitudes from 1e-8 to 1e4: the few large chunks dominate
    the dot product, the small ones must not be lost or overflow."""
    check_scaled_x(300, 4096, q, g, sss.GRID_SIGNED_SYM, 90 + q + g,
                   lambda i: 10.0 ** ((i * 7) % 13 - 8))
