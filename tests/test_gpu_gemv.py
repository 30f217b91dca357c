"""Parity of the CUDA decode GEMV with the fp64 oracle GEMV over the same
packed codes (packed by the oracle, so no input comes from the CUDA path)."""
import numpy as np
import pytest

import oracle
from paper_2607_08779_gb300 import inputs, sss

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from gpu_util import REL_TOL, qtensor_from_oracle, rel_err_per_row, to_dev, x_bits  # noqa: E402

QS = (2, 3, 4)
GRIDS = (sss.GRID_UNSIGNED_SYM, sss.GRID_SIGNED_SYM, sss.GRID_ASYM)


def run_case(n, k, q, g, grid, batch, seed, rows=None, outliers=True, tol=REL_TOL):
    W = inputs.student_t_weights(n, k, seed, outliers=outliers)
    codes, scales, mins, _, _ = oracle.quantize(W, q, g, grid)
    qt = qtensor_from_oracle(codes, scales, mins, n, k, q, g, grid)
    xb = x_bits(batch, k, seed + 1)
    x = to_dev(xb.view(np.int16)).view(torch.bfloat16)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    y = sss.sss_gemv(qt, x, dev_status=st)
    y2 = sss.sss_gemv(qt, x, dev_status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0, f"device status {int(st.item()):#x}"
    assert torch.equal(y, y2), "GEMV is not deterministic"
    y = y.cpu().numpy()
    if rows is None:
        yref = oracle.gemv(codes, scales, mins, n, k, q, g, grid, xb)
    else:
        r0, nr = rows
        yref = oracle.gemv(codes[r0:r0 + nr], scales[r0:r0 + nr],
                           None if mins is None else mins[r0:r0 + nr], nr, k, q, g, grid, xb)
        y = y[:, r0:r0 + nr]
    err = rel_err_per_row(y, yref)
    assert np.all(err <= tol), f"rel err {err.max():.3e} > {tol}"
    return err.max()


@pytest.mark.parametrize("grid", GRIDS)
@pytest.mark.parametrize("q", QS)
@pytest.mark.parametrize("g", [32, 64, 128])
def test_gemv_small_ragged(q, g, grid):
    # 75 rows (not a multiple of the 32-row tile), 11 groups per row (not a
    # multiple of the 8-group step)
    run_case(75, 11 * g, q, g, grid, 1, 7 * q + g)


@pytest.mark.parametrize("q", QS)
@pytest.mark.parametrize("n,k", [(1, 32), (16, 64), (33, 96), (128, 4096), (40, 4096 + 256)])
def test_gemv_shapes(q, n, k):
    run_case(n, k, q, 32, sss.GRID_SIGNED_SYM, 1, n + k + q)


@pytest.mark.parametrize("batch", [2, 3, 4, 5, 8, 13, 16])
@pytest.mark.parametrize("grid", GRIDS)
def test_gemv_batched(batch, grid):
    run_case(70, 1024 + 96, 4, 32, grid, batch, 3 * batch + grid)


@pytest.mark.parametrize("q", [2, 3])
@pytest.mark.parametrize("batch", [4, 16])
def test_gemv_batched_q(q, batch):
    run_case(64, 2048, q, 128, sss.GRID_ASYM, batch, 11 + q)


@pytest.mark.parametrize("batch", [5, 9, 16])
@pytest.mark.parametrize("q,grid", [(4, sss.GRID_SIGNED_SYM), (3, sss.GRID_ASYM), (2, sss.GRID_UNSIGNED_SYM)])
def test_gemv_batched_long_k_slabs(q, grid, batch):
    # k = 14336 (the down_proj width): at batch > 8 the staged activations
    # of all 56 units exceed shared memory, so the batched kernel runs the k
    # range in several slabs and adds each slab's result into y; 100 rows is
    # not a multiple of the 16-row tile
    run_case(100, 14336, q, 32, grid, batch, 900 + 10 * q + batch)


@pytest.mark.parametrize("batch", [2, 3, 8, 13])
@pytest.mark.parametrize("g", [32, 64, 128])
def test_gemv_batched_ragged_rows(g, batch):
    run_case(75, 2048, 4, g, sss.GRID_SIGNED_SYM, batch, 40 + g + batch)


@pytest.mark.parametrize("batch", [1, 16])
def test_gemv_qwen_down_width(batch):
    # the widest reduction of the configs (Qwen3-32B down_proj, k = 25600):
    # 100 units per row for the batch-1 kernel, eight x slabs for the
    # batched one; 264 rows (a ragged last tile), every output checked
    k = inputs.QWEN3_32B_LAYER["down_proj"][1]
    run_case(264, k, 2, 32, sss.GRID_SIGNED_SYM, batch, 4242 + batch)


def test_gemv_4096_square_q4_signed():
    """The 4096x4096 q=4 g=32 signed-symmetric case, every output checked."""
    run_case(4096, 4096, 4, 32, sss.GRID_SIGNED_SYM, 1, 1, outliers=False)


@pytest.mark.parametrize("q", QS)
@pytest.mark.parametrize("name", ["q_proj", "k_proj", "gate_proj", "down_proj"])
def test_gemv_llama_layer_shapes(q, name):
    n, k = inputs.LLAMA3_8B_LAYER[name]
    run_case(n, k, q, 32, sss.GRID_SIGNED_SYM, 1, inputs.weight_seed(2, 0, inputs.MATRIX_IDS[name]))


@pytest.mark.parametrize("grid", GRIDS)
@pytest.mark.parametrize("q", QS)
@pytest.mark.parametrize("g", [32, 128])
@pytest.mark.parametrize("batch", [1, 4, 16])
def test_gemv_grid_sweep_sampled(q, g, grid, batch):
    """The grid-comparison sweep shapes (4096 x 4096), rows sampled."""
    run_case(4096, 4096, q, g, grid, batch, 500 + q + g + grid, rows=(1000, 96))


def test_gemv_precision_is_far_inside_the_gate():
    """Products of integer codes and fp16 activations are exact; only the
    fp32 accumulation rounds, so the error sits orders below 1e-3."""
    e = run_case(1024, 4096, 4, 32, sss.GRID_SIGNED_SYM, 1, 77)
    assert e < 2e-5


def test_gemv_empty_k_and_n():
    qt = sss.empty_qtensor(0, 64, 4, 32, sss.GRID_SIGNED_SYM)
    x = torch.zeros((1, 64), dtype=torch.bfloat16, device="cuda")
    y = sss.sss_gemv(qt, x)
    assert y.shape == (1, 0)
