"""Parity of the tcgen05 prefill GEMM with the fp64 oracle matmul over the
dequantised weights (codes packed by the oracle).  Full-size shapes check
whole output rows (token vectors) for a few sampled tokens."""
import numpy as np
import pytest

import oracle
from paper_2607_08779_gb300 import inputs, sss

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from gpu_util import REL_TOL, qtensor_from_oracle, rel_err_per_row, to_dev  # noqa: E402

QS = (2, 3, 4)
GRIDS = (sss.GRID_UNSIGNED_SYM, sss.GRID_SIGNED_SYM, sss.GRID_ASYM)


def run_case(n, k, m, q, g, grid, seed, tokens=None, outliers=True, tol=REL_TOL):
    W = inputs.student_t_weights(n, k, seed, outliers=outliers)
    codes, scales, mins, _, _ = oracle.quantize(W, q, g, grid)
    qt = qtensor_from_oracle(codes, scales, mins, n, k, q, g, grid)
    Xb = inputs.normal_bf16_bits((m, k), seed + 1)
    X = to_dev(Xb.view(np.int16)).view(torch.bfloat16)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    Y = sss.sss_gemm(qt, X, dev_status=status)
    Y2 = sss.sss_gemm(qt, X)
    torch.cuda.synchronize()
    assert int(status.item()) == 0, "a bounded wait expired"
    assert torch.equal(Y, Y2), "GEMM is not deterministic"
    Y = Y.cpu().numpy()
    What = oracle.dequantize(codes, scales, mins, n, k, q, g, grid)
    rows = np.arange(m) if tokens is None else np.asarray(tokens)
    Yref = oracle.matmul_f64(What, Xb[rows])
    err = rel_err_per_row(Y[rows], Yref)
    assert np.all(err <= tol), f"rel err {err.max():.3e} > {tol}"
    return err.max()


@pytest.mark.parametrize("grid", GRIDS)
@pytest.mark.parametrize("q", QS)
@pytest.mark.parametrize("g", [32, 64, 128])
def test_gemm_small_ragged(q, g, grid):
    # 200 weight rows (ragged 128-row tile), 300 tokens (ragged token tile)
    run_case(200, 384, 300, q, g, grid, 13 * q + g + grid)


@pytest.mark.parametrize("m", [1, 7, 128, 129, 1100])
def test_gemm_token_counts(m):
    run_case(256, 512, m, 4, 32, sss.GRID_SIGNED_SYM, m)


@pytest.mark.parametrize("n,k", [(4, 64), (132, 64), (1024, 4096)])
def test_gemm_shapes(n, k):
    run_case(n, k, 256, 4, 32, sss.GRID_SIGNED_SYM, n + k)


@pytest.mark.parametrize("m", [512, 2048])
@pytest.mark.parametrize("name", list(inputs.LLAMA3_8B_LAYER))
def test_gemm_llama_prefill_shapes(name, m):
    """Llama3-8B layer shapes at q=4, g=32, prefill of 512 / 2048 tokens;
    whole output rows of 3 sampled tokens checked."""
    n, k = inputs.LLAMA3_8B_LAYER[name]
    toks = np.random.default_rng(m).choice(m, 3, replace=False)
    run_case(n, k, m, 4, 32, sss.GRID_SIGNED_SYM,
             inputs.weight_seed(3, 0, inputs.MATRIX_IDS[name]), tokens=toks)


def test_gemm_fp16_tile_precision():
    """fp16 weight tiles round s*c by <= 2^-11: the output error stays
    several times inside the 1e-3 gate."""
    e = run_case(1024, 4096, 256, 4, 32, sss.GRID_SIGNED_SYM, 5)
    assert e < 4e-4
