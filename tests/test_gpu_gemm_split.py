"""Parity of the GEMM's split-K path with the fp64 oracle.

When the output tiles leave SMs idle, sss_gemm splits K over CTAs (with a
workspace of sss_workspace_bytes) and the tile's last split sums the
partials in split order.  These shapes force 2, 4, 8 and 16 splits, ragged
row and token tiles, and a k whose k-blocks do not divide evenly among the
splits; run_case also checks that two calls give the same bits.  A
workspace that holds only the fp16 copy of X runs the same call unsplit,
and must agree within the tolerance.
"""
import numpy as np
import pytest

import oracle
from paper_2607_08779_gb300 import inputs, sss

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from gpu_util import REL_TOL, qtensor_from_oracle, rel_err_per_row, to_dev  # noqa: E402
from test_gpu_gemm import run_case  # noqa: E402


@pytest.mark.parametrize("n,k,m", [
    (1024, 4096, 512),   # k/v projection at 512 tokens: 32 tiles, 4 splits
    (300, 1088, 140),    # 6 ragged tiles, 17 k-blocks: splits of 9 and 8
    (128, 8192, 64),     # one tile, 128 k-blocks: 16 splits of 8
    (640, 2048, 300),    # 15 ragged tiles, 32 k-blocks
])
@pytest.mark.parametrize("q", [2, 3, 4])
def test_gemm_split_k_matches_oracle(n, k, m, q):
    run_case(n, k, m, q, 32, sss.GRID_SIGNED_SYM, n + k + m + q)


@pytest.mark.parametrize("grid", [sss.GRID_UNSIGNED_SYM, sss.GRID_ASYM])
def test_gemm_split_k_other_grids(grid):
    run_case(1024, 4096, 512, 4, 32, grid, 71 + grid)


def test_gemm_split_k_wide_tiles_down_proj():
    # down_proj at 512 tokens: 64 tiles of 256 tokens, 2 splits of 112
    # k-blocks; whole output rows of three tokens
    n, k = inputs.LLAMA3_8B_LAYER["down_proj"]
    run_case(n, k, 512, 4, 32, sss.GRID_SIGNED_SYM, 77, tokens=[0, 257, 511])


def test_gemm_minimal_workspace_runs_unsplit():
    n, k, m, q, g = 1024, 4096, 512, 4, 32
    W = inputs.student_t_weights(n, k, 81)
    codes, scales, mins, _, _ = oracle.quantize(W, q, g, oracle.GRID_SIGNED_SYM)
    qt = qtensor_from_oracle(codes, scales, mins, n, k, q, g, oracle.GRID_SIGNED_SYM)
    Xb = inputs.normal_bf16_bits((m, k), 82)
    X = to_dev(Xb.view(np.int16)).view(torch.bfloat16)
    full = sss.sss_workspace_bytes(qt, m, sss.OP_GEMM)
    small = m * k * 2
    assert full > small  # this shape splits K when the workspace allows it
    outs = []
    for nb in (full, small):
        ws = torch.empty(nb, dtype=torch.uint8, device="cuda")
        st = torch.zeros(1, dtype=torch.int32, device="cuda")
        outs.append(sss.sss_gemm(qt, X, workspace=ws, dev_status=st))
        torch.cuda.synchronize()
        assert int(st.item()) == 0
    toks = [0, 100, 511]
    What = oracle.dequantize(codes, scales, mins, n, k, q, g, oracle.GRID_SIGNED_SYM)
    Yref = oracle.matmul_f64(What, Xb[toks])
    for Y in outs:
        assert rel_err_per_row(Y.cpu().numpy()[toks], Yref).max() <= REL_TOL
    assert rel_err_per_row(outs[0].cpu().numpy(), outs[1].cpu().numpy()).max() <= REL_TOL
