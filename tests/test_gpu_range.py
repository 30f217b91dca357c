"""fp16 range of the weight operand in the batched GEMV and the GEMM.

Both kernels multiply w^ rounded to fp16 (times 2^p, p up to 4, in the
batched GEMV).  A group whose scale lets that operand reach 65520 must raise
SSS_FLAG_RANGE; every other group must give the oracle's result with no
flag.  The weights are seeded heavy-tailed rows with one group per chosen
row rescaled so its scale lands just below or above the bound.
"""
import numpy as np
import pytest

import oracle
from paper_2607_08779_gb300 import inputs, sss

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from gpu_util import REL_TOL, qtensor_from_oracle, rel_err_per_row, to_dev, x_bits  # noqa: E402

N, K, G = 64, 512, 32


def _weights(outlier, q, grid, seed):
    """Seeded rows; row 5's first group gets a negative outlier of magnitude
    `outlier` (so |s| = outlier / 2^(q-1) on the symmetric grids)."""
    W = inputs.student_t_weights(N, K, seed)
    W[5, 3] = -np.float32(outlier)
    codes, scales, mins, _, flags = oracle.quantize(W, q, G, grid)
    assert flags == 0
    return W, (codes, scales, mins)


def _bf16(bits):
    return to_dev(bits.view(np.int16)).view(torch.bfloat16)


def _gemv(pk, q, grid, batch, seed):
    codes, scales, mins = pk
    qt = qtensor_from_oracle(codes, scales, mins, N, K, q, G, grid)
    xb = x_bits(batch, K, seed)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    y = sss.sss_gemv(qt, _bf16(xb), dev_status=st)
    torch.cuda.synchronize()
    yref = oracle.gemv(codes, scales, mins, N, K, q, G, grid, xb)
    return int(st.item()), rel_err_per_row(y.cpu().numpy(), yref).max()


def _gemm(pk, q, grid, m, seed):
    codes, scales, mins = pk
    qt = qtensor_from_oracle(codes, scales, mins, N, K, q, G, grid)
    Xb = x_bits(m, K, seed)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    Y = sss.sss_gemm(qt, _bf16(Xb), dev_status=st)
    torch.cuda.synchronize()
    What = oracle.dequantize(codes, scales, mins, N, K, q, G, grid)
    Yref = oracle.matmul_f64(What, Xb)
    return int(st.item()), rel_err_per_row(Y.cpu().numpy(), Yref).max()


@pytest.mark.parametrize("q", [2, 3, 4])
def test_batched_gemv_range(q):
    grid = oracle.GRID_SIGNED_SYM
    half = 1 << (q - 1)
    # |s| * 2^(q-1) * 16 = outlier * 16: 65504 fits, 80000 does not
    for outlier, flagged in ((65504 / 16, False), (5000.0, True)):
        _, pk = _weights(outlier, q, grid, 40 + q)
        s = np.abs(pk[1].view(np.float16).astype(np.float64)).max()
        assert (s * half * 16 >= 65520) == flagged, s
        status, err = _gemv(pk, q, grid, 4, 3)
        if flagged:
            assert status & sss.FLAG_RANGE, status
        else:
            assert status == 0, status
            assert err <= REL_TOL, err


def test_batched_gemv_range_asym():
    grid = oracle.GRID_ASYM
    # min-max grid: (|s| (2^q - 1) + |m|) * 16 with m = the outlier
    _, pk = _weights(5000.0, 4, grid, 47)
    status, _ = _gemv(pk, 4, grid, 4, 5)
    assert status & sss.FLAG_RANGE, status
    _, pk = _weights(1000.0, 4, grid, 48)
    status, err = _gemv(pk, 4, grid, 4, 6)
    assert status == 0 and err <= REL_TOL, (status, err)


def test_batch1_gemv_exact_past_fp16_operand_range():
    # batch 1 applies the scale in fp32 to exact integer products: the same
    # weights that flag at batch 4 give the oracle's result and no flag
    _, pk = _weights(5000.0, 4, oracle.GRID_SIGNED_SYM, 44)
    status, err = _gemv(pk, 4, oracle.GRID_SIGNED_SYM, 1, 7)
    assert status == 0 and err <= REL_TOL, (status, err)


@pytest.mark.parametrize("q", [2, 4])
def test_gemm_range(q):
    grid = oracle.GRID_SIGNED_SYM
    # the GEMM operand is s*c itself: |s| * 2^(q-1) = outlier
    for outlier, flagged in ((5000.0, False), (65504.0, False), (70000.0, True)):
        _, pk = _weights(outlier, q, grid, 50 + q)
        status, err = _gemm(pk, q, grid, 40, 9)
        if flagged:
            assert status & sss.FLAG_RANGE, status
        else:
            assert status == 0, status
            assert err <= REL_TOL, err
