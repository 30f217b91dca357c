"""Q8_0 activations on the GPU (the paper's runtime pairing of the few-bit
weight formats with 8-bit activations, Sec. 5 "Composition with PTQ
methods", Appendix C): the standalone quantizer bit-exact with the oracle,
the GEMV that quantizes x while staging it, and the Q8_0 prefill GEMM,
both against the oracle's fp64 product over the same Q8_0 values."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import REL_TOL, qtensor_from_oracle, rel_err_per_row, to_dev, x_bits
from paper_2607_08779_gb300 import inputs, sss

pytestmark = pytest.mark.gpu

QS = (2, 3, 4)
GRIDS = (sss.GRID_UNSIGNED_SYM, sss.GRID_SIGNED_SYM, sss.GRID_ASYM)


def _x(bits):
    return to_dev(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)


def special_blocks(k=32 * 12):
    """Rows of bf16 activations whose blocks hit every case of the format:
    N(0,1), zeros, exact ties of x/d, a lone outlier, tiny and huge scales,
    NaN / Inf (non-finite) and a block whose d overflows fp16."""
    rng = np.random.default_rng(3)
    x = rng.standard_normal((3, k)).astype(np.float32)
    b = x[1].reshape(-1, 32)
    b[0] = 0.0                                     # zero block
    b[1] = np.arange(-16, 16) / 16.0                # M = 1: x/d near many half-integers
    b[1][0] = -1.0
    b[2] = 0.0
    b[2][5] = 3.0                                  # one outlier, the rest zero
    b[3] *= 1e-30                                  # tiny
    b[4] *= 1e30                                   # huge: d overflows fp16 (RANGE)
    b[5][7] = np.nan                               # non-finite
    b[6][3] = np.inf
    b[7] = np.array([127, 63.5, -63.5, 0.5, -0.5, 1.5, 2.5, -2.5] * 4, np.float32)  # d = 1: exact ties
    return inputs.f32_to_bf16_bits(x)


@pytest.mark.parametrize("rows,k", [(1, 4096), (7, 1024), (3, 14336)])
def test_quantize_act_q8_matches_oracle(rows, k):
    xb = x_bits(rows, k, 100 + rows)
    q_ref, d_ref, f_ref = oracle.quantize_act_q8(xb)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    q, d = sss.sss_quantize_act_q8(_x(xb), dev_status=st)
    torch.cuda.synchronize()
    assert np.array_equal(q.cpu().numpy(), q_ref)
    assert np.array_equal(d.cpu().numpy().view(np.uint16), d_ref)
    assert int(st.item()) == f_ref


def test_quantize_act_q8_special_blocks():
    xb = special_blocks()
    q_ref, d_ref, f_ref = oracle.quantize_act_q8(xb)
    assert f_ref & oracle.FLAG_NONFINITE and f_ref & oracle.FLAG_RANGE
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    q, d = sss.sss_quantize_act_q8(_x(xb), dev_status=st)
    torch.cuda.synchronize()
    assert np.array_equal(q.cpu().numpy(), q_ref)
    assert np.array_equal(d.cpu().numpy().view(np.uint16), d_ref)
    assert int(st.item()) == f_ref


def _gemv_q8_case(ns, k, q, g, grid, seed, flags=0):
    mats = []
    for i, n in enumerate(ns):
        W = inputs.student_t_weights(n, k, seed + 13 * i)
        codes, scales, mins, _, _ = oracle.quantize(W, q, g, grid)
        mats.append((qtensor_from_oracle(codes, scales, mins, n, k, q, g, grid),
                     (codes, scales, mins)))
    xb = x_bits(1, k, seed + 5)
    xq, xd, _ = oracle.quantize_act_q8(xb)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    ys = sss.sss_gemv_multi([m[0] for m in mats], _x(xb)[0], dev_status=st,
                            flags=flags | sss.GEMV_ACT_Q8)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    worst = 0.0
    for (qt, (codes, scales, mins)), y, n in zip(mats, ys, ns):
        yref = oracle.gemv_q8(codes, scales, mins, n, k, q, g, grid, xq, xd)
        err = rel_err_per_row(y.cpu().numpy()[None, :], yref)
        assert err.max() <= REL_TOL, f"rel err {err.max():.3e}"
        worst = max(worst, float(err.max()))
    return worst


@pytest.mark.parametrize("grid", GRIDS)
@pytest.mark.parametrize("q", QS)
@pytest.mark.parametrize("g", [32, 128])
def test_gemv_act_q8_matches_oracle(q, g, grid):
    # the integer dot of codes and Q8_0 values is exact: far inside the gate
    assert _gemv_q8_case([300, 45], 2048, q, g, grid, 200 + q + g + grid) < 1e-5


@pytest.mark.parametrize("q", QS)
def test_gemv_act_q8_llama_shapes(q):
    n_q, k = inputs.LLAMA3_8B_LAYER["q_proj"]
    _gemv_q8_case([n_q, 1024, 1024], k, q, 32, sss.GRID_SIGNED_SYM, 210 + q,
                  flags=sss.GEMV_PDL | sss.GEMV_WEIGHTS_READY)
    n, k = inputs.LLAMA3_8B_LAYER["down_proj"]
    _gemv_q8_case([n], k, q, 32, sss.GRID_SIGNED_SYM, 220 + q)


def test_gemv_act_q8_special_blocks_flags():
    k = 512  # the streaming kernel takes k % 256 == 0
    xb = special_blocks(k)[1:2]
    W = inputs.student_t_weights(64, k, 9)
    codes, scales, mins, _, _ = oracle.quantize(W, 4, 32, oracle.GRID_SIGNED_SYM)
    qt = qtensor_from_oracle(codes, scales, mins, 64, k, 4, 32, oracle.GRID_SIGNED_SYM)
    _, _, f_ref = oracle.quantize_act_q8(xb)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    sss.sss_gemv_multi([qt], _x(xb)[0], dev_status=st, flags=sss.GEMV_ACT_Q8)
    torch.cuda.synchronize()
    assert int(st.item()) == f_ref


def test_gemv_act_q8_unsupported_shape():
    k = 96  # not a multiple of 256: the general kernels take bf16 only
    W = inputs.student_t_weights(16, k, 2)
    codes, scales, mins, _, _ = oracle.quantize(W, 4, 32, oracle.GRID_SIGNED_SYM)
    qt = qtensor_from_oracle(codes, scales, mins, 16, k, 4, 32, oracle.GRID_SIGNED_SYM)
    with pytest.raises(sss.SssError):
        sss.sss_gemv_multi([qt], _x(x_bits(1, k, 1))[0], flags=sss.GEMV_ACT_Q8)


@pytest.mark.parametrize("grid", GRIDS)
@pytest.mark.parametrize("m", [1, 130])
def test_gemm_q8_matches_oracle(grid, m):
    n, k, q, g = 256, 1024, 4, 32
    W = inputs.student_t_weights(n, k, 230 + m + grid)
    codes, scales, mins, _, _ = oracle.quantize(W, q, g, grid)
    qt = qtensor_from_oracle(codes, scales, mins, n, k, q, g, grid)
    Xb = x_bits(m, k, 240 + m)
    xq, xd, _ = oracle.quantize_act_q8(Xb)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    Y = sss.sss_gemm_q8(qt, _x(Xb), dev_status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    Yref = oracle.gemv_q8(codes, scales, mins, n, k, q, g, grid, xq, xd)
    err = rel_err_per_row(Y.cpu().numpy(), Yref)
    assert err.max() <= REL_TOL, f"rel err {err.max():.3e}"


def test_gemm_q8_llama_gate_m512():
    n, k = inputs.LLAMA3_8B_LAYER["gate_proj"]
    W = inputs.student_t_weights(n, k, inputs.weight_seed(3, 0, 4))
    qt = sss.sss_quantize(to_dev(W), 4, 32, sss.GRID_SIGNED_SYM)
    Xb = x_bits(512, k, 250)
    Y = sss.sss_gemm_q8(qt, _x(Xb)).cpu().numpy()
    # sampled rows of the output, checked one by one
    rows = np.random.default_rng(1).choice(n, 64, replace=False)
    codes = qt.codes.cpu().numpy()[rows]
    scales = qt.scales.cpu().numpy().view(np.uint16)[rows]
    xq, xd, _ = oracle.quantize_act_q8(Xb)
    Yref = oracle.gemv_q8(codes, scales, None, len(rows), k, 4, 32, oracle.GRID_SIGNED_SYM, xq, xd)
    err = rel_err_per_row(Y[:, rows], Yref)
    assert err.max() <= REL_TOL, f"rel err {err.max():.3e}"
