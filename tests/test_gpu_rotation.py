"""Normalized Hadamard rotation of the weights before quantization (Sec. 5
"Composition with PTQ methods", Appendix C rotation graph): the GPU
rotation is bit-exact with the oracle's fp32 fast transform on both sides,
and the fused rotate-and-quantize gives exactly the oracle's quantization of
the oracle-rotated weights."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import to_dev
from paper_2607_08779_gb300 import inputs, sss

pytestmark = pytest.mark.gpu

QS = (2, 3, 4)
GRIDS = (sss.GRID_UNSIGNED_SYM, sss.GRID_SIGNED_SYM, sss.GRID_ASYM)


@pytest.mark.parametrize("b", [2, 32, 128, 1024, 4096, 8192])
def test_rotate_rows_bit_exact(b):
    n, k = 40, max(8192, 2 * b)
    W = inputs.student_t_weights(n, k, 400 + b)
    got = sss.sss_hadamard(to_dev(W), b, sss.ROTATE_INPUT).cpu().numpy()
    ref = oracle.rotate(W, b, "rows")
    assert np.array_equal(got.view(np.uint32), ref.view(np.uint32))


@pytest.mark.parametrize("b,k", [(16, 1024), (128, 192), (4096, 6), (2048, 12)])
def test_rotate_cols_bit_exact(b, k):
    n = 2 * b
    W = inputs.student_t_weights(n, k, 410 + b)
    got = sss.sss_hadamard(to_dev(W), b, sss.ROTATE_OUTPUT).cpu().numpy()
    ref = oracle.rotate(W, b, "cols")
    assert np.array_equal(got.view(np.uint32), ref.view(np.uint32))


def test_rotate_in_place_and_llama_q_proj_rows():
    n, k = inputs.LLAMA3_8B_LAYER["q_proj"]
    W = inputs.student_t_weights(n, k, inputs.weight_seed(2, 0, 0))
    w = to_dev(W)
    sss.sss_hadamard(w, 4096, sss.ROTATE_INPUT, out=w)  # R1 on the residual stream
    rows = np.random.default_rng(0).choice(n, 48, replace=False)
    assert np.array_equal(w.cpu().numpy()[rows].view(np.uint32),
                          oracle.rotate(W[rows], 4096, "rows").view(np.uint32))


@pytest.mark.parametrize("grid", GRIDS)
@pytest.mark.parametrize("q", QS)
@pytest.mark.parametrize("g,b", [(32, 32), (32, 128), (128, 4096), (64, 8192)])
def test_quantize_rotated_bit_exact(q, grid, g, b):
    n, k = 24, 8192
    W = inputs.student_t_weights(n, k, 420 + q + b)
    Wr = oracle.rotate(W, b, "rows")
    codes, scales, mins, clip, flags = oracle.quantize(Wr, q, g, grid, clip_counts=True)
    cc = torch.zeros((n, k // g, 2), dtype=torch.uint8, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    qt = sss.sss_quantize_rotated(to_dev(W), b, q, g, grid, clip_counts=cc, dev_status=st)
    torch.cuda.synchronize()
    assert np.array_equal(qt.codes.cpu().numpy(), codes)
    assert np.array_equal(qt.scales.cpu().numpy().view(np.uint16), scales)
    if mins is not None:
        assert np.array_equal(qt.mins.cpu().numpy().view(np.uint16), mins)
    if grid != sss.GRID_ASYM:
        assert np.array_equal(cc.cpu().numpy().reshape(clip.shape), clip)
    assert int(st.item()) == flags


def test_quantize_rotated_ragged_last_chunk():
    # n*k not a multiple of the 8192-value chunk: the last chunk is partial
    n, k, b = 7, 1024 + 512, 512
    W = inputs.student_t_weights(n, k, 430)
    codes, scales, _, _, _ = oracle.quantize(oracle.rotate(W, b, "rows"), 3, 32,
                                             oracle.GRID_SIGNED_SYM)
    qt = sss.sss_quantize_rotated(to_dev(W), b, 3, 32, sss.GRID_SIGNED_SYM)
    torch.cuda.synchronize()
    assert np.array_equal(qt.codes.cpu().numpy(), codes)
    assert np.array_equal(qt.scales.cpu().numpy().view(np.uint16), scales)


def test_rotation_rejects_bad_blocks():
    w = torch.zeros((8, 96), dtype=torch.float32, device="cuda")
    for b in (0, 3, 64, 16384):  # not a power of two, not dividing k, too large
        with pytest.raises(sss.SssError):
            sss.sss_hadamard(w, b)
