"""LSQ scale refinement on the GPU (Sec. 5 learned grid parameters;
Appendix C): codes and fp16 scales bit-exact with the oracle's data-free
LSQ steps, signed (s != 0) and conventional (s > 0) grids."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import to_dev
from paper_2607_08779_gb300 import inputs, sss

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("grid", [sss.GRID_SIGNED_SYM, sss.GRID_UNSIGNED_SYM])
@pytest.mark.parametrize("q", (2, 3, 4))
@pytest.mark.parametrize("g", [32, 64, 128])
@pytest.mark.parametrize("steps,lr", [(0, 0.01), (20, 0.01), (8, 3.0)])
def test_lsq_bit_exact(q, g, grid, steps, lr):
    n, k = 48, 1024
    W = inputs.student_t_weights(n, k, 600 + q + g + steps)
    W[2, :g] = 0.0  # an all-zero group keeps s = 0
    codes, scales, flags = oracle.lsq_quantize(W, q, g, grid, steps, lr)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    qt = sss.sss_quantize_lsq(to_dev(W), q, g, grid, steps, lr, dev_status=st)
    torch.cuda.synchronize()
    assert np.array_equal(qt.scales.cpu().numpy().view(np.uint16), scales)
    assert np.array_equal(qt.codes.cpu().numpy(), codes)
    assert int(st.item()) == flags


def test_lsq_zero_steps_equals_sss_quantize():
    W = inputs.student_t_weights(256, 4096, 610)
    w = to_dev(W)
    a = sss.sss_quantize(w, 3, 32, sss.GRID_SIGNED_SYM)
    b = sss.sss_quantize_lsq(w, 3, 32, sss.GRID_SIGNED_SYM, 0, 0.01)
    torch.cuda.synchronize()
    assert torch.equal(a.codes, b.codes) and torch.equal(a.scales, b.scales)


def test_lsq_llama_gate_rows_sampled():
    n, k = inputs.LLAMA3_8B_LAYER["gate_proj"]
    W = inputs.student_t_weights(n, k, inputs.weight_seed(2, 0, 4))
    qt = sss.sss_quantize_lsq(to_dev(W), 2, 32, sss.GRID_SIGNED_SYM, 20, 0.01)
    torch.cuda.synchronize()
    rows = np.sort(np.random.default_rng(3).choice(n, 32, replace=False))
    codes, scales, _ = oracle.lsq_quantize(W[rows], 2, 32, oracle.GRID_SIGNED_SYM, 20, 0.01)
    assert np.array_equal(qt.codes.cpu().numpy()[rows], codes)
    assert np.array_equal(qt.scales.cpu().numpy().view(np.uint16)[rows], scales)
