"""The bounded waits of the GEMM kernel, made to run out.

sss_test_set_stall leaves one mbarrier of the GEMM one arrive short, so the
wait on it expires after its bound (about one second).  The call must still
return SSS_OK, the device status word must carry SSS_FLAG_TIMEOUT, and a
normal call right after it must match the oracle: the kernel released its
tensor memory and the context is still usable.  The decode GEMV kernels
(batch 1 and batched) have no data-dependent waits (their warps meet only
at CTA-wide barriers), so their stall bits change nothing: checked too.
Nothing here faults, traps or hangs the GPU.
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import REL_TOL, qtensor_from_oracle, rel_err_per_row, to_dev, x_bits
from paper_2607_08779_gb300 import inputs, sss

pytestmark = pytest.mark.gpu

GRID = oracle.GRID_SIGNED_SYM


def _packed(n, k, q, g, seed):
    W = inputs.student_t_weights(n, k, seed)
    codes, scales, mins, _, _ = oracle.quantize(W, q, g, GRID)
    return qtensor_from_oracle(codes, scales, mins, n, k, q, g, GRID), (codes, scales, mins)


def _x(bits):
    return to_dev(bits.view(np.int16)).view(torch.bfloat16)


def _stalled(mask, call):
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    sss.sss_test_set_stall(mask)
    try:
        call(st)  # raises SssError on a non-OK return code
        torch.cuda.synchronize()
    finally:
        sss.sss_test_set_stall(0)
    return int(st.item())


def test_gemv_batch_has_no_waits_to_stall():
    # one 16-row tile whose 4096-code rows are split across the warps of the
    # CTA (their partial sums meet in shared memory after a CTA barrier) and
    # a k that takes two x slabs at batch 16: with the batched kernel's stall
    # bit set the calls still see no timeout and match the oracle
    n, q, g = 16, 4, 32
    for k, batch, seed in ((4096, 4, 21), (14336, 16, 26)):
        qt, (codes, scales, mins) = _packed(n, k, q, g, seed)
        xb = x_bits(batch, k, 5)
        x = _x(xb)
        y = torch.empty((batch, n), dtype=torch.float32, device="cuda")
        status = _stalled(sss.TEST_STALL_GEMV_BATCH,
                          lambda st: sss.sss_gemv(qt, x, y=y, dev_status=st))
        assert status == 0, status
        yref = oracle.gemv(codes, scales, mins, n, k, q, g, GRID, xb)
        assert rel_err_per_row(y.cpu().numpy(), yref).max() <= REL_TOL


def test_gemv_stream_has_no_waits_to_stall():
    # the same 16-row tile split across 16 warps (sss_gemv) and two matrices
    # in one launch (sss_gemv_multi): with the stream kernel's stall bit set
    # the calls still see no timeout and match the oracle
    n, k, q, g = 16, 4096, 3, 32
    qa, (ca, sa, ma) = _packed(n, k, q, g, 22)
    qb, (cb, sb, mb) = _packed(n, k, q, g, 23)
    xb = x_bits(1, k, 6)
    x = _x(xb)
    out = {}

    def call(st):
        out["one"] = sss.sss_gemv(qa, x, dev_status=st)
        out["multi"] = sss.sss_gemv_multi([qa, qb], x[0], dev_status=st,
                                          flags=sss.GEMV_PDL | sss.GEMV_WEIGHTS_READY)

    status = _stalled(sss.TEST_STALL_GEMV, call)
    assert status == 0, status
    ya, yb = out["multi"]
    for y, (c, s, m) in ((out["one"][0], (ca, sa, ma)), (ya, (ca, sa, ma)), (yb, (cb, sb, mb))):
        yref = oracle.gemv(c, s, m, n, k, q, g, GRID, xb)
        assert rel_err_per_row(y.cpu().numpy()[None], yref).max() <= REL_TOL


@pytest.mark.parametrize("noalloc", [False, True])
def test_gemm_wait_runs_out_then_recovers(noalloc):
    # 16 k-blocks of 64, more than the pipeline's stages, and two token tiles
    n, k, q, g, m = 256, 1024, 4, 32, 200
    qt, (codes, scales, mins) = _packed(n, k, q, g, 24)
    Xb = x_bits(m, k, 7)
    X = _x(Xb)
    Y = torch.empty((m, n), dtype=torch.float32, device="cuda")

    def call(st):
        if noalloc:
            sss.sss_gemm_noalloc(qt, X, Y, dev_status=st)
        else:
            sss.sss_gemm(qt, X, y=Y, dev_status=st)

    status = _stalled(sss.TEST_STALL_GEMM, call)
    assert status & sss.FLAG_TIMEOUT, status

    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    Y.fill_(float("nan"))
    call(st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    What = oracle.dequantize(codes, scales, mins, n, k, q, g, GRID)
    Yref = oracle.matmul_f64(What, Xb)
    assert rel_err_per_row(Y.cpu().numpy(), Yref).max() <= REL_TOL


def test_stall_mask_off_by_default():
    # the hook is process-wide: every test above clears it; a plain call here
    # must see no timeout
    n, k, q, g = 16, 4096, 2, 32
    qt, (codes, scales, mins) = _packed(n, k, q, g, 25)
    xb = x_bits(1, k, 8)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    y = sss.sss_gemv(qt, _x(xb), dev_status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    yref = oracle.gemv(codes, scales, mins, n, k, q, g, GRID, xb)
    assert rel_err_per_row(y.cpu().numpy(), yref).max() <= REL_TOL
