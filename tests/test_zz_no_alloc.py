"""sss_gemm_noalloc (the prefill GEMM with the library's static scratch)
against sss_gemm (caller workspace) on the same inputs, two calls in a row;
and its size limit.  Collected last on purpose: it must pass after every
other test in the process as well as alone."""
import numpy as np
import pytest

from paper_2607_08779_gb300 import inputs, sss

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from gpu_util import REL_TOL, rel_err_per_row, to_dev, x_bits  # noqa: E402


def _case(n, k, m, q, grid, seed):
    W = inputs.student_t_weights(n, k, seed)
    qt = sss.sss_quantize(to_dev(W), q, 32, grid)
    X = to_dev(x_bits(m, k, seed + 1).view(np.int16)).view(torch.bfloat16)
    return qt, X


@pytest.mark.parametrize("n,k,m,q,grid", [
    (256, 1024, 200, 4, sss.GRID_SIGNED_SYM),
    (512, 4096, 512, 3, sss.GRID_ASYM),
    (1024, 4096, 2048, 2, sss.GRID_UNSIGNED_SYM),
])
def test_noalloc_matches_workspace_gemm_twice(n, k, m, q, grid):
    qt, X = _case(n, k, m, q, grid, 700 + n + q)
    ref = sss.sss_gemm(qt, X).cpu().numpy()
    for _ in range(2):
        status = torch.zeros(1, dtype=torch.int32, device="cuda")
        y = torch.full((m, n), float("nan"), dtype=torch.float32, device="cuda")
        sss.sss_gemm_noalloc(qt, X, y, dev_status=status)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        err = rel_err_per_row(y.cpu().numpy(), ref)
        assert err.max() <= REL_TOL, f"rel err {err.max():.3e}"


def test_noalloc_rejects_sizes_beyond_the_scratch():
    limit = sss.sss_gemm_noalloc_max_scratch_bytes()
    assert limit == 32 << 20
    k = 1024
    m_ok = limit // (2 * k)          # exactly fills the scratch
    qt, _ = _case(64, k, 1, 4, sss.GRID_SIGNED_SYM, 9)
    # seeded N(0,1) activations, so the comparison below checks real values
    X = inputs.normal_bf16_cuda((m_ok + 1, k), 31)
    y = torch.zeros((m_ok + 1, 64), dtype=torch.float32, device="cuda")
    with pytest.raises(sss.SssError) as e:
        sss.sss_gemm_noalloc(qt, X, y)
    assert sss.STATUS_NAMES[e.value.status] == "SSS_E_WORKSPACE"
    assert "32 MiB" in str(e.value)
    # the largest accepted size runs
    sss.sss_gemm_noalloc(qt, X[:m_ok], y[:m_ok])
    torch.cuda.synchronize()
    ref = sss.sss_gemm(qt, X[:m_ok]).cpu().numpy()
    got = y[:m_ok].cpu().numpy()
    assert np.abs(ref).max() > 0
    # the static scratch may leave no room for split-K partials where a full
    # workspace has it, so the two may sum in different orders
    assert rel_err_per_row(got, ref).max() <= REL_TOL
