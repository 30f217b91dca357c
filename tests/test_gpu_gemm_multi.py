"""Parity of sss_gemm_multi (several packed matrices sharing X, one launch)
with the fp64 oracle matmul over the dequantised weights, and with sss_gemm
on each matrix alone where both calls take the same tile plan."""
import numpy as np
import pytest

import oracle
from paper_2607_08779_gb300 import inputs, sss

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from gpu_util import REL_TOL, qtensor_from_oracle, rel_err_per_row, to_dev  # noqa: E402


def _mats(ns, k, q, g, grid, seed):
    out = []
    for j, n in enumerate(ns):
        W = inputs.student_t_weights(n, k, seed + 17 * j) if n else np.zeros((0, k), np.float32)
        codes, scales, mins, _, _ = oracle.quantize(W, q, g, grid)
        out.append((qtensor_from_oracle(codes, scales, mins, n, k, q, g, grid), (codes, scales, mins)))
    return out


def _x(m, k, seed):
    Xb = inputs.normal_bf16_bits((m, k), seed)
    return Xb, to_dev(Xb.view(np.int16)).view(torch.bfloat16)


def run_multi(ns, k, m, q, g, grid, seed, tokens=None, workspace=None):
    mats = _mats(ns, k, q, g, grid, seed)
    Xb, X = _x(m, k, seed + 99)
    qts = [qt for qt, _ in mats]
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    Ys = sss.sss_gemm_multi(qts, X, workspace=workspace, dev_status=st)
    Ys2 = sss.sss_gemm_multi(qts, X, workspace=workspace)
    torch.cuda.synchronize()
    assert int(st.item()) == 0, "a bounded wait expired"
    rows = np.arange(m) if tokens is None else np.asarray(tokens)
    for (qt, (codes, scales, mins)), n, Y, Y2 in zip(mats, ns, Ys, Ys2):
        assert torch.equal(Y, Y2), "GEMM is not deterministic"
        if n == 0:
            continue
        What = oracle.dequantize(codes, scales, mins, n, k, q, g, grid)
        Yref = oracle.matmul_f64(What, Xb[rows])
        err = rel_err_per_row(Y.cpu().numpy()[rows], Yref)
        assert np.all(err <= REL_TOL), f"matrix n={n}: rel err {err.max():.3e}"
    return qts, X, Ys


@pytest.mark.parametrize("grid", [sss.GRID_UNSIGNED_SYM, sss.GRID_SIGNED_SYM, sss.GRID_ASYM])
@pytest.mark.parametrize("q", [2, 3, 4])
def test_gemm_multi_ragged(q, grid):
    # three matrices with ragged row tiles (132, 260 and 36 rows), 140
    # tokens and 17 k-blocks: 6 row tiles x 2 token tiles, so K is split (the
    # matrices' partial tiles share one padded array).  (A matrix of only 4
    # rows measures each token's error against the largest of 4 outputs,
    # where the fp16 weight rounding alone can reach the 1e-3 gate.)
    run_multi((132, 260, 36), 1088, 140, q, 32, grid, 300 + 10 * q + grid)


@pytest.mark.parametrize("g", [64, 128])
def test_gemm_multi_groups(g):
    run_multi((256, 128), 2048, 300, 4, g, sss.GRID_SIGNED_SYM, 400 + g)


def test_gemm_multi_llama_qkv():
    # q/k/v of a Llama3-8B layer at 512 tokens: whole output rows of three
    # tokens against the oracle, and every token of q against q alone (which
    # takes 128-token tiles where the fused call takes 256-token ones)
    dims = inputs.LLAMA3_8B_LAYER
    ns = [dims[nm][0] for nm in ("q_proj", "k_proj", "v_proj")]
    k = dims["q_proj"][1]
    qts, X, Ys = run_multi(ns, k, 512, 4, 32, sss.GRID_SIGNED_SYM, 500, tokens=[0, 301, 511])
    Yq = sss.sss_gemm(qts[0], X)
    torch.cuda.synchronize()
    err = rel_err_per_row(Ys[0].cpu().numpy(), Yq.cpu().numpy().astype(np.float64))
    assert err.max() <= REL_TOL


def test_gemm_multi_llama_gate_up_matches_single_calls():
    # gate/up at 512 tokens: both the fused call and each lone call take
    # 256-token tiles with K unsplit, so the outputs are the same bits
    # (each lone call is checked against the oracle in test_gpu_gemm)
    n, k = inputs.LLAMA3_8B_LAYER["gate_proj"]
    qts = [sss.sss_quantize(inputs.student_t_weights_cuda(n, k, 600 + j), 4, 32,
                            sss.GRID_SIGNED_SYM) for j in range(2)]
    _, X = _x(512, k, 601)
    Ys = sss.sss_gemm_multi(qts, X)
    for qt, Y in zip(qts, Ys):
        assert torch.equal(sss.sss_gemm(qt, X), Y)
    torch.cuda.synchronize()


def test_gemm_multi_skips_empty_matrices():
    run_multi((128, 0, 64), 512, 96, 4, 32, sss.GRID_SIGNED_SYM, 700)


def test_gemm_multi_minimal_workspace_runs_unsplit():
    # the preferred plan of this shape splits K (its workspace holds the
    # partial tiles); with room for the fp16 X only it runs unsplit and still
    # matches the oracle
    ns, m, k = (132, 260, 36), 140, 1088
    qts = [qt for qt, _ in _mats(ns, k, 4, 32, sss.GRID_SIGNED_SYM, 800)]
    assert sss.sss_gemm_multi_workspace_bytes(qts, m) > m * k * 2
    ws = torch.empty(m * k * 2, dtype=torch.uint8, device="cuda")
    run_multi(ns, k, m, 4, 32, sss.GRID_SIGNED_SYM, 800, workspace=ws)
