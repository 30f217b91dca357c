"""bench.py's CPU oracle baseline (the bench line's cpu_baseline) run on a
stand-in workload of CPU tensors: each leg (GEMV, quantize, GEMM) times the
unchanged oracle and reports a positive rate, its unit, the cores it used
and what its sample was."""
import numpy as np
import pytest

import bench
import oracle
from paper_2607_08779_gb300 import inputs, sss

torch = pytest.importorskip("torch")


class _Workload:
    """The fields cpu_baseline reads, as CPU tensors (the bench's are on the
    GPU and are copied to the host the same way)."""

    def __init__(self, n=128, k=512, m=32):
        self.torch = torch
        self.shapes = [("q_proj", (64, k)), ("gate_proj", (n, k))]
        W = inputs.student_t_weights(n, k, 3)
        codes, scales, _, _, _ = oracle.quantize(W, 4, bench.GROUP, oracle.GRID_SIGNED_SYM)
        qt = sss.QTensor(n, k, 4, bench.GROUP, sss.GRID_SIGNED_SYM, torch.from_numpy(codes),
                         torch.from_numpy(scales.view(np.int16)), None)
        self.stack = {4: [[None, qt]]}
        self.x = {k: torch.from_numpy(inputs.normal_bf16_bits((1, k), 5).view(np.int16))
                  .view(torch.bfloat16)}
        self.X = {k: torch.from_numpy(inputs.normal_bf16_bits((m, k), 6).view(np.int16))
                  .view(torch.bfloat16)}
        self.fresh = [[None, torch.from_numpy(W)]]


def test_oracle_gemm_rate_counts_the_products():
    n, k, m = 100, 256, 4
    W = inputs.student_t_weights(n, k, 7)
    codes, scales, _, _, _ = oracle.quantize(W, 4, bench.GROUP, oracle.GRID_SIGNED_SYM)
    xb = inputs.normal_bf16_bits((m, k), 8)
    rate, flops, el = bench.oracle_gemm_rate(codes, scales, n, k, 4, xb, 0.05)
    # whole blocks of 64 rows and a ragged one of 36, each 2 * rows * k * m
    assert flops > 0 and flops % (2 * k * m) == 0
    assert rate == pytest.approx(flops / el)


def test_cpu_baseline_reports_every_leg():
    cb = bench.cpu_baseline(_Workload(), seconds=0.4, cores=1)
    assert cb["kind"] == "oracle" and cb["cores"] == 1 and cb["unit"] == "GB/s"
    assert cb["value"] > 0 and cb["single_core_value"] == cb["value"]
    for leg, unit in (("quantize", "Gweights/s"), ("gemm", "TFLOP/s")):
        sub = cb[leg]
        assert sub["unit"] == unit and sub["cores"] == 1 and sub["value"] > 0, sub
        assert sub["single_core_value"] == pytest.approx(sub["value"], rel=1e-6)
        assert "oracle" in sub["sample"]
