"""Helpers shared by the GPU parity tests: move seeded inputs to the device,
run the CUDA path through the C ABI, run the oracle on the same bits."""
import numpy as np
import torch

import oracle
from paper_2607_08779_gb300 import inputs, sss

# Output tolerance of the GEMV and GEMM against the fp64 oracle: relative
# error 1e-3 per output vector, max|y - y_ref| / max|y_ref|.
REL_TOL = 1e-3

DEV = "cuda"


def to_dev(a: np.ndarray, dtype=None):
    t = torch.from_numpy(np.ascontiguousarray(a))
    if dtype is not None:
        t = t.view(dtype)
    return t.to(DEV)


def gpu_quantize(W: np.ndarray, q, g, grid, clip=True):
    w = to_dev(W)
    n, k = W.shape
    cc = torch.zeros((n, k // g, 2), dtype=torch.uint8, device=DEV) if clip else None
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    qt = sss.sss_quantize(w, q, g, grid, clip_counts=cc, dev_status=st)
    torch.cuda.synchronize()
    return qt, (cc.cpu().numpy() if clip else None), int(st.item())


def qtensor_from_oracle(codes, scales, mins, n, k, q, g, grid) -> sss.QTensor:
    return sss.QTensor(n, k, q, g, grid, to_dev(codes), to_dev(scales.view(np.int16)),
                       None if mins is None else to_dev(mins.view(np.int16)))


def rel_err_per_row(y: np.ndarray, yref: np.ndarray) -> np.ndarray:
    """max_n |y - y_ref| / max_n |y_ref| for each output vector (row)."""
    y = np.atleast_2d(y).astype(np.float64)
    yref = np.atleast_2d(yref)
    den = np.maximum(np.max(np.abs(yref), axis=1), 1e-300)
    return np.max(np.abs(y - yref), axis=1) / den


def x_bits(batch, k, seed):
    return inputs.normal_bf16_bits((batch, k), seed)
