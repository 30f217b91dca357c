"""Seeded synthetic inputs shared by the tests, the smoke check and the bench.

This module holds random-number recipes only -- none of the quantization
arithmetic.  It serves both the CUDA path and the CPU oracle, which receive
the exact same bits (generated here on the CPU, or generated on the GPU and
copied to the host).

Recipe (the paper's real-weight measurements use Llama3/Qwen3 linear layers,
Sec. 4 and Fig. 1; those weights are not available, so heavy-tailed synthetic
weights of the same shapes stand in):

* weights: Student-t with nu = 4 degrees of freedom, scaled by 0.02, drawn as
  t = Z / sqrt(V / 4) with V = Z1^2 + Z2^2 + Z3^2 + Z4^2 (an exact chi^2_4);
* outlier channels: round(0.005 * K) input channels (columns) chosen by a
  seeded permutation are multiplied by 20;
* activations: N(0, 1) rounded to bfloat16.

CPU draws use numpy's Philox4x32-10 bit generator; GPU draws use torch's CUDA
generator (also Philox4x32-10).  The two streams differ; whichever side
generates, the other side gets a copy of the same bits.
"""
from __future__ import annotations

import numpy as np

NU = 4
WEIGHT_SCALE = 0.02
OUTLIER_FRACTION = 0.005
OUTLIER_GAIN = 20.0

# Llama3-8B-shaped linear layers (out_features N, in_features K)
LLAMA3_8B_LAYER = {
    "q_proj": (4096, 4096),
    "k_proj": (1024, 4096),
    "v_proj": (1024, 4096),
    "o_proj": (4096, 4096),
    "gate_proj": (14336, 4096),
    "up_proj": (14336, 4096),
    "down_proj": (4096, 14336),
}
LLAMA3_8B_LAYERS = 32

# Qwen3-32B-shaped linear layers (hidden 5120, intermediate 25600,
# 64 query heads / 8 KV heads of dim 128)
QWEN3_32B_LAYER = {
    "q_proj": (8192, 5120),
    "k_proj": (1024, 5120),
    "v_proj": (1024, 5120),
    "o_proj": (5120, 8192),
    "gate_proj": (25600, 5120),
    "up_proj": (25600, 5120),
    "down_proj": (5120, 25600),
}
QWEN3_32B_LAYERS = 64

MATRIX_IDS = {name: i for i, name in enumerate(LLAMA3_8B_LAYER)}


def weight_seed(config: int, layer: int, matrix_id: int) -> int:
    return 0x55530000 + config * 1000 + layer * 16 + matrix_id


def n_outlier_channels(k: int) -> int:
    return int(round(OUTLIER_FRACTION * k))


def _rng(seed: int) -> np.random.Generator:
    return np.random.Generator(np.random.Philox(seed))


def student_t_weights(n: int, k: int, seed: int, outliers: bool = True,
                      nu: int = NU, scale: float = WEIGHT_SCALE) -> np.ndarray:
    """fp32 [n, k] heavy-tailed weights (CPU, numpy Philox)."""
    rng = _rng(seed)
    z = rng.standard_normal((n, k), dtype=np.float64)
    v = np.zeros((n, k), np.float64)
    for _ in range(nu):
        zi = rng.standard_normal((n, k), dtype=np.float64)
        v += zi * zi
    w = (z / np.sqrt(v / nu)) * scale
    if outliers:
        cols = rng.permutation(k)[: n_outlier_channels(k)]
        w[:, cols] *= OUTLIER_GAIN
    return w.astype(np.float32)


def normal_bf16_bits(shape, seed: int) -> np.ndarray:
    """N(0,1) rounded to bfloat16 (round to nearest even); returns uint16 bits."""
    rng = _rng(seed ^ 0x5A5A5A5A)
    x = rng.standard_normal(shape, dtype=np.float64).astype(np.float32)
    return f32_to_bf16_bits(x)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 to bfloat16 (nearest even; inputs are finite)."""
    b = np.ascontiguousarray(x, np.float32).view(np.uint32).astype(np.uint64)
    lsb = (b >> 16) & 1
    r = (b + 0x7FFF + lsb) >> 16
    return r.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(b, np.uint16).astype(np.uint32) << 16).view(np.float32)


# --------------------------------------------------------------------------
# GPU-side generation (bench-sized inputs); torch is imported lazily so the
# CPU-only tests never need it.
# --------------------------------------------------------------------------

def student_t_weights_cuda(n: int, k: int, seed: int, out=None, outliers=True,
                           nu: int = NU, scale: float = WEIGHT_SCALE,
                           device="cuda"):
    """fp32 [n, k] heavy-tailed weights generated on the GPU (torch Philox).

    Generated in row chunks to bound the temporary memory."""
    import torch

    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    if out is None:
        out = torch.empty((n, k), dtype=torch.float32, device=device)
    chunk = max(1, (1 << 26) // k)
    for r0 in range(0, n, chunk):
        r1 = min(n, r0 + chunk)
        z = torch.randn((r1 - r0, k), generator=gen, device=device)
        v = torch.zeros_like(z)
        for _ in range(nu):
            zi = torch.randn((r1 - r0, k), generator=gen, device=device)
            v.addcmul_(zi, zi)
        out[r0:r1] = z / torch.sqrt(v / nu) * scale
    if outliers:
        perm = torch.randperm(k, generator=gen, device=device)
        cols = perm[: n_outlier_channels(k)]
        out[:, cols] *= OUTLIER_GAIN
    return out


def normal_bf16_cuda(shape, seed: int, device="cuda"):
    import torch

    gen = torch.Generator(device=device)
    gen.manual_seed(seed ^ 0x5A5A5A5A)
    return torch.randn(shape, generator=gen, device=device).to(torch.bfloat16)
