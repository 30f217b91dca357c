"""The sign-rule diagnostics on the GPU (Sec. 4, rem:cardinality-margin,
fig:theory-diagnostics): the cardinality margin of every group bit-exact
with the oracle's clip counts, and the realised l2 gain exactly equal to
the exact rational value computed here from the oracle's quantization at
both signs."""
from fractions import Fraction as F

import numpy as np
import pytest
import torch

import oracle
from gpu_util import to_dev
from paper_2607_08779_gb300 import inputs, sss

pytestmark = pytest.mark.gpu

QS = (2, 3, 4)


def exact_gain(w, q):
    """g = ||w - Q_-gamma*(w)||^2 - ||w - Q_gamma*(w)||^2 in exact rationals,
    with each sign's stored fp16 scale, from the oracle's quantization."""
    r = oracle.quantize_group(w, q, oracle.GRID_SIGNED_SYM)
    gamma = r["gamma"]
    rp = oracle.quantize_group_gamma(w, q, gamma)
    rm = oracle.quantize_group_gamma(w, q, -gamma)
    sp = F(float(np.array([rp["s16"]], np.uint16).view(np.float16)[0]))
    sm = F(float(np.array([rm["s16"]], np.uint16).view(np.float16)[0]))
    ep = sum((F(float(x)) - sp * int(c)) ** 2 for x, c in zip(w, rp["c"]))
    em = sum((F(float(x)) - sm * int(c)) ** 2 for x, c in zip(w, rm["c"]))
    return em - ep, int(r["n_other"]) - int(r["n_self"])


@pytest.mark.parametrize("q", QS)
@pytest.mark.parametrize("g", [32, 64, 128])
def test_margin_and_gain_match_exact(q, g):
    n, k = 64, 1024
    W = inputs.student_t_weights(n, k, 300 + q + g)   # heavy tails, outlier channels
    W[3, :g] = 0.0                                    # an all-zero group
    W[5, g:2 * g] = np.linspace(-1, 1, g)             # a sign tie
    margin, gain, hist = sss.sss_sign_diagnostics(to_dev(W), q, g)
    torch.cuda.synchronize()
    margin, gain, hist = margin.cpu().numpy(), gain.cpu().numpy(), hist.cpu().numpy()
    flat = W.reshape(-1, g)
    rng = np.random.default_rng(q * g)
    sample = sorted(set(rng.choice(flat.shape[0], 160, replace=False)) | {3 * (k // g), 5 * (k // g) + 1})
    for G in sample:
        ge, me = exact_gain(flat[G], q)
        assert margin.ravel()[G] == me, G
        assert F(float(gain.ravel()[G])) == ge, (G, gain.ravel()[G], float(ge))
    # the histogram counts every group once, at its (margin, gain sign)
    ref = np.zeros_like(hist)
    for m, gg in zip(margin.ravel(), gain.ravel()):
        ref[m + g, 0 if gg < 0 else (1 if gg == 0 else 2)] += 1
    assert np.array_equal(hist, ref)
    assert hist.sum() == flat.shape[0]


def test_margins_equal_the_quantizer_clip_counts():
    n, k, q, g = 256, 4096, 3, 32
    W = inputs.student_t_weights(n, k, 311)
    _, _, _, clip, _ = oracle.quantize(W, q, g, oracle.GRID_SIGNED_SYM, clip_counts=True)
    margin, gain, hist = sss.sss_sign_diagnostics(to_dev(W), q, g)
    torch.cuda.synchronize()
    ref = clip[..., 1].astype(np.int32) - clip[..., 0].astype(np.int32)
    assert np.array_equal(margin.cpu().numpy().reshape(ref.shape), ref)


def test_nonfinite_groups_are_skipped_and_flagged():
    W = inputs.student_t_weights(4, 128, 5)
    W[1, 40] = np.nan
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    _, _, hist = sss.sss_sign_diagnostics(to_dev(W), 4, 32, dev_status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & sss.FLAG_NONFINITE
    assert int(hist.sum().item()) == 4 * 4 - 1
