"""Pins of the CPU oracle against what the paper and the mathematics fix.

Nothing here re-types the oracle's formulas: each check compares the
oracle's output with an independent statement -- a theorem or lemma of the
paper evaluated in exact rational arithmetic, a brute-force search over the
grid, a hand-worked fixture, or an independent library routine (numpy's
float16 conversion, numpy's float64 matmul).
"""
import itertools
import os
from fractions import Fraction as F

import numpy as np
import pytest

import oracle
from paper_2607_08779_gb300 import inputs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
QS = (2, 3, 4)
GRID_CODE = {"U": oracle.GRID_UNSIGNED_SYM, "S": oracle.GRID_SIGNED_SYM,
             "A": oracle.GRID_ASYM}


def alphabet(q):
    """A_q = {-2^(q-1), ..., 2^(q-1)-1} (Sec. 1, Notation)."""
    return range(-(1 << (q - 1)), 1 << (q - 1))


def nearest_index(w: F, base: F, step: F, idx):
    """Brute force: the a in idx minimising |w - (base + step*a)|; an exact
    tie between two neighbours goes to the even a."""
    best = None
    for a in idx:
        d = abs(w - (base + step * a))
        if best is None or d < best[0] or (d == best[0] and a % 2 == 0):
            best = (d, a)
    return best[1]


def is_midpoint(x: F) -> bool:
    return (x - F(1, 2)).denominator == 1


def dominant_outlier(w):
    """(index, value) of the largest-magnitude coordinate following the sign
    rule's reading: positive if max w > -min w, else negative."""
    mx, mn = float(np.max(w)), float(np.min(w))
    i = int(np.argmax(w)) if mx > -mn else int(np.argmin(w))
    return i, float(w[i])


def random_groups(n, g, seed, outliers=True):
    w = inputs.student_t_weights(n, g, seed, outliers=False)
    if outliers:
        # plant a few large coordinates, of random sign, as the outlier channels do
        rng = np.random.default_rng(seed)
        rows = rng.random(n) < 0.5
        cols = rng.integers(0, g, n)
        w[rows, cols[rows]] *= 20.0
    return w


def lattice_groups(d, den):
    vals = [F(i, den) for i in range(-den, den + 1)]
    for combo in itertools.product(vals, repeat=d):
        if any(v != 0 for v in combo):
            yield np.array([float(v) for v in combo], np.float32)


# --------------------------------------------------------------------------
# IEEE binary16 (the stored scale format of the Q-formats, Appendix)
# --------------------------------------------------------------------------

def test_f32_to_f16_matches_numpy():
    rng = np.random.default_rng(1)
    vals = list(rng.standard_normal(4000).astype(np.float32))
    vals += list((rng.standard_normal(4000) * 2.0 ** rng.integers(-30, 20, 4000))
                 .astype(np.float32))
    edges = [0.0, -0.0, 65504.0, 65519.0, 65519.99, 65520.0, -65520.0, 1e9,
             2.0 ** -24, 2.0 ** -25, 3 * 2.0 ** -26, 2.0 ** -14, 2.0 ** -15,
             (1 + 2.0 ** -11) * 2.0 ** -14, 1 + 2.0 ** -11, 1 + 3 * 2.0 ** -11,
             np.inf, -np.inf, 1e-40]
    vals += [np.float32(e) for e in edges]
    for x in vals:
        with np.errstate(over="ignore"):
            want = int(np.array([x], np.float32).astype(np.float16).view(np.uint16)[0])
        assert oracle.f32_to_f16(x) == want, x


def test_f16_to_f32_exhaustive():
    bits = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)
    ref = bits.view(np.float16).astype(np.float32)
    got = np.array([oracle.f16_to_f32(int(b)) for b in bits], np.float32)
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(got), nan)
    assert np.array_equal(got[~nan].view(np.uint32), ref[~nan].view(np.uint32))


# --------------------------------------------------------------------------
# Hand-worked fixtures and the paper's printed block sizes
# --------------------------------------------------------------------------

def _golden_records():
    for line in open(os.path.join(GOLDEN, "hand_groups.txt")):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        f = [x.strip() for x in line.split("|")]
        yield {
            "q": int(f[0]), "grid": GRID_CODE[f[1]],
            "w": np.array([float(v) for v in f[2].split()], np.float32),
            "c": [int(v) for v in f[3].split()],
            "u": [int(v) for v in f[4].split()],
            "s32": float(f[5]), "s16": int(f[6], 16),
            "m16": None if f[7] == "-" else int(f[7], 16),
            "packed": bytes.fromhex(f[8]),
        }


@pytest.mark.parametrize("rec", list(_golden_records()), ids=lambda r: f"q{r['q']}g{r['grid']}")
def test_hand_worked_groups(rec):
    r = oracle.quantize_group(rec["w"], rec["q"], rec["grid"])
    assert list(r["c"]) == rec["c"]
    assert list(r["u"]) == rec["u"]
    assert r["s32"] == rec["s32"]
    assert r["s16"] == rec["s16"]
    if rec["m16"] is not None:
        assert r["m16"] == rec["m16"]
    assert bytes(oracle.pack_group(r["u"], rec["q"])) == rec["packed"]


def test_paper_block_sizes():
    w = inputs.student_t_weights(1, 32, 7)
    for line in open(os.path.join(GOLDEN, "paper_block_sizes.txt")):
        if line.startswith("#") or not line.strip():
            continue
        q, kind, nbytes = [x.strip() for x in line.split("|")]
        q, nbytes = int(q), int(nbytes)
        grid = oracle.GRID_ASYM if kind == "asym" else oracle.GRID_SIGNED_SYM
        codes, scales, mins, _, _ = oracle.quantize(w, q, 32, grid)
        total = codes.nbytes + scales.nbytes + (mins.nbytes if mins is not None else 0)
        assert total == nbytes


# --------------------------------------------------------------------------
# eq:quantizer: rounding to nearest and clipping, by brute force
# --------------------------------------------------------------------------

@pytest.mark.parametrize("q", QS)
@pytest.mark.parametrize("d,den", [(2, 16), (3, 8)])
def test_symmetric_codes_are_nearest_grid_points(q, d, den):
    """Exhaustive dyadic lattice, both scale signs, exact ties included."""
    A = alphabet(q)
    for w in lattice_groups(d, den):
        for gamma in (1, -1):
            r = oracle.quantize_group_gamma(w, q, gamma)
            s = F(r["s32"])
            for j in range(d):
                assert r["c"][j] == nearest_index(F(float(w[j])), F(0), s, A)
                assert r["u"][j] == r["c"][j] + (1 << (q - 1))


@pytest.mark.parametrize("q", QS)
@pytest.mark.parametrize("g", [32, 128])
def test_symmetric_codes_random_groups(q, g):
    A = alphabet(q)
    W = random_groups(40, g, 11 * q + g)
    for w in W:
        for grid in (oracle.GRID_UNSIGNED_SYM, oracle.GRID_SIGNED_SYM):
            r = oracle.quantize_group(w, q, grid)
            s = F(r["s32"])
            for j in range(g):
                assert r["c"][j] == nearest_index(F(float(w[j])), F(0), s, A)


# --------------------------------------------------------------------------
# eq:sign_rule: brute force over both scale signs
# --------------------------------------------------------------------------

def _groups_for_sign_tests():
    out = [w for w in lattice_groups(3, 8)]
    out += list(random_groups(300, 32, 5))
    out += list(random_groups(100, 128, 6))
    return out


@pytest.mark.parametrize("q", QS)
def test_sign_rule_against_both_signs(q):
    half = 1 << (q - 1)
    for w in _groups_for_sign_tests():
        mx, mn = float(np.max(w)), float(np.min(w))
        sig = oracle.quantize_group(w, q, oracle.GRID_SIGNED_SYM)
        uns = oracle.quantize_group(w, q, oracle.GRID_UNSIGNED_SYM)
        both = {gm: oracle.quantize_group_gamma(w, q, gm) for gm in (1, -1)}
        # the signed grid is the gamma-quantizer at its chosen sign, and the
        # unsigned grid is the gamma = +1 quantizer (eq:signed_sym_quant)
        assert np.array_equal(sig["c"], both[sig["gamma"]]["c"])
        assert sig["s32"] == both[sig["gamma"]]["s32"]
        assert np.array_equal(uns["c"], both[1]["c"]) and uns["gamma"] == 1
        if mx == -mn:
            assert sig["gamma"] == 1  # tie reading
            continue
        i, wi = dominant_outlier(w)
        # exactly one sign represents the dominant outlier exactly
        exact = [gm for gm in (1, -1)
                 if F(both[gm]["s32"]) * both[gm]["c"][i] == F(wi)]
        assert exact == [sig["gamma"]]
        assert sig["c"][i] == -half
        # and it is -sign(w_i*)
        assert sig["gamma"] == (-1 if wi > 0 else 1)


@pytest.mark.parametrize("q", QS)
def test_negative_sign_is_the_unsigned_grid_on_the_negated_group(q):
    # Q_-1(w) = -Q_+1(-w): the quantizer with scale -alpha gives the same
    # codes as the unsigned grid applied to -w (the same exact quotient),
    # with the opposite scale.  The margin/gain sweep forms Q_-gamma* this
    # way from the unsigned grid.
    for w in _groups_for_sign_tests():
        neg = oracle.quantize_group_gamma(w, q, -1)
        flip = oracle.quantize_group(-np.asarray(w, np.float32), q, oracle.GRID_UNSIGNED_SYM)
        assert np.array_equal(neg["c"], flip["c"])
        assert np.array_equal(neg["c_pre"], flip["c_pre"])
        assert neg["s32"] == -flip["s32"]


@pytest.mark.parametrize("q", QS)
def test_unsigned_equals_signed_when_outlier_negative(q):
    W = random_groups(400, 32, 21)
    n_neg = 0
    for w in W:
        if float(np.max(w)) < -float(np.min(w)):
            n_neg += 1
            a = oracle.quantize_group(w, q, oracle.GRID_UNSIGNED_SYM)
            b = oracle.quantize_group(w, q, oracle.GRID_SIGNED_SYM)
            assert np.array_equal(a["u"], b["u"]) and a["s16"] == b["s16"]
    assert n_neg > 50


# --------------------------------------------------------------------------
# def:clipped-set, the structural properties, lem:error-separability,
# thm:worst-case-bound and cor:optimal-sign -- in exact arithmetic
# --------------------------------------------------------------------------

def _exact_group_terms(w, q, gamma, r):
    M = F(float(r["M"]))
    alpha = abs(F(r["s32"]))
    T = M * (1 - F(1, 1 << q))
    wf = [F(float(v)) for v in w]
    Qw = [F(r["s32"]) * c for c in r["c"]]
    return M, alpha, T, wf, Qw


@pytest.mark.parametrize("q", QS)
def test_clipped_set_and_lemma_and_bound(q):
    half = 1 << (q - 1)
    n_checked = 0
    for w in _groups_for_sign_tests():
        if float(np.max(np.abs(w))) == 0:
            continue
        res = {gm: oracle.quantize_group_gamma(w, q, gm) for gm in (1, -1)}
        for gm, r in res.items():
            M, alpha, T, wf, Qw = _exact_group_terms(w, q, gm, r)
            midpoint = any(is_midpoint(x / alpha) for x in wf)
            C = {j for j, cp in enumerate(r["c_pre"]) if cp == half}
            Cother = {j for j, cp in enumerate(r["c_pre"]) if cp == -half}
            assert r["n_self"] == len(C) and r["n_other"] == len(Cother)
            # the other sign's clipped set is this sign's lower-tail set
            assert Cother == {j for j, cp in enumerate(res[-gm]["c_pre"]) if cp == half}
            err = [(x - qx) ** 2 for x, qx in zip(wf, Qw)]
            # thm:worst-case-bound, total (holds at midpoints too)
            d = len(wf)
            assert sum(err) <= F(1, 1 << (2 * q)) * M * M * d * (1 + 3 * F(len(C), d))
            if midpoint:
                continue
            n_checked += 1
            # def:clipped-set: C_gamma = {i : gamma w_i > M (1 - 2^-q)}
            assert C == {j for j, x in enumerate(wf) if gm * x > T}
            # thm:worst-case-bound, per coordinate
            for j, e in enumerate(err):
                if j in C:
                    assert alpha * alpha / 4 < e <= alpha * alpha
                else:
                    assert e <= alpha * alpha / 4
            # lem:error-separability: ||w - Q||^2 = E(w) + 2 alpha sum_C (gamma w_i - T)
            E = sum((x - alpha * round(x / alpha)) ** 2 for x in wf)
            assert sum(err) == E + 2 * alpha * sum(gm * wf[j] - T for j in C)
        # cor:optimal-sign and rem:cardinality-margin, at gamma* of the sign rule
        mx, mn = float(np.max(w)), float(np.min(w))
        gs = -1 if mx > -mn else 1
        a, b = res[gs], res[-gs]
        margin = b["n_self"] - a["n_self"]
        bound = lambda r: F(1, 1 << (2 * q)) * F(float(r["M"])) ** 2 * len(w) * (1 + 3 * F(r["n_self"], len(w)))
        if margin >= 0:
            assert bound(a) <= bound(b)
        # structural: C_gamma* lies in {gamma* w_i > 0}
        assert all(gs * float(w[j]) > 0 for j, cp in enumerate(a["c_pre"]) if cp == half)
    assert n_checked > 500


# --------------------------------------------------------------------------
# thm:signed-asymmetric: Q(w; -alpha, 0) == Q(w; alpha, -1)
# --------------------------------------------------------------------------

@pytest.mark.parametrize("q", QS)
def test_sign_flip_is_unit_zero_point_shift(q):
    A = alphabet(q)
    n = 0
    groups = list(random_groups(300, 32, 5)) + list(lattice_groups(3, 8))[::7]
    for w in groups:
        if float(np.max(np.abs(w))) == 0:
            continue
        r = oracle.quantize_group_gamma(w, q, -1)
        alpha = -F(r["s32"])
        assert alpha > 0
        for j, x in enumerate(w):
            x = F(float(x))
            if is_midpoint(x / alpha):
                continue
            # Q(w; alpha, -1) = alpha * (clip(round(w/alpha - 1)) + 1): the
            # nearest point of the shifted grid alpha*(A_q + 1), by brute force
            rhs = alpha * (nearest_index(x, alpha, alpha, A) + 1)
            assert F(r["s32"]) * r["c"][j] == rhs
            n += 1
    assert n > 9000


def test_sign_flip_integer_identity_exhaustive():
    """-clip(-RNE(x)) == clip(RNE(x - 1)) + 1 for every non-midpoint x on a
    fine dyadic lattice (both sides give the nearest point of A_q + 1)."""
    for q in QS:
        lo, hi = -(1 << (q - 1)), (1 << (q - 1)) - 1
        for num in range(-40 * 64, 40 * 64 + 1):
            x = F(num, 64)
            if is_midpoint(x):
                continue
            lhs = -min(max(round(-x), lo), hi)
            rhs = min(max(round(x - 1), lo), hi) + 1
            assert lhs == rhs


# --------------------------------------------------------------------------
# code range, on-grid round trip
# --------------------------------------------------------------------------

@pytest.mark.parametrize("grid", [0, 1, 2])
@pytest.mark.parametrize("q", QS)
def test_code_range(q, grid):
    W = inputs.student_t_weights(64, 4096, 99 + q)
    codes, scales, mins, clip, flags = oracle.quantize(W, q, 32, grid, clip_counts=True)
    assert flags == 0
    u = np.stack([oracle.unpack_group(codes.reshape(-1, 32 * q // 8)[G], 32, q)
                  for G in range(codes.size // (32 * q // 8))])
    assert u.min() >= 0 and u.max() <= (1 << q) - 1


@pytest.mark.parametrize("q", QS)
def test_on_grid_round_trip(q):
    rng = np.random.default_rng(3)
    half = 1 << (q - 1)
    for _ in range(300):
        gamma = int(rng.choice([-1, 1]))
        alpha = 2.0 ** int(rng.integers(-12, 4))
        a = rng.integers(-half + 1, half, 32)
        a[int(rng.integers(0, 32))] = -half   # the dominant outlier at -2^(q-1)
        w = (gamma * alpha * a).astype(np.float32)
        r = oracle.quantize_group(w, q, oracle.GRID_SIGNED_SYM)
        assert r["gamma"] == gamma
        assert np.array_equal(r["c"], a)


# --------------------------------------------------------------------------
# eq:minmax asymmetric grid
# --------------------------------------------------------------------------

@pytest.mark.parametrize("q", QS)
def test_asym_codes_are_nearest_grid_points(q):
    umax = (1 << q) - 1
    groups = list(lattice_groups(3, 8)) + list(random_groups(200, 32, 17))
    for w in groups:
        r = oracle.quantize_group(w, q, oracle.GRID_ASYM)
        mn, mx = float(np.min(w)), float(np.max(w))
        if mx == mn:
            assert np.all(r["u"] == 0)
            continue
        s = F(r["s32"])
        assert s > 0
        # the stored min and scale are the fp16 roundings (numpy's conversion)
        assert r["m16"] == int(np.float16(np.float32(mn)).view(np.uint16))
        assert r["s16"] == int(np.float16(np.float32(r["s32"])).view(np.uint16))
        for j, x in enumerate(w):
            d = np.float32(x) - np.float32(mn)  # the fl32(w - min) of the reading
            u = nearest_index(F(float(d)), F(0), s, range(umax + 1))
            assert r["u"][j] == u
            if F(float(d)) == F(float(x)) - F(mn):  # exact subtraction
                assert abs(F(float(x)) - (F(mn) + s * r["u"][j])) <= s / 2
        assert r["u"][int(np.argmin(w))] == 0
        assert r["u"][int(np.argmax(w))] == umax


# --------------------------------------------------------------------------
# packed layout
# --------------------------------------------------------------------------

@pytest.mark.parametrize("q", QS)
@pytest.mark.parametrize("g", [8, 32, 128])
def test_pack_layout_bitwise(q, g):
    rng = np.random.default_rng(q * 1000 + g)
    for _ in range(50):
        u = rng.integers(0, 1 << q, g).astype(np.uint8)
        b = oracle.pack_group(u, q)
        assert b.size == g * q // 8
        bits = np.unpackbits(b, bitorder="little")
        if q == 4:
            got = bits.reshape(g, 4) @ (1 << np.arange(4))
        elif q == 2:
            got = bits.reshape(g, 2) @ (1 << np.arange(2))
        else:
            lo = bits[: 2 * g].reshape(g, 2) @ (1 << np.arange(2))
            hi = bits[2 * g:]
            got = lo + 4 * hi
        assert np.array_equal(got, u)
        assert np.array_equal(oracle.unpack_group(b, g, q), u)


def test_matrix_quantize_is_groupwise():
    for q in QS:
        for grid in (0, 1, 2):
            W = random_groups(6, 256, 31 + q)
            W = W.reshape(6, 256)
            codes, scales, mins, clip, _ = oracle.quantize(W, q, 32, grid, clip_counts=True)
            gb = 32 * q // 8
            flat = W.reshape(-1, 32)
            for G in range(flat.shape[0]):
                r = oracle.quantize_group(flat[G], q, grid)
                assert bytes(codes.reshape(-1, gb)[G]) == bytes(oracle.pack_group(r["u"], q))
                assert scales.ravel()[G] == r["s16"]
                if grid == 2:
                    assert mins.ravel()[G] == r["m16"]
                assert clip.reshape(-1, 2)[G, 0] == r["n_self"]
                assert clip.reshape(-1, 2)[G, 1] == r["n_other"]


# --------------------------------------------------------------------------
# dequantisation and the fp64 matmul reference
# --------------------------------------------------------------------------

def _numpy_dequant(codes, scales, mins, n, k, q, g, grid):
    gb = g * q // 8
    u = np.stack([oracle.unpack_group(cg, g, q) for cg in codes.reshape(-1, gb)])
    s = scales.reshape(-1, 1).view(np.float16).astype(np.float32)
    if grid == oracle.GRID_ASYM:
        m = mins.reshape(-1, 1).view(np.float16).astype(np.float32)
        return (s * u.astype(np.float32) + m).reshape(n, k)
    return (s * (u.astype(np.float32) - (1 << (q - 1)))).reshape(n, k)


@pytest.mark.parametrize("grid", [0, 1, 2])
@pytest.mark.parametrize("q", QS)
def test_dequantize_matches_numpy(q, grid):
    n, k, g = 16, 256, 32
    W = inputs.student_t_weights(n, k, 5 + q)
    codes, scales, mins, _, _ = oracle.quantize(W, q, g, grid)
    got = oracle.dequantize(codes, scales, mins, n, k, q, g, grid)
    ref = _numpy_dequant(codes, scales, mins, n, k, q, g, grid)
    assert np.array_equal(got.view(np.uint32), ref.view(np.uint32))
    part = oracle.dequantize(codes, scales, mins, n, k, q, g, grid, rows=(5, 3))
    assert np.array_equal(part, got[5:8])


def test_matmul_f64_matches_numpy():
    rng = np.random.default_rng(0)
    What = rng.standard_normal((40, 300)).astype(np.float32)
    xb = inputs.normal_bf16_bits((3, 300), 1)
    x = inputs.bf16_bits_to_f32(xb).astype(np.float64)
    ref = x @ What.astype(np.float64).T
    got = oracle.matmul_f64(What, xb)
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-12)
    # a one-hot activation picks one column of the weights exactly
    e = np.zeros((1, 300), np.float32)
    e[0, 17] = 1.0
    assert np.array_equal(oracle.matmul_f64(What, inputs.f32_to_bf16_bits(e))[0],
                          What[:, 17].astype(np.float64))


@pytest.mark.parametrize("grid", [0, 1, 2])
def test_gemv_is_matmul_of_dequantised(grid):
    n, k, q, g = 24, 512, 3, 32
    W = inputs.student_t_weights(n, k, 8)
    codes, scales, mins, _, _ = oracle.quantize(W, q, g, grid)
    xb = inputs.normal_bf16_bits((4, k), 2)
    y = oracle.gemv(codes, scales, mins, n, k, q, g, grid, xb)
    What = _numpy_dequant(codes, scales, mins, n, k, q, g, grid)
    ref = inputs.bf16_bits_to_f32(xb).astype(np.float64) @ What.astype(np.float64).T
    np.testing.assert_allclose(y, ref, rtol=1e-12, atol=1e-12)


# --------------------------------------------------------------------------
# flags and extreme magnitudes
# --------------------------------------------------------------------------

def test_nonfinite_and_range_flags():
    w = inputs.student_t_weights(1, 32, 3)[0]
    bad = w.copy()
    bad[5] = np.nan
    for grid in (0, 1, 2):
        assert oracle.quantize_group(bad, 4, grid)["flags"] & oracle.FLAG_NONFINITE
        assert oracle.quantize_group(w, 4, grid)["flags"] == 0
    big = (w / np.max(np.abs(w)) * 1e6).astype(np.float32)
    assert oracle.quantize_group(big, 2, 1)["flags"] & oracle.FLAG_RANGE


@pytest.mark.parametrize("q", QS)
@pytest.mark.parametrize("e", [-140, -130, -100, -20, 20, 60, 100])
def test_extreme_magnitudes_still_round_to_nearest(q, e):
    """Subnormal and huge groups: codes stay the nearest grid points for the
    scale the oracle used (eq:quantizer), for both signs."""
    A = alphabet(q)
    W = random_groups(20, 32, 1000 + e + q)
    for w in W:
        w = (w.astype(np.float64) * 2.0 ** e).astype(np.float32)
        if float(np.max(np.abs(w))) == 0:
            continue
        for gm in (1, -1):
            r = oracle.quantize_group_gamma(w, q, gm)
            s = F(r["s32"])
            if s == 0:
                continue
            for j in range(32):
                assert r["c"][j] == nearest_index(F(float(w[j])), F(0), s, A)


@pytest.mark.parametrize("q", QS)
def test_underflowed_alpha_is_a_zero_group(q):
    """alpha = M / 2^(q-1) of a subnormal M is rounded to a multiple of
    2^-149 (ties to the even multiple), so it is zero exactly when
    M = j * 2^-149 with j <= 2^(q-2).  Then no scale s != 0 exists
    (eq:absmax needs s != 0) and the group gets the all-zero group's
    outputs: every code 0 (stored 2^(q-1)) and a +0 scale, for both signs."""
    half = 1 << (q - 1)
    for j in range(1, 4 * half + 1):
        M = j * 2.0 ** -149
        for sign in (1.0, -1.0):
            w = np.zeros(32, np.float32)
            w[3] = np.float32(sign * M)
            w[7] = np.float32(-sign * 2.0 ** -149) if j > 1 else 0.0
            for grid in (oracle.GRID_UNSIGNED_SYM, oracle.GRID_SIGNED_SYM):
                r = oracle.quantize_group(w, q, grid)
                if F(j, half) <= F(1, 2):  # alpha rounds to zero
                    assert r["s32"] == 0.0 and r["s16"] == 0x0000, (j, sign)
                    assert np.all(r["u"] == half) and np.all(r["c"] == 0)
                    assert r["flags"] == 0
                else:
                    assert r["s32"] != 0.0
                    s = F(r["s32"])
                    for e in range(32):
                        assert r["c"][e] == nearest_index(F(float(w[e])), F(0), s, alphabet(q))


@pytest.mark.parametrize("q", QS)
def test_asym_zero_minimum_is_stored_as_plus_zero(q):
    """Reading of eq:minmax's stored minimum: a zero minimum is stored as +0
    (fp16 bits 0x0000), whichever zero the group holds or meets first."""
    base = np.linspace(0.0, 1.0, 32).astype(np.float32)
    for zeros in ([-0.0], [-0.0, 0.0], [0.0, -0.0]):
        w = base.copy()
        for i, z in enumerate(zeros):
            w[i] = np.float32(z)
        assert np.signbit(w[0]) == np.signbit(np.float32(zeros[0]))
        r = oracle.quantize_group(w, q, oracle.GRID_ASYM)
        assert r["m16"] == 0x0000, zeros
        assert r["u"][0] == 0 and r["u"][31] == (1 << q) - 1


# --------------------------------------------------------------------------
# Q8_0 activations (narrow range, blocks of 32): the runtime pairing of the
# weight formats (Sec. 5 "Composition with PTQ methods", Appendix C
# "Algorithm details")
# --------------------------------------------------------------------------

def _q8_hand_blocks():
    for line in open(os.path.join(GOLDEN, "q8_act_blocks.txt")):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        f = [v.strip() for v in line.split("|")]
        x = np.zeros(32, np.float32)
        xs = [float(v) for v in f[0].split()]
        x[:len(xs)] = xs
        q = np.zeros(32, np.int8)
        qs = [int(v) for v in f[1].split()]
        q[:len(qs)] = qs
        yield x, q, int(f[2], 16)


def test_q8_hand_worked_blocks():
    blocks = list(_q8_hand_blocks())
    assert len(blocks) == 4
    for x, q_want, d_want in blocks:
        xb = inputs.f32_to_bf16_bits(x)
        assert np.array_equal(inputs.bf16_bits_to_f32(xb), x)  # exact bf16 values
        q, d, flags = oracle.quantize_act_q8(xb[None, :])
        assert flags == 0
        assert np.array_equal(q[0], q_want)
        assert int(d[0, 0]) == d_want


def _q8_blocks(rng, count):
    """bf16 blocks of 32: normal, heavy-tailed, tiny, huge and tie-rich."""
    out = []
    for i in range(count):
        kind = i % 5
        if kind == 0:
            v = rng.standard_normal(32)
        elif kind == 1:
            v = rng.standard_t(3, 32) * 10.0
        elif kind == 2:
            v = rng.standard_normal(32) * 1e-30
        elif kind == 3:
            v = rng.standard_normal(32) * 1e30
        else:  # multiples of M/254 hit half-integer quotients
            v = rng.integers(-254, 255, 32) * 0.5
        out.append(inputs.f32_to_bf16_bits(v.astype(np.float32)))
    return np.stack(out)


def test_q8_codes_are_nearest_narrow_grid_points():
    rng = np.random.default_rng(8)
    xb = _q8_blocks(rng, 400)
    q, d16, flags = oracle.quantize_act_q8(xb.reshape(1, -1))
    # the huge blocks' scales overflow fp16 (flagged); their codes still
    # follow the fp32 scale
    assert flags == oracle.FLAG_RANGE
    q = q.reshape(-1, 32)
    x = inputs.bf16_bits_to_f32(xb)
    for i in range(x.shape[0]):
        M = float(np.max(np.abs(x[i])))
        d = F(float(np.float32(M) / np.float32(127.0)))  # fl32(M / 127)
        for j in range(32):
            t = F(float(x[i, j])) / d
            lo = t.numerator // t.denominator
            frac = t - lo
            want = lo + 1 if frac > F(1, 2) or (frac == F(1, 2) and lo % 2 == 1) else lo
            want = max(-127, min(127, want))
            assert q[i, j] == want, (i, j)
        # the block maximum lands on +-127, and -128 never appears
        jm = int(np.argmax(np.abs(x[i])))
        assert abs(int(q[i, jm])) == 127
        assert int(q[i].min()) >= -127


def test_q8_is_odd_and_its_error_is_bounded():
    rng = np.random.default_rng(9)
    xb = _q8_blocks(rng, 200).reshape(1, -1)
    q, d16, _ = oracle.quantize_act_q8(xb)
    qn, dn, _ = oracle.quantize_act_q8(xb ^ np.uint16(0x8000))  # -x
    assert np.array_equal(qn, -q) and np.array_equal(dn, d16)
    x = inputs.bf16_bits_to_f32(xb).reshape(-1, 32).astype(np.float64)
    qf = q.reshape(-1, 32).astype(np.float64)
    M = np.abs(x).max(axis=1)
    d32 = (M.astype(np.float32) / np.float32(127.0)).astype(np.float64)
    dh = np.array([oracle.f16_to_f32(int(v)) for v in d16.ravel()], np.float64)
    assert np.all(np.abs(x - d32[:, None] * qf) <= d32[:, None] / 2 * (1 + 1e-12))
    assert np.array_equal(dh, np.array([oracle.f16_to_f32(oracle.f32_to_f16(float(v)))
                                        for v in d32]))


def test_q8_flags():
    x = np.zeros((1, 64), np.float32)
    x[0, 3] = np.inf
    q, d, flags = oracle.quantize_act_q8(inputs.f32_to_bf16_bits(x))
    assert flags & oracle.FLAG_NONFINITE
    assert not q[0, :32].any() and d[0, 0] == 0
    y = np.zeros((1, 32), np.float32)
    y[0, 0] = 3.0e38  # d = 2.4e36 overflows fp16
    q, d, flags = oracle.quantize_act_q8(inputs.f32_to_bf16_bits(y))
    assert flags & oracle.FLAG_RANGE and (int(d[0, 0]) & 0x7fff) == 0x7c00 and q[0, 0] == 127


@pytest.mark.parametrize("grid", [oracle.GRID_SIGNED_SYM, oracle.GRID_ASYM])
def test_gemv_q8_is_matmul_of_dequantised_operands(grid):
    n, k, q, g = 24, 128, 4, 32
    W = inputs.student_t_weights(n, k, 77)
    codes, scales, mins, _, _ = oracle.quantize(W, q, g, grid)
    xb = inputs.normal_bf16_bits((3, k), 78)
    xq, xd, _ = oracle.quantize_act_q8(xb)
    y = oracle.gemv_q8(codes, scales, mins, n, k, q, g, grid, xq, xd)
    What = oracle.dequantize(codes, scales, mins, n, k, q, g, grid).astype(np.float64)
    dh = np.array([[oracle.f16_to_f32(int(v)) for v in row] for row in xd], np.float64)
    xh = xq.astype(np.float64) * np.repeat(dh, 32, axis=1)
    np.testing.assert_allclose(y, xh @ What.T, rtol=1e-12, atol=1e-12)


# --------------------------------------------------------------------------
# Normalized Hadamard rotation before quantization (Sec. 5 "Composition with
# PTQ methods", Appendix C): the fp32 fast transform against the fp64
# product with the Sylvester matrix of scipy, and its algebraic properties
# --------------------------------------------------------------------------

@pytest.mark.parametrize("b", [2, 8, 32, 128, 4096])
def test_fwht_is_the_normalized_sylvester_product(b):
    scipy_linalg = pytest.importorskip("scipy.linalg")
    H = scipy_linalg.hadamard(b).astype(np.float64)
    rng = np.random.default_rng(b)
    for trial in range(4):
        x = (rng.standard_t(4, b) * 0.02).astype(np.float32)
        y = oracle.fwht(x)
        ref = H @ x.astype(np.float64) / np.sqrt(b)
        # log2(b) fp32 butterfly stages on partial sums bounded by sum|x|,
        # plus the final multiply: a few ulps of sum|x| / sqrt(b)
        bound = (np.log2(b) + 2) * 2.0 ** -23 * np.sum(np.abs(x)) / np.sqrt(b)
        assert np.max(np.abs(y - ref)) <= bound
        # orthogonal: the norm is kept
        assert abs(np.linalg.norm(y.astype(np.float64)) / np.linalg.norm(x.astype(np.float64)) - 1) < 1e-5
        # an involution: the normalized transform is its own inverse
        assert np.max(np.abs(oracle.fwht(y) - x)) <= 2 * bound


@pytest.mark.parametrize("b", [4, 16, 64, 256])
def test_fwht_exact_cases(b):
    norm = np.float32(1.0 / np.sqrt(b))
    assert norm == np.float32(2.0 ** -(np.log2(b) / 2))  # b a power of 4: exact power of two
    # a one-hot input is one column of H/sqrt(b): +-norm exactly
    scipy_linalg = pytest.importorskip("scipy.linalg")
    H = scipy_linalg.hadamard(b)
    for j in (0, 1, b // 2 + 1, b - 1):
        e = np.zeros(b, np.float32)
        e[j] = 1.0
        assert np.array_equal(oracle.fwht(e), (H[:, j] * norm).astype(np.float32))
    # all ones: sqrt(b) in the first slot, zeros elsewhere, exactly
    y = oracle.fwht(np.ones(b, np.float32))
    assert y[0] == np.float32(b) * norm and np.all(y[1:] == 0)


def test_rotation_of_rows_and_columns_is_blockwise():
    rng = np.random.default_rng(7)
    W = rng.standard_normal((64, 256)).astype(np.float32)
    Wr = oracle.rotate(W, 32, "rows")
    for r in (0, 17, 63):
        for c0 in (0, 96, 224):
            assert np.array_equal(Wr[r, c0:c0 + 32], oracle.fwht(W[r, c0:c0 + 32]))
    Wc = oracle.rotate(W, 16, "cols")
    for c in (0, 5, 255):
        for r0 in (0, 48):
            assert np.array_equal(Wc[r0:r0 + 16, c], oracle.fwht(W[r0:r0 + 16, c]))
    # the product the rotations preserve: (W R)(R x) = W x for an orthogonal R
    scipy_linalg = pytest.importorskip("scipy.linalg")
    R = np.kron(np.eye(256 // 32), scipy_linalg.hadamard(32) / np.sqrt(32))
    x = rng.standard_normal(256)
    np.testing.assert_allclose(Wr.astype(np.float64) @ (R @ x), W.astype(np.float64) @ x,
                               rtol=1e-5, atol=1e-4)


# --------------------------------------------------------------------------
# Signed LSQ scale refinement (Sec. 5 learned grid parameters, Appendix C:
# LSQ with s != 0 for the signed formats, s > 0 for the conventional ones),
# in its data-free reading on each group's reconstruction loss
# --------------------------------------------------------------------------

def _recon_loss(w, s, q):
    """sum (w - s16 c)^2 in exact rationals, c = the nearest code of the
    exact quotient w/s (ties to even) clipped to A_q, s16 = fl16(s)."""
    A = alphabet(q)
    s16 = F(float(np.float16(np.float32(s))))
    tot = F(0)
    for x in w:
        c = nearest_index(F(float(x)), F(0), F(float(np.float32(s))), A)
        tot += (F(float(x)) - s16 * c) ** 2
    return tot


@pytest.mark.parametrize("grid", [oracle.GRID_UNSIGNED_SYM, oracle.GRID_SIGNED_SYM])
@pytest.mark.parametrize("q", QS)
def test_lsq_zero_steps_is_the_absmax_quantizer(q, grid):
    W = random_groups(12, 128, 500 + q).reshape(6, 256)
    codes, scales, _, _, flags = oracle.quantize(W, q, 32, grid)
    lc, ls, lf = oracle.lsq_quantize(W, q, 32, grid, 0, 0.01)
    assert np.array_equal(lc, codes) and np.array_equal(ls, scales) and lf == flags


@pytest.mark.parametrize("q", QS)
def test_lsq_on_grid_group_is_a_fixed_point(q):
    # w = s0 * c with the outlier on -2^(q-1): zero reconstruction error, so
    # every LSQ gradient term (2 e_i) d_i is zero and s never moves
    rng = np.random.default_rng(q)
    half = 1 << (q - 1)
    s0 = np.float32(-0.015625)
    c = rng.integers(-half + 1, half, 32)
    c[5] = -half
    w = (s0 * c).astype(np.float32)
    assert oracle.quantize_group(w, q, oracle.GRID_SIGNED_SYM)["s32"] == s0
    assert oracle.lsq_scale(w, q, True, 25, 0.05) == s0


@pytest.mark.parametrize("q", QS)
def test_lsq_keeps_the_sign_and_is_odd(q):
    W = random_groups(200, 32, 510 + q)
    for w in W:
        if np.max(w) == -np.min(w):
            continue  # a sign tie breaks the odd symmetry of the sign rule itself
        s0 = oracle.quantize_group(w, q, oracle.GRID_SIGNED_SYM)["s32"]
        s = oracle.lsq_scale(w, q, True, 20, 0.02)
        assert s != 0 and np.sign(s) == np.sign(s0)
        assert oracle.lsq_scale(-w, q, True, 20, 0.02) == -s       # exact odd symmetry
        su = oracle.lsq_scale(w, q, False, 20, 0.02)
        assert su > 0                                             # s > 0 stays positive
        # an aggressive rate must still never cross or reach zero
        assert np.sign(oracle.lsq_scale(w, q, True, 10, 50.0)) == np.sign(s0)


@pytest.mark.parametrize("q", QS)
def test_lsq_descends_the_reconstruction_loss(q):
    """Gradient steps on L(s) = ||w - s c||^2 with a small rate: the loss of
    the refined scale (exact rationals) is lower than the signed absmax loss
    on aggregate, and no worse on a clear majority of groups (the
    straight-through gradient is LSQ's estimate, not the loss's derivative,
    so single groups can get worse: measured 60-88 % improve at q = 2..4)."""
    W = random_groups(120, 32, 520 + q)
    better, before, after = 0, F(0), F(0)
    for w in W:
        s0 = oracle.quantize_group(w, q, oracle.GRID_SIGNED_SYM)["s32"]
        s = oracle.lsq_scale(w, q, True, 20, 0.01)
        l0, l1 = _recon_loss(w, s0, q), _recon_loss(w, s, q)
        better += l1 <= l0
        before += l0
        after += l1
    assert better >= 0.6 * len(W)
    assert after < before
