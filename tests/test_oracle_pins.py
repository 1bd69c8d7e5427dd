"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: a worked
example printed in the paper, hand-computed points of Algorithm 1, closed
forms of special rows, a textbook routine a special case reduces to, or an
invariant of the definition.
"""
import math
from fractions import Fraction
from pathlib import Path

import numpy as np
import pytest

import oracle

GOLDEN = Path(__file__).parent / "golden"


def _rows(name):
    out = []
    for line in (GOLDEN / name).read_text().splitlines():
        line = line.strip()
        if line and not line.startswith("#"):
            out.append(line.split())
    return out


# ---------------------------------------------------------------- I-Log2

def test_ilog2_worked_example():
    (bits, M, chi, res), = _rows("ilog2_worked_example.txt")
    x = int(bits, 2)
    assert x.bit_length() - 1 == int(M)
    assert (x >> (int(M) - 1)) & 1 == int(chi)
    assert oracle.ilog2(x) == int(res)


def test_ilog2_is_log2_rounded_at_one_and_a_half():
    # I-Log2 rounds log2 at 1.5 * 2^M: it counts the thresholds 2, 3, 6, 12, 24, ...
    # (T_1 = 2, T_k = 3 * 2^(k-2)) that x reaches.
    thresholds = [2] + [3 * 2 ** (k - 2) for k in range(2, 64)]
    xs = list(range(1, 1 << 14)) + [(1 << k) + o for k in range(14, 62) for o in (-1, 0, 1)] \
        + [3 << k for k in range(13, 60)] + [(3 << k) - 1 for k in range(13, 60)]
    for x in xs:
        assert oracle.ilog2(x) == sum(1 for t in thresholds if x >= t), x


# ---------------------------------------------------------------- i-exp

def test_iexp_hand_points():
    rows = _rows("iexp_s0p1.txt")
    assert rows[0][0] == "consts"
    assert oracle.iexp_consts(0.1) == tuple(int(v) for v in rows[0][1:])
    for q, val in rows[1:]:
        assert oracle.iexp(int(q), 0.1) == int(val), q


def test_polynomial_gap_matches_supplement():
    # Eq. 31: L(p) = 0.3585 (p + 1.353)^2 + 0.344 approximates exp(p) on (-ln2, 0].
    # The supplement prints a largest gap of 1.9e-3; evaluating the printed
    # constants gives 2.128e-3 at p ~ -0.138.
    p = np.linspace(-math.log(2), 0, 2_000_001)
    gap = np.abs(0.3585 * (p + 1.353) ** 2 + 0.344 - np.exp(p))
    assert 1.8e-3 < gap.max() < 2.2e-3


@pytest.mark.parametrize("s", [1 / 256, 0.01, 0.0425, 0.17])
def test_iexp_tracks_exp(s):
    # Algorithm 1 splits q s = z (q_ln2 s) + q_p s and returns L(q_p s) / 2^z in
    # units of a s^2 / 2^n.  Against 2^-z exp(q_p s) the error is the polynomial
    # gap (<= 2.2e-3) plus the flooring of q_b and q_c (O(s)); against exp(q s)
    # it also carries exp(z (q_ln2 s + ln2)), the drift of the floored q_ln2.
    s = float(np.float32(s))
    q_ln2, q_b, q_c = oracle.iexp_consts(s)
    scale = 0.3585 * s * s / 2.0 ** 15
    drift = q_ln2 * s + math.log(2)
    assert -s < drift <= 0
    for q in range(0, 15 * q_ln2 - 1, -1):
        z = q // q_ln2
        qp = q - z * q_ln2
        approx = oracle.iexp(q, s) * scale
        assert abs(approx - 2.0 ** (-z) * math.exp(qp * s)) <= (2.2e-3 + 4.5 * s) * 2.0 ** (-z), q
        exact = math.exp(s * q)
        assert abs(approx * math.exp(z * drift) - exact) <= (2.2e-3 + 4.5 * s) * 2.0 ** (-z) * 1.01, q


@pytest.mark.parametrize("s", [0.0078125, 0.03, 0.1, 0.5])
def test_iexp_halves_per_band(s):
    # Algorithm 1: stepping q by q_ln2 increments z and halves the output exactly.
    q_ln2, _, _ = oracle.iexp_consts(s)
    for q in range(0, 14 * q_ln2, -1):
        assert oracle.iexp(q, s) == 2 * oracle.iexp(q + q_ln2, s)


# ---------------------------------------------------------------- Log-Int-Softmax

def test_lis_uniform_rows():
    for L, code in _rows("lis_uniform_rows.txt"):
        L, code = int(L), int(code)
        for val in (-128, 0, 127):
            codes, S = oracle.lis_softmax(np.full((1, L), val, np.int8), L, 0.05)
            assert set(codes[0].tolist()) == {code}
        # Eq. 14 float form gives the same
        assert code == min(15, round(math.log2(L)))


@pytest.mark.parametrize("L", [2, 49, 197, 577, 1024])
def test_lis_one_hot_row(L):
    # one logit far above the rest: its share is ~1 -> code 0; the others'
    # shares are below 2^-15.5 -> clipped to 15.
    s = 0.1  # 255 * s = 25.5 > 15 ln2 * ... makes the others negligible
    row = np.full((1, L), -128, np.int8)
    row[0, L // 3] = 127
    codes, S = oracle.lis_softmax(row, L, s)
    assert codes[0, L // 3] == 0
    assert all(codes[0, j] == 15 for j in range(L) if j != L // 3)


def test_lis_shift_and_permutation_invariance():
    rng = np.random.default_rng(7)
    L = 197
    base = rng.integers(-100, 60, size=(16, L)).astype(np.int8)
    c0, S0 = oracle.lis_softmax(base, L, 0.04)
    c1, S1 = oracle.lis_softmax((base.astype(np.int16) + 40).astype(np.int8), L, 0.04)
    assert np.array_equal(c0, c1) and np.array_equal(S0, S1)
    perm = rng.permutation(L)
    c2, S2 = oracle.lis_softmax(np.ascontiguousarray(base[:, perm]), L, 0.04)
    assert np.array_equal(c2, c0[:, perm]) and np.array_equal(S2, S0)


def test_lis_codes_monotone_in_logit():
    rng = np.random.default_rng(8)
    L = 577
    x = rng.integers(-128, 128, size=(8, L)).astype(np.int8)
    for s in (0.01, 0.05, 0.2):
        codes, _ = oracle.lis_softmax(x, L, s)
        for r in range(x.shape[0]):
            order = np.argsort(x[r].astype(np.int32), kind="stable")
            assert np.all(np.diff(codes[r][order].astype(np.int32)) <= 0)


def _ref_ilog2(x):
    m = x.bit_length() - 1
    return m + ((x >> (m - 1)) & 1 if m >= 1 else 0)


def test_lis_brute_force_pairs():
    # every row of length 2 (up to the shift invariance): exact rational
    # reciprocal rounded half up, then I-Log2, then clip
    for s in (0.0078125, 0.05, 0.3):
        q_ln2, q_b, q_c = oracle.iexp_consts(s)
        rows = np.zeros((256, 2), np.int8)
        rows[:, 0] = 127
        rows[:, 1] = np.arange(127, -129, -1)
        codes, S = oracle.lis_softmax(rows, 2, s)
        for r in range(256):
            e = [oracle.iexp(int(rows[r, j]) - 127, s) for j in range(2)]
            tot = sum(e)
            assert S[r] == tot
            for j in range(2):
                qrev = math.floor(Fraction(tot, e[j]) + Fraction(1, 2))
                assert codes[r, j] == min(15, _ref_ilog2(qrev))


def test_lis_agrees_with_float_log2_quantizer():
    # Eq. 14 in floating point: clip(round(-log2 softmax), 0, 15).  LIS rounds
    # linearly (1.5 * 2^M) where Eq. 14 rounds in the log domain (sqrt2 * 2^M),
    # and i-exp is approximate, so codes may differ by one; nearly all agree.
    rng = np.random.default_rng(9)
    L = 197
    x = np.clip(np.rint(rng.normal(0, 25, size=(64, L))), -128, 127).astype(np.int8)
    s = 0.0425
    codes, _ = oracle.lis_softmax(x, L, s)
    z = s * x.astype(np.float64)
    p = np.exp(z - z.max(axis=1, keepdims=True))
    p /= p.sum(axis=1, keepdims=True)
    ref = np.clip(np.rint(-np.log2(p)), 0, 15)
    diff = np.abs(codes.astype(np.int64) - ref)
    assert diff.max() <= 1
    assert (diff == 0).mean() > 0.85


def test_lis_relpos_bias():
    rng = np.random.default_rng(10)
    L, H, w = 49, 3, 7
    x = rng.integers(-128, 128, size=(2 * H * L, L)).astype(np.int8)
    zero = np.zeros((H, 169), np.int8)
    c0, _ = oracle.lis_softmax(x, L, 0.05)
    c1, _ = oracle.lis_softmax(x, L, 0.05, bias=zero, heads=H, window=w)
    assert np.array_equal(c0, c1)
    # a bias that is constant over each head leaves every code unchanged (max subtraction)
    const = np.repeat(np.array([[-16], [5], [16]], np.int8), 169, axis=1)
    c2, _ = oracle.lis_softmax(x, L, 0.05, bias=const, heads=H, window=w)
    assert np.array_equal(c0, c2)
    # a bias equals adding the looked-up table entry to the logit
    tab = rng.integers(-16, 17, size=(H, 169)).astype(np.int8)
    c3, _ = oracle.lis_softmax(x, L, 0.05, bias=tab, heads=H, window=w)
    ii, jj = np.meshgrid(np.arange(L), np.arange(L), indexing="ij")
    idx = (ii // w - jj // w + w - 1) * (2 * w - 1) + (ii % w - jj % w + w - 1)
    xb = x.reshape(2, H, L, L).astype(np.int16) + tab[None, :, idx]
    # with a bias the logit leaves int8; a shift by a per-row constant keeps it in range
    xb = xb - xb.max(axis=-1, keepdims=True) + 127
    assert xb.min() >= -160
    clipped = np.maximum(xb, -128).astype(np.int8).reshape(-1, L)
    c4, _ = oracle.lis_softmax(clipped, L, 0.05)
    safe = (xb >= -128).reshape(-1, L).all(axis=1)
    assert safe.sum() > 0
    assert np.array_equal(c3[safe], c4[safe])


# ---------------------------------------------------------------- BitShift Attn.V

def test_attn_v_is_power_of_two_matmul():
    # Eq. 15: (V - zp) << (15 - code) summed over keys == matmul with 2^(15-code)
    rng = np.random.default_rng(11)
    BH, L, d = 3, 67, 32
    codes = rng.integers(0, 16, size=(BH * L, L)).astype(np.uint8)
    v = rng.integers(-128, 128, size=(BH, L, d)).astype(np.int8)
    for zp in (0, 5):
        acc, ov = oracle.lis_attn_v(codes, v, zp)
        w = (2 ** (15 - codes.astype(np.int64))).reshape(BH, L, L)
        ref = np.matmul(w, v.astype(np.int64) - zp)
        assert not ov
        assert np.array_equal(acc.astype(np.int64), ref)


def test_attn_v_special_rows():
    rng = np.random.default_rng(12)
    BH, L, d = 2, 49, 64
    v = rng.integers(-128, 128, size=(BH, L, d)).astype(np.int8)
    all15 = np.full((BH * L, L), 15, np.uint8)
    acc, _ = oracle.lis_attn_v(all15, v)
    assert np.array_equal(acc, np.repeat(v.astype(np.int64).sum(axis=1, keepdims=True), L, axis=1))
    onehot = np.full((BH * L, L), 15, np.uint8)
    onehot[:, 10] = 0
    acc, _ = oracle.lis_attn_v(onehot, v)
    ref = v.astype(np.int64).sum(axis=1, keepdims=True) + (2 ** 15 - 1) * v[:, 10:11].astype(np.int64)
    assert np.array_equal(acc, np.repeat(ref, L, axis=1))


# ---------------------------------------------------------------- PTF

def _minmax_codes(x):
    # Eqs. 3-5, layer-wise MinMax, fp32 throughout
    x = x.astype(np.float32)
    lo, hi = x.min(), x.max()
    s = np.float32(hi - lo) / np.float32(255)
    zp = int(np.clip(np.rint(np.float32(-lo) / s), 0, 255))
    q = np.clip(np.rint(x / s) + zp, 0, 255).astype(np.uint8)
    return s, zp, q


def _channels(seed, rows=300, C=40):
    rng = np.random.default_rng(seed)
    r = np.exp(rng.normal(0, 1, C)) * 2
    m = rng.normal(0, 0.25, C) * r
    return (m + r / 6 * rng.normal(0, 1, (rows, C))).astype(np.float32)


def test_minmax_range_is_the_data_range():
    # Eqs. 4-5 over all calibration elements, the range not widened to include 0: all-positive
    # data keeps its own minimum, and extremes anywhere (the first row away from its first
    # element, the last row) are found; K = 0 then gives s = (7 - 3) / 255 and zp = clip(-191) = 0
    rng = np.random.default_rng(12)
    x = rng.uniform(3.5, 6.5, (50, 7)).astype(np.float32)
    x[0, 5] = 7.0
    x[49, 6] = 3.0
    assert oracle.calibrate_minmax(x) == (3.0, 7.0)
    x2 = x.copy()
    x2[0, 3] = 2.5
    assert oracle.calibrate_minmax(x2) == (2.5, 7.0)
    s, zp, _, _ = oracle.calibrate_ptf(x, K=0)
    assert np.float32(s) == np.float32(np.float32(4.0) / np.float32(255.0)) and zp == 0


def test_ptf_k0_is_minmax():
    x = _channels(1)
    s, zp, alpha, sse = oracle.calibrate_ptf(x, K=0)
    s_mm, zp_mm, q_mm = _minmax_codes(x)
    assert np.all(alpha == 0)
    assert np.float32(s) == s_mm and zp == zp_mm
    assert np.array_equal(oracle.ptf_quantize(x, s, zp, alpha), q_mm)


@pytest.mark.parametrize("K", [1, 3, 5])
def test_ptf_all_factors_k_is_minmax(K):
    # 2^K s equals the MinMax scale exactly, so alpha_c = K for all c is MinMax
    x = _channels(2)
    s, zp, _, _ = oracle.calibrate_ptf(x, K=K)
    s_mm, zp_mm, q_mm = _minmax_codes(x)
    assert np.float32(s) * np.float32(2 ** K) == s_mm and zp == zp_mm
    q = oracle.ptf_quantize(x, s, zp, np.full(x.shape[1], K, np.uint8))
    assert np.array_equal(q, q_mm)


def test_ptf_factor_follows_channel_range():
    # channel j spans 0.9 * R / 2^j around 0: alpha = K - j is the finest factor
    # whose grid does not clip it (coarser wastes resolution, finer clips)
    rng = np.random.default_rng(3)
    R, K, rows = 10.0, 3, 4000
    cols = []
    for j in range(6):
        c = rng.uniform(-0.9, 0.9, rows) * R / 2 ** j
        c[:2] = [-0.9 * R / 2 ** j, 0.9 * R / 2 ** j]
        cols.append(c)
    x = np.stack(cols, axis=1).astype(np.float32)
    x[0, 0], x[1, 0] = -R, R  # the widest channel sets min / max
    s, zp, alpha, sse = oracle.calibrate_ptf(x, K=K)
    assert alpha.tolist() == [3, 2, 1, 0, 0, 0]
    assert np.array_equal(alpha, np.argmin(sse, axis=1))


def test_ptf_ties_take_the_smallest_factor():
    # a channel of zeros and a channel on the coarsest grid (values -s0, 0, s0 with s0 = 2^K s)
    # quantize without error for every factor: Eq. 10's minimum is attained by every alpha, and
    # the reading breaks the tie toward the smallest
    rng = np.random.default_rng(9)
    K, rows = 3, 500
    x = rng.uniform(-5.0, 5.0, (rows, 3)).astype(np.float32)
    x[0, 0], x[1, 0] = -5.0, 5.0
    s0 = np.float32(np.float32(10.0) / np.float32(255.0))
    x[:, 1] = 0.0
    x[:, 2] = rng.integers(-1, 2, rows).astype(np.float32) * s0
    s, zp, alpha, sse = oracle.calibrate_ptf(x, K=K)
    assert np.float32(s) * np.float32(2 ** K) == s0
    assert np.all(sse[1] == 0.0) and np.all(sse[2] == 0.0)
    assert alpha[1] == 0 and alpha[2] == 0


def test_ptf_sse_definition():
    x = _channels(4, rows=200, C=8)
    K = 3
    s, zp, alpha, sse = oracle.calibrate_ptf(x, K=K)
    for c in range(x.shape[1]):
        for a in range(K + 1):
            sa = np.float32(s) * np.float32(2 ** a)
            q = np.clip(np.rint(x[:, c] / sa), -zp, 255 - zp).astype(np.float32)
            d = (x[:, c] - q * sa).astype(np.float64)
            assert abs(sse[c, a] - np.sum(d * d)) <= 1e-9 * max(1.0, sse[c, a])


# ---------------------------------------------------------------- integer LayerNorm

def _ln_case(seed, rows=256, C=192, K=3):
    x = _channels(seed, rows=rows, C=C)
    s, zp, alpha, _ = oracle.calibrate_ptf(x, K=K)
    xq = oracle.ptf_quantize(x, s, zp, alpha)
    rng = np.random.default_rng(seed + 100)
    gamma = (1 + 0.1 * rng.normal(size=C)).astype(np.float32)
    beta = (0.1 * rng.normal(size=C)).astype(np.float32)
    return x, s, zp, alpha, xq, gamma, beta


def test_ln_integer_statistics():
    x, s, zp, alpha, xq, gamma, beta = _ln_case(5)
    y, m1, m2 = oracle.ptf_layernorm(xq, zp, alpha, gamma, beta, 0.02, 128)
    xh = (xq.astype(np.int64) - zp) * (2 ** alpha.astype(np.int64))
    assert np.array_equal(m1, xh.sum(axis=1))
    assert np.array_equal(m2, (xh * xh).sum(axis=1))
    assert np.all(xq.shape[1] * m2 - m1 * m1 >= 0)


def test_ln_matches_textbook_layernorm():
    # dequantized input -> fp64 LayerNorm (eps -> 0) -> output quantizer, vs the
    # integer path: the dyadic A (8-bit N2) and the rounding of B give at most a
    # couple of output steps
    x, s, zp, alpha, xq, gamma, beta = _ln_case(6, rows=512, C=384)
    s_out, zp_out = 0.03, 120
    y, _, _ = oracle.ptf_layernorm(xq, zp, alpha, gamma, beta, s_out, zp_out)
    xd = (xq.astype(np.float64) - zp) * (2.0 ** alpha) * s
    mu = xd.mean(axis=1, keepdims=True)
    sd = xd.std(axis=1, keepdims=True)
    yf = (xd - mu) / sd * gamma + beta
    ref = np.clip(np.rint(yf / s_out) + zp_out, 0, 255)
    diff = np.abs(y.astype(np.int64) - ref)
    assert diff.max() <= 2
    assert (diff == 0).mean() > 0.9


def test_ln_gamma_zero_and_constant_row():
    x, s, zp, alpha, xq, gamma, beta = _ln_case(7, rows=32, C=96)
    gamma = gamma.copy()
    gamma[5] = 0.0
    xq = xq.copy()
    xq[3, :] = 77
    alpha = alpha.copy()
    alpha[:] = 0
    s_out, zp_out = 0.01, 100
    y, _, _ = oracle.ptf_layernorm(xq, zp, alpha, gamma, beta, s_out, zp_out)
    beta_q = np.clip(np.rint((beta.astype(np.float64) / s_out).astype(np.float32)) + zp_out, 0, 255)
    assert np.all(y[:, 5] == beta_q[5])
    assert np.array_equal(y[3], beta_q.astype(np.uint8))


def test_ln_exact_row_by_hand():
    # A row whose statistics are exact: x - zp_in = +-64 on 8 channels (alpha = 0), so M1 = 0,
    # D = 8 * 8 * 64^2 = 2^18, sqrt(D) = 512, C / sqrt(D) = 2^-6, and the mean term vanishes.
    # With s_out = 2^-6, gamma = +-129.5 2^-6 and beta = 0: A = +-2.0234375 (nine significant
    # bits), and the supplement's output stage gives N1 = 7 - floor(log2 |A|) = 6 and
    # N2 = floor(129.5) = 129 (eight bits), Y = floor((sign(A) 129 X + 32) / 64) + zp_out:
    # the quotient is +-129.5 or +-128.5 and rounds to +-129, the sign that of A X, so
    # Y = clip(+-129 + zp_out).
    C = 8
    xq = np.array([[192, 64] * 4], np.uint8)
    alpha = np.zeros(C, np.uint8)
    beta = np.zeros(C, np.float32)
    s_out = 2.0 ** -6
    for sign, zp_out, want in ((1, 0, [129, 0]), (1, 126, [255, 0]), (-1, 200, [71, 255]), (-1, 129, [0, 255])):
        gamma = np.full(C, sign * 129.5 * 2.0 ** -6, np.float32)
        y, m1, m2 = oracle.ptf_layernorm(xq, 128, alpha, gamma, beta, s_out, zp_out)
        assert int(m1[0]) == 0 and int(m2[0]) == 8 * 64 * 64
        assert y[0].tolist() == want * 4, (sign, zp_out)


def test_ln_shift_by_factor_equals_minmax_path():
    # alpha = K everywhere with scale s equals alpha = 0 with scale 2^K s:
    # X_hat differs by the factor 2^K, which cancels in A X_hat and M1/sqrt(D);
    # only the 8-bit N2 of A and the rounding of B see the scale, so the
    # outputs agree within one step
    x, s, zp, alpha, xq, gamma, beta = _ln_case(8, rows=256, C=192)
    yk, _, _ = oracle.ptf_layernorm(xq, zp, np.full(192, 3, np.uint8), gamma, beta, 0.03, 128)
    y0, _, _ = oracle.ptf_layernorm(xq, zp, np.zeros(192, np.uint8), gamma, beta, 0.03, 128)
    assert np.abs(yk.astype(int) - y0.astype(int)).max() <= 1
