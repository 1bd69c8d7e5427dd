"""Pins of the oracle's MinMax Linear layer (Sec. 3: uniform MinMax for Linear layers;
Sec. 4.1: symmetric channel-wise weights, asymmetric layer-wise activations; the output
quantizer applied with the dyadic multiplier of the supplement's LayerNorm output stage).

Each pin checks or_linear_q against something other than itself:
- closed forms of the integer product: permutation weights (N != K, so a transposed weight
  matrix or a swapped index fails), all-ones weights, and an input equal to its zero point;
- exact multipliers (M_n = 1, 2^-3, 2^-30 and 3 2^-32 at the N1 cap, 300 and 4096 for
  N1 <= 0, 1 + 2^-8 and 255 2^-10 for the 8-bit truncation of M_n), where the dyadic
  requantization reduces to a rounded shift or a product;
- the one-sided bounds of a truncated multiplier for scales of many significant bits;
- the real-valued layer in fp64, within the 8-bit multiplier's error bound;
- the int32 overflow report and the argument checks.
"""
import numpy as np
import pytest

import oracle


@pytest.fixture(scope="module", autouse=True)
def _built():
    oracle.build()


def _rng(seed):
    return np.random.default_rng(seed)


def test_permutation_weights_closed_form():
    """w[n][perm[n]] = c_n, zero elsewhere: acc[m][n] = (x[m][perm[n]] - zp_x) c_n + b[n]."""
    rng = _rng(1)
    M, K, N = 7, 13, 9
    zp = 77
    x = rng.integers(0, 256, size=(M, K)).astype(np.uint8)
    perm = np.array([5, 0, 12, 3, 7, 1, 10, 2, 8])   # not an involution: perm[1] = 0, perm[0] = 5
    c = np.array([1, -1, 127, -128, 3, -7, 64, 2, -33])
    w = np.zeros((N, K), np.int8)
    for n in range(N):
        w[n, perm[n]] = c[n]
    b = rng.integers(-1000, 1000, size=N).astype(np.int32)
    s_w = np.full(N, 0.01, np.float32)
    _, acc = oracle.linear_q(x, zp, 0.02, w, s_w, b, 0.05, 128)
    for m in range(M):
        for n in range(N):
            assert acc[m, n] == (int(x[m, perm[n]]) - zp) * int(c[n]) + int(b[n]), (m, n)


def test_all_ones_and_zero_point_input():
    rng = _rng(2)
    M, K, N = 5, 300, 4
    zp = 200
    x = rng.integers(0, 256, size=(M, K)).astype(np.uint8)
    w = np.ones((N, K), np.int8)
    s_w = np.full(N, 0.003, np.float32)
    _, acc = oracle.linear_q(x, zp, 0.1, w, s_w, None, 1.0, 0)
    for m in range(M):
        assert np.all(acc[m] == int(x[m].astype(np.int64).sum()) - zp * K)
    # an input equal to its zero point leaves only the bias
    xz = np.full((M, K), zp, np.uint8)
    wr = rng.integers(-128, 128, size=(N, K)).astype(np.int8)
    b = np.array([5, -6, 0, 2 ** 30], np.int32)
    _, acc = oracle.linear_q(xz, zp, 0.1, wr, s_w, b, 1.0, 0)
    assert np.all(acc == b[None, :])


def _one_hot(M, zp, vals):
    """x with x[m][0] - zp = vals[m], the rest at the zero point; w = e_0 (one channel)."""
    x = np.full((M, 3), zp, np.uint8)
    x[:, 0] = np.array(vals) + zp
    w = np.zeros((1, 3), np.int8)
    w[0, 0] = 1
    return x, w


@pytest.mark.parametrize("zp_y", [0, 100, 255])
def test_unit_multiplier_is_identity(zp_y):
    """s_x s_w / s_y = 1 exactly (N1 = 7, N2 = 128): y = clip(acc + zp_y)."""
    vals = list(range(-128, 128))
    x, w = _one_hot(len(vals), 128, vals)
    y, acc = oracle.linear_q(x, 128, 0.5, w, np.array([4.0], np.float32), None, 2.0, zp_y)
    assert np.array_equal(acc[:, 0], vals)
    assert np.array_equal(y[:, 0], np.clip(np.array(vals) + zp_y, 0, 255))


def test_power_of_two_multiplier_rounds_half_up():
    """M = 2^-3 (N1 = 10, N2 = 128): y = floor((acc + 4) / 8) + zp_y, ties toward +inf."""
    vals = list(range(-128, 128))
    x, w = _one_hot(len(vals), 128, vals)
    y, _ = oracle.linear_q(x, 128, 0.25, w, np.array([0.5], np.float32), None, 1.0, 50)
    want = [min(255, max(0, (v + 4) // 8 + 50)) for v in vals]
    assert y[:, 0].tolist() == want
    # the ties: acc = 4 -> 1, acc = -4 -> 0, acc = -12 -> -1
    assert y[vals.index(4), 0] == 51 and y[vals.index(-4), 0] == 50 and y[vals.index(-12), 0] == 49


def test_multiplier_shift_cap():
    """M = 2^-30: N1 = 37 is capped at 31, N2 = floor(2^-30 2^31) = 2: y = floor((2 acc + 2^30) / 2^31)."""
    M, K = 2, 20000
    x = np.full((M, K), 255, np.uint8)
    w = np.full((1, K), 127, np.int8)
    b = np.array([2 ** 30 - 255 * 127 * K], np.int32)
    y, acc = oracle.linear_q(x, 0, 2.0 ** -15, w, np.array([2.0 ** -15], np.float32), b, 1.0, 10)
    a = int(acc[0, 0])
    assert a == 2 ** 30
    assert int(y[0, 0]) == (2 * a + 2 ** 30) // 2 ** 31 + 10 == 11


@pytest.mark.parametrize("Mval,factor", [(300.0, 300), (4096.0, 4096)])
def test_large_multiplier_branch(Mval, factor):
    """M >= 256 takes N1 <= 0: 300 = 150 * 2^1 (N1 = -1), 4096 = 128 * 2^5 (N1 = -5): y = clip(M acc + zp)."""
    vals = [-1, 0, 1]
    x, w = _one_hot(3, 128, vals)
    s_w = np.array([Mval], np.float32)
    y, _ = oracle.linear_q(x, 128, 1.0, w, s_w, None, 1.0, 7)
    assert y[:, 0].tolist() == [max(0, min(255, factor * v + 7)) for v in vals]
    # acc = 0 except through the bias: 300 * 0 + 7
    y, _ = oracle.linear_q(np.full((1, 3), 128, np.uint8), 128, 1.0, w, s_w, np.array([0], np.int32), 1.0, 7)
    assert int(y[0, 0]) == 7


def test_agrees_with_real_valued_layer():
    """The integer layer against the fp64 product of the dequantized operands, quantized with
    s_y and zp_y: the dyadic multiplier N2 / 2^N1 is within a relative 2^-7 of M_n (N2 >= 128),
    so the codes differ by at most 1 + |acc M_n| 2^-7 + the half step of each rounding."""
    rng = _rng(3)
    M, K, N = 64, 384, 96
    xf = rng.normal(0.3, 1.0, size=(M, K))
    s_x = np.float32((xf.max() - xf.min()) / 255.0)
    zp_x = int(np.clip(np.rint(-xf.min() / s_x), 0, 255))
    x = np.clip(np.rint(xf / s_x) + zp_x, 0, 255).astype(np.uint8)
    wf = rng.normal(0.0, 0.05, size=(N, K)) * rng.uniform(0.2, 3.0, size=(N, 1))
    s_w = (np.abs(wf).max(axis=1) / 127.0).astype(np.float32)
    w = np.clip(np.rint(wf / s_w[:, None]), -127, 127).astype(np.int8)
    bf = rng.normal(0.0, 0.2, size=N)
    b = np.rint(bf / (float(s_x) * s_w.astype(np.float64))).astype(np.int32)
    real = ((x.astype(np.float64) - zp_x) * float(s_x)) @ (w.astype(np.float64) * s_w[:, None]).T \
        + b * (float(s_x) * s_w.astype(np.float64))
    s_y = np.float32((real.max() - real.min()) / 255.0)
    zp_y = int(np.clip(np.rint(-real.min() / s_y), 0, 255))
    y, acc = oracle.linear_q(x, zp_x, float(s_x), w, s_w, b, float(s_y), zp_y)
    ref = np.rint(real / float(s_y)) + zp_y
    inside = (ref >= 0) & (ref <= 255)
    Mn = (float(s_x) * s_w.astype(np.float64)) / float(s_y)
    bound = 1.0 + np.abs(acc * Mn[None, :]) / 128.0
    diff = np.abs(y.astype(np.float64) - ref)
    assert np.all(diff[inside] <= bound[inside])
    assert diff[inside].mean() < 0.6
    assert np.all(y[ref < 0] == 0) and np.all(y[ref > 255] == 255)
    # the integer product itself is the real product divided by s_x s_w[n], exactly
    assert np.allclose(acc * (float(s_x) * s_w.astype(np.float64))[None, :], real, rtol=1e-12, atol=1e-12)


def test_overflow_and_argument_checks():
    K = 70000  # K * 255 * 127 > 2^31
    x = np.full((1, K), 255, np.uint8)
    w = np.full((1, K), 127, np.int8)
    with pytest.raises(OverflowError):
        oracle.linear_q(x, 0, 1.0, w, np.array([1.0], np.float32), None, 1.0, 0)
    x = np.zeros((2, 4), np.uint8)
    w = np.zeros((3, 4), np.int8)
    for s_w in ([1.0, 0.0, 1.0], [1.0, -1.0, 1.0], [1.0, np.nan, 1.0], [1.0, np.inf, 1.0]):
        with pytest.raises(ValueError):
            oracle.linear_q(x, 0, 1.0, w, np.array(s_w, np.float32), None, 1.0, 0)
    with pytest.raises(ValueError):
        oracle.linear_q(x, 0, 0.0, w, np.ones(3, np.float32), None, 1.0, 0)
    with pytest.raises(ValueError):  # M_n >= 1e30
        oracle.linear_q(x, 0, 1e20, w, np.full(3, 1e20, np.float32), None, 1.0, 0)


def test_eight_bit_truncation_of_the_multiplier():
    """The reading keeps 8 significant bits of M_n.  M = 1 + 2^-8: N1 = 7, N2 = floor(128.5) = 128,
    so the multiplier is exactly 1 and y = acc for acc in 0 .. 254 (where M itself would round
    acc >= 128 up by one).  M = 255 2^-10 (8 bits): N1 = 10, N2 = 255,
    y = floor(255 acc / 1024 + 1/2) + zp_y."""
    vals = list(range(0, 128))
    x, w = _one_hot(len(vals), 128, vals)
    w[0, 0] = 2  # acc = 2 v, 0 .. 254
    y, _ = oracle.linear_q(x, 128, 1.0, w, np.array([1.0 + 2.0 ** -8], np.float32), None, 1.0, 0)
    assert y[:, 0].tolist() == [2 * v for v in vals]
    vals = list(range(-128, 128))
    x, w = _one_hot(len(vals), 128, vals)
    w[0, 0] = 127  # acc = 127 v, up to 16129 in magnitude
    acc_v = [127 * v for v in vals]
    y, _ = oracle.linear_q(x, 128, 1.0, w, np.array([255 * 2.0 ** -10], np.float32), None, 1.0, 128)
    assert y[:, 0].tolist() == [min(255, max(0, (255 * a + 512) // 1024 + 128)) for a in acc_v]


def test_shift_cap_truncates_the_multiplier():
    """M = 3 2^-32: N1 = 38 is capped at 31, N2 = floor(1.5) = 1: y = floor((acc + 2^30) / 2^31) + zp_y."""
    x = np.full((1, 3), 9, np.uint8)  # x = zp_x: acc is the bias alone
    w = np.ones((1, 3), np.int8)
    for b, want in ((3 * 2 ** 29, 1), (2 ** 30 - 1, 0), (-(2 ** 30), 0), (-(2 ** 30) - 1, -1)):
        y, acc = oracle.linear_q(x, 9, 2.0 ** -15, w, np.array([3 * 2.0 ** -17], np.float32),
                                 np.array([b], np.int32), 1.0, 20)
        assert int(acc[0, 0]) == b and int(y[0, 0]) == 20 + want, b


def test_multiplier_truncates():
    """N2 / 2^N1 lies in (M (1 - 2^-7), M]: for acc >= 0 and scales of many significant bits,
    floor(M acc (1 - 2^-7) + 1/2) <= y - zp_y <= floor(M acc + 1/2), with M the fp32 value of
    (s_x s_w[n]) / s_y in exact rational arithmetic."""
    from fractions import Fraction
    import math
    rng = _rng(7)
    M_, K, N = 40, 16, 24
    x = rng.integers(100, 256, size=(M_, K)).astype(np.uint8)      # x - zp_x >= 0
    w = rng.integers(0, 128, size=(N, K)).astype(np.int8)           # w >= 0
    s_x, s_y = np.float32(0.0173), np.float32(0.91)
    s_w = (rng.uniform(0.5, 2.0, size=N) * 2.9e-3).astype(np.float32)
    y, acc = oracle.linear_q(x, 100, float(s_x), w, s_w, None, float(s_y), 0)
    assert acc.min() >= 0
    for n in range(N):
        Mn = Fraction(float(np.float32(np.float32(s_x * s_w[n]) / s_y)))
        for m in range(M_):
            a = int(acc[m, n])
            hi = math.floor(Mn * a + Fraction(1, 2))
            lo = math.floor(Mn * a * (1 - Fraction(1, 128)) + Fraction(1, 2))
            assert hi <= 255 and lo <= int(y[m, n]) <= hi, (m, n)
