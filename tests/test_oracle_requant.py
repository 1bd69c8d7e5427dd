"""Pins of the oracle's 8-bit requantization of the attention output.

The multiplier is M = (s_v / s_out) / 2^15, applied as the dyadic N2 / 2^N1
of the LayerNorm output stage (8 significant bits) with the division
rounding half up.  Where M itself has at most 8 significant bits the dyadic
form is exact, so the result must equal the exactly rounded product, computed
here with rational arithmetic; for any M it stays within the truncation bound
of the 8-bit multiplier; and it is monotone in the accumulator.
"""
from fractions import Fraction
import math

import numpy as np
import pytest

import oracle


@pytest.fixture(scope="module", autouse=True)
def _build():
    oracle.build()


def _exact(acc, M: Fraction, zp):
    # floor(acc M + 1/2) + zp, clipped to 8 bits, in exact arithmetic
    out = []
    for a in np.asarray(acc).ravel().tolist():
        v = math.floor(Fraction(a) * M + Fraction(1, 2)) + zp
        out.append(min(255, max(0, v)))
    return np.array(out, np.int64).reshape(np.shape(acc))


def _accs(seed, n=4000, span=2 ** 24):
    rng = np.random.default_rng(seed)
    a = rng.integers(-span, span, size=n)
    a[:8] = [0, 1, -1, 2, -2, span - 1, -span, 12345]
    return a.astype(np.int32)


# s_v / s_out chosen so that the fp32 division is exact and M = k 2^e has at most 8 significant bits
@pytest.mark.parametrize("k,e", [(1, 0), (3, -4), (5, 2), (129, -7), (255, -8), (1, 22), (1, 24), (3, 23),
                                 (1, -15), (7, 10)])
def test_exact_for_multipliers_of_eight_bits(k, e):
    s_out = 2.0 ** -3
    s_v = float(k) * 2.0 ** (e - 3)
    assert np.float32(s_v) == s_v and np.float32(s_v / s_out) == s_v / s_out
    M = Fraction(k) * Fraction(2) ** (e - 15)
    for zp in (0, 128, 255):
        acc = _accs(100 * k + e + zp)
        got = oracle.attn_requant(acc.reshape(-1, 40), s_v, s_out, zp).ravel()
        assert np.array_equal(got.astype(np.int64), _exact(acc, M, zp)), (k, e, zp)


def test_multiplier_keeps_eight_bits():
    # M = 1 + 2^-8 (nine significant bits): N1 = 7, N2 = floor(128.5) = 128, so the multiplier is
    # exactly 1 and y = acc + zp_out for acc in 0 .. 254, where M itself would round acc >= 128 up
    s_out = 2.0 ** -10
    s_v = (1 + 2.0 ** -8) * 32.0
    assert float(np.float32(np.float32(s_v) / np.float32(s_out))) * 2.0 ** -15 == 1 + 2.0 ** -8
    acc = np.arange(0, 255, dtype=np.int32).reshape(-1, 5)
    got = oracle.attn_requant(acc, s_v, s_out, 0)
    assert np.array_equal(got.astype(np.int64), acc.astype(np.int64))


def test_cap_of_the_shift_for_tiny_multipliers():
    # M = 2^-30: N1 = 37 capped at 31, N2 = 2: still the exactly rounded product
    s_out = 1.0
    s_v = 2.0 ** -15
    acc = _accs(7, span=2 ** 31 - 1)
    got = oracle.attn_requant(acc.reshape(-1, 40), s_v, s_out, 3).ravel()
    assert np.array_equal(got.astype(np.int64), _exact(acc, Fraction(1, 2 ** 30), 3))


@pytest.mark.parametrize("s_v,s_out,zp", [(0.05, 0.02, 128), (0.0371, 0.1123, 17), (1.7, 0.013, 240),
                                          (0.3, 7.0, 0)])
def test_within_the_bound_of_an_eight_bit_multiplier(s_v, s_out, zp):
    M = Fraction(float(np.float32(np.float32(s_v) / np.float32(s_out)))) / 2 ** 15
    acc = _accs(int(s_v * 1e4), span=int(min(2 ** 24, 300 / float(M))))
    y = oracle.attn_requant(acc.reshape(-1, 40), s_v, s_out, zp).ravel().astype(np.int64)
    exact = _exact(acc, M, zp)
    # N2 / 2^N1 truncates M by less than 2^-7 relative: |acc M| (unclipped, at most ~255 + |zp|)
    # times 2^-7, plus the rounding
    bound = np.array([float(abs(Fraction(int(a)) * M)) * 2.0 ** -7 + 1.0 for a in acc])
    assert np.all(np.abs(y - exact) <= bound)
    # monotone in the accumulator
    order = np.argsort(acc, kind="stable")
    assert np.all(np.diff(y[order]) >= 0)


def test_zero_point_and_clip():
    acc = np.array([[0, 10 ** 9, -10 ** 9, 0]], np.int32)
    y = oracle.attn_requant(acc, 0.05, 0.02, 77)
    assert y.tolist() == [[77, 255, 0, 77]]
