"""Pins of the oracle's Q K^T logits (MinMax 8-bit output of the MatMul, the
dyadic multiplier of the LayerNorm output stage).

* With M = s_q s_k / (sqrt(d) s_logit) = 1 (d = 64, powers of two) the logit is
  the exact integer product, clipped: numpy's int64 matmul of the
  zero-point-shifted operands (a transposed operand, a wrong zero point or a
  dropped term shows up, the products are not symmetric).
* Where M has at most 8 significant bits (including N1 <= 0 and the N1 = 31
  cap) the result is the exactly rounded product floor(P M + 1/2), computed
  with rational arithmetic; M = 1 + 2^-8 keeps 8 bits (the multiplier is 1).
* For any scales it stays within the truncation bound of an 8-bit multiplier
  of the exact real logit, and it is monotone in P.
* Log-Int-Softmax only sees differences: moving the zero point leaves the
  codes unchanged while nothing clips.
"""
from fractions import Fraction
import math

import numpy as np
import pytest

import oracle


@pytest.fixture(scope="module", autouse=True)
def _build():
    oracle.build()


def _qk(seed, BH, L, d, lo=-128, hi=128):
    rng = np.random.default_rng(seed)
    q = rng.integers(lo, hi, size=(BH, L, d), dtype=np.int16).astype(np.int8)
    k = rng.integers(lo, hi, size=(BH, L, d), dtype=np.int16).astype(np.int8)
    return q, k


def _product(q, k, zp_q, zp_k):
    a = q.astype(np.int64) - zp_q
    b = k.astype(np.int64) - zp_k
    return np.einsum("hid,hjd->hij", a, b)


@pytest.mark.parametrize("zp_q,zp_k", [(0, 0), (-128, 0), (17, -55), (127, 127)])
def test_unit_multiplier_is_the_integer_product(zp_q, zp_k):
    # s_q s_k = 2^-7, sqrt(64) s_logit = 8 2^-10 = 2^-7: M = 1 exactly (N1 = 7, N2 = 128)
    small = zp_q == 0 and zp_k == 0
    q, k = _qk(1000 + zp_q, 3, 21, 64, lo=-2 if small else -8, hi=3 if small else 8)
    got = oracle.qk_logits(q, k, zp_q, zp_k, 2.0 ** -3, 2.0 ** -4, 2.0 ** -10, 0, ld=32)
    P3 = _product(q, k, zp_q, zp_k)
    P = P3.reshape(3 * 21, 21)
    assert np.array_equal(got[:, :21].astype(np.int64), np.clip(P, -128, 127))
    assert np.all(got[:, 21:] == 0)
    if small:
        # the small operands keep P inside int8: nothing clipped, the logits are P itself, and
        # P is not symmetric (a transposed product would differ)
        assert np.abs(P).max() <= 127 and not np.array_equal(P3, P3.transpose(0, 2, 1))


def _exact(P, M: Fraction, zp):
    out = [min(127, max(-128, math.floor(Fraction(int(x)) * M + Fraction(1, 2)) + zp)) for x in P.ravel()]
    return np.array(out, np.int64).reshape(P.shape)


# M = kk 2^e with at most 8 significant bits: s_q = kk 2^(e+1), s_k = 2^-4, s_logit = 2^-6, d = 64
@pytest.mark.parametrize("kk,e", [(1, -8), (3, -12), (255, -20), (129, -14), (5, -3), (1, 3), (7, 2), (1, -30),
                                  (3, -35)])
def test_exact_rounding_for_multipliers_of_eight_bits(kk, e):
    s_q = float(kk) * 2.0 ** (e + 1)
    s_k, s_logit = 2.0 ** -4, 2.0 ** -6
    a = np.float32(s_q) * np.float32(s_k)
    c = np.float32(8.0) * np.float32(s_logit)
    assert np.float32(a / c) == kk * 2.0 ** e
    M = Fraction(kk) * Fraction(2) ** e
    q, k = _qk(kk * 100 + 50 - e, 2, 19, 64)
    for zp_l in (0, -128, 45):
        got = oracle.qk_logits(q, k, 3, -9, s_q, s_k, s_logit, zp_l)
        P = _product(q, k, 3, -9).reshape(-1, 19)
        assert np.array_equal(got.astype(np.int64), _exact(P, M, zp_l)), (kk, e, zp_l)


def test_multiplier_keeps_eight_bits():
    """M = 1 + 2^-8 (nine significant bits): N1 = 7 and N2 = floor(128.5) = 128, so the
    multiplier is exactly 1 and every unclipped logit is P + zp_l; most P here are at least 128,
    where M itself would round P up by one."""
    rng = np.random.default_rng(21)
    q = rng.integers(1, 3, size=(2, 17, 64)).astype(np.int8)
    k = rng.integers(1, 3, size=(2, 17, 64)).astype(np.int8)
    s_q = (1 + 2.0 ** -8) * 2.0 ** -3
    assert np.float32(np.float32(s_q) * np.float32(2.0 ** -4)) / np.float32(2.0 ** -7) == 1 + 2.0 ** -8
    got = oracle.qk_logits(q, k, 0, 0, s_q, 2.0 ** -4, 2.0 ** -10, -100)
    P = _product(q, k, 0, 0).reshape(-1, 17)
    assert P.min() >= 100 and (P >= 128).mean() > 0.5
    assert np.array_equal(got.astype(np.int64), np.clip(P - 100, -128, 127))


@pytest.mark.parametrize("d,s_q,s_k,s_logit", [(64, 0.031, 0.027, 0.0441), (32, 0.5, 0.011, 0.37),
                                               (64, 0.0123, 0.0456, 0.0031), (16, 1.7, 0.9, 13.0)])
def test_within_the_bound_of_an_eight_bit_multiplier(d, s_q, s_k, s_logit):
    q, k = _qk(d, 2, 33, d)
    got = oracle.qk_logits(q, k, 0, 0, s_q, s_k, s_logit, 0).astype(np.int64)
    P = _product(q, k, 0, 0).reshape(-1, 33)
    f32 = np.float32
    M = Fraction(float(f32(f32(s_q) * f32(s_k)) / f32(f32(math.sqrt(d)) * f32(s_logit))))
    exact = _exact(P, M, 0)
    # N2 / 2^N1 truncates M by less than 2^-7 relative (|P M| of an unclipped logit is below ~128)
    bound = np.array([float(abs(Fraction(int(x)) * M)) * 2.0 ** -7 + 1.0 for x in P.ravel()]).reshape(P.shape)
    assert np.all(np.abs(got - exact) <= bound)
    order = np.argsort(P.ravel(), kind="stable")
    assert np.all(np.diff(got.ravel()[order]) >= 0)


def test_softmax_codes_ignore_the_zero_point():
    q, k = _qk(5, 2, 49, 32, lo=-40, hi=40)
    a = oracle.qk_logits(q, k, 0, 0, 0.05, 0.05, 0.06, -20, ld=64)
    b = oracle.qk_logits(q, k, 0, 0, 0.05, 0.05, 0.06, 7, ld=64)
    assert int(a[:, :49].max()) + 27 <= 127 and int(a[:, :49].min()) >= -128  # no clipping either way
    assert np.array_equal(b[:, :49].astype(np.int64), a[:, :49].astype(np.int64) + 27)
    ca, _ = oracle.lis_softmax(a, 49, 0.06)
    cb, _ = oracle.lis_softmax(b, 49, 0.06)
    assert np.array_equal(ca, cb)


def test_rejects_bad_arguments():
    q, k = _qk(0, 1, 4, 8)
    with pytest.raises(ValueError):
        oracle.qk_logits(q, k, 0, 0, 0.0, 1.0, 1.0, 0)
    with pytest.raises(ValueError):
        oracle.qk_logits(q, k, 0, 0, 1.0, 1.0, 1.0, 0, ld=3)
