"""Pins of the oracle's shifted-window mask (Swin attention, not in the paper).

Key j of query i gets mask_value added to its logit when their region ids in
the row's window differ; rows are ordered [batch][window][head][query].  The
pins rest on the unmasked oracle (pinned elsewhere) and on Algorithm 1's
clamp: a zero mask or a single region changes nothing, a small mask is the
same as lowering the masked logits, and a mask far below the clamp leaves a
query alone with its own key (code 0) and every other key at code 15.
"""
import numpy as np
import pytest

import oracle


@pytest.fixture(scope="module", autouse=True)
def _build():
    oracle.build()


def _rows(seed, n_rows, L, ld, lo=-60, hi=60):
    rng = np.random.default_rng(seed)
    x = np.zeros((n_rows, ld), np.int8)
    x[:, :L] = rng.integers(lo, hi, size=(n_rows, L), dtype=np.int8)
    return x


@pytest.mark.parametrize("s", [0.0078125, 0.0347, 0.17, 0.5])
def test_zero_mask_or_one_region_changes_nothing(s):
    L, heads, nw = 49, 3, 4
    rng = np.random.default_rng(1)
    x = _rows(2, 2 * nw * heads * L, L, 64)
    bias = rng.integers(-16, 17, size=(heads, 169), dtype=np.int8)
    region = rng.integers(0, 9, size=(nw, L), dtype=np.uint8)
    c0, S0 = oracle.lis_softmax(x, L, s, bias=bias, heads=heads, window=7)
    c1, S1 = oracle.lis_softmax(x, L, s, bias=bias, heads=heads, window=7, region=region, mask_value=0)
    assert np.array_equal(c0, c1) and np.array_equal(S0, S1)
    one = np.full((nw, L), 5, np.uint8)
    c2, S2 = oracle.lis_softmax(x, L, s, bias=bias, heads=heads, window=7, region=one, mask_value=-3000)
    assert np.array_equal(c0, c2) and np.array_equal(S0, S2)


@pytest.mark.parametrize("mask_value", [-1, -5, -37])
def test_small_mask_is_a_lowered_logit(mask_value):
    """Adding the mask is adding to the integer logit: the same row with the masked keys'
    logits lowered (kept inside int8 here) gives the same codes and row sum."""
    L = 16
    x = _rows(3, 40, L, 16, lo=-80, hi=80)
    region = np.zeros((1, L), np.uint8)
    region[0, L // 2:] = 1
    c1, S1 = oracle.lis_softmax(x, L, 0.05, region=region, mask_value=mask_value)
    y = x.copy()
    for r in range(40):
        i = r % L
        for j in range(L):
            if region[0, i] != region[0, j]:
                y[r, j] = np.int8(int(x[r, j]) + mask_value)
    c2, S2 = oracle.lis_softmax(y, L, 0.05)
    assert np.array_equal(c1, c2) and np.array_equal(S1, S2)


@pytest.mark.parametrize("s", [0.0078125, 0.0347, 0.5])
def test_mask_far_below_the_clamp(s):
    """Every token in its own region, mask far below n q_ln2: the query's own key is the row
    maximum (e(0)), every other key sits at the clamp (e(n q_ln2)); when (L-1) e_clamp < e(0)/2
    the query's code is 0 and every other code is 15."""
    L = 49
    x = _rows(4, 3 * L, L, 64)
    region = np.arange(L, dtype=np.uint8)[None, :]
    codes, S = oracle.lis_softmax(x, L, s, region=region, mask_value=-100000)
    e0 = oracle.iexp(0, s)
    q_ln2 = oracle.iexp_consts(s)[0]
    ec = oracle.iexp(15 * q_ln2, s)
    assert np.all(S == e0 + (L - 1) * ec)
    assert (L - 1) * ec * 2 < e0
    for r in range(3 * L):
        i = r % L
        assert codes[r, i] == 0
        assert np.all(np.delete(codes[r], i) == 15)


def test_rows_take_their_window_region_row():
    """Rows are [batch][window][head][query]: window 0 has one region (no masking), window 1
    one region per token; with two heads the window index is (row / (L heads)) % n_windows."""
    L, heads, nw = 9, 2, 2
    x = _rows(5, 2 * nw * heads * L, L, 16)
    region = np.stack([np.zeros(L, np.uint8), np.arange(L, dtype=np.uint8)])
    codes, _ = oracle.lis_softmax(x, L, 0.1, heads=heads, region=region, mask_value=-100000)
    plain, _ = oracle.lis_softmax(x, L, 0.1)
    for r in range(x.shape[0]):
        w = (r // (L * heads)) % nw
        if w == 0:
            assert np.array_equal(codes[r], plain[r])
        else:
            i = r % L
            assert codes[r, i] == 0 and np.all(np.delete(codes[r], i) == 15)
