"""Fused Log-Int-Softmax + BitShift attention times values for short rows
(at most 64 keys, two heads per tensor-core tile): windowed attention with
and without the relative-position bias, against the oracle bit for bit, and
against the CUDA-core path on the same inputs.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2111_13824_gb300 import build as fbuild
from paper_2111_13824_gb300 import fqvit, synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"

# scales: the smallest and largest supported, two whose floored i-exp constants make
# e(d) rise once per period (Algorithm 1), and the scales of the synthetic window stages
SCALES = (0.0078125, float(np.float32(0.008350185749701165)), float(np.float32(0.01732846078509329)),
          0.0347, 0.17, 0.5)


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    fbuild.build()
    fqvit.load()
    oracle.build()


def _logits(rng, rows, L, ld, spread):
    x = np.zeros((rows, ld), np.int8)
    centre = rng.uniform(-60, 60, size=(rows, 1))
    x[:, :L] = np.clip(np.rint(rng.normal(centre, spread, size=(rows, L))), -128, 127)
    return x


def _oracle(x, L, s, v, zp, bias=None, heads=1, window=0):
    co, _ = oracle.lis_softmax(x, L, s, bias=bias, heads=heads, window=window or 7)
    ao, ov = oracle.lis_attn_v(co, v, zp)
    assert not ov
    return ao


def _gpu(x, s, v, zp, bias=None, heads=1, window=0):
    b = torch.from_numpy(bias).to(DEV) if bias is not None else None
    acc = fqvit.lis_attention(torch.from_numpy(x).to(DEV), s, torch.from_numpy(v).to(DEV), zp, bias=b,
                              heads=heads, window=window)
    fqvit.sync_status()
    return acc.cpu().numpy()


def _cuda_core(monkeypatch, *args, **kw):
    monkeypatch.setenv("FQVIT_ATTN_PATH", "cuda_core")
    try:
        return _gpu(*args, **kw)
    finally:
        monkeypatch.delenv("FQVIT_ATTN_PATH")


@pytest.mark.parametrize("L", [1, 2, 3, 4, 9, 16, 17, 33, 36, 48, 49, 63, 64])
@pytest.mark.parametrize("d", [32, 64])
def test_short_rows_match_oracle(L, d, monkeypatch):
    rng = np.random.default_rng(100 * L + d)
    for BH, s, spread in ((1, 0.0347, 20.0), (5, 0.17, 60.0), (6, 0.0078125, 90.0)):
        ld = (L + 15) // 16 * 16
        x = _logits(rng, BH * L, L, ld, spread)
        v = rng.integers(-128, 128, size=(BH, L, d), dtype=np.int8)
        ao = _oracle(x, L, s, v, 0)
        assert np.array_equal(_gpu(x, s, v, 0), ao), (L, d, BH, s)
        assert np.array_equal(_cuda_core(monkeypatch, x, s, v, 0), ao)


@pytest.mark.parametrize("window", [1, 2, 3, 4, 6, 7, 8])
@pytest.mark.parametrize("brange", [16, 128])
def test_relpos_bias_match_oracle(window, brange, monkeypatch):
    """Bias from the synthetic range [-16, 16] and the full int8 range (distances to the row
    maximum up to 510: the whole i-exp table, or its clamp at 15 |q_ln2|)."""
    L = window * window
    rng = np.random.default_rng(7 * window + brange)
    heads = 3 if window % 2 else 5
    BH = heads * 3
    nb = (2 * window - 1) ** 2
    ld = (L + 15) // 16 * 16
    for s in SCALES:
        bias = rng.integers(-brange, min(brange, 127) + 1, size=(heads, nb), dtype=np.int8)
        x = _logits(rng, BH * L, L, ld, 40.0)
        v = rng.integers(-128, 128, size=(BH, L, 32), dtype=np.int8)
        ao = _oracle(x, L, s, v, 0, bias=bias, heads=heads, window=window)
        got = _gpu(x, s, v, 0, bias=bias, heads=heads, window=window)
        assert np.array_equal(got, ao), (window, brange, s)
        assert np.array_equal(_cuda_core(monkeypatch, x, s, v, 0, bias=bias, heads=heads, window=window), ao)
    # d = 64 with the bias (zero point 0)
    v = rng.integers(-128, 128, size=(BH, L, 64), dtype=np.int8)
    ao = _oracle(x, L, 0.0347, v, 0, bias=bias, heads=heads, window=window)
    assert np.array_equal(_gpu(x, 0.0347, v, 0, bias=bias, heads=heads, window=window), ao)


@pytest.mark.parametrize("zp", [-255, -77, 1, 128, 255])
def test_v_zero_point(zp):
    """acc = P V - zp_V (P 1), the row sums of P taken from a column of ones of B (d = 32)."""
    rng = np.random.default_rng(500 + zp)
    heads, window = 3, 7
    L, BH = 49, 9
    bias = rng.integers(-16, 17, size=(heads, 169), dtype=np.int8)
    x = _logits(rng, BH * L, L, 64, 30.0)
    v = rng.integers(-128, 128, size=(BH, L, 32), dtype=np.int8)
    for s in (0.0347, 0.5, 0.0078125):
        for b in (None, bias):
            ao = _oracle(x, L, s, v, zp, bias=b, heads=heads, window=window)
            got = _gpu(x, s, v, zp, bias=b, heads=heads, window=window if b is not None else 0)
            assert np.array_equal(got, ao), (zp, s, b is None)


@pytest.mark.parametrize("d", [32, 64])
def test_accumulator_bound_rows(d):
    """Rows whose sum_j 2^(15-code_j) |V| comes closest to the exactness bound: k equal top logits
    and the rest far below, V = -128 or +127 everywhere; one-hot and uniform rows."""
    L, ld = 49, 64
    rows = []
    for k in (1, 2, 3, 5, 11, 23, 47, 49):
        r = np.full(ld, -128, np.int8)
        r[:k] = 127
        rows.append(r)
    rows.append(np.full(ld, 3, np.int8))
    BH = 2
    x = np.full((BH * L, ld), -128, np.int8)
    for i, r in enumerate(rows):
        x[i] = r
        x[L + i] = r
    zero_bias = np.zeros((1, 169), np.int8)
    for s, vv in ((0.5, -128), (0.5, 127), (0.1, -128), (0.0078125, -128)):
        v = np.full((BH, L, d), vv, np.int8)
        for b in (None, zero_bias):
            ao = _oracle(x, L, s, v, 0, bias=b, heads=1, window=7)
            got = _gpu(x, s, v, 0, bias=b, heads=1, window=7 if b is not None else 0)
            assert np.array_equal(got, ao), (s, vv, b is None)
            assert np.abs(ao).max() < 2 ** 24


def test_row_padding_and_strides_are_ignored():
    """Bytes of a logit row past L and V columns past d are not read as data."""
    rng = np.random.default_rng(3)
    L, BH = 49, 7
    x = _logits(rng, BH * L, L, 96, 30.0)
    xg = x.copy()
    xg[:, L:] = rng.integers(-128, 128, size=(BH * L, 96 - L), dtype=np.int8)
    vbig = rng.integers(-128, 128, size=(BH, L, 64), dtype=np.int8)
    v = np.ascontiguousarray(vbig[:, :, :32])
    ao = _oracle(x, L, 0.0347, v, 0)
    assert np.array_equal(_gpu(xg, 0.0347, v, 0), ao)
    # V as a strided view (row stride 64 bytes, 32 used)
    vd = torch.from_numpy(vbig).to(DEV)[:, :, :32]
    acc = fqvit.lis_attention(torch.from_numpy(xg).to(DEV), 0.0347, vd, 0)
    fqvit.sync_status()
    assert np.array_equal(acc.cpu().numpy(), ao)


def test_many_tiles_per_group(monkeypatch):
    """More heads than one pass of the CTAs' groups, an odd head count (the last tile holds
    one head): the whole output against the CUDA-core path, sampled heads against the oracle."""
    rng = np.random.default_rng(9)
    heads, window, L = 3, 7, 49
    BH = 4011  # odd, a multiple of the heads
    bias = rng.integers(-16, 17, size=(heads, 169), dtype=np.int8)
    x = _logits(rng, BH * L, L, 64, 25.0)
    v = rng.integers(-128, 128, size=(BH, L, 32), dtype=np.int8)
    s = 0.0347
    got = _gpu(x, s, v, 0, bias=bias, heads=heads, window=window)
    assert np.array_equal(got, _cuda_core(monkeypatch, x, s, v, 0, bias=bias, heads=heads, window=window))
    for bh in sorted(set(rng.integers(0, BH, size=40).tolist()) | {0, BH - 1}):
        # one head alone: the head index of its bias table is bh % heads
        hb = bias[[bh % heads]]
        ao = _oracle(x[bh * L:(bh + 1) * L], L, s, v[bh:bh + 1], 0, bias=hb, heads=1, window=window)
        assert np.array_equal(got[bh], ao[0]), bh


def test_window_stage_at_full_size_sampled(monkeypatch):
    """The first window stage of the synthetic Swin-S workload at full size (4096 windows x
    3 heads per batch of 64), as the benchmark runs it: sampled heads against the oracle and
    the whole output against the CUDA-core path."""
    cfg = synth.CONFIGS["swin_s"]
    a = synth.attn_inputs(cfg, 0)
    L, heads = a["L"], a["heads"]
    x, v, bias = a["logits"].numpy(), a["v"].numpy(), a["bias"].numpy()
    got = _gpu(x, a["s_logit"], v, 0, bias=bias, heads=heads, window=a["window"])
    ref = _cuda_core(monkeypatch, x, a["s_logit"], v, 0, bias=bias, heads=heads, window=a["window"])
    assert np.array_equal(got, ref)
    rng = np.random.default_rng(0)
    for bh in rng.integers(0, a["BH"], size=24).tolist():
        hb = bias[[bh % heads]]
        ao = _oracle(x[bh * L:(bh + 1) * L], L, a["s_logit"], v[bh:bh + 1], 0, bias=hb, heads=1,
                     window=a["window"])
        assert np.array_equal(got[bh], ao[0]), bh
