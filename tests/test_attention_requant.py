"""Fused attention with its output requantized to 8 bits (fqvit_lis_attention_q)
against the oracle: the oracle's accumulators, then its requantization, bit
for bit, on every kernel path (rows of up to 640 keys on the tensor cores,
short rows with the relative-position bias on the tensor cores, CUDA cores).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2111_13824_gb300 import build as fbuild
from paper_2111_13824_gb300 import fqvit, synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"

# (s_v, s_out, zp_out): a typical pair, a multiplier of 8 bits, N1 <= 0 (M = 512), the shift cap
# (M = 2^-30), a small output scale that saturates often
REQ = [(0.05, 0.02, 128), (3 * 2 ** -10, 2 ** -3, 7), (2.0 ** 21, 2 ** -3, 100), (2.0 ** -18, 2 ** -3, 250),
       (0.9, 0.0007, 60)]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    fbuild.build()
    fqvit.load()
    oracle.build()


def _want(x, L, s, v, zp_v, s_v, s_out, zp_out, bias=None, heads=1, window=7):
    co, _ = oracle.lis_softmax(x, L, s, bias=bias, heads=heads, window=window)
    ao, ov = oracle.lis_attn_v(co, v, zp_v)
    assert not ov
    return oracle.attn_requant(ao, s_v, s_out, zp_out)


def _got(x, s, v, zp_v, s_v, s_out, zp_out, bias=None, heads=1, window=0):
    b = torch.from_numpy(bias).to(DEV) if bias is not None else None
    out = fqvit.lis_attention_q(torch.from_numpy(x).to(DEV), s, torch.from_numpy(v).to(DEV), zp_v, s_v, s_out,
                                zp_out, bias=b, heads=heads, window=window)
    fqvit.sync_status()
    return out.cpu().numpy()


@pytest.fixture(params=["auto", "cuda_core"])
def path(request, monkeypatch):
    if request.param == "cuda_core":
        monkeypatch.setenv("FQVIT_ATTN_PATH", "cuda_core")
    return request.param


@pytest.mark.parametrize("name,bh,sigma", [("deit_s", 5, 1.0), ("vit_l384", 3, 2.0), ("vit_b", 4, 1.0)])
def test_long_rows(name, bh, sigma, path):
    a = synth.attn_inputs(synth.CONFIGS[name], 0, bh=bh, sigma=sigma)
    x, v, L, s = a["logits"].numpy(), a["v"].numpy(), a["L"], a["s_logit"]
    for s_v, s_out, zp_out in REQ:
        want = _want(x, L, s, v, 0, s_v, s_out, zp_out)
        assert np.array_equal(_got(x, s, v, 0, s_v, s_out, zp_out), want), (name, s_v, s_out, zp_out)


def test_windows_with_bias(path):
    a = synth.attn_inputs(synth.CONFIGS["swin_s"], 0, bh=3 * 7)
    x, v, s = a["logits"].numpy(), a["v"].numpy(), a["s_logit"]
    bias = a["bias"].numpy()
    for s_v, s_out, zp_out in REQ:
        want = _want(x, 49, s, v, 0, s_v, s_out, zp_out, bias=bias, heads=3, window=7)
        got = _got(x, s, v, 0, s_v, s_out, zp_out, bias=bias, heads=3, window=7)
        assert np.array_equal(got, want), (s_v, s_out, zp_out)


@pytest.mark.parametrize("L,d", [(49, 64), (17, 32), (64, 64)])
def test_short_rows_without_bias(L, d, path):
    rng = np.random.default_rng(L + d)
    BH, ld = 5, (L + 15) // 16 * 16
    x = np.zeros((BH * L, ld), np.int8)
    x[:, :L] = rng.integers(-128, 128, size=(BH * L, L), dtype=np.int8)
    v = rng.integers(-128, 128, size=(BH, L, d), dtype=np.int8)
    for s_v, s_out, zp_out in REQ[:3]:
        want = _want(x, L, 0.06, v, 0, s_v, s_out, zp_out)
        assert np.array_equal(_got(x, 0.06, v, 0, s_v, s_out, zp_out), want), (L, d, s_v)


@pytest.mark.parametrize("zp_v", [-77, 128])
def test_with_v_zero_point(zp_v, path):
    """Asymmetric V (acc = P (V - zp_V)) then the requantization, on the long-row and short-row kernels."""
    rng = np.random.default_rng(900 + zp_v)
    for L, d in ((197, 64), (49, 32)):
        BH, ld = 4, (L + 15) // 16 * 16
        x = np.zeros((BH * L, ld), np.int8)
        x[:, :L] = rng.integers(-128, 128, size=(BH * L, L), dtype=np.int8)
        v = rng.integers(-128, 128, size=(BH, L, d), dtype=np.int8)
        for s_v, s_out, zp_out in REQ[:2]:
            want = _want(x, L, 0.06, v, zp_v, s_v, s_out, zp_out)
            assert np.array_equal(_got(x, 0.06, v, zp_v, s_v, s_out, zp_out), want), (L, zp_v, s_v)
