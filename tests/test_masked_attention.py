"""Shifted-window (Swin) attention mask on the GPU against the oracle, bit for bit:
Log-Int-Softmax codes and row sums (fqvit_lis_softmax_masked) and the fused
attention (fqvit_lis_attention_masked) on the short-row tensor-core kernel and
on the CUDA-core path; mask values from 0 to -32768, the shifted-window region
pattern of each Swin-S stage, random region ids, and scales on both sides of
the short-row kernel's limit (15 |q_ln2| <= 510, past which the CUDA-core path
takes over).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2111_13824_gb300 import build as fbuild
from paper_2111_13824_gb300 import fqvit, synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
MASKS = (0, -1, -5, -37, -300, -510, -511, -1023, -1024, -1025, -2857, -32768)


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    fbuild.build()
    fqvit.load()
    oracle.build()


@pytest.fixture(params=["auto", "cuda_core"])
def path(request, monkeypatch):
    if request.param == "cuda_core":
        monkeypatch.setenv("FQVIT_ATTN_PATH", "cuda_core")
    return request.param


def _unpack(packed, L):
    out = np.stack([packed & 0x0F, packed >> 4], axis=-1).reshape(packed.shape[0], -1)
    return out[:, :L]


def _logits(rng, rows, L, ld, spread=40.0):
    x = np.zeros((rows, ld), np.int8)
    centre = rng.uniform(-60, 60, size=(rows, 1))
    x[:, :L] = np.clip(np.rint(rng.normal(centre, spread, size=(rows, L))), -128, 127)
    return x


def _oracle(x, L, s, v, zp, region, mask_value, bias=None, heads=1, window=7):
    co, S = oracle.lis_softmax(x, L, s, bias=bias, heads=heads, window=window, region=region,
                               mask_value=mask_value)
    ao, ov = oracle.lis_attn_v(co, v, zp)
    assert not ov
    return co, S, ao


def _gpu(x, s, v, zp, region, mask_value, bias=None, heads=1, window=0):
    L = v.shape[1]
    b = torch.from_numpy(bias).to(DEV) if bias is not None else None
    r = torch.from_numpy(region).to(DEV) if region is not None else None
    codes = torch.empty(x.shape[0], (L + 1) // 2, dtype=torch.uint8, device=DEV)
    acc = fqvit.lis_attention_masked(torch.from_numpy(x).to(DEV), s, torch.from_numpy(v).to(DEV), r, mask_value,
                                     zp, codes=codes, bias=b, heads=heads, window=window)
    fqvit.sync_status()
    return _unpack(codes.cpu().numpy(), L), acc.cpu().numpy()


@pytest.mark.parametrize("layer,side", [(1, 56), (3, 28), (5, 14)])
def test_swin_shifted_stages(layer, side, path):
    """The odd (shifted) block of each Swin-S stage whose side exceeds the window: synthetic
    logits, bias and V of that layer, the stage's region ids, the mask of -100 in logit units."""
    cfg = synth.CONFIGS["swin_s"]
    st = synth.layer_stage(cfg, layer)
    region = synth.shifted_window_regions(side, 7).numpy()
    nw = region.shape[0]
    assert nw == (side // 7) ** 2 and region.max() == 8
    bh = nw * st.H * (2 if nw < 16 else 1)
    a = synth.attn_inputs(cfg, layer, bh=bh)
    x, v, s = a["logits"].numpy(), a["v"].numpy(), a["s_logit"]
    bias = a["bias"].numpy()
    mv = synth.swin_mask_value(s)
    co, _, ao = _oracle(x, 49, s, v, 0, region, mv, bias=bias, heads=st.H)
    gc, ga = _gpu(x, s, v, 0, region, mv, bias=bias, heads=st.H, window=7)
    assert np.array_equal(gc, co) and np.array_equal(ga, ao), (layer, mv)
    # the mask matters: the unmasked codes differ
    plain, _ = oracle.lis_softmax(x, 49, s, bias=bias, heads=st.H, window=7)
    assert not np.array_equal(plain, co)


@pytest.mark.parametrize("s", [0.0078125, 0.0347, 0.17, 0.5])
def test_mask_values(s, path):
    """Every mask value from 0 to -32768 with random region ids: the short-row kernel clamps the
    mask at -1024 (exact while 15 |q_ln2| <= 510); at s = 2^-7 (15 |q_ln2| = 1320) the CUDA-core
    path runs."""
    rng = np.random.default_rng(int(s * 1e4))
    heads, nw, L, d = 3, 3, 49, 32
    bias = rng.integers(-16, 17, size=(heads, 169), dtype=np.int8)
    region = rng.integers(0, 9, size=(nw, L), dtype=np.uint8)
    region[1] = np.arange(L, dtype=np.uint8)  # every token alone: only the self key is unmasked
    region[2] = 4                             # one region: nothing masked
    BH = 2 * nw * heads
    x = _logits(rng, BH * L, L, 64)
    v = rng.integers(-128, 128, size=(BH, L, d), dtype=np.int8)
    for mv in MASKS:
        co, _, ao = _oracle(x, L, s, v, 0, region, mv, bias=bias, heads=heads)
        gc, ga = _gpu(x, s, v, 0, region, mv, bias=bias, heads=heads, window=7)
        assert np.array_equal(gc, co) and np.array_equal(ga, ao), (s, mv)


@pytest.mark.parametrize("window,d", [(4, 64), (7, 64), (8, 32), (3, 32)])
def test_full_range_bias_and_zero_point(window, d, path):
    """Bias over the whole int8 range (distances to the maximum up to 510 before the mask), a V zero
    point, head dimension 64; window sides other than 7."""
    rng = np.random.default_rng(7 * window + d)
    L, heads, nw = window * window, 2, 4
    bias = rng.integers(-128, 128, size=(heads, (2 * window - 1) ** 2), dtype=np.int8)
    region = rng.integers(0, 4, size=(nw, L), dtype=np.uint8)
    BH = nw * heads
    ld = (L + 15) // 16 * 16
    x = _logits(rng, BH * L, L, ld, spread=80.0)
    v = rng.integers(-128, 128, size=(BH, L, d), dtype=np.int8)
    for s, mv, zp in ((0.0347, -2857, 0), (0.17, -300, -19), (0.5, -1025, 77)):
        co, _, ao = _oracle(x, L, s, v, zp, region, mv, bias=bias, heads=heads, window=window)
        gc, ga = _gpu(x, s, v, zp, region, mv, bias=bias, heads=heads, window=window)
        assert np.array_equal(gc, co) and np.array_equal(ga, ao), (window, s, mv, zp)


@pytest.mark.parametrize("L", [49, 64, 197])
def test_mask_without_bias(L, path):
    """A mask without a bias (one head per window row group): the CUDA-core path."""
    rng = np.random.default_rng(L)
    nw, d = 2, 64
    region = rng.integers(0, 3, size=(nw, L), dtype=np.uint8)
    BH = 2 * nw
    ld = (L + 15) // 16 * 16
    x = _logits(rng, BH * L, L, ld)
    v = rng.integers(-128, 128, size=(BH, L, d), dtype=np.int8)
    for mv in (-7, -2000):
        co, _, ao = _oracle(x, L, 0.05, v, 0, region, mv)
        gc, ga = _gpu(x, 0.05, v, 0, region, mv)
        assert np.array_equal(gc, co) and np.array_equal(ga, ao), (L, mv)


def test_softmax_masked_codes_and_row_sums():
    """fqvit_lis_softmax_masked: packed codes and the i-exp row sums of Algorithm 2, rows in
    [batch][window][head][query] order with a ragged batch count."""
    rng = np.random.default_rng(5)
    heads, nw, L = 3, 4, 49
    bias = rng.integers(-16, 17, size=(heads, 169), dtype=np.int8)
    region = synth.shifted_window_regions(14, 7).numpy()
    assert region.shape == (nw, L)
    rows = 3 * nw * heads * L
    x = _logits(rng, rows, L, 64)
    for s, mv in ((0.0347, -2882), (0.0078125, -12800), (0.3, -3)):
        co, So = oracle.lis_softmax(x, L, s, bias=bias, heads=heads, window=7, region=region, mask_value=mv)
        rs = torch.empty(rows, dtype=torch.int64, device=DEV)
        codes = fqvit.lis_softmax_masked(torch.from_numpy(x).to(DEV), L, s, torch.from_numpy(region).to(DEV), mv,
                                         rowsum=rs, bias=torch.from_numpy(bias).to(DEV), heads=heads, window=7)
        fqvit.sync_status()
        assert np.array_equal(_unpack(codes.cpu().numpy(), L), co), (s, mv)
        assert np.array_equal(rs.cpu().numpy().astype(np.uint64), np.asarray(So, np.uint64)), (s, mv)


def test_null_mask_is_the_plain_call():
    a = synth.attn_inputs(synth.CONFIGS["swin_s"], 0, bh=2 * 3 * 7)
    x = a["logits"].to(DEV)
    v = a["v"].to(DEV)
    b = a["bias"].to(DEV)
    want = fqvit.lis_attention(x, a["s_logit"], v, bias=b, heads=3, window=7)
    got = fqvit.lis_attention_masked(x, a["s_logit"], v, None, 0, bias=b, heads=3, window=7)
    fqvit.sync_status()
    assert torch.equal(got, want)


def test_masked_requantized_output(path):
    """fqvit_lis_attention_masked_q: the masked accumulators of the oracle, then its 8-bit
    requantization."""
    rng = np.random.default_rng(11)
    heads, L, d = 3, 49, 32
    region = synth.shifted_window_regions(14, 7).numpy()
    nw = region.shape[0]
    bias = rng.integers(-16, 17, size=(heads, 169), dtype=np.int8)
    BH = 2 * nw * heads
    x = _logits(rng, BH * L, L, 64)
    v = rng.integers(-128, 128, size=(BH, L, d), dtype=np.int8)
    for s, mv, (s_v, s_out, zp_out) in ((0.0347, -2882, (0.05, 0.02, 128)), (0.17, -588, (3 * 2 ** -10, 2 ** -3, 7)),
                                        (0.0078125, -12800, (0.9, 0.0007, 60))):
        _, _, ao = _oracle(x, L, s, v, 0, region, mv, bias=bias, heads=heads)
        want = oracle.attn_requant(ao, s_v, s_out, zp_out)
        out = fqvit.lis_attention_masked_q(torch.from_numpy(x).to(DEV), s, torch.from_numpy(v).to(DEV),
                                           torch.from_numpy(region).to(DEV), mv, 0, s_v, s_out, zp_out,
                                           bias=torch.from_numpy(bias).to(DEV), heads=heads, window=7)
        fqvit.sync_status()
        assert np.array_equal(out.cpu().numpy(), want), (s, mv)
