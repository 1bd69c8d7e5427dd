"""Attention from 8-bit Q and K on the GPU against the oracle, bit for bit:
the Q K^T logits with their MinMax 8-bit output quantizer (fqvit_qk_logits, on
the tensor cores) and the chained attention Q, K, V -> logits -> Log-Int-Softmax
-> BitShift attn.V (fqvit_qk_lis_attention, in groups of heads), for ragged and
full shapes, zero points, multipliers that take the 32-bit and the 64-bit
epilogue, the Swin windows with bias and mask, and both Log-Int-Softmax paths.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2111_13824_gb300 import build as fbuild
from paper_2111_13824_gb300 import fqvit, synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    fbuild.build()
    fqvit.load()
    oracle.build()


def _codes(rng, BH, L, d, lo=-128, hi=128):
    return rng.integers(lo, hi, size=(BH, L, d), dtype=np.int16).astype(np.int8)


def _gpu_logits(q, k, zp_q, zp_k, s_q, s_k, s_l, zp_l):
    out = fqvit.qk_logits(torch.from_numpy(q).to(DEV), torch.from_numpy(k).to(DEV), zp_q, zp_k, s_q, s_k, s_l, zp_l)
    fqvit.sync_status()
    return out.cpu().numpy()


# (s_q, s_k, s_logit): a typical set; M = 1 exactly; M = 2^-30 (shift cap N1 = 31); M = 300 (N1 < 0: the
# 64-bit epilogue); M with 8 significant bits
SCALES = [(0.031, 0.027, 0.0441), (2.0 ** -3, 2.0 ** -4, 2.0 ** -10), (2.0 ** -20, 2.0 ** -13, 8.0),
          (30.0, 80.0, 1.0), (255 * 2.0 ** -9, 2.0 ** -4, 2.0 ** -6)]


@pytest.mark.parametrize("BH,L,d", [(3, 577, 64), (5, 197, 64), (4, 49, 32), (2, 1, 64), (3, 17, 16), (2, 640, 64),
                                    (3, 129, 64), (2, 128, 8), (2, 255, 40), (1, 513, 64)])
def test_qk_logits_match_oracle(BH, L, d):
    rng = np.random.default_rng(BH * 1000 + L + d)
    q, k = _codes(rng, BH, L, d), _codes(rng, BH, L, d)
    ld = (L + 15) // 16 * 16
    for zp_q, zp_k, zp_l in ((0, 0, 0), (-128, 127, 5), (17, -55, -100)):
        for s_q, s_k, s_l in SCALES:
            want = oracle.qk_logits(q, k, zp_q, zp_k, s_q, s_k, s_l, zp_l, ld=ld)
            got = _gpu_logits(q, k, zp_q, zp_k, s_q, s_k, s_l, zp_l)
            bad = np.argwhere(got != want)
            assert bad.size == 0, (BH, L, d, zp_q, zp_k, zp_l, s_q, bad[:4], got[tuple(bad[0])], want[tuple(bad[0])])


def test_qk_logits_full_size_sampled():
    """ViT-L/384 (512 heads of 577 x 577, d = 64) from the synthetic generator in one launch;
    heads sampled across the launch (first, both ends of the CTAs' ranges, last) against the oracle."""
    a = synth.attn_inputs(synth.CONFIGS["vit_l384"], 0)
    q, k = a["q"], a["k"]
    BH = q.shape[0]
    out = fqvit.qk_logits(q.to(DEV), k.to(DEV), 0, 0, a["s_q"], a["s_k"], a["s_logit"], a["zp_logit"])
    fqvit.sync_status()
    got = out.cpu().numpy().reshape(BH, 577, -1)
    for h in (0, 1, 3, 4, 255, 256, 509, 510, 511):
        want = oracle.qk_logits(q[h:h + 1].numpy(), k[h:h + 1].numpy(), 0, 0, a["s_q"], a["s_k"], a["s_logit"],
                                a["zp_logit"], ld=got.shape[2])
        assert np.array_equal(got[h], want), h
    # the integer path agrees with the generator's real-valued logits within the 8-bit multiplier's bound
    diff = np.abs(got[:4, :, :577].astype(np.int64) - a["logits"].numpy().reshape(BH, 577, -1)[:4, :, :577])
    assert diff.max() <= 3


def _chain(q, k, v, zp_q, zp_k, s_q, s_k, s_l, zp_l, zp_v=0, bias=None, heads=1, window=7, region=None,
           mask_value=0):
    BH, L, d = q.shape
    lg = oracle.qk_logits(q, k, zp_q, zp_k, s_q, s_k, s_l, zp_l, ld=(L + 15) // 16 * 16)
    co, _ = oracle.lis_softmax(lg, L, s_l, bias=bias, heads=heads, window=window, region=region,
                               mask_value=mask_value)
    ao, ov = oracle.lis_attn_v(co, v, zp_v)
    assert not ov
    return ao


@pytest.fixture(params=["auto", "cuda_core"])
def path(request, monkeypatch):
    if request.param == "cuda_core":
        monkeypatch.setenv("FQVIT_ATTN_PATH", "cuda_core")
    return request.param


@pytest.mark.parametrize("name,bh,group", [("vit_l384", 5, 2), ("vit_l384", 3, 0), ("deit_s", 7, 3),
                                           ("vit_b", 4, 1)])
def test_chained_attention_from_qkv(name, bh, group, path):
    a = synth.attn_inputs(synth.CONFIGS[name], 1, bh=bh)
    q, k, v = a["q"].numpy(), a["k"].numpy(), a["v"].numpy()
    want = _chain(q, k, v, 0, 0, a["s_q"], a["s_k"], a["s_logit"], a["zp_logit"])
    acc = fqvit.qk_lis_attention(a["q"].to(DEV), a["k"].to(DEV), a["v"].to(DEV), 0, 0, a["s_q"], a["s_k"],
                                 a["s_logit"], a["zp_logit"], group_heads=group)
    fqvit.sync_status()
    assert np.array_equal(acc.cpu().numpy(), want), (name, bh, group)


@pytest.mark.parametrize("zp_q,zp_k,zp_v", [(-128, 127, 0), (40, -3, -77)])
def test_chained_attention_with_zero_points(zp_q, zp_k, zp_v, path):
    rng = np.random.default_rng(200 + zp_q)
    BH, L, d = 4, 197, 64
    q, k, v = _codes(rng, BH, L, d), _codes(rng, BH, L, d), _codes(rng, BH, L, d)
    s = (0.02, 0.03, 0.35)
    want = _chain(q, k, v, zp_q, zp_k, *s, -20, zp_v=zp_v)
    acc = fqvit.qk_lis_attention(torch.from_numpy(q).to(DEV), torch.from_numpy(k).to(DEV),
                                 torch.from_numpy(v).to(DEV), zp_q, zp_k, *s, -20, zp_v=zp_v, group_heads=3)
    fqvit.sync_status()
    assert np.array_equal(acc.cpu().numpy(), want)


def test_chained_swin_windows_with_bias_and_mask(path):
    """Swin-S stage 3 (12 heads, d = 32, 7 x 7 windows): bias, and the shifted-window mask; the
    groups are whole (window, head) units."""
    cfg = synth.CONFIGS["swin_s"]
    st = synth.layer_stage(cfg, 5)
    region = synth.layer_window_mask(cfg, 5).numpy()
    nw = region.shape[0]
    a = synth.attn_inputs(cfg, 5, bh=2 * nw * st.H)
    q, k, v = a["q"].numpy(), a["k"].numpy(), a["v"].numpy()
    bias = a["bias"].numpy()
    mv = synth.swin_mask_value(a["s_logit"])
    args = (a["s_q"], a["s_k"], a["s_logit"], a["zp_logit"])
    for reg, m in ((None, 0), (region, mv)):
        want = _chain(q, k, v, 0, 0, *args, bias=bias, heads=st.H, region=reg, mask_value=m)
        acc = fqvit.qk_lis_attention(a["q"].to(DEV), a["k"].to(DEV), a["v"].to(DEV), 0, 0, *args,
                                     group_heads=nw * st.H, bias=a["bias"].to(DEV), heads=st.H, window=7,
                                     region=None if reg is None else torch.from_numpy(reg).to(DEV), mask_value=m)
        fqvit.sync_status()
        assert np.array_equal(acc.cpu().numpy(), want), m


def test_workspace_too_small_is_an_error():
    BH, L, d = 4, 49, 32
    z = torch.zeros(BH, L, d, dtype=torch.int8, device=DEV)
    ws = torch.empty(L * 64 - 16, dtype=torch.int8, device=DEV)
    with pytest.raises(fqvit.FqvitError):
        fqvit.qk_lis_attention(z, z, z, 0, 0, 0.1, 0.1, 0.1, 0, workspace=ws)
