"""Full-size layers in the launch configuration the bench times, checked against the oracle.

Every config's attention runs over all of its heads at once, as in the timed step, so every CTA
walks its whole range of tiles: the next tile's copy while the current one is computed, heads
changing inside a CTA's range (V converted again), and with tiles packed across heads (rows of
128 .. 384 keys: DeiT-S, ViT-B) tiles that hold the end of one head and the start of the next.
The oracle checks sampled heads element by element: the first and last head of sampled CTA
ranges, heads that share a tile with a neighbour, and random heads.  Layer 0 and the last layer
of each config (their inputs come from different seeds).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2111_13824_gb300 import build as fbuild
from paper_2111_13824_gb300 import fqvit, synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
TM = 128  # query rows per tile of the tensor-core attention


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    fbuild.build()
    fqvit.load()
    oracle.build()


def np_(t):
    return t.detach().cpu().numpy()


def sampled_heads(BH: int, L: int, n_random: int = 6, seed: int = 0) -> list[int]:
    """Heads at the edges of the CTAs' tile ranges of the tensor-core attention (one CTA per SM,
    contiguous ranges), heads whose tile is shared with the next head (packed tiles), and random
    heads."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    packed = TM <= L <= 384
    ntiles = -(-BH * L // TM) if packed else BH * -(-L // TM)
    grid = min(ntiles, sms)
    heads = set()

    def head_of_tile(t: int, last_row: bool) -> int:
        if packed:
            row = min(t * TM + (TM - 1 if last_row else 0), BH * L - 1)
            return row // L
        return t // -(-L // TM)

    for b in list(range(0, grid, max(1, grid // 8))) + [grid - 1]:
        t0, t1 = b * ntiles // grid, (b + 1) * ntiles // grid - 1
        heads.update({head_of_tile(t0, False), head_of_tile(t0, True), head_of_tile(t1, False),
                      head_of_tile(t1, True)})
    if packed:
        split = [t for t in range(ntiles) if (t * TM) // L != min(t * TM + TM - 1, BH * L - 1) // L]
        for t in split[:: max(1, len(split) // 6)]:
            heads.update({(t * TM) // L, (t * TM) // L + 1})
    rng = np.random.default_rng(seed)
    heads.update(int(h) for h in rng.integers(0, BH, n_random))
    return sorted(h for h in heads if 0 <= h < BH)


def _check_heads(acc, logits, v, L, s_logit, heads):
    for h in heads:
        x = np_(logits[h * L:(h + 1) * L])
        co, _ = oracle.lis_softmax(x, L, s_logit)
        ao, ov = oracle.lis_attn_v(co, np_(v[h:h + 1]), 0)
        assert not ov
        got = np_(acc[h:h + 1])
        bad = np.argwhere(got != ao)
        assert bad.size == 0, (h, bad[:4])


@pytest.mark.parametrize("name", ["deit_s", "vit_b", "vit_l384"])
@pytest.mark.parametrize("which", ["first", "last"])
def test_full_layer_attention(name, which):
    cfg = synth.CONFIGS[name]
    layer = 0 if which == "first" else cfg.layers - 1
    a = synth.attn_inputs(cfg, layer, device=DEV)
    acc = fqvit.lis_attention(a["logits"], a["s_logit"], a["v"], 0)
    fqvit.sync_status()
    heads = sampled_heads(a["BH"], a["L"], seed=layer)
    assert len(heads) >= 10
    _check_heads(acc, a["logits"], a["v"], a["L"], a["s_logit"], heads)


@pytest.mark.parametrize("name", ["deit_s", "vit_b"])
def test_full_layer_attention_8bit_output(name):
    """The 8-bit requantized output on the packed tiles, full layer, sampled heads."""
    cfg = synth.CONFIGS[name]
    a = synth.attn_inputs(cfg, 1, device=DEV)
    s_v, s_out, zp_out = 1.0 / 127.0, 0.9 / 127.0, 128
    out = fqvit.lis_attention_q(a["logits"], a["s_logit"], a["v"], 0, s_v, s_out, zp_out)
    fqvit.sync_status()
    L = a["L"]
    for h in sampled_heads(a["BH"], L, n_random=3, seed=1):
        co, _ = oracle.lis_softmax(np_(a["logits"][h * L:(h + 1) * L]), L, a["s_logit"])
        ao, _ = oracle.lis_attn_v(co, np_(a["v"][h:h + 1]), 0)
        yo = oracle.attn_requant(ao, s_v, s_out, zp_out)
        assert np.array_equal(np_(out[h:h + 1]), yo), h


@pytest.mark.parametrize("name", ["deit_s", "vit_l384"])
def test_full_layer_attention_from_qkv(name):
    """Attention from the int8 Q, K, V of a full layer (Q K^T on the tensor cores, head group by
    head group through the workspace), sampled heads against the oracle's Q K^T, softmax and
    attn.V."""
    cfg = synth.CONFIGS[name]
    layer = cfg.layers - 1
    a = synth.attn_inputs(cfg, layer, device=DEV)
    acc = fqvit.qk_lis_attention(a["q"], a["k"], a["v"], 0, 0, a["s_q"], a["s_k"], a["s_logit"], a["zp_logit"])
    fqvit.sync_status()
    L = a["L"]
    for h in sampled_heads(a["BH"], L, n_random=3, seed=layer)[::2]:
        x = oracle.qk_logits(np_(a["q"][h:h + 1]), np_(a["k"][h:h + 1]), 0, 0, a["s_q"], a["s_k"], a["s_logit"],
                             a["zp_logit"], ld=synth.ld_pad(L))
        co, _ = oracle.lis_softmax(x, L, a["s_logit"])
        ao, _ = oracle.lis_attn_v(co, np_(a["v"][h:h + 1]), 0)
        assert np.array_equal(np_(acc[h:h + 1]), ao), h


@pytest.mark.parametrize("layer", [1, 5, 21, 23])
def test_full_swin_layer_attention(layer):
    """A full Swin-S layer (windowed attention with the relative-position bias, and the shifted-window
    mask on odd blocks), whole images sampled so that the bias and mask indexing line up."""
    cfg = synth.CONFIGS["swin_s"]
    st = synth.layer_stage(cfg, layer)
    a = synth.attn_inputs(cfg, layer, device=DEV)
    region = synth.layer_window_mask(cfg, layer, device=DEV)
    mv = synth.swin_mask_value(a["s_logit"])
    kw = dict(bias=a["bias"], heads=a["heads"], window=a["window"])
    if region is not None:
        acc = fqvit.lis_attention_masked(a["logits"], a["s_logit"], a["v"], region, mv, 0, **kw)
    else:
        acc = fqvit.lis_attention(a["logits"], a["s_logit"], a["v"], 0, **kw)
    fqvit.sync_status()
    L, H = a["L"], a["heads"]
    heads_per_image = a["BH"] // 64
    bias = np_(a["bias"])
    reg = np_(region) if region is not None else None
    for img in (0, 37, 63):
        h0, h1 = img * heads_per_image, (img + 1) * heads_per_image
        x = np_(a["logits"][h0 * L:h1 * L])
        co, _ = oracle.lis_softmax(x, L, a["s_logit"], bias=bias, heads=H, window=a["window"], region=reg,
                                   mask_value=mv if reg is not None else 0)
        ao, _ = oracle.lis_attn_v(co, np_(a["v"][h0:h1]), 0)
        assert np.array_equal(np_(acc[h0:h1]), ao), (layer, img, st.C)


@pytest.mark.parametrize("name,layer", [("deit_s", 11), ("vit_b", 6), ("vit_l384", 23), ("swin_s", 20)])
def test_full_layer_layernorm(name, layer):
    """The PTF LayerNorm of a full later layer (every row) against the oracle."""
    cfg = synth.CONFIGS[name]
    d = synth.ln_inputs(cfg, layer, device=DEV)
    s, zp, alpha = fqvit.calibrate_ptf(d["x_calib"], K=cfg.K)
    xq = fqvit.ptf_quantize(d["x"], float(s.item()), int(zp.item()), alpha)
    y = fqvit.ptf_layernorm(xq, int(zp.item()), alpha, d["gamma"], d["beta"], d["s_out"], d["zp_out"])
    fqvit.sync_status()
    so, zo, ao, _ = oracle.calibrate_ptf(np_(d["x_calib"]), K=cfg.K)
    assert np.float32(so) == np.float32(s.item()) and zo == zp.item() and np.array_equal(ao, np_(alpha))
    xqo = oracle.ptf_quantize(np_(d["x"]), so, zo, ao)
    assert np.array_equal(np_(xq), xqo)
    yo, _, _ = oracle.ptf_layernorm(xqo, zo, ao, np_(d["gamma"]), np_(d["beta"]), d["s_out"], d["zp_out"])
    assert np.array_equal(np_(y), yo)
