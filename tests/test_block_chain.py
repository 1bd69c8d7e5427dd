"""One fully quantized transformer block, end to end on the GPU through the library's public calls,
against the oracle functions chained the same way, bit for bit at every stage:

    norm1 (PTF LayerNorm) -> QKV Linear -> head split -> Q K^T (8-bit logits) -> Log-Int-Softmax +
    BitShift attn.V (8-bit output) -> head merge -> proj Linear -> norm2 -> fc1 Linear -> fc2 Linear

(Sec. 3: MinMax for Linear and MatMul, PTF for LayerNorm inputs, Log-Int-Softmax; Sec. 4.1: weights
symmetric channel-wise, activations asymmetric layer-wise; the supplement's integer LayerNorm and
Algorithms 1-2; Eq. 15).  GELU and the residual additions have no integer form in the paper and are
left out: fc1's output feeds fc2, and proj's output feeds norm2 as a PTF input with every alpha 0
(the MinMax quantizer).

Every output scale is calibrated the paper's way, MinMax over the stage's real-valued output, with
the real values taken from the oracle's exact integer accumulators on the same inputs.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2111_13824_gb300 import build as fbuild
from paper_2111_13824_gb300 import fqvit

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    fbuild.build()
    fqvit.load()
    oracle.build()


def np_(t):
    return t.detach().cpu().numpy()


def minmax_u8(v):
    """MinMax asymmetric 8-bit quantizer of a real-valued range (Sec. 4.1): (scale, zero point)."""
    lo, hi = float(min(v.min(), 0.0)), float(max(v.max(), 0.0))
    s = np.float32(max(hi - lo, 1e-6) / 255.0)
    zp = int(np.clip(np.rint(-lo / float(s)), 0, 255))
    return float(s), zp


def linear_params(rng, N, K, bias=True):
    w = rng.integers(-127, 128, size=(N, K)).astype(np.int8)
    s_w = (rng.uniform(0.5, 1.5, size=N) / (127.0 * np.sqrt(K))).astype(np.float32)
    b = rng.integers(-2000, 2000, size=N).astype(np.int32) if bias else None
    return w, s_w, b


def calibrated_linear(x, zp_x, s_x, w, s_w, b):
    """Output scale of a Linear layer from the exact accumulators, then the layer itself (oracle)."""
    _, acc = oracle.linear_q(x, zp_x, s_x, w, s_w, b, 1.0, 0)
    s_y, zp_y = minmax_u8(acc.astype(np.float64) * s_x * s_w.astype(np.float64)[None, :])
    y, _ = oracle.linear_q(x, zp_x, s_x, w, s_w, b, s_y, zp_y)
    return y, s_y, zp_y


def split_np(qkv, B, L, H, d):
    """[B L, 3 H d] uint8 -> three int8 [B H, L, d] (code - 128), as fqvit_split_qkv."""
    t = qkv.reshape(B, L, 3, H, d).transpose(2, 0, 3, 1, 4).reshape(3, B * H, L, d)
    return [(t[p].astype(np.int16) - 128).astype(np.int8) for p in range(3)]


def merge_np(o, B, L, H, d):
    return o.reshape(B, H, L, d).transpose(0, 2, 1, 3).reshape(B * L, H * d)


def oracle_block(seed, B, L, H, d):
    """The block on the oracle: inputs, calibrated scales, and every stage's codes."""
    rng = np.random.default_rng(seed)
    C, M = H * d, B * L
    # norm1's input: channel ranges that differ by up to 16x (PTF picks alpha per channel)
    ch = np.where(rng.random(C) < 0.05, rng.uniform(4, 16, C), rng.uniform(0.5, 1.5, C))
    x = (rng.normal(size=(M, C)) * ch[None, :] + rng.normal(size=C)[None, :] * 0.3).astype(np.float32)
    s_in, zp_in, alpha, _ = oracle.calibrate_ptf(x, K=3)
    xq = oracle.ptf_quantize(x, s_in, zp_in, alpha)
    g1 = (1 + 0.1 * rng.normal(size=C)).astype(np.float32)
    b1 = (0.1 * rng.normal(size=C)).astype(np.float32)
    st = {}
    # LayerNorm output range: gamma * (+-4 sigma) + beta
    s_n1, zp_n1 = minmax_u8(np.array([-4.0 * np.abs(g1).max() + b1.min(), 4.0 * np.abs(g1).max() + b1.max()]))
    y1, _, _ = oracle.ptf_layernorm(xq, zp_in, alpha, g1, b1, s_n1, zp_n1)
    st["norm1"] = y1
    wq, sq, bq = linear_params(rng, 3 * C, C)
    qkv, s_qkv, zp_qkv = calibrated_linear(y1, zp_n1, s_n1, wq, sq, bq)
    st["qkv"] = qkv
    q, k, v = split_np(qkv, B, L, H, d)
    zp_s = zp_qkv - 128
    # logit scale: MinMax of Q K^T / sqrt(d), within the range Log-Int-Softmax takes
    P = np.einsum("bid,bjd->bij", q.astype(np.int64) - zp_s, k.astype(np.int64) - zp_s)
    real = P.astype(np.float64) * s_qkv * s_qkv / np.sqrt(d)
    s_logit = float(np.float32(np.clip((real.max() - real.min()) / 255.0, 2.0 ** -7, 0.5)))
    zp_logit = int(np.clip(np.rint(-real.min() / s_logit), 0, 255)) - 128
    ld = (L + 15) // 16 * 16
    logits = oracle.qk_logits(q, k, zp_s, zp_s, s_qkv, s_qkv, s_logit, zp_logit, ld=ld)
    st["logits"] = logits
    codes, _ = oracle.lis_softmax(logits, L, s_logit)
    acc, ov = oracle.lis_attn_v(codes, v, zp_s)
    assert not ov
    s_att, zp_att = minmax_u8(acc.astype(np.float64) * s_qkv / 32768.0)
    att = oracle.attn_requant(acc, s_qkv, s_att, zp_att)
    st["attn"] = att
    am = merge_np(att, B, L, H, d)
    wp, sp, bp = linear_params(rng, C, C)
    proj, s_p, zp_p = calibrated_linear(am, zp_att, s_att, wp, sp, bp)
    st["proj"] = proj
    g2 = (1 + 0.1 * rng.normal(size=C)).astype(np.float32)
    b2 = (0.1 * rng.normal(size=C)).astype(np.float32)
    s_n2, zp_n2 = minmax_u8(np.array([-4.0 * np.abs(g2).max() + b2.min(), 4.0 * np.abs(g2).max() + b2.max()]))
    alpha0 = np.zeros(C, np.uint8)
    y2, _, _ = oracle.ptf_layernorm(proj, zp_p, alpha0, g2, b2, s_n2, zp_n2)
    st["norm2"] = y2
    w1, s1, bb1 = linear_params(rng, 4 * C, C)
    f1, s_f1, zp_f1 = calibrated_linear(y2, zp_n2, s_n2, w1, s1, bb1)
    st["fc1"] = f1
    w2, s2, bb2 = linear_params(rng, C, 4 * C)
    f2, s_f2, zp_f2 = calibrated_linear(f1, zp_f1, s_f1, w2, s2, bb2)
    st["fc2"] = f2
    prm = dict(xq=xq, zp_in=zp_in, alpha=alpha, g1=g1, b1=b1, s_n1=s_n1, zp_n1=zp_n1, wq=wq, sq=sq, bq=bq,
               s_qkv=s_qkv, zp_qkv=zp_qkv, s_logit=s_logit, zp_logit=zp_logit, s_att=s_att, zp_att=zp_att,
               wp=wp, sp=sp, bp=bp, s_p=s_p, zp_p=zp_p, g2=g2, b2=b2, s_n2=s_n2, zp_n2=zp_n2, w1=w1, s1=s1,
               bb1=bb1, s_f1=s_f1, zp_f1=zp_f1, w2=w2, s2=s2, bb2=bb2, s_f2=s_f2, zp_f2=zp_f2)
    return prm, st


def gpu_block(prm, B, L, H, d):
    """The same block through the library on cuda:0; every stage's codes."""
    T = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(DEV)  # noqa: E731
    C = H * d
    st = {}
    y1 = fqvit.ptf_layernorm(T(prm["xq"]), prm["zp_in"], T(prm["alpha"]), T(prm["g1"]), T(prm["b1"]),
                             prm["s_n1"], prm["zp_n1"])
    st["norm1"] = y1

    def lin(x, zp_x, s_x, w, s_w, b, s_y, zp_y):
        return fqvit.linear_q(x, zp_x, s_x, fqvit.linear_pack_weight(T(w)), T(s_w), None if b is None else T(b),
                              s_y, zp_y)

    qkv = lin(y1, prm["zp_n1"], prm["s_n1"], prm["wq"], prm["sq"], prm["bq"], prm["s_qkv"], prm["zp_qkv"])
    st["qkv"] = qkv
    q, k, v = fqvit.split_qkv(qkv, B, L, H, d)
    zp_s = prm["zp_qkv"] - 128
    logits = fqvit.qk_logits(q, k, zp_s, zp_s, prm["s_qkv"], prm["s_qkv"], prm["s_logit"], prm["zp_logit"])
    st["logits"] = logits
    att = fqvit.lis_attention_q(logits, prm["s_logit"], v, zp_s, prm["s_qkv"], prm["s_att"], prm["zp_att"])
    st["attn"] = att
    am = fqvit.merge_heads(att, B, L, H)
    proj = lin(am, prm["zp_att"], prm["s_att"], prm["wp"], prm["sp"], prm["bp"], prm["s_p"], prm["zp_p"])
    st["proj"] = proj
    y2 = fqvit.ptf_layernorm(proj, prm["zp_p"], torch.zeros(C, dtype=torch.uint8, device=DEV), T(prm["g2"]),
                             T(prm["b2"]), prm["s_n2"], prm["zp_n2"])
    st["norm2"] = y2
    f1 = lin(y2, prm["zp_n2"], prm["s_n2"], prm["w1"], prm["s1"], prm["bb1"], prm["s_f1"], prm["zp_f1"])
    st["fc1"] = f1
    f2 = lin(f1, prm["zp_f1"], prm["s_f1"], prm["w2"], prm["s2"], prm["bb2"], prm["s_f2"], prm["zp_f2"])
    st["fc2"] = f2
    fqvit.sync_status()
    return st


@pytest.mark.parametrize("B,L,H,d", [(2, 197, 6, 64), (1, 577, 16, 64)])
def test_block_chain_matches_oracle(B, L, H, d):
    prm, want = oracle_block(B * 1000 + L, B, L, H, d)
    got = gpu_block(prm, B, L, H, d)
    for stage in ("norm1", "qkv", "logits", "attn", "proj", "norm2", "fc1", "fc2"):
        g = np_(got[stage]).reshape(want[stage].shape)
        bad = np.argwhere(g != want[stage])
        assert bad.size == 0, (stage, bad[:4])
    # the stages carry information: no stage collapsed to a constant code
    for stage in ("qkv", "attn", "proj", "fc1", "fc2"):
        assert len(np.unique(want[stage])) > 16, stage


def test_split_and_merge_heads_are_inverse_layouts():
    """fqvit_split_qkv and fqvit_merge_heads against numpy reshapes, with padded head rows."""
    B, L, H, d = 3, 37, 5, 32
    rng = np.random.default_rng(5)
    qkv = rng.integers(0, 256, size=(B * L, 3 * H * d + 16)).astype(np.uint8)
    t = torch.from_numpy(qkv).to(DEV)
    q, k, v = fqvit.split_qkv(t[:, : 3 * H * d], B, L, H, d, ld_head=48)
    want = split_np(qkv[:, : 3 * H * d], B, L, H, d)
    for got, w in zip((q, k, v), want):
        assert np.array_equal(np_(got), w)
    heads = torch.from_numpy((want[2].astype(np.int16) + 128).astype(np.uint8)).to(DEV)
    m = fqvit.merge_heads(heads, B, L, H)
    assert np.array_equal(np_(m), qkv[:, 2 * H * d: 3 * H * d])
