"""Back-to-back dependent launches on one stream, with no host synchronisation between them.

The step's kernels are launched with programmatic dependent launch: each may start while the
previous kernel finishes, and waits before its first access to global memory.  These tests put
a kernel right behind the one that writes its input (read after write), or behind one that
still reads the buffer it overwrites (write after read), and compare with the oracle: a wait
placed too late would read stale or half-written data.
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


def _ln_case(seed, rows, C):
    rng = np.random.default_rng(seed)
    xq = rng.integers(0, 256, size=(rows, C), dtype=np.int32).astype(np.uint8)
    alpha = rng.integers(0, 4, size=C).astype(np.uint8)
    gamma = (1.0 + 0.1 * rng.standard_normal(C)).astype(np.float32)
    beta = (0.1 * rng.standard_normal(C)).astype(np.float32)
    return xq, alpha, gamma, beta


def test_layernorm_chain_read_after_write():
    """LayerNorm of a LayerNorm's output, eight times over, launched back to back."""
    rows, C = 20000, 768
    xq, alpha, gamma, beta = _ln_case(1, rows, C)
    zp, s_out, zp_out = 37, 0.021, 101
    d = [torch.from_numpy(t).to(DEV) for t in (xq, alpha, gamma, beta)]
    bufs = [d[0]] + [torch.empty(rows, C, dtype=torch.uint8, device=DEV) for _ in range(8)]
    torch.cuda.synchronize()
    for i in range(8):  # each launch reads the previous one's output
        fqvit.ptf_layernorm(bufs[i], zp, d[1], d[2], d[3], s_out, zp_out, out=bufs[i + 1])
    torch.cuda.synchronize()
    want = xq
    for i in range(8):
        want, _, _ = oracle.ptf_layernorm(want, zp, alpha, gamma, beta, s_out, zp_out)
        assert np.array_equal(bufs[i + 1].cpu().numpy(), want), i


def test_layernorm_write_after_read():
    """A LayerNorm that overwrites the input of the LayerNorm launched just before it."""
    rows, C = 20000, 1024
    xq, alpha, gamma, beta = _ln_case(2, rows, C)
    zp, s_out, zp_out = 5, 0.03, 90
    a = torch.from_numpy(xq).to(DEV)
    b = torch.empty_like(a)
    al, g, be = (torch.from_numpy(t).to(DEV) for t in (alpha, gamma, beta))
    torch.cuda.synchronize()
    fqvit.ptf_layernorm(a, zp, al, g, be, s_out, zp_out, out=b)   # reads a
    fqvit.ptf_layernorm(b, zp, al, g, be, s_out, zp_out, out=a)   # writes a
    torch.cuda.synchronize()
    y1, _, _ = oracle.ptf_layernorm(xq, zp, alpha, gamma, beta, s_out, zp_out)
    y2, _, _ = oracle.ptf_layernorm(y1, zp, alpha, gamma, beta, s_out, zp_out)
    assert np.array_equal(b.cpu().numpy(), y1)
    assert np.array_equal(a.cpu().numpy(), y2)


@pytest.mark.parametrize("name,bh", [("vit_l384", 6), ("deit_s", 9), ("swin_s", 12)])
def test_attention_reads_logits_written_just_before(name, bh):
    """Logits produced by a kernel on the stream (Q K^T, or a device copy for the window path)
    and the fused attention launched right after on them."""
    a = synth.attn_inputs(synth.CONFIGS[name], 0, bh=bh)
    x = a["logits"].to(DEV)
    v = a["v"].to(DEV)
    bias = a["bias"].to(DEV) if a["bias"] is not None else None
    L = a["L"]
    kw = dict(bias=bias, heads=a["heads"], window=a["window"])
    if name == "swin_s":
        src = torch.zeros_like(x)
        torch.cuda.synchronize()
        src.copy_(x)  # written on the stream right before the attention
        acc = fqvit.lis_attention(src, a["s_logit"], v, 0, **kw)
        co, _ = oracle.lis_softmax(a["logits"].numpy(), L, a["s_logit"], bias=a["bias"].numpy(), heads=a["heads"],
                                   window=a["window"])
    else:
        logits = torch.zeros_like(x)
        torch.cuda.synchronize()
        fqvit.qk_logits(a["q"].to(DEV), a["k"].to(DEV), 0, 0, a["s_q"], a["s_k"], a["s_logit"], a["zp_logit"],
                        out=logits)
        acc = fqvit.lis_attention(logits, a["s_logit"], v, 0, **kw)
        lo = oracle.qk_logits(a["q"].numpy(), a["k"].numpy(), 0, 0, a["s_q"], a["s_k"], a["s_logit"], a["zp_logit"],
                              ld=a["ld_logit"])
        co, _ = oracle.lis_softmax(lo, L, a["s_logit"])
    fqvit.sync_status()
    ao, ov = oracle.lis_attn_v(co, a["v"].numpy(), 0)
    assert not ov
    assert np.array_equal(acc.cpu().numpy(), ao)
