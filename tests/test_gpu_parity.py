"""CUDA path vs CPU oracle, element by element, on seeded inputs.

Every integer tensor must match bit for bit: PTF codes, alpha, s / zp (as
bits), the LayerNorm statistics and output, the i-exp row sums, the 4-bit
codes and the attention accumulators.  Calls go through the C ABI
(paper_2111_13824_gb300.fqvit).
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


def unpack_codes(packed: np.ndarray, L: int) -> np.ndarray:
    lo = packed & 0x0F
    hi = packed >> 4
    out = np.stack([lo, hi], axis=-1).reshape(packed.shape[0], -1)
    return out[:, :L]


def np_(t):
    return t.detach().cpu().numpy()


# ---------------------------------------------------------------- PTF

def _channels(seed, rows, C, spread=40.0):
    rng = np.random.default_rng(seed)
    r = np.exp(rng.normal(0, 1, C))
    med = np.median(r)
    r = np.exp(np.log(med) + (np.log(r) - np.log(med)) * np.log(spread) / (np.log(r.max()) - np.log(med)))
    m = 0.25 * r * rng.normal(size=C)
    return (m + r / 6 * rng.normal(size=(rows, C))).astype(np.float32)


@pytest.mark.parametrize("rows,C,K", [(6304, 192, 3), (1000, 96, 0), (777, 384, 7), (300, 100, 3), (1, 64, 3)])
def test_calibrate_and_quantize(rows, C, K):
    x = _channels(rows * 7 + C, rows, C)
    s_o, zp_o, a_o, sse_o = oracle.calibrate_ptf(x, K=K)
    xd = torch.from_numpy(x).to(DEV)
    sse = torch.empty(C, K + 1, dtype=torch.float64, device=DEV)
    s, zp, alpha = fqvit.calibrate_ptf(xd, K=K, sse=sse)
    torch.cuda.synchronize()
    assert np.float32(s_o).view(np.uint32) == np_(s).view(np.uint32)[0]
    assert zp_o == int(zp.item())
    assert np.array_equal(a_o, np_(alpha))
    assert np.array_equal(sse_o.view(np.uint64), np_(sse).view(np.uint64))
    q = fqvit.ptf_quantize(xd, float(s.item()), int(zp.item()), alpha)
    assert np.array_equal(oracle.ptf_quantize(x, s_o, zp_o, a_o), np_(q))


def test_calibrate_strided_and_constant():
    x = _channels(3, 500, 64)
    big = np.zeros((500, 80), np.float32)
    big[:, :64] = x
    xd = torch.from_numpy(big).to(DEV)[:, :64]
    s, zp, alpha = fqvit.calibrate_ptf(xd, K=3)
    s_o, zp_o, a_o, _ = oracle.calibrate_ptf(x, K=3)
    assert np.float32(s_o) == np.float32(s.item()) and zp_o == zp.item()
    assert np.array_equal(a_o, np_(alpha))
    c = np.full((40, 16), 0.75, np.float32)  # degenerate range
    s, zp, alpha = fqvit.calibrate_ptf(torch.from_numpy(c).to(DEV), K=2)
    s_o, zp_o, a_o, _ = oracle.calibrate_ptf(c, K=2)
    assert np.float32(s_o) == np.float32(s.item()) and zp_o == zp.item()
    assert np.array_equal(a_o, np_(alpha))


# ---------------------------------------------------------------- LayerNorm

def _ln_case(seed, rows, C, K=3, s_out=0.03, zp_out=120):
    x = _channels(seed, rows, C)
    s, zp, alpha, _ = oracle.calibrate_ptf(x, K=K)
    xq = oracle.ptf_quantize(x, s, zp, alpha)
    rng = np.random.default_rng(seed + 1)
    gamma = (1 + 0.1 * rng.normal(size=C)).astype(np.float32)
    beta = (0.1 * rng.normal(size=C)).astype(np.float32)
    return xq, zp, alpha, gamma, beta, s_out, zp_out


def _run_ln(xq, zp, alpha, gamma, beta, s_out, zp_out, ld_in=None, ld_out=None):
    rows, C = xq.shape
    ld_in = ld_in or C
    ld_out = ld_out or C
    buf = torch.zeros(rows, ld_in, dtype=torch.uint8, device=DEV)
    buf[:, :C] = torch.from_numpy(xq).to(DEV)
    out = torch.zeros(rows, ld_out, dtype=torch.uint8, device=DEV)
    m1 = torch.empty(rows, dtype=torch.int64, device=DEV)
    m2 = torch.empty(rows, dtype=torch.int64, device=DEV)
    fqvit.ptf_layernorm(buf[:, :C], zp, torch.from_numpy(alpha).to(DEV), torch.from_numpy(gamma).to(DEV),
                        torch.from_numpy(beta).to(DEV), s_out, zp_out, out=out[:, :C], m1=m1, m2=m2)
    torch.cuda.synchronize()
    return np_(out[:, :C]), np_(m1), np_(m2)


def _assert_ln(case, **kw):
    y, m1, m2 = _run_ln(*case, **kw)
    yo, m1o, m2o = oracle.ptf_layernorm(*case)
    assert np.array_equal(m1, m1o)
    assert np.array_equal(m2, m2o)
    bad = np.argwhere(y != yo)
    assert bad.size == 0, (bad[:5], y[tuple(bad[0])], yo[tuple(bad[0])])


@pytest.mark.parametrize("rows,C", [(1003, 192), (517, 384), (300, 768), (257, 1024), (64, 96), (33, 4096),
                                    (129, 100), (17, 8192), (1, 16)])
def test_layernorm_matches_oracle(rows, C):
    _assert_ln(_ln_case(rows + C, rows, C))


@pytest.mark.parametrize("rows,C", [(1001, 32), (777, 48), (513, 64), (2049, 80), (333, 128), (99, 256),
                                    (50001, 96), (40003, 192), (7, 16), (3, 48)])
def test_layernorm_rows_per_warp(rows, C):
    """Short rows share a warp (a segment of lanes per row): every segment width, row counts
    that leave the last warp partly empty, and enough rows for many passes per warp."""
    _assert_ln(_ln_case(rows * 7 + C, rows, C))


@pytest.mark.parametrize("rows,C", [(3001, 1024), (6007, 768), (10001, 384), (4000, 4096)])
def test_layernorm_two_rows_per_segment(rows, C):
    """Row counts between the thresholds of the rows-per-segment choice: on a 152-SM GPU these
    take 2 rows per segment (the most that still gives half of the grid's warps a group), the
    other counts of these tests 4 or 1."""
    _assert_ln(_ln_case(rows + 3 * C, rows, C))


def test_layernorm_strided_rows():
    _assert_ln(_ln_case(5, 200, 192), ld_in=208, ld_out=224)
    _assert_ln(_ln_case(6, 200, 192), ld_in=193, ld_out=195)


def test_layernorm_edge_rows():
    xq, zp, alpha, gamma, beta, s_out, zp_out = _ln_case(9, 256, 384, K=7)
    gamma = gamma.copy()
    gamma[3] = 0.0                 # A == 0 channel
    gamma[5] = -1.5                # negative A
    gamma[7] = 1e-6                # large N1
    gamma[11] = 3e4                # N1 < 0
    beta = beta.copy()
    beta[13] = 1e5                 # huge B
    xq = xq.copy()
    xq[0, :] = 77                  # constant row (D == 0)
    xq[1, :] = 0
    xq[1, 5] = 1                   # near-constant row: tiny D, large A
    alpha = alpha.copy()
    alpha[:4] = 7
    _assert_ln((xq, zp, alpha, gamma, beta, s_out, zp_out))
    _assert_ln((xq, zp, alpha, gamma, beta, 1e-4, 0))
    _assert_ln((xq, 255, alpha, gamma, beta, 5.0, 255))


@pytest.mark.parametrize("zp", [0, 128, 255])
def test_layernorm_extreme_values(zp):
    """Bytes 0 and 255 only with alpha = 3 on every channel: |Xh| = 2040 at its largest, the bound of
    the exact squares of the fp32 statistics path; rows of C = 1024 and 4096."""
    rng = np.random.default_rng(zp)
    for C in (1024, 4096):
        rows = 67
        xq = (rng.integers(0, 2, size=(rows, C)) * 255).astype(np.uint8)
        xq[0, :] = 255 - zp if zp in (0, 255) else 255
        alpha = np.full(C, 3, np.uint8)
        gamma = (1 + 0.1 * rng.normal(size=C)).astype(np.float32)
        beta = (0.1 * rng.normal(size=C)).astype(np.float32)
        _assert_ln((xq, zp, alpha, gamma, beta, 0.02, 128))


def test_layernorm_synthetic_configs():
    for name in ("deit_s", "vit_b", "swin_s"):
        cfg = synth.CONFIGS[name]
        d = synth.ln_inputs(cfg, 0, rows=2048)
        x = d["x"].numpy()
        s, zp, alpha, _ = oracle.calibrate_ptf(d["x_calib"].numpy(), K=cfg.K)
        xq = oracle.ptf_quantize(x, s, zp, alpha)
        _assert_ln((xq, zp, alpha, d["gamma"].numpy(), d["beta"].numpy(), d["s_out"], d["zp_out"]))


# ---------------------------------------------------------------- Log-Int-Softmax

SCALES = [0.0078125, 0.008350185749701165, 0.01732846078509329, 0.0425, 0.17, 0.5]


def _rand_logits(seed, n_rows, L, spread):
    rng = np.random.default_rng(seed)
    ld = (L + 15) // 16 * 16
    x = np.zeros((n_rows, ld), np.int8)
    x[:, :L] = np.clip(np.rint(rng.normal(rng.uniform(-40, 40), spread, size=(n_rows, L))), -128, 127)
    return x


@pytest.mark.parametrize("L", [1, 2, 3, 17, 49, 197, 577, 1024])
@pytest.mark.parametrize("s", SCALES)
def test_lis_softmax_matches_oracle(L, s):
    n_rows = 37 if L > 500 else 131
    x = _rand_logits(L * 1000 + int(s * 1e4), n_rows, L, spread=60.0)
    xd = torch.from_numpy(x).to(DEV)
    rowsum = torch.empty(n_rows, dtype=torch.int64, device=DEV)
    codes = fqvit.lis_softmax(xd, L, s, rowsum=rowsum)
    torch.cuda.synchronize()
    co, So = oracle.lis_softmax(x, L, s)
    assert np.array_equal(np_(rowsum).view(np.uint64), So)
    got = unpack_codes(np_(codes), L)
    bad = np.argwhere(got != co)
    assert bad.size == 0, bad[:5]
    if L % 2:
        assert np.all((np_(codes)[:, -1] >> 4) == 0)


def test_lis_softmax_special_rows():
    L = 577
    x = np.full((4, 592), -128, np.int8)
    x[0, 100] = 127                       # one-hot
    x[1, :L] = 5                          # uniform
    x[2, :L] = np.arange(L) % 256 - 128   # ramp
    x[3, :L] = 127
    for s in (0.1, 0.5, 0.0078125):
        codes = fqvit.lis_softmax(torch.from_numpy(x).to(DEV), L, s)
        torch.cuda.synchronize()
        co, _ = oracle.lis_softmax(x, L, s)
        assert np.array_equal(unpack_codes(np_(codes), L), co)
    got = unpack_codes(np_(fqvit.lis_softmax(torch.from_numpy(x).to(DEV), L, 0.1)), L)
    assert got[0, 100] == 0 and (np.delete(got[0], 100) == 15).all()
    assert (got[1] == 9).all() and (got[3] == 9).all()


def test_lis_softmax_relpos_bias():
    cfg = synth.CONFIGS["swin_s"]
    a = synth.attn_inputs(cfg, 0, bh=2 * 3)
    x = a["logits"].numpy()
    bias = a["bias"].numpy()
    for s in (a["s_logit"], 0.0078125, 0.3):
        codes = fqvit.lis_softmax(torch.from_numpy(x).to(DEV), 49, s, bias=torch.from_numpy(bias).to(DEV),
                                  heads=3, window=7)
        torch.cuda.synchronize()
        co, _ = oracle.lis_softmax(x, 49, s, bias=bias, heads=3, window=7)
        assert np.array_equal(unpack_codes(np_(codes), 49), co)


# ---------------------------------------------------------------- BitShift Attn.V

def _pack(codes: np.ndarray) -> np.ndarray:
    n, L = codes.shape
    c = np.zeros((n, (L + 1) // 2 * 2), np.uint8)
    c[:, :L] = codes
    return (c[:, 0::2] | (c[:, 1::2] << 4)).astype(np.uint8)


@pytest.mark.parametrize("L,d,zp", [(1, 64, 0), (49, 32, 0), (197, 64, 0), (577, 64, 0), (200, 64, 7),
                                    (61, 32, -3), (1024, 64, 0)])
def test_attn_v_matches_oracle(L, d, zp):
    rng = np.random.default_rng(L * 10 + d)
    BH = 3
    codes = rng.integers(0, 16, size=(BH * L, L)).astype(np.uint8)
    codes[:, ::7] = rng.integers(8, 16, size=codes[:, ::7].shape)
    v = rng.integers(-128, 128, size=(BH, L, d)).astype(np.int8)
    acc = fqvit.lis_attn_v(torch.from_numpy(_pack(codes)).to(DEV), torch.from_numpy(v).to(DEV), zp)
    torch.cuda.synchronize()
    ao, ov = oracle.lis_attn_v(codes, v, zp)
    if not ov:
        assert np.array_equal(np_(acc), ao)


def test_attn_v_range_flag():
    L, d = 1024, 64
    codes = np.zeros((L, L), np.uint8)  # every weight 2^15: sums leave int32
    v = np.full((1, L, d), -128, np.int8)
    flag = torch.zeros(1, dtype=torch.int32, device=DEV)
    fqvit.lis_attn_v(torch.from_numpy(_pack(codes)).to(DEV), torch.from_numpy(v).to(DEV), 0, range_flag=flag)
    torch.cuda.synchronize()
    assert flag.item() == 1
    _, ov = oracle.lis_attn_v(codes, v, 0)
    assert ov


# ---------------------------------------------------------------- fused and block

def _attn_case(name, layer=0, bh=None, sigma=1.0):
    cfg = synth.CONFIGS[name]
    return synth.attn_inputs(cfg, layer, bh=bh, sigma=sigma)


def _oracle_attention(a):
    x = a["logits"].numpy()
    bias = a["bias"].numpy() if a["bias"] is not None else None
    co, _ = oracle.lis_softmax(x, a["L"], a["s_logit"], bias=bias, heads=a["heads"], window=a["window"] or 7)
    ao, ov = oracle.lis_attn_v(co, a["v"].numpy(), 0)
    assert not ov
    return co, ao


@pytest.mark.parametrize("name,bh,sigma", [("deit_t", None, 1.0), ("deit_s", 7, 2.0), ("vit_l384", 3, 1.0),
                                           ("vit_l384", 2, 2.0), ("swin_s", 12, 1.0)])
def test_lis_attention_matches_oracle(name, bh, sigma, cuda_core_path):
    a = _attn_case(name, bh=bh, sigma=sigma)
    co, ao = _oracle_attention(a)
    L = a["L"]
    bias = a["bias"].to(DEV) if a["bias"] is not None else None
    codes = torch.zeros(a["BH"] * L, (L + 1) // 2, dtype=torch.uint8, device=DEV)
    acc = fqvit.lis_attention(a["logits"].to(DEV), a["s_logit"], a["v"].to(DEV), 0, codes=codes, bias=bias,
                              heads=a["heads"], window=a["window"])
    torch.cuda.synchronize()
    assert np.array_equal(unpack_codes(np_(codes), L), co)
    assert np.array_equal(np_(acc), ao)
    acc2 = fqvit.lis_attention(a["logits"].to(DEV), a["s_logit"], a["v"].to(DEV), 0, bias=bias,
                               heads=a["heads"], window=a["window"])
    torch.cuda.synchronize()
    assert np.array_equal(np_(acc2), ao)


def test_block_int_matches_oracle():
    cfg = synth.CONFIGS["deit_t"]
    d = synth.ln_inputs(cfg, 0)
    a = synth.attn_inputs(cfg, 0)
    s, zp, alpha, _ = oracle.calibrate_ptf(d["x_calib"].numpy(), K=3)
    xq = oracle.ptf_quantize(d["x"].numpy(), s, zp, alpha)
    yo, _, _ = oracle.ptf_layernorm(xq, zp, alpha, d["gamma"].numpy(), d["beta"].numpy(), d["s_out"], d["zp_out"])
    _, ao = _oracle_attention(a)
    yq = torch.empty_like(torch.from_numpy(xq)).to(DEV)
    acc = torch.empty(a["BH"], a["L"], a["d"], dtype=torch.int32, device=DEV)
    fqvit.block_int(torch.from_numpy(xq).to(DEV), zp, torch.from_numpy(alpha).to(DEV), d["gamma"].to(DEV),
                    d["beta"].to(DEV), d["s_out"], d["zp_out"], yq, a["logits"].to(DEV), a["ld_logit"],
                    a["s_logit"], a["v"].to(DEV), 0, acc)
    torch.cuda.synchronize()
    assert np.array_equal(np_(yq), yo)
    assert np.array_equal(np_(acc), ao)


def test_full_size_vit_l_layer_sampled():
    """ViT-L/384 layer at full size (BH = 512, L = 577, 18464 x 1024 LayerNorm),
    in the launch configuration the bench uses; the oracle checks sampled heads
    of the attention and every LayerNorm row."""
    cfg = synth.CONFIGS["vit_l384"]
    a = synth.attn_inputs(cfg, 0, device=DEV)
    acc = fqvit.lis_attention(a["logits"], a["s_logit"], a["v"], 0)
    torch.cuda.synchronize()
    L = a["L"]
    for h in (0, 137, 511):
        rows = slice(h * L, (h + 1) * L)
        x = np_(a["logits"][rows])
        co, _ = oracle.lis_softmax(x, L, a["s_logit"])
        ao, _ = oracle.lis_attn_v(co, np_(a["v"][h:h + 1]), 0)
        assert np.array_equal(np_(acc[h:h + 1]), ao), h
    d = synth.ln_inputs(cfg, 0, device=DEV)
    xd = d["x"]
    s, zp, alpha = fqvit.calibrate_ptf(d["x_calib"], K=3)
    xq = fqvit.ptf_quantize(xd, float(s.item()), int(zp.item()), alpha)
    y = fqvit.ptf_layernorm(xq, int(zp.item()), alpha, d["gamma"], d["beta"], d["s_out"], d["zp_out"])
    torch.cuda.synchronize()
    so, zo, ao_, _ = oracle.calibrate_ptf(np_(d["x_calib"]), K=3)
    assert np.float32(so) == np.float32(s.item()) and zo == zp.item() and np.array_equal(ao_, np_(alpha))
    xqo = oracle.ptf_quantize(np_(xd), so, zo, ao_)
    assert np.array_equal(np_(xq), xqo)
    yo, _, _ = oracle.ptf_layernorm(xqo, zo, ao_, np_(d["gamma"]), np_(d["beta"]), d["s_out"], d["zp_out"])
    assert np.array_equal(np_(y), yo)


# ---------------------------------------------------------------- tensor-core path

@pytest.fixture
def cuda_core_path(monkeypatch):
    monkeypatch.setenv("FQVIT_ATTN_PATH", "cuda_core")


@pytest.mark.parametrize("name,bh,sigma", [("deit_s", 5, 1.0), ("vit_b", 3, 2.0), ("vit_l384", 4, 1.0),
                                           ("vit_l384", 3, 2.0)])
def test_tensor_core_path_matches_oracle(name, bh, sigma):
    a = _attn_case(name, bh=bh, sigma=sigma)
    co, ao = _oracle_attention(a)
    acc = fqvit.lis_attention(a["logits"].to(DEV), a["s_logit"], a["v"].to(DEV), 0)
    fqvit.sync_status()
    assert np.array_equal(np_(acc), ao)


def test_tensor_core_and_cuda_core_agree(monkeypatch):
    a = _attn_case("vit_l384", bh=6, sigma=1.5)
    acc_tc = fqvit.lis_attention(a["logits"].to(DEV), a["s_logit"], a["v"].to(DEV), 0)
    fqvit.sync_status()
    monkeypatch.setenv("FQVIT_ATTN_PATH", "cuda_core")
    acc_cc = fqvit.lis_attention(a["logits"].to(DEV), a["s_logit"], a["v"].to(DEV), 0)
    fqvit.sync_status()
    assert torch.equal(acc_tc, acc_cc)


@pytest.mark.parametrize("L", [1, 2, 17, 64, 65, 128, 129, 197, 577, 592])
def test_tensor_core_exact_at_the_accumulator_bound(L):
    """Rows that push sum_j 2^(15-code_j) |V| toward its bound: k equal top
    logits (I-Log2 rounds k up to 1.5 * 2^M, so k 2^-code approaches 1.5),
    the rest far below, every V = -128 or +127; uniform rows; one-hot rows."""
    ld = (L + 15) // 16 * 16
    ks = [k for k in (1, 2, 3, 5, 11, 23, 47, 95, 191, 383) if k <= L]
    rows = []
    for k in ks:
        r = np.full(ld, -128, np.int8)
        r[:k] = 127
        rows.append(r)
    rows.append(np.full(ld, 3, np.int8))
    n = (len(rows) + L - 1) // L * L
    BH = max(1, n // L)
    x = np.full((BH * L, ld), -128, np.int8)
    for i, r in enumerate(rows):
        x[i] = r
    for s, vv in ((0.5, -128), (0.5, 127), (0.1, -128), (0.0078125, -128)):
        v = np.full((BH, L, 64), vv, np.int8)
        acc = fqvit.lis_attention(torch.from_numpy(x).to(DEV), s, torch.from_numpy(v).to(DEV), 0)
        fqvit.sync_status()
        co, _ = oracle.lis_softmax(x, L, s)
        ao, ov = oracle.lis_attn_v(co, v, 0)
        assert not ov
        assert np.array_equal(np_(acc), ao), (L, s, vv)
        assert np.abs(ao).max() < 2 ** 24


# scales whose floored i-exp constants (Algorithm 1) make e(d) rise once per
# period of d: there the 4-bit code is not monotone in the logit
_RISING_SCALES = (float(np.float32(0.008350185749701165)), float(np.float32(0.01732846078509329)))


@pytest.mark.parametrize("s", _RISING_SCALES + (0.5, 0.3, 0.0625, 0.0078125))
def test_tensor_core_operand_table_at_any_scale(s):
    """Per-row operand tables against the oracle: large scales change the code
    every few logit steps, and at the rising scales codes may fall back."""
    if s in _RISING_SCALES:
        e = [oracle.iexp(-d, s) for d in range(256)]
        assert any(e[i] < e[i + 1] for i in range(255))
    rng = np.random.default_rng(11)
    L, BH, ld = 300, 4, 304
    x = rng.integers(-128, 128, (BH * L, ld), dtype=np.int8)
    x[::3] = rng.integers(60, 90, (x[::3].shape), dtype=np.int8)          # narrow rows
    x[1::7] = rng.integers(-128, -100, (x[1::7].shape), dtype=np.int8)    # rows far below 0
    v = rng.integers(-128, 128, (BH, L, 64), dtype=np.int8)
    acc = fqvit.lis_attention(torch.from_numpy(x).to(DEV), s, torch.from_numpy(v).to(DEV), 0)
    fqvit.sync_status()
    co, _ = oracle.lis_softmax(x, L, s)
    ao, ov = oracle.lis_attn_v(co, v, 0)
    assert not ov
    assert np.array_equal(np_(acc), ao)


@pytest.mark.parametrize("L", [63, 64, 65, 577])
def test_tensor_core_ignores_row_padding(L):
    """Bytes of a logit row past L (up to the row stride) are not keys: filling them with
    random values must not change anything."""
    rng = np.random.default_rng(L)
    BH = 3
    ld = (L + 15) // 16 * 16 + 32
    x = np.zeros((BH * L, ld), np.int8)
    x[:, :L] = rng.integers(-128, 128, (BH * L, L), dtype=np.int8)
    v = rng.integers(-128, 128, (BH, L, 64), dtype=np.int8)
    xg = x.copy()
    xg[:, L:] = rng.integers(-128, 128, (BH * L, ld - L), dtype=np.int8)
    for s in (0.05, 0.3):
        a0 = fqvit.lis_attention(torch.from_numpy(x).to(DEV), s, torch.from_numpy(v).to(DEV), 0)
        a1 = fqvit.lis_attention(torch.from_numpy(xg).to(DEV), s, torch.from_numpy(v).to(DEV), 0)
        fqvit.sync_status()
        co, _ = oracle.lis_softmax(x, L, s)
        ao, _ = oracle.lis_attn_v(co, v, 0)
        assert np.array_equal(np_(a0), ao) and np.array_equal(np_(a1), ao)


@pytest.mark.parametrize("zp", [-255, -7, 3, 128, 255])
def test_fused_attention_with_v_zero_point(zp, monkeypatch):
    """acc = sum_j 2^(15-code) (V - zp_V) with an asymmetric V (Eq. 15): the tensor-core
    path (P V - zp P 1) and the CUDA-core path against the oracle."""
    rng = np.random.default_rng(1000 + zp)
    for L in (49, 197, 577):
        BH = 2
        ld = (L + 15) // 16 * 16
        x = np.zeros((BH * L, ld), np.int8)
        x[:, :L] = rng.integers(-128, 128, (BH * L, L), dtype=np.int8)
        v = rng.integers(-128, 128, (BH, L, 64), dtype=np.int8)
        co, _ = oracle.lis_softmax(x, L, 0.06)
        ao, ov = oracle.lis_attn_v(co, v, zp)
        assert not ov
        acc = fqvit.lis_attention(torch.from_numpy(x).to(DEV), 0.06, torch.from_numpy(v).to(DEV), zp)
        fqvit.sync_status()
        assert np.array_equal(np_(acc), ao), (L, zp)
        monkeypatch.setenv("FQVIT_ATTN_PATH", "cuda_core")
        acc2 = fqvit.lis_attention(torch.from_numpy(x).to(DEV), 0.06, torch.from_numpy(v).to(DEV), zp)
        fqvit.sync_status()
        monkeypatch.delenv("FQVIT_ATTN_PATH")
        assert np.array_equal(np_(acc2), ao), (L, zp)
