"""Planted mistakes in the oracle, on the CPU.

Each mutant is a copy of the oracle's C source with one plausible mistake planted in one
function: a dropped term, a wrong sign, a wrong index or operand, a missing rounding half, an
exponent off by one, a truncation turned into a rounding up.  The copy is compiled into a
temporary library.  The pins of that function (the tests of the ``test_oracle_*.py`` module
that pins it, every parametrization) then run against it, and at least one must fail.
The oracle itself is never altered; the harness is first checked to pass every pin on it.
Every mutant keeps its indexes in bounds and defines every shift and division (none may
crash the test process).
"""
import ctypes
import importlib.util
import itertools
import re
import subprocess
from pathlib import Path

import pytest

import oracle

ROOT = Path(__file__).resolve().parents[1]
SRC = ROOT / "oracle" / "fqvit_oracle.c"

PINS = "test_oracle_pins"
LIS_PINS = ("test_oracle_pins", "test_oracle_mask")

# (pin module(s), oracle function, planted text replaced, by, the mistake)
MUTANTS = [
    # PTF calibration and quantizer (Eqs. 7-10)
    (PINS, "or_calibrate_scale", "float t = -mn / s0;", "float t = mn / s0;", "zero point of the wrong sign"),
    (PINS, "or_calibrate_scale", "*s_out = ldexpf(s0, -K);", "*s_out = ldexpf(s0, K);", "2^K multiplied, not divided"),
    (PINS, "or_calibrate_sse", "q = clamp_f32(q, (float)(-zp), (float)(255 - zp));", "(void)zp;",
     "Eq. 10 without the quantizer's clip"),
    (PINS, "or_calibrate_sse", "float sa = ldexpf(s0, a - K);", "float sa = ldexpf(s0, a);", "factor 2^a on s0, not s"),
    (PINS, "or_calibrate_sse", "err += (double)d * (double)d;", "err += fabs((double)d);", "absolute, not squared error"),
    (PINS, "or_calibrate_ptf", "if (e[a] < e[best_a]) best_a = a;", "if (e[a] <= e[best_a]) best_a = a;",
     "ties to the largest factor"),
    (PINS, "or_calibrate_minmax", "float mn = x[0], mx = x[0];", "float mn = 0.0f, mx = x[0];",
     "minimum started at zero"),
    (PINS, "or_calibrate_minmax", "for (int64_t r = 0; r < rows; ++r)", "for (int64_t r = 1; r < rows; ++r)",
     "first row skipped"),
    (PINS, "or_ptf_quantize", "float q = rintf(x[r * ld_x + c] / sa);", "float q = truncf(x[r * ld_x + c] / sa);",
     "codes truncated, not rounded"),
    (PINS, "or_ptf_quantize", "float sa = ldexpf(s, alpha[c]);", "float sa = s;", "factor ignored"),
    (PINS, "or_ptf_quantize", "xq[r * ld_q + c] = (uint8_t)((int32_t)q + zp);", "xq[r * ld_q + c] = (uint8_t)((int32_t)q);",
     "zero point dropped"),
    # integer LayerNorm (Eqs. 11-13, the supplement's LayerNorm)
    (PINS, "or_ptf_layernorm", "M2 += xh * xh;", "M2 += xh;", "second moment not squared"),
    (PINS, "or_ptf_layernorm", "int64_t D = (int64_t)C * M2 - M1 * M1;", "int64_t D = (int64_t)C * M2 - M1;",
     "mean not squared in D"),
    (PINS, "or_ptf_layernorm", "tf = (float)M1 / sd;", "tf = 0.0f;", "mean dropped"),
    (PINS, "or_ptf_layernorm", "float B = bs - gt;", "float B = bs + gt;", "sign of the mean term"),
    (PINS, "or_ptf_layernorm", "if (A < 0.0f) sgn = -1;", "(void)sgn;", "sign of A lost"),
    (PINS, "or_ptf_layernorm", "N1 = 7 - ilogbf(A);", "N1 = 6 - ilogbf(A);", "N1 one too small (7-bit N2)"),
    (PINS, "or_ptf_layernorm", "N1 = 7 - ilogbf(A);", "N1 = 8 - ilogbf(A);", "N1 one too large (9-bit N2)"),
    (PINS, "or_ptf_layernorm", "R = floor_div_pow2(num + ((int64_t)1 << (N1 - 1)), N1);",
     "R = floor_div_pow2(num, N1);", "no half in the rounding"),
    (PINS, "or_ptf_layernorm", "int64_t xh = ((int64_t)xr[c] - zp_in) * ((int64_t)1 << alpha[c]);\n            float gs",
     "int64_t xh = ((int64_t)xr[c] - zp_in);\n            float gs", "PTF shift missing in the output"),
    (PINS, "or_ptf_layernorm", "clamp_i64(R + zp_out, 0, 255)", "clamp_i64(R - zp_out, 0, 255)",
     "output zero point subtracted"),
    (PINS, "or_ptf_layernorm", "float bqf = clamp_f32(rintf(bsc),", "float bqf = clamp_f32(floorf(bsc),",
     "B 2^N1 floored, not rounded"),
    # i-exp (Algorithm 1) and I-Log2 (Algorithm 2)
    (PINS, "or_iexp_consts", "*q_ln2 = (int64_t)floor(-OR_LN2 / sd);", "*q_ln2 = (int64_t)ceil(-OR_LN2 / sd);",
     "q_ln2 rounded up"),
    (PINS, "or_iexp_consts", "*q_b = (int64_t)floor(1.353 / sd);", "*q_b = (int64_t)ceil(1.353 / sd);",
     "q_b rounded up"),
    (PINS, "or_iexp_consts", "*q_c = (int64_t)floor(0.344 / (0.3585 * (sd * sd)));",
     "*q_c = (int64_t)floor(0.344 / (0.3585 * sd));", "q_c over s, not s^2"),
    (PINS, "or_iexp", "int64_t qL = (qp + q_b) * (qp + q_b) + q_c;", "int64_t qL = (q + q_b) * (q + q_b) + q_c;",
     "the listing's (q + q_b) read literally"),
    (PINS, "or_iexp", "return (uint64_t)qL << (n - z);", "return (uint64_t)qL << (n - z + 1);",
     "output scale doubled"),
    (PINS, "or_ilog2", "int32_t chi = (M >= 1) ? (int32_t)((x >> (M - 1)) & 1u) : 0;", "int32_t chi = 0;",
     "the rounding bit dropped (floor of log2)"),
    (PINS, "or_ilog2", "int32_t chi = (M >= 1) ? (int32_t)((x >> (M - 1)) & 1u) : 0;",
     "int32_t chi = (M >= 2) ? (int32_t)((x >> (M - 2)) & 1u) : 0;", "the second bit taken for the first"),
    # Log-Int-Softmax (Algorithm 2, Eqs. 16-17, 33) with the bias and the mask
    (LIS_PINS, "or_lis_softmax_masked", "uint64_t qrev = (2 * S + ev[j]) / (2 * ev[j]);",
     "uint64_t qrev = S / ev[j];", "reciprocal truncated, not rounded"),
    (LIS_PINS, "or_lis_softmax_masked", "if (code > 15) code = 15;", "if (code > 14) code = 14;", "clip at 14"),
    (LIS_PINS, "or_lis_softmax_masked", "S += ev[j];", "if (j + 1 < L) S += ev[j];", "last key left out of the sum"),
    (LIS_PINS, "or_lis_softmax_masked", "ev[j] = or_iexp((int64_t)qv[j] - m, n, q_ln2, q_b, q_c);",
     "ev[j] = or_iexp((int64_t)qv[j] - m - 1, n, q_ln2, q_b, q_c);", "maximum off by one"),
    (LIS_PINS, "or_lis_softmax_masked", "relpos_index(i, j, window)", "relpos_index(j, i, window)",
     "bias index transposed"),
    (LIS_PINS, "or_lis_softmax_masked", "int32_t h = bias ? (int32_t)((r / L) % heads) : 0;",
     "int32_t h = bias ? (int32_t)(r % heads) : 0;", "head of a row taken from the query index"),
    (LIS_PINS, "or_lis_softmax_masked", "if (reg && reg[i] != reg[j]) q += mask_value;",
     "if (reg && reg[i] == reg[j]) q += mask_value;", "mask on equal regions"),
    (LIS_PINS, "or_lis_softmax_masked", "% n_windows) * L : NULL;", "% n_windows) * 0 : NULL;",
     "every row takes the first window"),
    # BitShift attention V (Eq. 15)
    (PINS, "or_lis_attn_v", "int64_t w = (int64_t)1 << (15 - crow[j]);", "int64_t w = (int64_t)1 << crow[j];",
     "shift by the code, not 15 - code"),
    (PINS, "or_lis_attn_v", "a[t] += ((int64_t)vh[(int64_t)j * ld_v + t] - zp_v) * w;",
     "a[t] += ((int64_t)vh[(int64_t)t * 0 + j] - zp_v) * w;", "V read along the wrong axis"),
    (PINS, "or_lis_attn_v", "a[t] += ((int64_t)vh[(int64_t)j * ld_v + t] - zp_v) * w;",
     "a[t] += ((int64_t)vh[(int64_t)j * ld_v + t]) * w;", "V zero point dropped"),
    # 8-bit attention output (Eq. 3 with the dyadic multiplier)
    ("test_oracle_requant", "or_attn_requant", "const float M = ldexpf(s_v / s_out, -15);",
     "const float M = ldexpf(s_v / s_out, -14);", "2^15 of the BitShift scale off by one"),
    ("test_oracle_requant", "or_attn_requant", "R = floor_div_pow2(num + ((int64_t)1 << (N1 - 1)), N1);",
     "R = floor_div_pow2(num, N1);", "no half in the rounding"),
    ("test_oracle_requant", "or_attn_requant", "int N1 = 7 - ilogbf(M);", "int N1 = 6 - ilogbf(M);",
     "N1 one too small (7-bit N2)"),
    ("test_oracle_requant", "or_attn_requant", "int N1 = 7 - ilogbf(M);", "int N1 = 8 - ilogbf(M);",
     "N1 one too large (9-bit N2)"),
    # MinMax Linear layer and Q K^T
    ("test_oracle_linear", "or_linear_q", "((int64_t)xm[k] - zp_x)", "((int64_t)xm[k])",
     "activation zero point dropped"),
    ("test_oracle_linear", "or_linear_q", "(int64_t)wn[k]", "(int64_t)wn[K - 1 - k]", "weight index reversed"),
    ("test_oracle_linear", "or_linear_q", "const uint8_t *xm = x + m * ld_x;",
     "const uint8_t *xm = x + (M - 1 - m) * ld_x;", "activation row reversed"),
    ("test_oracle_linear", "or_linear_q", "if (bias) s += bias[n];", "(void)bias;", "bias dropped"),
    ("test_oracle_linear", "or_linear_q", "const float a = s_x * s_w[n];", "const float a = s_x;",
     "channel scale dropped"),
    ("test_oracle_linear", "or_linear_q", "const float Mn = a / s_y;", "const float Mn = s_y / a;",
     "multiplier inverted"),
    ("test_oracle_linear", "or_linear_q", "num + ((int64_t)1 << (n1[n] - 1))", "num", "no half in the rounding"),
    ("test_oracle_linear", "or_linear_q", "int e = 7 - ilogbf(Mn);", "int e = 6 - ilogbf(Mn);",
     "N1 one too small (7-bit N2)"),
    ("test_oracle_linear", "or_linear_q", "int e = 7 - ilogbf(Mn);", "int e = 8 - ilogbf(Mn);",
     "N1 one too large (9-bit N2)"),
    ("test_oracle_linear", "or_linear_q", "if (e > 31) e = 31;", "if (e > 30) e = 30;", "shift cap at 30"),
    ("test_oracle_linear", "or_linear_q", "floorf(ldexpf(Mn, e))", "ceilf(ldexpf(Mn, e))", "N2 rounded up"),
    ("test_oracle_linear", "or_linear_q", "R = num * ((int64_t)1 << sh);", "R = num;",
     "N1 <= 0 branch without its power of two"),
    ("test_oracle_linear", "or_linear_q", "clamp_i64(R + zp_y, 0, 255)", "clamp_i64(R - zp_y, 0, 255)",
     "output zero point subtracted"),
    ("test_oracle_qk", "or_qk_logits", "((int64_t)qi[t] - zp_q)", "((int64_t)qi[t])", "query zero point dropped"),
    ("test_oracle_qk", "or_qk_logits", "const int8_t *kj = k + (bh * L + j) * ld_k;",
     "const int8_t *kj = k + (bh * L + i) * ld_k;", "key indexed by the query"),
    ("test_oracle_qk", "or_qk_logits", "P += ((int64_t)qi[t] - zp_q) * ((int64_t)kj[t] - zp_k);",
     "P += ((int64_t)(q + (bh * L + j) * ld_q)[t] - zp_q) * ((int64_t)(k + (bh * L + i) * ld_k)[t] - zp_k);",
     "product transposed"),
    ("test_oracle_qk", "or_qk_logits", "num + ((int64_t)1 << (N1 - 1))", "num", "no half in the rounding"),
    ("test_oracle_qk", "or_qk_logits", "int N1 = 7 - ilogbf(M);", "int N1 = 6 - ilogbf(M);",
     "N1 one too small (7-bit N2)"),
    ("test_oracle_qk", "or_qk_logits", "int N1 = 7 - ilogbf(M);", "int N1 = 8 - ilogbf(M);",
     "N1 one too large (9-bit N2)"),
    ("test_oracle_qk", "or_qk_logits", "const float c = r * s_logit;", "const float c = s_logit;",
     "1/sqrt(d) dropped"),
    ("test_oracle_qk", "or_qk_logits", "clamp_i64(R + zp_l, -128, 127)", "clamp_i64(R, -128, 127)",
     "output zero point dropped"),
]


def _module(name):
    spec = importlib.util.spec_from_file_location(f"_pins_{name}", Path(__file__).parent / f"{name}.py")
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _pin_calls(mod):
    """Every test function of a pin module with every combination of its parametrizations."""
    for name in sorted(dir(mod)):
        if not name.startswith("test_"):
            continue
        fn = getattr(mod, name)
        grids = []
        for mark in getattr(fn, "pytestmark", []):
            if mark.name != "parametrize":
                continue
            names, values = mark.args[0], mark.args[1]
            names = [n.strip() for n in names.split(",")] if isinstance(names, str) else list(names)
            grids.append([dict(zip(names, v if len(names) > 1 else (v,))) for v in values])
        for combo in itertools.product(*grids):
            kw = {}
            for d in combo:
                kw.update(d)
            yield f"{name}{kw or ''}", fn, kw


def _failing_pins(mods):
    failed = []
    for label, fn, kw in (c for m in mods for c in _pin_calls(m)):
        try:
            fn(**kw)
        except (AssertionError, ValueError, OverflowError, pytest.fail.Exception):
            failed.append(label)
    return failed


def _mutant_lib(tmp, function, old, new):
    text = SRC.read_text()
    start = re.search(rf"OR_EXPORT \w+ {function}\(", text).start()
    end = text.find("\nOR_EXPORT", start + 1)
    end = len(text) if end < 0 else end
    body = text[start:end]
    assert body.count(old) == 1, (function, old)
    src = tmp / "mutant.c"
    src.write_text(text[:start] + body.replace(old, new) + text[end:])
    lib = tmp / "libmutant.so"
    subprocess.run(["gcc", *oracle._CFLAGS, "-o", str(lib), str(src), "-lm"], check=True, capture_output=True)
    return oracle._declare(ctypes.CDLL(str(lib)))


def _modules(pins):
    return [_module(p) for p in ((pins,) if isinstance(pins, str) else pins)]


@pytest.mark.parametrize("pins", ["test_oracle_pins", "test_oracle_mask", "test_oracle_requant",
                                  "test_oracle_linear", "test_oracle_qk"])
def test_every_pin_passes_on_the_oracle(pins):
    oracle.build()
    assert _failing_pins(_modules(pins)) == []


@pytest.mark.parametrize("pins,function,old,new,why", MUTANTS, ids=[f"{m[1]}: {m[4]}" for m in MUTANTS])
def test_planted_mistake_fails_a_pin(tmp_path, monkeypatch, pins, function, old, new, why):
    monkeypatch.setattr(oracle, "_lib", _mutant_lib(tmp_path, function, old, new))
    assert _failing_pins(_modules(pins)), f"no pin of {pins} fails with the planted mistake: {why}"
