"""Planted mistakes in the oracle, on the CPU.

Each mutant is a copy of the oracle's C source with one plausible mistake planted in one
function: a dropped term, a wrong sign, a wrong index or operand, a missing rounding half, an
exponent off by one, a truncation turned into a rounding up.  The copy is compiled into a
temporary library.  The pins of that function (the tests of ``test_oracle_linear.py`` or
``test_oracle_qk.py``, every parametrization) then run against it, and at least one must fail.
The oracle itself is never altered; the harness is first checked to pass every pin on it.
Every mutant keeps its indexes in bounds.
"""
import ctypes
import importlib.util
import itertools
import subprocess
from pathlib import Path

import pytest

import oracle

ROOT = Path(__file__).resolve().parents[1]
SRC = ROOT / "oracle" / "fqvit_oracle.c"

# (pin module, oracle function, planted text replaced, by, the mistake)
MUTANTS = [
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


def _failing_pins(mod):
    failed = []
    for label, fn, kw in _pin_calls(mod):
        try:
            fn(**kw)
        except (AssertionError, ValueError, OverflowError, pytest.fail.Exception):
            failed.append(label)
    return failed


def _mutant_lib(tmp, function, old, new):
    text = SRC.read_text()
    start = text.index(f"OR_EXPORT int {function}(")
    end = text.find("\nOR_EXPORT", start + 1)
    end = len(text) if end < 0 else end
    body = text[start:end]
    assert body.count(old) == 1, (function, old)
    src = tmp / "mutant.c"
    src.write_text(text[:start] + body.replace(old, new) + text[end:])
    lib = tmp / "libmutant.so"
    subprocess.run(["gcc", *oracle._CFLAGS, "-o", str(lib), str(src), "-lm"], check=True, capture_output=True)
    return oracle._declare(ctypes.CDLL(str(lib)))


@pytest.mark.parametrize("pins", ["test_oracle_linear", "test_oracle_qk"])
def test_every_pin_passes_on_the_oracle(pins):
    oracle.build()
    assert _failing_pins(_module(pins)) == []


@pytest.mark.parametrize("pins,function,old,new,why", MUTANTS, ids=[f"{m[1]}: {m[4]}" for m in MUTANTS])
def test_planted_mistake_fails_a_pin(tmp_path, monkeypatch, pins, function, old, new, why):
    monkeypatch.setattr(oracle, "_lib", _mutant_lib(tmp_path, function, old, new))
    assert _failing_pins(_module(pins)), f"no pin of {pins} fails with the planted mistake: {why}"
