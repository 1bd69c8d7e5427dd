"""The C-ABI library loads, exports every symbol include/fqvit.h declares, and
rejects bad arguments on the host before launching anything (no GPU needed)."""
import ctypes
import re
from pathlib import Path

import pytest

from paper_2111_13824_gb300 import build as fbuild
from paper_2111_13824_gb300 import fqvit

HEADER = Path(__file__).resolve().parents[1] / "include" / "fqvit.h"


@pytest.fixture(scope="module")
def lib():
    fbuild.build()
    return fqvit.load()


def declared_functions():
    text = HEADER.read_text()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(fqvit_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_path():
    names = declared_functions()
    for n in ("fqvit_calibrate_ptf", "fqvit_ptf_layernorm", "fqvit_lis_softmax", "fqvit_lis_attn_v",
              "fqvit_block_int", "fqvit_lis_attention", "fqvit_ptf_quantize"):
        assert n in names


def test_exports_every_declared_symbol(lib):
    raw = ctypes.CDLL(str(fqvit.library_path()))
    for name in declared_functions():
        assert hasattr(raw, name), name
    assert set(fqvit.EXPORTS) == set(declared_functions())


def test_version(lib):
    assert lib.fqvit_version() >= 1


def test_workspace_size_alias(lib):
    # the planned interface's fqvit_workspace_size(C, K) is the calibration workspace, which does
    # not depend on the number of rows
    for C, K in ((192, 3), (1024, 3), (4096, 7), (1, 0)):
        w = lib.fqvit_workspace_size(C, K)
        assert w > 0 and all(w == lib.fqvit_calibrate_workspace_size(rows, C, K) for rows in (1, 577, 10 ** 6))
    assert lib.fqvit_workspace_size(0, 3) == 0 and lib.fqvit_workspace_size(64, 8) == 0


def _err(lib):
    return lib.fqvit_last_error().decode()


def test_null_and_shape_checks(lib):
    P = ctypes.c_void_p
    fake = P(4096)  # never dereferenced: validation fails first
    assert lib.fqvit_ptf_layernorm(None, 10, 64, 64, 0, fake, fake, fake, 0.1, 0, fake, 64, None, None, None) == 1
    assert "NULL" in _err(lib)
    assert lib.fqvit_ptf_layernorm(fake, 10, 64, 32, 0, fake, fake, fake, 0.1, 0, fake, 64, None, None, None) == 1
    assert lib.fqvit_ptf_layernorm(fake, 10, 64, 64, 300, fake, fake, fake, 0.1, 0, fake, 64, None, None, None) == 1
    assert lib.fqvit_ptf_layernorm(fake, 10, 64, 64, 0, fake, fake, fake, -1.0, 0, fake, 64, None, None, None) == 1
    assert lib.fqvit_lis_softmax(fake, 10, 2000, 2048, 0.05, 15, None, fake, 1024, None, None) == 2
    assert lib.fqvit_lis_softmax(fake, 10, 197, 197, 0.05, 15, None, fake, 100, None, None) == 1
    assert "aligned" in _err(lib)
    assert lib.fqvit_lis_softmax(fake, 10, 197, 208, 0.05, 14, None, fake, 100, None, None) == 2
    assert lib.fqvit_lis_softmax(fake, 10, 197, 208, 0.001, 15, None, fake, 100, None, None) == 2
    assert lib.fqvit_lis_softmax(fake, 10, 197, 208, 0.05, 15, None, fake, 50, None, None) == 1
    assert lib.fqvit_lis_attn_v(fake, 25, fake, 48, 0, 2, 49, 48, fake, 48, None, None) == 2
    assert lib.fqvit_lis_attn_v(fake, 25, fake, 64, 300, 2, 49, 64, fake, 64, None, None) == 2
    assert lib.fqvit_calibrate_ptf(fake, 10, 64, 64, 4, 3, fake, fake, fake, None, fake, 1 << 20, None) == 2
    assert lib.fqvit_calibrate_ptf(fake, 10, 64, 64, 8, 9, fake, fake, fake, None, fake, 1 << 20, None) == 2
    assert lib.fqvit_calibrate_ptf(fake, 10, 64, 64, 8, 3, fake, fake, fake, None, fake, 16, None) == 1
    assert "workspace" in _err(lib)
    assert lib.fqvit_block_int(None, None) == 1


def test_relpos_bias_checks(lib):
    fake = ctypes.c_void_p(4096)
    # only invalid descriptors here: a valid one would launch on the fake pointers
    bad = fqvit.RelposBias(fake, 3, 6)
    assert lib.fqvit_lis_softmax(fake, 3 * 49, 49, 64, 0.05, 15, ctypes.byref(bad), fake, 25, None, None) == 1
    b2 = fqvit.RelposBias(fake, 4, 7)
    assert lib.fqvit_lis_softmax(fake, 3 * 49, 49, 64, 0.05, 15, ctypes.byref(b2), fake, 25, None, None) == 1


def test_requantized_attention_checks(lib):
    """fqvit_lis_attention_q rejects bad output arguments before any launch."""
    fake = ctypes.c_void_p(4096)
    args = lambda s_v, s_out, zp, out, ld: lib.fqvit_lis_attention_q(  # noqa: E731
        fake, 208, 0.05, 15, None, fake, 64, 0, 2, 197, 64, s_v, s_out, zp, out, ld, None)
    assert args(0.05, 0.02, 0, None, 64) == 1
    assert "NULL" in _err(lib)
    assert args(0.05, 0.02, 0, fake, 32) == 1          # ld_out < d
    assert args(0.0, 0.02, 0, fake, 64) == 1           # s_v not positive
    assert args(0.05, float("inf"), 0, fake, 64) == 1  # s_out not finite
    assert args(0.05, 0.02, 256, fake, 64) == 1        # zp_out outside 0..255
    assert "zp_out" in _err(lib)
    assert args(1e30, 1e-30, 0, fake, 64) == 2         # M leaves the fp32 range


def test_window_mask_checks(lib):
    """The masked entry points reject a bad mask before any launch; heads come from the bias."""
    fake = ctypes.c_void_p(4096)
    b = fqvit.RelposBias(fake, 3, 7)
    soft = lambda m, rows=2 * 3 * 49: lib.fqvit_lis_softmax_masked(  # noqa: E731
        fake, rows, 49, 64, 0.05, 15, ctypes.byref(b), m, fake, 25, None, None)
    assert soft(ctypes.byref(fqvit.WindowMask(None, 2, -100))) == 1        # NULL region
    assert "mask" in _err(lib)
    assert soft(ctypes.byref(fqvit.WindowMask(fake, 0, -100))) == 1        # no windows
    assert soft(ctypes.byref(fqvit.WindowMask(fake, 2, 1))) == 2           # positive mask value
    assert soft(ctypes.byref(fqvit.WindowMask(fake, 2, -32769))) == 2      # below -32768
    assert soft(ctypes.byref(fqvit.WindowMask(fake, 4, -100))) == 1        # rows not a multiple of 3*49*4
    assert "n_windows" in _err(lib)
    att = lambda m: lib.fqvit_lis_attention_masked(  # noqa: E731
        fake, 64, 0.05, 15, ctypes.byref(b), m, fake, 32, 0, 2 * 3, 49, 32, fake, 32, None, 0, None)
    assert att(ctypes.byref(fqvit.WindowMask(None, 2, -100))) == 1
    assert att(ctypes.byref(fqvit.WindowMask(fake, 4, -100))) == 1
    assert att(ctypes.byref(fqvit.WindowMask(fake, 2, -32769))) == 2
    attq = lambda m, zp=0: lib.fqvit_lis_attention_masked_q(  # noqa: E731
        fake, 64, 0.05, 15, ctypes.byref(b), m, fake, 32, 0, 2 * 3, 49, 32, 0.05, 0.02, zp, fake, 32, None)
    assert attq(ctypes.byref(fqvit.WindowMask(fake, 4, -100))) == 1
    assert attq(ctypes.byref(fqvit.WindowMask(fake, 2, -100)), zp=300) == 1
    assert "zp_out" in _err(lib)


def test_qk_checks(lib):
    """fqvit_qk_logits / fqvit_qk_lis_attention reject bad arguments before any launch."""
    fake = ctypes.c_void_p(4096)
    f = lambda *a: lib.fqvit_qk_logits(*a)  # noqa: E731
    ok = [fake, 64, 0, fake, 64, 0, 2, 197, 64, 0.03, 0.03, 0.04, 0, fake, 208, None]
    assert f(*[None] + ok[1:]) == 1                                     # NULL q
    bad = list(ok); bad[7] = 641; bad[14] = 656
    assert f(*bad) == 2 and "L=641" in _err(lib)                        # L > 640
    bad = list(ok); bad[8] = 12; bad[1] = 12; bad[4] = 12
    assert f(*bad) == 2                                                 # d not a multiple of 8
    bad = list(ok); bad[14] = 200
    assert f(*bad) == 1                                                 # ld_logit not a multiple of 16
    bad = list(ok); bad[2] = 128
    assert f(*bad) == 1 and "zero points" in _err(lib)                  # zp_q outside -128..127
    bad = list(ok); bad[11] = 0.0
    assert f(*bad) == 1                                                 # s_logit not positive
    bad = list(ok); bad[9] = 1e30; bad[10] = 1e30; bad[11] = 1e-30
    assert f(*bad) == 2                                                 # M leaves the fp32 range
    assert lib.fqvit_qk_workspace_size(4, 49, 3) == 3 * 49 * 64
    assert lib.fqvit_qk_workspace_size(0, 49, 3) == 0
    # the library's choice: every head in one group, up to 1 GiB of logits
    assert lib.fqvit_qk_workspace_size(512, 577, 0) == 512 * 577 * 592
    assert lib.fqvit_qk_workspace_size(10 ** 6, 577, 0) <= 1 << 30
    g = lambda ws_bytes, v=fake: lib.fqvit_qk_lis_attention(  # noqa: E731
        fake, 64, 0, fake, 64, 0, 0.03, 0.03, 0.04, 0, 15, None, None, v, 64, 0, 4, 197, 64, fake, 64, fake,
        ws_bytes, 0, None)
    assert g(197 * 208 - 1) == 1 and "workspace" in _err(lib)          # less than one head
    assert g(10 ** 8, v=None) == 1                                      # NULL V


def test_linear_checks(lib):
    """fqvit_linear_q / fqvit_linear_pack_weight reject bad arguments before any launch."""
    fake = ctypes.c_void_p(4096)
    M, K, N = 300, 384, 1152
    ws = lib.fqvit_linear_workspace_size(M, K)
    # the fp16 copy of x, rounded up to 256 bytes, then 4096 int32 weight sums
    assert ws == (M * K * 2 + 255) // 256 * 256 + 4 * 4096 and lib.fqvit_linear_workspace_size(0, K) == 0
    f = lambda *a: lib.fqvit_linear_q(*a)  # noqa: E731
    ok = [fake, M, K, K, 128, 0.04, fake, N, fake, None, 0.03, 120, fake, N, None, 0, fake, ws, None]
    assert f(*[None] + ok[1:]) == 1                                     # NULL x
    bad = list(ok); bad[8] = None
    assert f(*bad) == 1                                                 # NULL s_w
    bad = list(ok); bad[2] = 100; bad[3] = 100
    assert f(*bad) == 2 and "K=100" in _err(lib)                        # K not a multiple of 8
    bad = list(ok); bad[7] = 1160; bad[13] = 1168
    assert f(*bad) == 2                                                 # N not a multiple of 16
    bad = list(ok); bad[7] = 4112; bad[13] = 4112
    assert f(*bad) == 2                                                 # N > 4096
    bad = list(ok); bad[2] = 16392; bad[3] = 16392
    assert f(*bad) == 2                                                 # K > 16384
    bad = list(ok); bad[4] = 256
    assert f(*bad) == 1 and "zero points" in _err(lib)                  # zp_x outside 0..255
    bad = list(ok); bad[10] = float("inf")
    assert f(*bad) == 1                                                 # s_y not finite
    bad = list(ok); bad[13] = N + 8
    assert f(*bad) == 1                                                 # ld_y not a multiple of 16
    bad = list(ok); bad[3] = K + 4
    assert f(*bad) == 1                                                 # ld_x not a multiple of 8
    bad = list(ok); bad[14] = fake; bad[15] = N - 4
    assert f(*bad) == 1                                                 # ld_acc below N
    bad = list(ok); bad[17] = ws - 1
    assert f(*bad) == 1 and "workspace" in _err(lib)                    # small workspace
    p = lambda *a: lib.fqvit_linear_pack_weight(*a)  # noqa: E731
    assert p(None, N, K, K, fake, None) == 1
    assert p(fake, N, 100, 100, fake, None) == 2
    assert p(fake, N, K, K, ctypes.c_void_p(4104), None) == 1           # w_h not 16-byte aligned
