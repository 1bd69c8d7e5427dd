"""CPU oracle for the FQ-ViT integer inference path (test infrastructure).

This package is the checker, not the product.  Only ``tests/``, the smoke
check in ``__graft_entry__`` and the CPU-baseline leg of ``bench.py`` may
import it.  It wraps ``fqvit_oracle.c`` (plain C, fp32/fp64 IEEE arithmetic,
int64 integers) through ctypes and takes / returns numpy arrays.  It shares
no code with the CUDA library.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from pathlib import Path

import numpy as np

_HERE = Path(__file__).resolve().parent
_SRC = _HERE / "fqvit_oracle.c"
_LIB = _HERE / "liboracle.so"
_CFLAGS = ["-O2", "-ffp-contract=off", "-fno-fast-math", "-fopenmp", "-fPIC",
           "-shared", "-Wall", "-Wextra"]

_lib = None


def build(force: bool = False) -> Path:
    """Compile the oracle shared object next to its source."""
    if force or not _LIB.exists() or _LIB.stat().st_mtime < _SRC.stat().st_mtime:
        tmp = _LIB.with_suffix(f".so.{os.getpid()}")
        subprocess.run(["gcc", *_CFLAGS, "-o", str(tmp), str(_SRC), "-lm"], check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is not None:
        return _lib
    build()
    _lib = _declare(ctypes.CDLL(str(_LIB)))
    return _lib


def _declare(lib):
    """Declare the C signatures on a loaded copy of the oracle (also used by the tests' planted
    mistakes, which compile altered copies of the source)."""
    P = ctypes.c_void_p
    i64, i32, f32 = ctypes.c_int64, ctypes.c_int32, ctypes.c_float
    lib.or_calibrate_ptf.argtypes = [P, i64, i32, i64, i32, P, P, P, P]
    lib.or_calibrate_ptf.restype = ctypes.c_int
    lib.or_calibrate_minmax.argtypes = [P, i64, i32, i64, P, P]
    lib.or_calibrate_minmax.restype = ctypes.c_int
    lib.or_calibrate_scale.argtypes = [f32, f32, i32, P, P, P]
    lib.or_calibrate_scale.restype = None
    lib.or_calibrate_sse.argtypes = [P, i64, i32, i64, i32, f32, f32, P]
    lib.or_calibrate_sse.restype = ctypes.c_int
    lib.or_ptf_quantize.argtypes = [P, i64, i32, i64, f32, i32, P, P, i64]
    lib.or_ptf_quantize.restype = ctypes.c_int
    lib.or_ptf_layernorm.argtypes = [P, i64, i32, i64, i32, P, P, P, f32, i32, P, i64, P, P]
    lib.or_ptf_layernorm.restype = ctypes.c_int
    lib.or_iexp_consts.argtypes = [f32, P, P, P]
    lib.or_iexp_consts.restype = None
    lib.or_iexp.argtypes = [i64, i32, i64, i64, i64]
    lib.or_iexp.restype = ctypes.c_uint64
    lib.or_ilog2.argtypes = [ctypes.c_uint64]
    lib.or_ilog2.restype = i32
    lib.or_lis_softmax.argtypes = [P, i64, i32, i64, f32, i32, P, i32, i32, P, i64, P]
    lib.or_lis_softmax_masked.restype = ctypes.c_int
    lib.or_lis_softmax_masked.argtypes = [P, i64, i32, i64, f32, i32, P, i32, i32, P, i32, i32, P, i64, P]
    lib.or_lis_softmax.restype = ctypes.c_int
    lib.or_lis_attn_v.argtypes = [P, i64, P, i64, i32, i64, i32, i32, P, i64]
    lib.or_attn_requant.restype = ctypes.c_int
    lib.or_attn_requant.argtypes = [P, i64, i32, i64, f32, f32, i32, P, i64]
    lib.or_qk_logits.restype = ctypes.c_int
    lib.or_qk_logits.argtypes = [P, i64, i32, P, i64, i32, i64, i32, i32, f32, f32, f32, i32, P, i64]
    lib.or_lis_attn_v.restype = ctypes.c_int
    lib.or_linear_q.restype = ctypes.c_int
    lib.or_linear_q.argtypes = [P, i64, i32, i64, i32, f32, P, i32, i64, P, P, f32, i32, P, i64, P, i64]
    lib.or_num_threads.argtypes = []
    lib.or_num_threads.restype = ctypes.c_int
    lib.or_set_num_threads.argtypes = [ctypes.c_int]
    lib.or_set_num_threads.restype = None
    return lib


def _ptr(a: np.ndarray | None):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    a = np.asarray(a)
    if a.dtype != dtype:
        raise TypeError(f"expected {dtype}, got {a.dtype}")
    if not a.flags.c_contiguous:
        a = np.ascontiguousarray(a)
    return a


def num_threads() -> int:
    return int(_load().or_num_threads())


def set_num_threads(n: int) -> None:
    _load().or_set_num_threads(int(n))


def calibrate_ptf(x: np.ndarray, K: int = 3):
    """Eqs. 8-10: returns (s, zp, alpha[C] uint8, sse[C, K+1] float64)."""
    x = _c(x, np.float32)
    rows, C = x.shape
    s = np.zeros(1, np.float32)
    zp = np.zeros(1, np.int32)
    alpha = np.zeros(C, np.uint8)
    sse = np.zeros((C, K + 1), np.float64)
    rc = _load().or_calibrate_ptf(_ptr(x), rows, C, C, K, _ptr(s), _ptr(zp), _ptr(alpha), _ptr(sse))
    if rc:
        raise ValueError("or_calibrate_ptf rejected its arguments")
    return float(s[0]), int(zp[0]), alpha, sse


def calibrate_minmax(x: np.ndarray):
    """Exact fp32 (min, max) over every element of x."""
    x = _c(x, np.float32)
    rows, C = x.shape
    mn = np.zeros(1, np.float32)
    mx = np.zeros(1, np.float32)
    if _load().or_calibrate_minmax(_ptr(x), rows, C, C, _ptr(mn), _ptr(mx)):
        raise ValueError("or_calibrate_minmax rejected its arguments")
    return float(mn[0]), float(mx[0])


def calibrate_scale(mn: float, mx: float, K: int = 3):
    """Eqs. 8-9 from a range: (s0 = 2^K s, s, zp)."""
    s0 = np.zeros(1, np.float32)
    s = np.zeros(1, np.float32)
    zp = np.zeros(1, np.int32)
    _load().or_calibrate_scale(mn, mx, K, _ptr(s0), _ptr(s), _ptr(zp))
    return float(s0[0]), float(s[0]), int(zp[0])


def calibrate_sse(x: np.ndarray, K: int, mn: float, mx: float) -> np.ndarray:
    """Eq. 10 over the rows of x (ascending, fp64) for the range (mn, mx): [C, K+1]."""
    x = _c(x, np.float32)
    rows, C = x.shape
    sse = np.zeros((C, K + 1), np.float64)
    if _load().or_calibrate_sse(_ptr(x), rows, C, C, K, mn, mx, _ptr(sse)):
        raise ValueError("or_calibrate_sse rejected its arguments")
    return sse


def calibrate_ptf_sharded(shards, K: int = 3):
    """Eqs. 8-10 over a calibration batch split by rows into shards (rank order).

    The range is the min / max over all shards (exact, so any split gives the
    unsplit range and hence the same s and zp).  Each shard sums its own rows
    in ascending order in fp64; the per-shard sums are then added in shard
    order, starting from 0.0, and alpha_c is the smallest factor with the
    least total.  One shard reproduces ``calibrate_ptf`` exactly.
    Returns (s, zp, alpha[C] uint8, sse[C, K+1] float64).
    """
    shards = [s for s in shards if s.shape[0] > 0]
    if not shards:
        raise ValueError("no calibration rows")
    ranges = [calibrate_minmax(x) for x in shards]
    mn = min(r[0] for r in ranges)
    mx = max(r[1] for r in ranges)
    _, s, zp = calibrate_scale(mn, mx, K)
    total = np.zeros((shards[0].shape[1], K + 1), np.float64)
    for x in shards:
        total = total + calibrate_sse(x, K, mn, mx)
    alpha = np.zeros(total.shape[0], np.uint8)
    for c in range(total.shape[0]):
        best = 0
        for a in range(1, K + 1):
            if total[c, a] < total[c, best]:
                best = a
        alpha[c] = best
    return s, zp, alpha, total


def ptf_quantize(x: np.ndarray, s: float, zp: int, alpha: np.ndarray) -> np.ndarray:
    """Eq. 7: fp32 [rows, C] -> uint8 codes."""
    x = _c(x, np.float32)
    alpha = _c(alpha, np.uint8)
    rows, C = x.shape
    out = np.zeros((rows, C), np.uint8)
    rc = _load().or_ptf_quantize(_ptr(x), rows, C, C, np.float32(s), zp, _ptr(alpha), _ptr(out), C)
    if rc:
        raise ValueError("or_ptf_quantize rejected its arguments")
    return out


def ptf_layernorm(xq, zp_in, alpha, gamma, beta, s_out, zp_out):
    """Supplement LayerNorm: returns (Y_Q uint8 [rows, C], M1 int64, M2 int64)."""
    xq = _c(xq, np.uint8)
    alpha = _c(alpha, np.uint8)
    gamma = _c(gamma, np.float32)
    beta = _c(beta, np.float32)
    rows, C = xq.shape
    y = np.zeros((rows, C), np.uint8)
    m1 = np.zeros(rows, np.int64)
    m2 = np.zeros(rows, np.int64)
    rc = _load().or_ptf_layernorm(_ptr(xq), rows, C, C, zp_in, _ptr(alpha), _ptr(gamma), _ptr(beta),
                                  np.float32(s_out), zp_out, _ptr(y), C, _ptr(m1), _ptr(m2))
    if rc:
        raise ValueError("or_ptf_layernorm rejected its arguments")
    return y, m1, m2


def iexp_consts(s: float):
    a, b, c = ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int64()
    _load().or_iexp_consts(np.float32(s), ctypes.byref(a), ctypes.byref(b), ctypes.byref(c))
    return a.value, b.value, c.value


def iexp(q: int, s: float, n: int = 15) -> int:
    """Algorithm 1 on one non-positive integer q."""
    a, b, c = iexp_consts(s)
    return int(_load().or_iexp(int(q), n, a, b, c))


def ilog2(x: int) -> int:
    """Algorithm 2's I-Log2."""
    return int(_load().or_ilog2(int(x)))


def lis_softmax(logits: np.ndarray, L: int, s: float, n: int = 15, bias=None, heads: int = 1,
                window: int = 7, region=None, mask_value: int = 0):
    """Algorithm 2 over rows of int8 logits [n_rows, >=L], with the optional relative-position
    bias [heads, (2w-1)^2] and the optional shifted-window mask (region ids [n_windows, L]:
    mask_value added where the query's and the key's regions differ).

    Returns (codes uint8 [n_rows, L], rowsum uint64 [n_rows])."""
    logits = _c(logits, np.int8)
    n_rows, ld = logits.shape
    codes = np.zeros((n_rows, L), np.uint8)
    rowsum = np.zeros(n_rows, np.uint64)
    b = None if bias is None else _c(bias, np.int8)
    reg = None if region is None else _c(region, np.uint8)
    nw = 1 if reg is None else reg.shape[0]
    rc = _load().or_lis_softmax_masked(_ptr(logits), n_rows, L, ld, np.float32(s), n, _ptr(b),
                                       heads, window, _ptr(reg), nw, int(mask_value), _ptr(codes), L,
                                       _ptr(rowsum))
    if rc:
        raise ValueError("or_lis_softmax rejected its arguments")
    return codes, rowsum


def qk_logits(q: np.ndarray, k: np.ndarray, zp_q: int, zp_k: int, s_q: float, s_k: float, s_logit: float,
              zp_l: int, ld: int | None = None) -> np.ndarray:
    """The MatMul Q K^T and its MinMax 8-bit output quantizer with the dyadic multiplier of the
    LayerNorm output stage: q, k int8 [BH, L, d] -> int8 logits [BH*L, ld] (ld >= L, zero padding)."""
    q = _c(q, np.int8)
    k = _c(k, np.int8)
    BH, L, d = q.shape
    assert k.shape == q.shape
    ld = L if ld is None else ld
    out = np.zeros((BH * L, ld), np.int8)
    rc = _load().or_qk_logits(_ptr(q), d, int(zp_q), _ptr(k), d, int(zp_k), BH, L, d, np.float32(s_q),
                              np.float32(s_k), np.float32(s_logit), int(zp_l), _ptr(out), ld)
    if rc:
        raise ValueError("or_qk_logits rejected its arguments")
    return out


def lis_attn_v(codes: np.ndarray, v: np.ndarray, zp_v: int = 0):
    """Eq. 15: codes uint8 [BH*L, L], v int8 [BH, L, d] -> int32 [BH, L, d].

    Returns (acc, overflowed)."""
    codes = _c(codes, np.uint8)
    v = _c(v, np.int8)
    BH, L, d = v.shape
    assert codes.shape[0] == BH * L and codes.shape[1] >= L
    acc = np.zeros((BH, L, d), np.int32)
    rc = _load().or_lis_attn_v(_ptr(codes), codes.shape[1], _ptr(v), d, zp_v, BH, L, d, _ptr(acc), d)
    if rc not in (0, 3):
        raise ValueError("or_lis_attn_v rejected its arguments")
    return acc, rc == 3


def attn_requant(acc: np.ndarray, s_v: float, s_out: float, zp_out: int) -> np.ndarray:
    """8-bit requantization of the attention output (Eq. 3 with the dyadic multiplier of the
    LayerNorm output stage): int32 [..., d] -> uint8 [..., d]."""
    acc = _c(acc, np.int32)
    d = acc.shape[-1]
    rows = acc.size // d
    y = np.zeros(acc.shape, np.uint8)
    rc = _load().or_attn_requant(_ptr(acc), rows, d, d, float(s_v), float(s_out), int(zp_out), _ptr(y), d)
    if rc != 0:
        raise ValueError("or_attn_requant rejected its arguments")
    return y


def linear_q(x: np.ndarray, zp_x: int, s_x: float, w: np.ndarray, s_w: np.ndarray, bias: np.ndarray | None,
             s_y: float, zp_y: int):
    """A MinMax Linear layer (Sec. 3; Sec. 4.1: symmetric channel-wise weights, asymmetric
    layer-wise activations) with its dyadic output multipliers: x uint8 [M, K], w int8 [N, K],
    s_w float32 [N], bias int32 [N] or None -> (y uint8 [M, N], acc int32 [M, N])."""
    x = _c(x, np.uint8)
    w = _c(w, np.int8)
    s_w = _c(s_w, np.float32)
    b = None if bias is None else _c(bias, np.int32)
    M, K = x.shape
    N = w.shape[0]
    assert w.shape[1] == K and s_w.shape == (N,)
    y = np.zeros((M, N), np.uint8)
    acc = np.zeros((M, N), np.int32)
    rc = _load().or_linear_q(_ptr(x), M, K, K, int(zp_x), np.float32(s_x), _ptr(w), N, K, _ptr(s_w), _ptr(b),
                             np.float32(s_y), int(zp_y), _ptr(y), N, _ptr(acc), N)
    if rc == 1:
        raise ValueError("or_linear_q rejected its arguments")
    if rc == 3:
        raise OverflowError("or_linear_q: an accumulator does not fit int32")
    return y, acc
