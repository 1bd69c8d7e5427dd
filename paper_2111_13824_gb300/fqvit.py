"""Thin Python binding of libfqvit.so (include/fqvit.h).

Argument marshalling only: every function passes torch tensors' device
pointers and the current CUDA stream to the C ABI of the same name and
raises ``FqvitError`` on a non-OK status.  There is no fallback: if the
library is missing or was not built, loading fails loudly.
"""
from __future__ import annotations

import ctypes
from pathlib import Path

import torch

_LIB_PATH = Path(__file__).resolve().parent / "libfqvit.so"
_lib = None

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_RANGE, ERR_CUDA, ERR_TIMEOUT = 0, 1, 2, 3, 4, 5


class FqvitError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"fqvit error {code}: {msg}")
        self.code = code


class RelposBias(ctypes.Structure):
    _fields_ = [("table", ctypes.c_void_p), ("heads", ctypes.c_int32), ("window", ctypes.c_int32)]


class WindowMask(ctypes.Structure):
    _fields_ = [("region", ctypes.c_void_p), ("n_windows", ctypes.c_int32), ("mask_value", ctypes.c_int32)]


class BlockDesc(ctypes.Structure):
    _fields_ = [
        ("xq", ctypes.c_void_p), ("rows", ctypes.c_int64), ("C", ctypes.c_int32), ("zp_in", ctypes.c_int32),
        ("alpha", ctypes.c_void_p), ("gamma", ctypes.c_void_p), ("beta", ctypes.c_void_p),
        ("s_out", ctypes.c_float), ("zp_out", ctypes.c_int32), ("yq", ctypes.c_void_p),
        ("logits", ctypes.c_void_p), ("ld_logit", ctypes.c_int64), ("s_logit", ctypes.c_float),
        ("v", ctypes.c_void_p), ("zp_v", ctypes.c_int32), ("BH", ctypes.c_int64), ("L", ctypes.c_int32),
        ("d", ctypes.c_int32), ("bias", ctypes.c_void_p), ("acc", ctypes.c_void_p),
    ]


EXPORTS = (
    "fqvit_version", "fqvit_last_error", "fqvit_calibrate_workspace_size", "fqvit_workspace_size",
    "fqvit_calibrate_ptf",
    "fqvit_ptf_quantize", "fqvit_ptf_layernorm", "fqvit_lis_softmax", "fqvit_lis_attn_v",
    "fqvit_lis_attention", "fqvit_lis_attention_q", "fqvit_block_int", "fqvit_sync_status",
    "fqvit_calibrate_ptf_noalloc",
    "fqvit_calibrate_minmax", "fqvit_calibrate_sse_partial", "fqvit_calibrate_combine",
    "fqvit_lis_softmax_masked", "fqvit_lis_attention_masked", "fqvit_lis_attention_masked_q",
    "fqvit_qk_logits", "fqvit_qk_workspace_size", "fqvit_qk_lis_attention",
    "fqvit_linear_pack_weight", "fqvit_linear_workspace_size", "fqvit_linear_q",
    "fqvit_split_qkv", "fqvit_merge_heads",
    "fqvit_selftest_bounded_wait",
)


def library_path() -> Path:
    return _LIB_PATH


def load(path: str | Path | None = None):
    """Load libfqvit.so and declare its signatures (raises if it is missing)."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = Path(path) if path else _LIB_PATH
    if not p.exists():
        raise FileNotFoundError(f"{p} is missing: build it with paper_2111_13824_gb300.build.build()")
    lib = ctypes.CDLL(str(p))
    P, i64, i32, f32, sz = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_float, ctypes.c_size_t
    sig = {
        "fqvit_version": ([], ctypes.c_int),
        "fqvit_last_error": ([], ctypes.c_char_p),
        "fqvit_calibrate_workspace_size": ([i64, i32, i32], sz),
        "fqvit_workspace_size": ([i32, i32], sz),
        "fqvit_calibrate_ptf": ([P, i64, i32, i64, i32, i32, P, P, P, P, P, sz, P], ctypes.c_int),
        "fqvit_ptf_quantize": ([P, i64, i32, i64, f32, i32, P, P, i64, P], ctypes.c_int),
        "fqvit_ptf_layernorm": ([P, i64, i32, i64, i32, P, P, P, f32, i32, P, i64, P, P, P], ctypes.c_int),
        "fqvit_lis_softmax": ([P, i64, i32, i64, f32, i32, P, P, i64, P, P], ctypes.c_int),
        "fqvit_lis_attn_v": ([P, i64, P, i64, i32, i64, i32, i32, P, i64, P, P], ctypes.c_int),
        "fqvit_lis_attention_q": ([P, i64, f32, i32, P, P, i64, i32, i64, i32, i32, f32, f32, i32, P, i64, P],
                                  ctypes.c_int),
        "fqvit_lis_attention": ([P, i64, f32, i32, P, P, i64, i32, i64, i32, i32, P, i64, P, i64, P],
                                ctypes.c_int),
        "fqvit_lis_softmax_masked": ([P, i64, i32, i64, f32, i32, P, P, P, i64, P, P], ctypes.c_int),
        "fqvit_lis_attention_masked": ([P, i64, f32, i32, P, P, P, i64, i32, i64, i32, i32, P, i64, P, i64, P],
                                       ctypes.c_int),
        "fqvit_lis_attention_masked_q": ([P, i64, f32, i32, P, P, P, i64, i32, i64, i32, i32, f32, f32, i32, P,
                                          i64, P], ctypes.c_int),
        "fqvit_qk_logits": ([P, i64, i32, P, i64, i32, i64, i32, i32, f32, f32, f32, i32, P, i64, P], ctypes.c_int),
        "fqvit_qk_workspace_size": ([i64, i32, i64], sz),
        "fqvit_qk_lis_attention": ([P, i64, i32, P, i64, i32, f32, f32, f32, i32, i32, P, P, P, i64, i32, i64, i32,
                                    i32, P, i64, P, sz, i64, P], ctypes.c_int),
        "fqvit_selftest_bounded_wait": ([P], ctypes.c_int),
        "fqvit_linear_pack_weight": ([P, i32, i32, i64, P, P], ctypes.c_int),
        "fqvit_linear_workspace_size": ([i64, i32], sz),
        "fqvit_linear_q": ([P, i64, i32, i64, i32, f32, P, i32, P, P, f32, i32, P, i64, P, i64, P, sz, P],
                           ctypes.c_int),
        "fqvit_block_int": ([P, P], ctypes.c_int),
        "fqvit_split_qkv": ([P, i64, i32, i32, i32, i64, P, P, P, i64, P], ctypes.c_int),
        "fqvit_merge_heads": ([P, i64, i32, i32, i32, i64, P, i64, P], ctypes.c_int),
        "fqvit_sync_status": ([P], ctypes.c_int),
        "fqvit_calibrate_ptf_noalloc": ([P, i64, i32, i64, i32, i32, P, P, P, P, P], ctypes.c_int),
        "fqvit_calibrate_minmax": ([P, i64, i32, i64, P, P, sz, P], ctypes.c_int),
        "fqvit_calibrate_sse_partial": ([P, i64, i32, i64, i32, i32, P, P, P, sz, P], ctypes.c_int),
        "fqvit_calibrate_combine": ([P, i32, i32, i32, f32, f32, P, P, P, P], ctypes.c_int),
    }
    for name, (args, res) in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    if path is None:
        _lib = lib
    return lib


def _check(rc: int):
    if rc != OK:
        raise FqvitError(rc, load().fqvit_last_error().decode())


def _p(t):
    if t is None:
        return None
    if not isinstance(t, torch.Tensor):
        raise TypeError("expected a torch.Tensor")
    if not t.is_cuda:
        raise ValueError("libfqvit takes device tensors (got a CPU tensor)")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _ld(t: torch.Tensor) -> int:
    return t.stride(0) if t.dim() >= 2 else t.shape[-1]


def _bias(bias, heads, window):
    if bias is None:
        return None
    b = RelposBias(ctypes.c_void_p(bias.data_ptr()), heads, window)
    return b


def sync_status(stream=None) -> None:
    """Synchronize the stream; raise FqvitError if a kernel abandoned a bounded wait."""
    _check(load().fqvit_sync_status(_stream(stream)))


def selftest_bounded_wait(stream=None) -> None:
    """One CTA waits on a barrier nothing completes (fqvit_selftest_bounded_wait); the next
    sync_status raises FqvitError with ERR_TIMEOUT."""
    _check(load().fqvit_selftest_bounded_wait(_stream(stream)))


def version() -> int:
    return int(load().fqvit_version())


def calibrate_workspace_size(rows: int, C: int, K: int) -> int:
    return int(load().fqvit_calibrate_workspace_size(rows, C, K))


def calibrate_ptf(x: torch.Tensor, K: int = 3, bits: int = 8, sse: torch.Tensor | None = None,
                  workspace: torch.Tensor | None = None, stream=None):
    """Eqs. 8-10 on the device; returns device tensors (s[1] f32, zp[1] i32, alpha[C] u8)."""
    rows, C = x.shape
    dev = x.device
    s = torch.empty(1, dtype=torch.float32, device=dev)
    zp = torch.empty(1, dtype=torch.int32, device=dev)
    alpha = torch.empty(C, dtype=torch.uint8, device=dev)
    nbytes = calibrate_workspace_size(rows, C, K)
    if workspace is None:
        workspace = torch.empty(max(nbytes, 8) // 8 + 1, dtype=torch.float64, device=dev)
    _check(load().fqvit_calibrate_ptf(_p(x), rows, C, _ld(x), bits, K, _p(s), _p(zp), _p(alpha), _p(sse),
                                      _p(workspace), workspace.numel() * workspace.element_size(),
                                      _stream(stream)))
    return s, zp, alpha


def calibrate_ptf_noalloc(x: torch.Tensor, K: int = 3, bits: int = 8, sse: torch.Tensor | None = None,
                          stream=None):
    """fqvit_calibrate_ptf_noalloc: calibration with the library's fixed scratch (no workspace)."""
    rows, C = x.shape
    dev = x.device
    s = torch.empty(1, dtype=torch.float32, device=dev)
    zp = torch.empty(1, dtype=torch.int32, device=dev)
    alpha = torch.empty(C, dtype=torch.uint8, device=dev)
    _check(load().fqvit_calibrate_ptf_noalloc(_p(x), rows, C, _ld(x), bits, K, _p(s), _p(zp), _p(alpha), _p(sse),
                                              _stream(stream)))
    return s, zp, alpha


def _workspace(rows: int, C: int, K: int, dev) -> torch.Tensor:
    nbytes = calibrate_workspace_size(rows, C, K)
    return torch.empty(max(nbytes, 64) // 8 + 1, dtype=torch.float64, device=dev)


def calibrate_minmax(x: torch.Tensor, workspace: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """Stage 1 of sharded calibration: device float32[2] = (min, max) of x."""
    rows, C = x.shape
    mnmx = torch.empty(2, dtype=torch.float32, device=x.device)
    if workspace is None:
        workspace = _workspace(rows, C, 0, x.device)
    _check(load().fqvit_calibrate_minmax(_p(x), rows, C, _ld(x), _p(mnmx), _p(workspace),
                                         workspace.numel() * workspace.element_size(), _stream(stream)))
    return mnmx


def calibrate_sse_partial(x: torch.Tensor, K: int, mnmx: torch.Tensor, bits: int = 8,
                          sse: torch.Tensor | None = None, workspace: torch.Tensor | None = None,
                          stream=None) -> torch.Tensor:
    """Stage 2: device float64[C, K+1] of Eq. 10 over the rows of x for the global range mnmx."""
    rows, C = x.shape
    if sse is None:
        sse = torch.empty(C, K + 1, dtype=torch.float64, device=x.device)
    if workspace is None:
        workspace = _workspace(rows, C, 0, x.device)
    _check(load().fqvit_calibrate_sse_partial(_p(x), rows, C, _ld(x), bits, K, _p(mnmx), _p(sse), _p(workspace),
                                              workspace.numel() * workspace.element_size(), _stream(stream)))
    return sse


def calibrate_combine(sse_parts: torch.Tensor, mn: float, mx: float, K: int):
    """Stage 3 (host, no GPU): sse_parts float64 [world, C, K+1] on the CPU, in rank order.

    Returns (s float, zp int, alpha uint8[C] CPU tensor, sse_total float64 [C, K+1] CPU tensor).
    """
    if sse_parts.device.type != "cpu" or sse_parts.dtype != torch.float64 or sse_parts.dim() != 3:
        raise ValueError("sse_parts must be a CPU float64 tensor [world, C, K+1]")
    parts = sse_parts.contiguous()
    world, C, k1 = parts.shape
    if k1 != K + 1:
        raise ValueError("sse_parts has the wrong factor count")
    s = ctypes.c_float()
    zp = ctypes.c_int32()
    alpha = torch.empty(C, dtype=torch.uint8)
    total = torch.empty(C, K + 1, dtype=torch.float64)
    _check(load().fqvit_calibrate_combine(ctypes.c_void_p(parts.data_ptr()), world, C, K, float(mn), float(mx),
                                          ctypes.byref(s), ctypes.byref(zp), ctypes.c_void_p(alpha.data_ptr()),
                                          ctypes.c_void_p(total.data_ptr())))
    return float(s.value), int(zp.value), alpha, total


def ptf_quantize(x: torch.Tensor, s: float, zp: int, alpha: torch.Tensor, out: torch.Tensor | None = None,
                 stream=None) -> torch.Tensor:
    rows, C = x.shape
    if out is None:
        out = torch.empty(rows, C, dtype=torch.uint8, device=x.device)
    _check(load().fqvit_ptf_quantize(_p(x), rows, C, _ld(x), float(s), int(zp), _p(alpha), _p(out), _ld(out),
                                     _stream(stream)))
    return out


def ptf_layernorm(xq: torch.Tensor, zp_in: int, alpha, gamma, beta, s_out: float, zp_out: int,
                  out: torch.Tensor | None = None, m1: torch.Tensor | None = None, m2: torch.Tensor | None = None,
                  stream=None) -> torch.Tensor:
    rows, C = xq.shape
    if out is None:
        out = torch.empty(rows, C, dtype=torch.uint8, device=xq.device)
    _check(load().fqvit_ptf_layernorm(_p(xq), rows, C, _ld(xq), int(zp_in), _p(alpha), _p(gamma), _p(beta),
                                      float(s_out), int(zp_out), _p(out), _ld(out), _p(m1), _p(m2),
                                      _stream(stream)))
    return out


def lis_softmax(logits: torch.Tensor, L: int, s_logit: float, codes: torch.Tensor | None = None,
                rowsum: torch.Tensor | None = None, bias: torch.Tensor | None = None, heads: int = 1,
                window: int = 0, n_shift: int = 15, stream=None) -> torch.Tensor:
    n_rows = logits.shape[0]
    if codes is None:
        codes = torch.empty(n_rows, (L + 1) // 2, dtype=torch.uint8, device=logits.device)
    b = _bias(bias, heads, window)
    _check(load().fqvit_lis_softmax(_p(logits), n_rows, L, _ld(logits), float(s_logit), n_shift,
                                    ctypes.byref(b) if b is not None else None, _p(codes), _ld(codes),
                                    _p(rowsum), _stream(stream)))
    return codes


def lis_attn_v(codes: torch.Tensor, v: torch.Tensor, zp_v: int = 0, acc: torch.Tensor | None = None,
               range_flag: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    BH, L, d = v.shape
    if acc is None:
        acc = torch.empty(BH, L, d, dtype=torch.int32, device=v.device)
    _check(load().fqvit_lis_attn_v(_p(codes), _ld(codes), _p(v), v.stride(1), int(zp_v), BH, L, d, _p(acc),
                                   acc.stride(1), _p(range_flag), _stream(stream)))
    return acc


def lis_attention(logits: torch.Tensor, s_logit: float, v: torch.Tensor, zp_v: int = 0,
                  acc: torch.Tensor | None = None, codes: torch.Tensor | None = None,
                  bias: torch.Tensor | None = None, heads: int = 1, window: int = 0, n_shift: int = 15,
                  stream=None) -> torch.Tensor:
    BH, L, d = v.shape
    if acc is None:
        acc = torch.empty(BH, L, d, dtype=torch.int32, device=v.device)
    b = _bias(bias, heads, window)
    _check(load().fqvit_lis_attention(_p(logits), _ld(logits), float(s_logit), n_shift,
                                      ctypes.byref(b) if b is not None else None, _p(v), v.stride(1), int(zp_v),
                                      BH, L, d, _p(acc), acc.stride(1), _p(codes),
                                      _ld(codes) if codes is not None else 0, _stream(stream)))
    return acc


def lis_attention_q(logits: torch.Tensor, s_logit: float, v: torch.Tensor, zp_v: int, s_v: float, s_out: float,
                    zp_out: int, out: torch.Tensor | None = None, bias: torch.Tensor | None = None, heads: int = 1,
                    window: int = 0, n_shift: int = 15, stream=None) -> torch.Tensor:
    """Fused attention with the output requantized to 8 bits (fqvit_lis_attention_q): uint8 [BH, L, d]."""
    BH, L, d = v.shape
    if out is None:
        out = torch.empty(BH, L, d, dtype=torch.uint8, device=v.device)
    b = _bias(bias, heads, window)
    _check(load().fqvit_lis_attention_q(_p(logits), _ld(logits), float(s_logit), n_shift,
                                        ctypes.byref(b) if b is not None else None, _p(v), v.stride(1), int(zp_v),
                                        BH, L, d, float(s_v), float(s_out), int(zp_out), _p(out), out.stride(1),
                                        _stream(stream)))
    return out


def _mask(region, mask_value):
    if region is None:
        return None
    if not isinstance(region, torch.Tensor) or not region.is_cuda or region.dtype != torch.uint8:
        raise ValueError("region: a uint8 device tensor [n_windows, L]")
    if not region.is_contiguous():
        raise ValueError("region must be contiguous")
    return WindowMask(ctypes.c_void_p(region.data_ptr()), region.shape[0], int(mask_value))


def lis_softmax_masked(logits: torch.Tensor, L: int, s_logit: float, region: torch.Tensor | None,
                       mask_value: int, codes: torch.Tensor | None = None, rowsum: torch.Tensor | None = None,
                       bias: torch.Tensor | None = None, heads: int = 1, window: int = 0, n_shift: int = 15,
                       stream=None) -> torch.Tensor:
    """LIS codes with a shifted-window mask (fqvit_lis_softmax_masked); region uint8 [n_windows, L]."""
    n_rows = logits.shape[0]
    if codes is None:
        codes = torch.empty(n_rows, (L + 1) // 2, dtype=torch.uint8, device=logits.device)
    b = _bias(bias, heads, window)
    m = _mask(region, mask_value)
    _check(load().fqvit_lis_softmax_masked(_p(logits), n_rows, L, _ld(logits), float(s_logit), n_shift,
                                           ctypes.byref(b) if b is not None else None,
                                           ctypes.byref(m) if m is not None else None, _p(codes), _ld(codes),
                                           _p(rowsum), _stream(stream)))
    return codes


def lis_attention_masked(logits: torch.Tensor, s_logit: float, v: torch.Tensor, region: torch.Tensor | None,
                         mask_value: int, zp_v: int = 0, acc: torch.Tensor | None = None,
                         codes: torch.Tensor | None = None, bias: torch.Tensor | None = None, heads: int = 1,
                         window: int = 0, n_shift: int = 15, stream=None) -> torch.Tensor:
    """Fused attention with a shifted-window mask (fqvit_lis_attention_masked): int32 [BH, L, d]."""
    BH, L, d = v.shape
    if acc is None:
        acc = torch.empty(BH, L, d, dtype=torch.int32, device=v.device)
    b = _bias(bias, heads, window)
    m = _mask(region, mask_value)
    _check(load().fqvit_lis_attention_masked(_p(logits), _ld(logits), float(s_logit), n_shift,
                                             ctypes.byref(b) if b is not None else None,
                                             ctypes.byref(m) if m is not None else None, _p(v), v.stride(1),
                                             int(zp_v), BH, L, d, _p(acc), acc.stride(1), _p(codes),
                                             _ld(codes) if codes is not None else 0, _stream(stream)))
    return acc


def lis_attention_masked_q(logits: torch.Tensor, s_logit: float, v: torch.Tensor, region: torch.Tensor | None,
                           mask_value: int, zp_v: int, s_v: float, s_out: float, zp_out: int,
                           out: torch.Tensor | None = None, bias: torch.Tensor | None = None, heads: int = 1,
                           window: int = 0, n_shift: int = 15, stream=None) -> torch.Tensor:
    """Masked fused attention, output requantized to 8 bits (fqvit_lis_attention_masked_q): uint8 [BH, L, d]."""
    BH, L, d = v.shape
    if out is None:
        out = torch.empty(BH, L, d, dtype=torch.uint8, device=v.device)
    b = _bias(bias, heads, window)
    m = _mask(region, mask_value)
    _check(load().fqvit_lis_attention_masked_q(_p(logits), _ld(logits), float(s_logit), n_shift,
                                               ctypes.byref(b) if b is not None else None,
                                               ctypes.byref(m) if m is not None else None, _p(v), v.stride(1),
                                               int(zp_v), BH, L, d, float(s_v), float(s_out), int(zp_out), _p(out),
                                               out.stride(1), _stream(stream)))
    return out


def qk_logits(q: torch.Tensor, k: torch.Tensor, zp_q: int, zp_k: int, s_q: float, s_k: float, s_logit: float,
              zp_logit: int, out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """Q K^T and its 8-bit output quantizer (fqvit_qk_logits): int8 [BH, L, d] x 2 -> int8 [BH*L, ld]."""
    BH, L, d = q.shape
    if out is None:
        out = torch.empty(BH * L, (L + 15) // 16 * 16, dtype=torch.int8, device=q.device)
    _check(load().fqvit_qk_logits(_p(q), q.stride(1), int(zp_q), _p(k), k.stride(1), int(zp_k), BH, L, d,
                                  float(s_q), float(s_k), float(s_logit), int(zp_logit), _p(out), _ld(out),
                                  _stream(stream)))
    return out


def qk_workspace_size(BH: int, L: int, group_heads: int = 0) -> int:
    return int(load().fqvit_qk_workspace_size(BH, L, group_heads))


def qk_lis_attention(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, zp_q: int, zp_k: int, s_q: float, s_k: float,
                     s_logit: float, zp_logit: int, zp_v: int = 0, acc: torch.Tensor | None = None,
                     workspace: torch.Tensor | None = None, group_heads: int = 0, bias: torch.Tensor | None = None,
                     heads: int = 1, window: int = 0, region: torch.Tensor | None = None, mask_value: int = 0,
                     n_shift: int = 15, stream=None) -> torch.Tensor:
    """Attention from int8 Q, K, V (fqvit_qk_lis_attention): int32 [BH, L, d]."""
    BH, L, d = v.shape
    if acc is None:
        acc = torch.empty(BH, L, d, dtype=torch.int32, device=v.device)
    if workspace is None:
        workspace = torch.empty(qk_workspace_size(BH, L, group_heads), dtype=torch.int8, device=v.device)
    b = _bias(bias, heads, window)
    m = _mask(region, mask_value)
    _check(load().fqvit_qk_lis_attention(_p(q), q.stride(1), int(zp_q), _p(k), k.stride(1), int(zp_k), float(s_q),
                                         float(s_k), float(s_logit), int(zp_logit), n_shift,
                                         ctypes.byref(b) if b is not None else None,
                                         ctypes.byref(m) if m is not None else None, _p(v), v.stride(1), int(zp_v),
                                         BH, L, d, _p(acc), acc.stride(1), _p(workspace),
                                         workspace.numel() * workspace.element_size(), int(group_heads),
                                         _stream(stream)))
    return acc


def linear_pack_weight(w: torch.Tensor, out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """int8 weight codes [N, K] -> the fp16 copy [N, K] fqvit_linear_q takes (fqvit_linear_pack_weight)."""
    N, K = w.shape
    if out is None:
        out = torch.empty(N, K, dtype=torch.float16, device=w.device)
    _check(load().fqvit_linear_pack_weight(_p(w), N, K, _ld(w), _p(out), _stream(stream)))
    return out


def linear_workspace_size(M: int, K: int) -> int:
    return int(load().fqvit_linear_workspace_size(int(M), int(K)))


def linear_q(x: torch.Tensor, zp_x: int, s_x: float, w_h: torch.Tensor, s_w: torch.Tensor,
             bias: torch.Tensor | None, s_y: float, zp_y: int, out: torch.Tensor | None = None,
             acc: torch.Tensor | None = None, workspace: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """A MinMax Linear layer (fqvit_linear_q): uint8 x [M, K] (zp_x, s_x), packed fp16 weights
    [N, K] with per-channel scales s_w [N] and int32 bias [N] -> uint8 y [M, N] (s_y, zp_y);
    acc, if given, receives the int32 accumulators."""
    M, K = x.shape
    N = w_h.shape[0]
    if w_h.dtype != torch.float16 or w_h.shape[1] != K or not w_h.is_contiguous():
        raise ValueError("w_h must be the contiguous fp16 [N, K] array of linear_pack_weight")
    if out is None:
        out = torch.empty(M, N, dtype=torch.uint8, device=x.device)
    if workspace is None:
        workspace = torch.empty(linear_workspace_size(M, K), dtype=torch.uint8, device=x.device)
    _check(load().fqvit_linear_q(_p(x), M, K, _ld(x), int(zp_x), float(s_x), _p(w_h), N, _p(s_w), _p(bias),
                                 float(s_y), int(zp_y), _p(out), _ld(out), _p(acc),
                                 _ld(acc) if acc is not None else 0, _p(workspace), workspace.numel(),
                                 _stream(stream)))
    return out


def split_qkv(qkv: torch.Tensor, B: int, L: int, H: int, d: int, ld_head: int | None = None, stream=None):
    """The QKV Linear's uint8 output [B*L, >= 3 H d] -> int8 q, k, v [B*H, L, d] (codes minus 128)
    (fqvit_split_qkv); ld_head pads the head rows (then the views are [B*H, L, ld_head][..., :d])."""
    ld = d if ld_head is None else ld_head
    outs = [torch.empty(B * H, L, ld, dtype=torch.int8, device=qkv.device) for _ in range(3)]
    _check(load().fqvit_split_qkv(_p(qkv), int(B), int(L), int(H), int(d), _ld(qkv), _p(outs[0]), _p(outs[1]),
                                  _p(outs[2]), ld, _stream(stream)))
    return tuple(o[..., :d] for o in outs)


def merge_heads(heads: torch.Tensor, B: int, L: int, H: int, out: torch.Tensor | None = None, stream=None):
    """Head-major uint8 rows [B*H, L, d] -> token rows [B*L, H d] (fqvit_merge_heads)."""
    d = heads.shape[-1]
    if out is None:
        out = torch.empty(B * L, H * d, dtype=torch.uint8, device=heads.device)
    _check(load().fqvit_merge_heads(_p(heads), int(B), int(L), int(H), int(d), heads.stride(-2), _p(out), _ld(out),
                                    _stream(stream)))
    return out


def block_int(xq, zp_in, alpha, gamma, beta, s_out, zp_out, yq, logits, ld_logit, s_logit, v, zp_v, acc,
              bias=None, heads=1, window=0, stream=None):
    """One layer: LayerNorm then fused LIS attention (fqvit_block_int)."""
    BH, L, d = v.shape
    b = _bias(bias, heads, window)
    desc = BlockDesc(xq.data_ptr(), xq.shape[0], xq.shape[1], int(zp_in), alpha.data_ptr(), gamma.data_ptr(),
                     beta.data_ptr(), float(s_out), int(zp_out), yq.data_ptr(), logits.data_ptr(), int(ld_logit),
                     float(s_logit), v.data_ptr(), int(zp_v), BH, L, d,
                     ctypes.cast(ctypes.pointer(b), ctypes.c_void_p) if b is not None else None, acc.data_ptr())
    _check(load().fqvit_block_int(ctypes.byref(desc), _stream(stream)))
    return yq, acc
