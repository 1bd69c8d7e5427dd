"""fqvit_calibrate_ptf_noalloc: PTF calibration for callers that cannot
allocate device memory (a fixed memory budget after start-up, or device memory
owned by another allocator).  It must give exactly what fqvit_calibrate_ptf
gives with a caller-provided workspace, call after call, although every call
reuses the same library-owned scratch array.

Called through the C ABI with ctypes.  This file is collected last so that a
run stopping at the first failure has already run every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2111_13824_gb300 import build as fbuild
from paper_2111_13824_gb300 import fqvit

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    fbuild.build()
    return fqvit.load()


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr()) if t is not None else None


def _noalloc(lib, x, K, with_sse=True):
    """The call with (or, with_sse=False, without) a caller buffer for the error sums; without one
    the sums are kept in the library's array and only s, zp and alpha come back."""
    rows, C = x.shape
    s = torch.empty(1, dtype=torch.float32, device=x.device)
    zp = torch.empty(1, dtype=torch.int32, device=x.device)
    alpha = torch.empty(C, dtype=torch.uint8, device=x.device)
    sse = torch.empty(C, K + 1, dtype=torch.float64, device=x.device) if with_sse else None
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    rc = lib.fqvit_calibrate_ptf_noalloc(_ptr(x), rows, C, x.stride(0), 8, K, _ptr(s), _ptr(zp), _ptr(alpha),
                                         _ptr(sse), stream)
    assert rc == 0, lib.fqvit_last_error().decode()
    return s, zp, alpha, sse


def _with_workspace(x, K):
    rows, C = x.shape
    sse = torch.empty(C, K + 1, dtype=torch.float64, device=x.device)
    s, zp, alpha = fqvit.calibrate_ptf(x, K=K, sse=sse)
    return s, zp, alpha, sse


def _channels(seed, rows, C):
    rng = np.random.default_rng(seed)
    r = np.exp(rng.normal(0, 1, C)) * 2
    m = 0.25 * r * rng.normal(size=C)
    return torch.from_numpy((m + r / 6 * rng.normal(size=(rows, C))).astype(np.float32)).to("cuda:0")


def test_noalloc_matches_workspace_calibration_twice(lib):
    # two calls in a row on different problems: the second must not see the first's leftovers
    cases = [(_channels(1, 3000, 384), 3), (_channels(2, 517, 96), 7), (_channels(3, 4096, 4096), 3)]
    for x, K in cases:
        got = _noalloc(lib, x, K)
        ref = _with_workspace(x, K)
        torch.cuda.synchronize()
        for a, b in zip(got, ref):
            assert torch.equal(a, b)
        # the same problem again right away
        again = _noalloc(lib, x, K)
        torch.cuda.synchronize()
        for a, b in zip(again, ref):
            assert torch.equal(a, b)


def test_noalloc_sums_in_the_library_array(lib):
    """Without a caller sse buffer the error sums live in the fixed array: its largest use (C = 4096
    at K = 3, 16384 sums), then a smaller problem right after it, then the largest again; s, zp and
    alpha bit for bit as with a workspace.  After the first call no call takes device memory."""
    cases = [(_channels(5, 2000, 4096), 3), (_channels(6, 700, 192), 5), (_channels(7, 1500, 4096), 3)]
    refs = [_with_workspace(x, K) for x, K in cases]
    outs = [(torch.empty(1, dtype=torch.float32, device=x.device), torch.empty(1, dtype=torch.int32, device=x.device),
             torch.empty(x.shape[1], dtype=torch.uint8, device=x.device)) for x, _ in cases]
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)

    def call(i):
        x, K = cases[i]
        s, zp, alpha = outs[i]
        rc = lib.fqvit_calibrate_ptf_noalloc(_ptr(x), x.shape[0], x.shape[1], x.stride(0), 8, K, _ptr(s), _ptr(zp),
                                             _ptr(alpha), None, stream)
        assert rc == 0, lib.fqvit_last_error().decode()

    call(1)  # the first call may load the library's code (and so reserve its array)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for i in range(len(cases)):
        call(i)
        torch.cuda.synchronize()
        assert torch.cuda.mem_get_info()[0] == free0  # nothing allocated by the call
        rs, rzp, ralpha, _ = refs[i]
        s, zp, alpha = outs[i]
        assert torch.equal(s.view(torch.int32), rs.view(torch.int32))
        assert torch.equal(zp, rzp) and torch.equal(alpha, ralpha)


def test_noalloc_with_caller_sums_takes_any_size(lib):
    """With the caller's sse buffer the array holds only the small min/max part, so C (K + 1) may
    exceed 16384."""
    x = _channels(8, 300, 8192)
    got = _noalloc(lib, x, 3)
    ref = _with_workspace(x, 3)
    torch.cuda.synchronize()
    for a, b in zip(got, ref):
        assert torch.equal(a, b)


def test_noalloc_rejects_problems_beyond_its_scratch(lib):
    x = _channels(4, 8, 4096)
    s = torch.empty(1, dtype=torch.float32, device=x.device)
    zp = torch.empty(1, dtype=torch.int32, device=x.device)
    alpha = torch.empty(4096, dtype=torch.uint8, device=x.device)
    rc = lib.fqvit_calibrate_ptf_noalloc(_ptr(x), 8, 4096, 4096, 8, 4, _ptr(s), _ptr(zp), _ptr(alpha), None,
                                         None)
    assert rc == fqvit.ERR_UNSUPPORTED
    assert "16384" in lib.fqvit_last_error().decode()
