"""The failure path of the bounded device waits, without a fault: a CTA waits on an mbarrier
that nothing completes (fqvit_selftest_bounded_wait), gives up after its two-second limit and
records the timeout; fqvit_sync_status reports FQVIT_ERR_TIMEOUT once, and the context stays
usable (a LayerNorm and a Linear layer afterwards still match the oracle bit for bit).
"""
import time

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


def test_bounded_wait_gives_up_and_the_context_survives():
    fqvit.sync_status()  # nothing pending
    t0 = time.monotonic()
    fqvit.selftest_bounded_wait()
    with pytest.raises(fqvit.FqvitError) as e:
        fqvit.sync_status()
    waited = time.monotonic() - t0
    assert e.value.code == fqvit.ERR_TIMEOUT
    assert 1.5 < waited < 60.0
    fqvit.sync_status()  # the status word was cleared

    rng = np.random.default_rng(3)
    xq = rng.integers(0, 256, size=(300, 384)).astype(np.uint8)
    alpha = rng.integers(0, 4, size=384).astype(np.uint8)
    gamma = (1.0 + 0.1 * rng.standard_normal(384)).astype(np.float32)
    beta = (0.1 * rng.standard_normal(384)).astype(np.float32)
    y = fqvit.ptf_layernorm(torch.from_numpy(xq).to(DEV), 100, torch.from_numpy(alpha).to(DEV),
                            torch.from_numpy(gamma).to(DEV), torch.from_numpy(beta).to(DEV), 0.02, 120)
    w = rng.integers(-128, 128, size=(96, 384)).astype(np.int8)
    s_w = (rng.uniform(0.5, 2.0, size=96) * 1e-3).astype(np.float32)
    out = fqvit.linear_q(y, 120, 0.02, fqvit.linear_pack_weight(torch.from_numpy(w).to(DEV)),
                         torch.from_numpy(s_w).to(DEV), None, 0.05, 128)
    fqvit.sync_status()
    y_want, _, _ = oracle.ptf_layernorm(xq, 100, alpha, gamma, beta, 0.02, 120)
    out_want, _ = oracle.linear_q(y_want, 120, 0.02, w, s_w, None, 0.05, 128)
    assert np.array_equal(y.cpu().numpy(), y_want)
    assert np.array_equal(out.cpu().numpy(), out_want)
