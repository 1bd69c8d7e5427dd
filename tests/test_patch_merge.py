"""PTF LayerNorm of Swin's patch merging (4C channels: the 2x2 neighbours of a
token concatenated) on the GPU against the oracle, at the full Swin-S batch
for each of the three merges: PTF calibration (Eqs. 8-10) on the merged
calibration batch, the quantizer (Eq. 7), then the integer LayerNorm with its
per-row M1 / M2, all bit for bit.
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


@pytest.mark.parametrize("stage", [0, 1, 2])
def test_patch_merge_layernorm_full_batch(stage):
    cfg = synth.CONFIGS["swin_s"]
    st = cfg.stages[stage]
    d = synth.merge_ln_inputs(cfg, stage)
    assert d["C"] == 4 * st.C and d["rows"] == 64 * (st.side // 2) ** 2
    xc = d["x_calib"].numpy()
    s_o, zp_o, a_o, _ = oracle.calibrate_ptf(xc, K=cfg.K)
    s, zp, alpha = fqvit.calibrate_ptf(d["x_calib"].to(DEV), K=cfg.K)
    torch.cuda.synchronize()
    assert np.float32(s_o) == np.float32(s.item()) and zp_o == int(zp.item())
    assert np.array_equal(a_o, alpha.cpu().numpy())
    # the factors differ across channels (the point of PTF) and repeat the stage's channel
    # model in each of the four neighbour blocks
    assert len(set(a_o.tolist())) > 1
    xq_o = oracle.ptf_quantize(d["x"].numpy(), s_o, zp_o, a_o)
    xq = fqvit.ptf_quantize(d["x"].to(DEV), float(s.item()), int(zp.item()), alpha)
    assert np.array_equal(xq.cpu().numpy(), xq_o)
    gamma, beta = d["gamma"].numpy(), d["beta"].numpy()
    yo, m1o, m2o = oracle.ptf_layernorm(xq_o, zp_o, a_o, gamma, beta, d["s_out"], d["zp_out"])
    m1 = torch.empty(d["rows"], dtype=torch.int64, device=DEV)
    m2 = torch.empty(d["rows"], dtype=torch.int64, device=DEV)
    y = fqvit.ptf_layernorm(xq, int(zp.item()), alpha, d["gamma"].to(DEV), d["beta"].to(DEV), d["s_out"],
                            d["zp_out"], m1=m1, m2=m2)
    torch.cuda.synchronize()
    assert np.array_equal(m1.cpu().numpy(), m1o) and np.array_equal(m2.cpu().numpy(), m2o)
    assert np.array_equal(y.cpu().numpy(), yo)
