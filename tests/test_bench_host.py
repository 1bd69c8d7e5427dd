"""Host logic of bench.py and of the input generator, on the CPU: the reference arm's JSON
line (the oracle timed on the host), the step's byte and element model, and the structure
of the Swin inputs (shifted-window regions, patch merging) that the GPU tests and the bench
rely on.
"""
import json
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2111_13824_gb300 import synth  # noqa: E402


def test_reference_arm_prints_one_json_line():
    """`bench.py --impl reference` runs the oracle on the host and prints the contract's line."""
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                          "--warmup", "3", "--config", "deit_t"], capture_output=True, text=True, timeout=600,
                         cwd=ROOT)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [ln for ln in out.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["unit"] == "tokens/s" and d["higher_is_better"] is True
    assert d["value"] > 0 and d["steps"] == 1 and d["warmup"] == 3 and d["n_gpus"] == 1
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"] == {"value": d["value"], "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    assert d["config"]["workload"].startswith("deit_t")
    # the measured step is layer 0; the stack's rate is extrapolated from it, and says so
    assert d["extrapolated_from"] == "layer 0"
    assert d["ms_per_step"] * d["steps"] / 1e3 <= d["wall_s"] + 0.05
    assert d["step_extrapolated_ms"] >= d["ms_per_step"]


class _Args:
    qk = False
    out8 = False
    sigma = 1.0


def test_oracle_leg_parity_verdict():
    """The cpu_baseline leg's parity check: outputs equal to the oracle's read as bit-exact, one
    planted wrong element as a mismatch (host tensors stand in for the GPU step's)."""
    import oracle

    oracle.build()
    cfg = synth.CONFIGS["deit_t"]
    ly = bench.make_host_layer0(cfg, _Args)
    leg = bench.OracleLeg(cfg, [ly], _Args)
    ly["yq"] = torch.from_numpy(leg._ln(ly, slice(None)))
    ly["acc"] = torch.from_numpy(leg._attn(ly, 0, ly["BH"]))
    leg.layer0_all_cores()
    leg.other_layers()
    assert leg.verdict().startswith("bit-exact"), leg.verdict()
    ly["acc"][1, 5, 7] += 1
    leg2 = bench.OracleLeg(cfg, [ly], _Args)
    leg2.layer0_all_cores()
    assert leg2.verdict().startswith("MISMATCH") and "attention" in leg2.verdict()


def test_metric_names():
    class A:
        config, qk = "vit_l384", False
    assert bench.metric_name(A) == bench.METRIC
    A.qk = True
    assert "Q K^T" in bench.metric_name(A)
    A.config, A.qk = "swin_s", False
    assert bench.metric_name(A).endswith("swin_s")


def test_algorithmic_bytes():
    # one ViT-L/384 layer: 1 B per logit, 1 B per V element, 4 B per accumulator
    BH, L, d = 512, 577, 64
    assert bench.attn_bytes(BH, L, d) == BH * (L * L + L * d + 4 * L * d) == 264995328
    # from Q and K: their bytes replace the logits'
    assert bench.attn_bytes(BH, L, d, qk=True) == BH * (2 * L * d + L * d + 4 * L * d)
    # the 8-bit output
    assert bench.attn_bytes(BH, L, d, out_bytes=1) == BH * (L * L + 2 * L * d)
    assert bench.ln_bytes(18464, 1024) == 2 * 18464 * 1024 + 9 * 1024


def test_step_elements():
    ln, logits = bench.step_elements(synth.CONFIGS["vit_l384"])
    assert ln == 24 * 32 * 577 * 1024 and logits == 24 * 512 * 577 * 577
    ln, logits = bench.step_elements(synth.CONFIGS["swin_s"])
    # 24 blocks of LayerNorm plus the three patch mergings (4C channels on a quarter of the tokens)
    blocks = 64 * (2 * 3136 * 96 + 2 * 784 * 192 + 18 * 196 * 384 + 2 * 49 * 768)
    merges = 64 * (784 * 384 + 196 * 768 + 49 * 1536)
    assert ln == blocks + merges
    assert logits == 49 * 49 * (2 * 12288 + 2 * 6144 + 18 * 3072 + 2 * 1536)


def test_shifted_window_regions():
    """Three bands per axis after the cyclic shift: the last window of the map sees four regions
    (its lower-right block mixes the wrapped rows and columns), the first window one."""
    for side in (56, 28, 14):
        r = synth.shifted_window_regions(side, 7).numpy()
        nw = side // 7
        assert r.shape == (nw * nw, 49)
        assert set(np.unique(r[0]).tolist()) == {0}
        assert set(np.unique(r[-1]).tolist()) == {4, 5, 7, 8}
        # a window on the right edge (not bottom): bands 1 and 2 along x only
        assert set(np.unique(r[nw - 1]).tolist()) == {1, 2}
        last = r[-1].reshape(7, 7)
        assert np.all(last[:4, :4] == 4) and np.all(last[4:, 4:] == 8)
    # one window covering the map: no shifted layer
    assert synth.layer_window_mask(synth.CONFIGS["swin_s"], 23) is None


def test_layer_window_mask_pattern():
    cfg = synth.CONFIGS["swin_s"]
    masked = [l for l in range(cfg.layers) if synth.layer_window_mask(cfg, l) is not None]
    # odd blocks of stages 1-3 (2, 2, 18 blocks); stage 4 is one window
    assert masked == [1, 3] + list(range(5, 22, 2))
    assert synth.layer_window_mask(synth.CONFIGS["vit_l384"], 1) is None


def test_patch_merge_order():
    x = torch.arange(2 * 16 * 3, dtype=torch.float32).reshape(32, 3)  # 2 images, 4 x 4 tokens, C = 3
    y = synth.patch_merge(x, 4)
    assert y.shape == (8, 12)
    # neighbours (y, x), (y + 1, x), (y, x + 1), (y + 1, x + 1) of token (0, 0): rows 0, 4, 1, 5
    assert y[0].tolist() == x[[0, 4, 1, 5]].reshape(-1).tolist()
    # token (0, 1) of the second image: rows 16 + 2, 16 + 6, 16 + 3, 16 + 7
    assert y[5].tolist() == x[[18, 22, 19, 23]].reshape(-1).tolist()


def test_swin_mask_value():
    assert synth.swin_mask_value(0.035) == -2857
    assert synth.swin_mask_value(0.001) == -32768
    assert synth.swin_mask_value(1e9) == 0


@pytest.mark.parametrize("name", ["vit_l384", "deit_s", "swin_s"])
def test_qk_inputs_are_codes_and_scales(name):
    a = synth.attn_inputs(synth.CONFIGS[name], 0, bh=2)
    assert a["q"].dtype == torch.int8 and a["k"].dtype == torch.int8 and a["q"].shape == (2, a["L"], a["d"])
    assert int(a["q"].abs().max()) <= 127 and a["s_q"] > 0 and a["s_k"] > 0
    assert -128 <= a["zp_logit"] <= 127


@pytest.mark.parametrize("name,kind", [("deit_t", "qkv"), ("deit_t", "fc2"), ("swin_s", "fc1"), ("vit_b", "proj")])
def test_linear_inputs_structure(name, kind):
    """The Linear generator: shapes of the block's layers, symmetric per-channel weight codes,
    asymmetric activation codes, an int32 bias and a MinMax output quantizer."""
    cfg = synth.CONFIGS[name]
    a = synth.linear_inputs(cfg, 0, kind, rows=300)
    C = synth.layer_stage(cfg, 0).C
    N, K = {"qkv": (3 * C, C), "proj": (C, C), "fc1": (4 * C, C), "fc2": (C, 4 * C)}[kind]
    assert (a["M"], a["N"], a["K"]) == (300, N, K)
    assert a["x"].dtype == torch.uint8 and a["x"].shape == (300, K)
    assert a["w"].dtype == torch.int8 and a["w"].shape == (N, K) and int(a["w"].abs().max()) <= 127
    # every channel reaches its own maximum code (symmetric MinMax per channel)
    assert torch.all(a["w"].abs().amax(dim=1) == 127)
    assert a["s_w"].dtype == torch.float32 and bool(torch.all(a["s_w"] > 0))
    assert a["bias"].dtype == torch.int32 and a["bias"].shape == (N,)
    assert 0 <= a["zp_x"] <= 255 and 0 <= a["zp_y"] <= 255 and a["s_x"] > 0 and a["s_y"] > 0
    # GELU's input to fc2 sits above -0.17: its zero point is near the bottom of the range
    if kind == "fc2":
        assert a["zp_x"] < 32
    else:
        assert 96 < a["zp_x"] < 160
    # the activation codes span the range (MinMax of the draw)
    assert int(a["x"].min()) == 0 and int(a["x"].max()) == 255
