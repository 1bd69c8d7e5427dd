"""Seeded synthetic workloads shaped like the paper's DeiT / ViT / Swin layers.

This module only draws inputs; it holds none of the integer path's arithmetic
(no PTF quantizer, no integer LayerNorm, no i-exp, no log2 code, no
BitShift).  Both the CUDA path and the CPU oracle consume what it returns.

Recipe (per layer l of a config with seed S, generator seeded with
S * 1000 + l, draws in this fixed order):

* LayerNorm input (fp32, ``[rows, C]``): per-channel range r_c drawn
  log-normal(0, 1), then stretched in the log domain so that
  max(r) / median(r) = 40 (the inter-channel variation reported for vision
  transformers, Sec. 3.2).  ``outliers`` channels are then forced to
  U(40, 60) x median.  Channel centre m_c ~ N(0, (r_c / 4)^2); values
  m_c + (r_c / 6) N(0, 1).
* Calibration batch: 32 images' worth of rows (``32 * tokens``) from the
  same channel model.
* gamma ~ N(1, 0.1^2), beta ~ N(0, 0.1^2).
* Output quantizer of the LayerNorm: the min / max of a textbook fp64
  LayerNorm of the calibration batch mapped to 0..255 (MinMax, as the paper
  uses for activations).
* Q, K ~ N(0, sigma^2) fp32 ``[BH, L, d]``, rounded symmetrically to int8;
  the exact integer Q K^T times s_q s_k / sqrt(d) is mapped onto the full
  int8 range by its min / max (``s_logit``).  sigma = 1 is the literal
  config, sigma = 2 the "peaked" variant whose rows put most mass on a few
  keys (Sec. 3.3: 98.8 % of ViT-L attention values are below 1/16).
  The int8 codes of Q and K, their scales and the logits' zero point
  (round(-min / s_logit) - 128, signed) are returned too: the inputs of the
  Q K^T path.
* V: int8 uniform in [-128, 127], zero point 0.
* Swin relative-position bias: int8 ``[H, (2w-1)^2]`` uniform in [-16, 16].
* Swin patch merging (after stages 1-3): the stage's channel model drawn
  on its side x side map (generator seed S * 1000 + 500 + stage), each 2x2
  neighbourhood concatenated into one token of 4C channels (``patch_merge``),
  then gamma, beta and the output quantizer as for a layer.
* Swin shifted-window mask (odd blocks of a stage whose side exceeds the
  window): region ids ``[n_windows, w*w]`` of the cyclically shifted map
  (three bands per axis: below side - w, below side - shift, the rest;
  id = 3 band_y + band_x), windows in raster order, tokens in raster order
  inside a window; the mask value is -100 in real units, rounded to logit
  units (``swin_mask_value``).

Rows of logits are padded to a multiple of 16 bytes (``ld_logit``).
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import torch


@dataclass(frozen=True)
class Stage:
    """One attention / LayerNorm shape inside a config."""
    rows: int          # LayerNorm rows (tokens in the batch)
    C: int             # channels
    BH: int            # attention problems (batch x windows x heads)
    H: int             # heads
    L: int             # tokens per attention row
    d: int             # head dimension
    layers: int        # how many layers of this shape
    calib_rows: int    # calibration rows (32 images)
    window: int = 0    # Swin window side (0 = no relative-position bias)
    side: int = 0      # Swin feature-map side (tokens per image = side^2)


@dataclass(frozen=True)
class Config:
    name: str
    seed: int
    stages: tuple
    K: int = 3
    outliers: int = 0
    first_tokens: int = 0   # tokens of the first layer per image x batch
    note: str = ""

    @property
    def layers(self) -> int:
        return sum(s.layers for s in self.stages)


def _vit(name, seed, B, L, C, H, d, layers, outliers=0, note=""):
    st = Stage(rows=B * L, C=C, BH=B * H, H=H, L=L, d=d, layers=layers, calib_rows=32 * L)
    return Config(name=name, seed=seed, stages=(st,), outliers=outliers, first_tokens=B * L, note=note)


def _swin():
    B, w = 64, 7
    stages = []
    for C, H, depth, side in ((96, 3, 2, 56), (192, 6, 2, 28), (384, 12, 18, 14), (768, 24, 2, 7)):
        tokens = side * side
        nwin = (side // w) ** 2
        stages.append(Stage(rows=B * tokens, C=C, BH=B * nwin * H, H=H, L=w * w, d=32,
                            layers=depth, calib_rows=32 * tokens, window=w, side=side))
    return Config(name="swin_s", seed=4, stages=tuple(stages), first_tokens=B * 56 * 56,
                  note="Swin-S, 7x7 windows, relative-position bias")


CONFIGS = {
    "deit_t": _vit("deit_t", 0, 1, 197, 192, 3, 64, 1, note="DeiT-T block, batch 1"),
    "deit_s": _vit("deit_s", 1, 64, 197, 384, 6, 64, 12, note="DeiT-S stack, batch 64"),
    "vit_b": _vit("vit_b", 2, 64, 197, 768, 12, 64, 12, outliers=8, note="ViT-B/16 stack, batch 64"),
    "vit_l384": _vit("vit_l384", 3, 32, 577, 1024, 16, 64, 24, note="ViT-L/16 at 384 px, batch 32"),
    "swin_s": _swin(),
}


def ld_pad(n: int, align: int = 16) -> int:
    return (n + align - 1) // align * align


def layer_stage(cfg: Config, layer: int) -> Stage:
    for st in cfg.stages:
        if layer < st.layers:
            return st
        layer -= st.layers
    raise IndexError("layer out of range")


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def _channel_model(g, C, outliers, device):
    r = torch.exp(torch.randn(C, generator=g, device=device, dtype=torch.float64))
    med = torch.median(r)
    lmax, lmed = torch.log(r.max()), torch.log(med)
    if float(lmax - lmed) > 0:
        r = torch.exp(lmed + (torch.log(r) - lmed) * (math.log(40.0) / (lmax - lmed)))
    if outliers:
        idx = torch.randperm(C, generator=g, device=device)[:outliers]
        r[idx] = med * (40.0 + 20.0 * torch.rand(outliers, generator=g, device=device, dtype=torch.float64))
    m = 0.25 * r * torch.randn(C, generator=g, device=device, dtype=torch.float64)
    return r, m


def _channel_values(g, rows, r, m):
    z = torch.randn(rows, r.numel(), generator=g, device=r.device, dtype=torch.float64)
    return (m + (r / 6.0) * z).to(torch.float32)


def ln_inputs(cfg: Config, layer: int, device="cpu", rows: int | None = None):
    """LayerNorm-side inputs of one layer: x, calibration x, gamma, beta, s_out, zp_out."""
    st = layer_stage(cfg, layer)
    g = _gen(cfg.seed * 1000 + layer, device)
    r, m = _channel_model(g, st.C, cfg.outliers, device)
    n = st.rows if rows is None else rows
    x = _channel_values(g, n, r, m)
    xc = _channel_values(g, st.calib_rows, r, m)
    gamma = (1.0 + 0.1 * torch.randn(st.C, generator=g, device=device)).to(torch.float32)
    beta = (0.1 * torch.randn(st.C, generator=g, device=device)).to(torch.float32)
    s_out, zp_out = _ln_output_quantizer(xc, gamma, beta)
    return dict(x=x, x_calib=xc, gamma=gamma, beta=beta, s_out=s_out, zp_out=zp_out, C=st.C, rows=n)


def _ln_output_quantizer(xc, gamma, beta):
    """MinMax (0..255) of a textbook fp64 LayerNorm of the calibration batch: (s_out fp32, zp_out)."""
    xd = xc.double()
    mu = xd.mean(dim=1, keepdim=True)
    var = xd.var(dim=1, unbiased=False, keepdim=True)
    yf = (xd - mu) / torch.sqrt(var + 1e-6) * gamma.double() + beta.double()
    lo, hi = float(yf.min()), float(yf.max())
    s_out = (hi - lo) / 255.0
    zp_out = int(min(255, max(0, round(-lo / s_out))))
    return float(torch.tensor(s_out, dtype=torch.float32)), zp_out


def merge_stages(cfg: Config) -> tuple:
    """Indices of the stages followed by a patch merging (every Swin stage but the last)."""
    return tuple(i for i, st in enumerate(cfg.stages[:-1]) if st.window and st.side >= 2)


def patch_merge(x: torch.Tensor, side: int) -> torch.Tensor:
    """[images * side^2, C] tokens in raster order -> [images * (side/2)^2, 4C]: each merged token
    is the concatenation of its 2x2 neighbours (y, x), (y+1, x), (y, x+1), (y+1, x+1)."""
    C = x.shape[1]
    g = x.reshape(-1, side // 2, 2, side // 2, 2, C)       # image, y/2, y%2, x/2, x%2, c
    return g.permute(0, 1, 3, 4, 2, 5).reshape(-1, 4 * C)  # neighbour order: (x%2, y%2) = 00, 01, 10, 11


def merge_ln_inputs(cfg: Config, stage: int, device="cpu", images: int | None = None):
    """Inputs of the LayerNorm of the patch merging after Swin stage ``stage`` (4C channels):
    tokens of the stage's channel model on its side x side map, gathered 2x2.  ``images``
    defaults to the batch (the stage's rows / side^2); the calibration batch is 32 images.
    Generator seeded with seed * 1000 + 500 + stage; draws: channel model, tokens,
    calibration tokens, gamma, beta."""
    st = cfg.stages[stage]
    g = _gen(cfg.seed * 1000 + 500 + stage, device)
    r, m = _channel_model(g, st.C, cfg.outliers, device)
    nimg = st.rows // (st.side * st.side) if images is None else images
    x = patch_merge(_channel_values(g, nimg * st.side * st.side, r, m), st.side)
    xc = patch_merge(_channel_values(g, 32 * st.side * st.side, r, m), st.side)
    C4 = 4 * st.C
    gamma = (1.0 + 0.1 * torch.randn(C4, generator=g, device=device)).to(torch.float32)
    beta = (0.1 * torch.randn(C4, generator=g, device=device)).to(torch.float32)
    s_out, zp_out = _ln_output_quantizer(xc, gamma, beta)
    return dict(x=x.contiguous(), x_calib=xc.contiguous(), gamma=gamma, beta=beta, s_out=s_out, zp_out=zp_out,
                C=C4, rows=x.shape[0])


def attn_inputs(cfg: Config, layer: int, device="cpu", sigma: float = 1.0, bh: int | None = None):
    """Attention-side inputs of one layer: int8 logits [BH*L, ld], s_logit, int8 V [BH, L, d], bias."""
    st = layer_stage(cfg, layer)
    g = _gen(cfg.seed * 1000 + layer, device)
    # skip the LayerNorm draws so that the attention draws follow them in the fixed order
    r, m = _channel_model(g, st.C, cfg.outliers, device)
    _ = torch.randn(st.rows + st.calib_rows, st.C, generator=g, device=device, dtype=torch.float64)
    _ = torch.randn(2 * st.C, generator=g, device=device)
    BH = st.BH if bh is None else bh
    L, d = st.L, st.d
    q = sigma * torch.randn(BH, L, d, generator=g, device=device)
    k = sigma * torch.randn(BH, L, d, generator=g, device=device)
    v = torch.randint(-128, 128, (BH, L, d), generator=g, device=device, dtype=torch.int16).to(torch.int8)
    bias = None
    if st.window:
        nb = (2 * st.window - 1) ** 2
        bias = torch.randint(-16, 17, (st.H, nb), generator=g, device=device, dtype=torch.int16).to(torch.int8)
    sq = float(q.abs().max()) / 127.0
    sk = float(k.abs().max()) / 127.0
    qi = torch.clamp(torch.round(q / sq), -127, 127)
    ki = torch.clamp(torch.round(k / sk), -127, 127)
    prod = torch.bmm(qi, ki.transpose(1, 2))  # exact integers (|sum| < 2^24 in fp32)
    real = prod * (sq * sk / math.sqrt(d))
    lo, hi = float(real.min()), float(real.max())
    s_logit = max(hi - lo, 1e-6) / 255.0
    s_logit = float(torch.tensor(s_logit, dtype=torch.float32))
    qq = torch.clamp(torch.round((real - lo) / s_logit), 0, 255) - 128
    ld = ld_pad(L)
    logits = torch.zeros(BH * L, ld, dtype=torch.int8, device=device)
    logits[:, :L] = qq.reshape(BH * L, L).to(torch.int8)
    # the int8 Q and K codes (symmetric MinMax) and the logits' MinMax zero point, signed
    # (the 8-bit zero point round(-lo / s_logit) minus 128): the inputs of the Q K^T path
    zp_logit = int(min(255, max(0, round(-lo / s_logit)))) - 128
    return dict(logits=logits, ld_logit=ld, s_logit=s_logit, v=v.contiguous(), bias=bias,
                heads=st.H, window=st.window, BH=BH, L=L, d=d,
                q=qi.to(torch.int8).contiguous(), k=ki.to(torch.int8).contiguous(),
                s_q=float(torch.tensor(sq, dtype=torch.float32)), s_k=float(torch.tensor(sk, dtype=torch.float32)),
                zp_logit=zp_logit)


def layer_window_mask(cfg: Config, layer: int, device="cpu"):
    """(region ids uint8 [n_windows, L], n_windows) of a shifted-window layer, else None: in a
    Swin stage the odd blocks shift their windows by window // 2, unless one window covers the map."""
    st = layer_stage(cfg, layer)
    if not st.window or st.side <= st.window:
        return None
    block = layer
    for prev in cfg.stages:
        if prev is st:
            break
        block -= prev.layers
    if block % 2 == 0:
        return None
    return shifted_window_regions(st.side, st.window).to(device)


def shifted_window_regions(side: int, window: int, shift: int | None = None) -> torch.Tensor:
    """Region ids uint8 [n_windows, window^2] of a side x side map shifted by ``shift``
    (default window // 2); every token of a window carries its band pair 3 band_y + band_x."""
    shift = window // 2 if shift is None else shift

    def band(t):
        return 0 if t < side - window else (1 if t < side - shift else 2)

    nw = side // window
    out = torch.empty(nw * nw, window * window, dtype=torch.uint8)
    for wy in range(nw):
        for wx in range(nw):
            for ty in range(window):
                for tx in range(window):
                    y, x = wy * window + ty, wx * window + tx
                    out[wy * nw + wx, ty * window + tx] = 3 * band(y) + band(x)
    return out


def swin_mask_value(s_logit: float, real: float = -100.0) -> int:
    """The Swin mask (-100 in real units) in logit units, kept inside -32768 .. 0."""
    return max(-32768, min(0, int(round(real / s_logit))))


# ---- MinMax Linear layers of the block -------------------------------------

LINEAR_KINDS = ("qkv", "proj", "fc1", "fc2")


def linear_shape(C: int, kind: str) -> tuple[int, int]:
    """(N, K) of a block's Linear layer: QKV C -> 3C, projection C -> C, MLP C -> 4C -> C."""
    return {"qkv": (3 * C, C), "proj": (C, C), "fc1": (4 * C, C), "fc2": (C, 4 * C)}[kind]


def linear_inputs(cfg: Config, layer: int, kind: str, device="cpu", rows: int | None = None,
                  calib_rows: int = 512):
    """Inputs of one MinMax Linear layer (generator seed S * 1000 + 700 + 4 layer + kind index).

    * activations, real ``[rows, K]``: N(0, 1) for the LayerNorm outputs (QKV, fc1) and the
      attention output (projection); GELU of N(0, 1) for the MLP's hidden layer (fc2), so its
      zero point sits near the bottom of the range.  Quantized asymmetric, layer-wise, by the
      min / max of the draw (Sec. 4.1).
    * weights ``[N, K]``: N(0, 0.02^2) times a per-channel factor U(0.5, 2), quantized
      symmetric, channel-wise (s_w = max |w_n| / 127, codes in -127 .. 127).
    * bias: N(0, 0.02^2), as an integer at scale s_x s_w[n].
    * output quantizer: min / max of the real-valued layer over the first ``calib_rows`` rows,
      mapped to 0 .. 255 (MinMax).
    """
    st = layer_stage(cfg, layer)
    N, K = linear_shape(st.C, kind)
    M = st.rows if rows is None else rows
    g = _gen(cfg.seed * 1000 + 700 + 4 * layer + LINEAR_KINDS.index(kind), device)
    xr = torch.randn(M, K, generator=g, device=device, dtype=torch.float32)
    if kind == "fc2":
        xr = torch.nn.functional.gelu(xr)
    lo, hi = float(xr.min()), float(xr.max())
    s_x = float(torch.tensor((hi - lo) / 255.0, dtype=torch.float32))
    zp_x = int(min(255, max(0, round(-lo / s_x))))
    x = torch.clamp(torch.round(xr / s_x) + zp_x, 0, 255).to(torch.uint8)
    del xr
    wr = 0.02 * torch.randn(N, K, generator=g, device=device, dtype=torch.float32)
    wr *= 0.5 + 1.5 * torch.rand(N, 1, generator=g, device=device)
    s_w = (wr.abs().amax(dim=1) / 127.0).to(torch.float32)
    w = torch.clamp(torch.round(wr / s_w[:, None]), -127, 127).to(torch.int8)
    br = 0.02 * torch.randn(N, generator=g, device=device, dtype=torch.float64)
    bias = torch.round(br / (s_x * s_w.double())).to(torch.int32)
    c = min(M, calib_rows)
    real = ((x[:c].double() - zp_x) * s_x) @ (w.double() * s_w.double()[:, None]).T + bias.double() * (s_x * s_w.double())
    ylo, yhi = float(real.min()), float(real.max())
    s_y = float(torch.tensor((yhi - ylo) / 255.0, dtype=torch.float32))
    zp_y = int(min(255, max(0, round(-ylo / s_y))))
    return dict(x=x.contiguous(), zp_x=zp_x, s_x=s_x, w=w.contiguous(), s_w=s_w.contiguous(),
                bias=bias.contiguous(), s_y=s_y, zp_y=zp_y, M=M, N=N, K=K)
