"""Throughput of the FQ-ViT integer hot path on GB300.

One step = the whole hot path over one batch: for each of the config's
layers, the PTF integer LayerNorm (norm1) and the fused Log-Int-Softmax
attention (codes -> BitShift attn.V), on per-layer synthetic inputs already
resident in HBM (7.4 GB for ViT-L/384, far above the 129 MB L2, so no flush
is needed between steps).  Swin-S adds its shifted-window mask on the odd
blocks of stages 1-3 and the LayerNorm of each patch merging (4C channels)
before stages 2-4.  Calibration and quantization of the LayerNorm
input are offline (setup), as in post-training quantization.

Algorithmic bytes per layer: LayerNorm 2 bytes per element (int8 in and out)
plus 9 bytes of per-channel parameters; attention 1 byte per logit, 1 per V
element and 4 per int32 accumulator (the 4-bit codes stay on chip).  The K
timed steps run as one CUDA graph holding only the kernels, which are
launched with programmatic dependent launch (a kernel's set-up overlaps the
previous kernel's tail); the per-kernel times come from a second graph of up to
three steps with timing events around each kernel (--no-graph: eager launches).
Event nodes between kernels serialise them and add their own gaps, so each kernel
kind is also timed alone: its launches of those steps back to back between one
pair of events (`back_to_back`, the launches overlapping as in the step).

Prints ONE JSON line (rank 0).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--config vit_l384]
                  [--impl reference] [--no-e2e] [--no-cpu]
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2111_13824_gb300 import synth  # noqa: E402

METRIC = "tokens/s and achieved HBM GB/s (% of GB300 peak) for PTF-LN + LIS attention, ViT-L/384"


def _dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def tensor_peak():
    """Dense fp16 / bf16 tensor-core TFLOP/s for a kernel timed alone (the burst figure; the two
    types have the same dense rate on this GPU)."""
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        if "bf16_tflops" in d:
            return float(d["bf16_tflops"]), "measured"
    return 1900.0, "fallback"


def bench_linear(fqvit, cfg, dev):
    """The block's four MinMax Linear layers (QKV, projection, fc1, fc2) of layer 0 at the
    config's token count, each call (the fp16 copy of X, then the tensor-core product and its
    requantization) timed alone with CUDA events: 10 calls after 3."""
    peak, kind = tensor_peak()
    out, tot_ms, tot_flop = {}, 0.0, 0
    for k in synth.LINEAR_KINDS:
        a = synth.linear_inputs(cfg, 0, k, device=dev)
        wh = fqvit.linear_pack_weight(a["w"])
        ws = torch.empty(fqvit.linear_workspace_size(a["M"], a["K"]), dtype=torch.uint8, device=dev)
        y = torch.empty(a["M"], a["N"], dtype=torch.uint8, device=dev)
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(10)]
        for i in range(13):
            if i >= 3:
                evs[i - 3][0].record()
            fqvit.linear_q(a["x"], a["zp_x"], a["s_x"], wh, a["s_w"], a["bias"], a["s_y"], a["zp_y"], out=y,
                           workspace=ws)
            if i >= 3:
                evs[i - 3][1].record()
        torch.cuda.synchronize()
        fqvit.sync_status()
        ms = statistics.mean(e0.elapsed_time(e1) for e0, e1 in evs)
        flop = 2 * a["M"] * a["N"] * a["K"]
        tf = flop / (ms / 1e3) / 1e12
        out[k] = {"M": a["M"], "N": a["N"], "K": a["K"], "ms_per_call": round(ms, 5), "tflops": round(tf, 1),
                  "frac": round(tf / peak, 4)}
        tot_ms += ms
        tot_flop += flop
        del a, wh, ws, y
    tf = tot_flop / (tot_ms / 1e3) / 1e12
    out["block"] = {"ms": round(tot_ms, 5), "tflops": round(tf, 1), "frac": round(tf / peak, 4),
                    "peak_tflops": peak, "peak_source": f"{kind} (MEASURED_PEAKS.json bf16_tflops)"
                    if kind == "measured" else "fallback"}
    out["how"] = ("fqvit_linear_q per layer of block 0 (fp16 copy of X + tcgen05 product + per-channel "
                  "requantization), 10 calls after 3, outside the timed step; FLOP = 2 M N K")
    return out


# ------------------------------------------------------------------ byte model

def ln_bytes(rows, C):
    """Algorithmic bytes of one LayerNorm launch: u8 in + u8 out + 9 B / channel of parameters."""
    return 2 * rows * C + 9 * C


OUT8_SV = 1.0 / 127.0  # V's scale for the 8-bit output option (any value: the work is the same)


def metric_name(args):
    if args.config == "vit_l384" and not args.qk:
        return METRIC
    return f"tokens/s, PTF-LN + {'Q K^T + ' if args.qk else ''}LIS attention, {args.config}"


def attn_bytes(BH, L, d, out_bytes=4, qk=False):
    """Algorithmic bytes of one fused attention launch: 1 B / logit + 1 B / V element + 4 B / acc element
    (1 B / output element with the 8-bit requantized output).  From Q and K (--qk): 1 B per Q and per K
    element instead of the logits, which stay on chip and in L2."""
    return BH * ((2 * L * d if qk else L * L) + L * d + out_bytes * L * d)


def recorded_traffic(config, kernel):
    """DRAM bytes per launch (mean over the step's layers) from the committed ncu record of this
    config, if the kernel's sources are unchanged since that capture (else None)."""
    import hashlib

    path = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        rec = json.load(f).get(config, {}).get(kernel)
    if not rec:
        return None
    h = hashlib.sha256()
    for src in rec["sources"]:
        if not os.path.exists(os.path.join(ROOT, src)):
            return None  # a source of the captured kernel is gone: the record is stale
        with open(os.path.join(ROOT, src), "rb") as f:
            h.update(f.read())
    return rec["dram_bytes_per_launch"] if h.hexdigest()[:16] == rec["source_sha"] else None


# ------------------------------------------------------------------ workload

def make_layers(cfg, device, sigma=1.0, limit=0, qk=False):
    from paper_2111_13824_gb300 import fqvit

    layers = []
    ws = None  # --qk: one logits workspace, reused group after group and layer after layer
    for l in range(cfg.layers if limit <= 0 else min(limit, cfg.layers)):
        st = synth.layer_stage(cfg, l)
        d = synth.ln_inputs(cfg, l, device=device)
        s, zp, alpha = fqvit.calibrate_ptf(d["x_calib"], K=cfg.K)
        zp_i, s_f = int(zp.item()), float(s.item())
        xq = fqvit.ptf_quantize(d["x"], s_f, zp_i, alpha)
        a = synth.attn_inputs(cfg, l, device=device, sigma=sigma)
        if qk and ws is None:
            ws = torch.empty(fqvit.qk_workspace_size(a["BH"], a["L"]), dtype=torch.int8, device=device)
        layers.append(dict(
            qk=qk, q=a["q"] if qk else None, k=a["k"] if qk else None, s_q=a["s_q"], s_k=a["s_k"],
            zp_logit=a["zp_logit"], workspace=ws,
            xq=xq, zp=zp_i, alpha=alpha, gamma=d["gamma"], beta=d["beta"], s_out=d["s_out"], zp_out=d["zp_out"],
            yq=torch.empty_like(xq), logits=None if qk else a["logits"], s_logit=a["s_logit"], v=a["v"],
            bias=a["bias"],
            heads=a["heads"], window=a["window"],
            region=synth.layer_window_mask(cfg, l, device=device), mask_value=synth.swin_mask_value(a["s_logit"]),
            acc=torch.empty(a["BH"], a["L"], a["d"], dtype=torch.int32, device=device),
            out8=torch.empty(a["BH"], a["L"], a["d"], dtype=torch.uint8, device=device),
            rows=st.rows, C=st.C, BH=st.BH, L=st.L, d=st.d, merge=None))
        del d, a
    # Swin: the patch merging after stage i runs its LayerNorm (4C channels) before stage i+1
    first = 0
    for i, st in enumerate(cfg.stages):
        if i > 0 and (i - 1) in synth.merge_stages(cfg) and first < len(layers):
            layers[first]["merge"] = make_merge(cfg, i - 1, device)
        first += st.layers
    torch.cuda.synchronize()
    return layers


def make_merge(cfg, stage, device):
    from paper_2111_13824_gb300 import fqvit

    d = synth.merge_ln_inputs(cfg, stage, device=device)
    s, zp, alpha = fqvit.calibrate_ptf(d["x_calib"], K=cfg.K)
    zp_i, s_f = int(zp.item()), float(s.item())
    xq = fqvit.ptf_quantize(d["x"], s_f, zp_i, alpha)
    return dict(xq=xq, zp=zp_i, alpha=alpha, gamma=d["gamma"], beta=d["beta"], s_out=d["s_out"], zp_out=d["zp_out"],
                yq=torch.empty_like(xq), rows=d["rows"], C=d["C"])


def qk_group(ly):
    """Heads per group of the chained --qk attention (the library's choice for the layer's shape)."""
    from paper_2111_13824_gb300 import fqvit

    return max(1, fqvit.qk_workspace_size(ly["BH"], ly["L"]) // (ly["L"] * synth.ld_pad(ly["L"])))


def layernorm(fq, m):
    fq.ptf_layernorm(m["xq"], m["zp"], m["alpha"], m["gamma"], m["beta"], m["s_out"], m["zp_out"], out=m["yq"])


def attention(fq, ly, out8=False):
    """The layer's fused attention; Swin's shifted blocks take their window mask.  --qk: from the
    int8 Q, K and V (Q K^T on the tensor cores, then the fused attention, head group by group)."""
    kw = dict(bias=ly["bias"], heads=ly["heads"], window=ly["window"])
    if ly["qk"]:
        fq.qk_lis_attention(ly["q"], ly["k"], ly["v"], 0, 0, ly["s_q"], ly["s_k"], ly["s_logit"], ly["zp_logit"],
                            acc=ly["acc"], workspace=ly["workspace"], region=ly["region"],
                            mask_value=ly["mask_value"], **kw)
    elif ly["region"] is not None:
        if out8:  # the output requantized to 8 bits (output scale = V's: M = 2^-15)
            fq.lis_attention_masked_q(ly["logits"], ly["s_logit"], ly["v"], ly["region"], ly["mask_value"], 0,
                                      OUT8_SV, OUT8_SV, 128, out=ly["out8"], **kw)
        else:
            fq.lis_attention_masked(ly["logits"], ly["s_logit"], ly["v"], ly["region"], ly["mask_value"], 0,
                                    acc=ly["acc"], **kw)
    elif out8:
        fq.lis_attention_q(ly["logits"], ly["s_logit"], ly["v"], 0, OUT8_SV, OUT8_SV, 128, out=ly["out8"], **kw)
    else:
        fq.lis_attention(ly["logits"], ly["s_logit"], ly["v"], 0, acc=ly["acc"], **kw)


def run_layer(fq, ly, ev=None):
    if ly["merge"] is not None:
        layernorm(fq, ly["merge"])
    layernorm(fq, ly)
    if ev is not None:
        ev[0].record()
    attention(fq, ly)
    if ev is not None:
        ev[1].record()


# ------------------------------------------------------------------ clocks

class ClockSampler:
    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits", "-lms", "100",
                 "-i", str(self.index)], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        self.proc.terminate()
        out, _ = self.proc.communicate(timeout=10)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 8:
                continue
            try:
                sm.append(float(f[0]))
                mx.append(float(f[1]))
            except ValueError:
                continue
            for n, val in zip(names, f[4:8]):
                if val.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------------------ CPU oracle baseline

def step_elements(cfg):
    """(LayerNorm elements, attention logits) of one step over the whole config."""
    ln = sum(st.layers * st.rows * st.C for st in cfg.stages)
    for i in synth.merge_stages(cfg):
        st = cfg.stages[i]
        ln += (st.rows // 4) * 4 * st.C
    return ln, sum(st.layers * st.BH * st.L * st.L for st in cfg.stages)


def _host(t):
    return t.detach().cpu().numpy()


class OracleLeg:
    """The oracle, as it stands, on this host's cores, fed the GPU step's own resident inputs.

    Timing: all of layer 0 (every LayerNorm row and every attention head) on all cores, and a
    bounded part of it (256 rows, 2 heads; Swin: one image) on one core; each is scaled by the
    step's LayerNorm elements and attention logits to the whole step.  Parity: the same layer-0
    outputs, and sampled LayerNorm rows and heads of every other layer, compared element by
    element with what the GPU step wrote."""

    def __init__(self, cfg, layers, args):
        import oracle

        self.o, self.cfg, self.layers, self.args = oracle, cfg, layers, args
        self.mismatch = []
        self.checked_rows = self.checked_heads = 0

    # -- the oracle on part of one layer, from that layer's resident inputs
    def _ln(self, m, rows):
        xq = _host(m["xq"][rows])
        return self.o.ptf_layernorm(xq, m["zp"], _host(m["alpha"]), _host(m["gamma"]), _host(m["beta"]), m["s_out"],
                                    m["zp_out"])[0]

    def _attn(self, ly, h0, h1):
        """Outputs of heads h0 .. h1 - 1 (Swin: whole images, so that bias and mask line up)."""
        o, L = self.o, ly["L"]
        if ly["qk"]:
            x = o.qk_logits(_host(ly["q"][h0:h1]), _host(ly["k"][h0:h1]), 0, 0, ly["s_q"], ly["s_k"], ly["s_logit"],
                            ly["zp_logit"], ld=synth.ld_pad(L))
        else:
            x = _host(ly["logits"][h0 * L:h1 * L])
        bias = _host(ly["bias"]) if ly["bias"] is not None else None
        reg = _host(ly["region"]) if ly["region"] is not None else None
        co, _ = o.lis_softmax(x, L, ly["s_logit"], bias=bias, heads=ly["heads"], window=ly["window"] or 7, region=reg,
                              mask_value=ly["mask_value"] if reg is not None else 0)
        acc, _ = o.lis_attn_v(co, _host(ly["v"][h0:h1]), 0)
        if self.args.out8:
            return o.attn_requant(acc, OUT8_SV, OUT8_SV, 128)
        return acc

    def _gpu_attn(self, ly, h0, h1):
        return _host((ly["out8"] if self.args.out8 else ly["acc"])[h0:h1])

    def _head_unit(self, ly):
        """Heads per independent unit: one head, or (windowed attention) one image's heads."""
        return ly["BH"] // 64 if ly["window"] else 1

    def _compare(self, what, got, want):
        if not np.array_equal(got, want):
            self.mismatch.append(f"{what}: {int((got != want).sum())} elements differ")

    # -- the legs
    def layer0_all_cores(self):
        """Seconds of the LayerNorm and of the attention of all of layer 0, all cores; checks them."""
        o, ly = self.o, self.layers[0]
        o.set_num_threads(os.cpu_count() or 1)
        t0 = time.perf_counter()
        yo = self._ln(ly, slice(None))
        t1 = time.perf_counter()
        ao = self._attn(ly, 0, ly["BH"])
        t2 = time.perf_counter()
        self._compare("layer 0 LayerNorm", _host(ly["yq"]), yo)
        self._compare("layer 0 attention", self._gpu_attn(ly, 0, ly["BH"]), ao)
        self.checked_rows += ly["rows"]
        self.checked_heads += ly["BH"]
        return t1 - t0, t2 - t1

    def layer0_one_core(self, rows=256, units=2):
        o, ly = self.o, self.layers[0]
        o.set_num_threads(1)
        hu = self._head_unit(ly)
        t0 = time.perf_counter()
        self._ln(ly, slice(0, rows))
        t1 = time.perf_counter()
        self._attn(ly, 0, units * hu)
        t2 = time.perf_counter()
        o.set_num_threads(os.cpu_count() or 1)
        return (t1 - t0) * ly["rows"] / rows, (t2 - t1) * ly["BH"] / (units * hu)

    def other_layers(self, rows=64, units=2):
        """Sampled rows and heads of every layer but 0 (and of every patch merging's LayerNorm)."""
        for i, ly in enumerate(self.layers):
            for m, tag in ((ly, f"layer {i}"), (ly["merge"], f"merge before layer {i}")):
                if m is None or (i == 0 and m is ly):
                    continue
                sel = np.linspace(0, m["rows"] - 1, rows).astype(np.int64)
                self._compare(f"{tag} LayerNorm", _host(m["yq"][torch.from_numpy(sel).to(m["yq"].device)]),
                              self._ln(m, torch.from_numpy(sel).to(m["xq"].device)))
                self.checked_rows += rows
            if i == 0:
                continue
            hu = self._head_unit(ly)
            nunit = ly["BH"] // hu
            for u in sorted({(i * 7919) % nunit, nunit - 1 - (i * 104729) % nunit})[:units]:
                self._compare(f"layer {i} attention unit {u}", self._gpu_attn(ly, u * hu, (u + 1) * hu),
                              self._attn(ly, u * hu, (u + 1) * hu))
                self.checked_heads += hu

    def verdict(self):
        n = len(self.layers)
        if self.mismatch:
            return "MISMATCH: " + "; ".join(self.mismatch[:4])
        return (f"bit-exact against the oracle: all of layer 0, sampled rows and heads of the other {n - 1} "
                f"layer(s) ({self.checked_rows} LayerNorm rows, {self.checked_heads} attention heads)")


# ------------------------------------------------------------------ main arms

def time_config(fqvit, cfg, layers, args, steps, warmup, dev, ws, sample_clocks=False):
    """Times `steps` steps of the config's stack (one CUDA graph of the kernels, launched with
    programmatic dependent launch), then a second pass with timing events around each kernel.
    Returns the step time, the per-kernel times and byte rates, and the clock record."""
    for _ in range(warmup):
        for ly in layers:
            run_layer(fqvit, ly)
    torch.cuda.synchronize()

    use_graph = not args.no_graph
    ev_kw = dict(enable_timing=True)
    if use_graph:
        try:
            torch.cuda.Event(enable_timing=True, external=True)
            ev_kw["external"] = True
        except TypeError:
            use_graph = False
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    merges = [ly["merge"] for ly in layers if ly["merge"] is not None]
    ev_steps = min(steps, 3)  # steps of the per-kernel timing pass
    ev = {}

    def new_events(kw):
        ev["attn"] = [(torch.cuda.Event(**kw), torch.cuda.Event(**kw)) for _ in range(ev_steps * len(layers))]
        ev["ln"] = [(torch.cuda.Event(**kw), torch.cuda.Event(**kw)) for _ in range(ev_steps * len(layers))]
        ev["merge"] = [(torch.cuda.Event(**kw), torch.cuda.Event(**kw)) for _ in range(ev_steps * len(merges))]

    new_events(ev_kw)

    def enqueue_steps(n, events):
        """The step's launches; with events, each kernel between a pair of timing events (which
        serialise the kernels: the timed step runs without them)."""
        k = km = 0

        def mark(name, idx, j):
            if events:
                ev[name][idx][j].record()

        for _ in range(n):
            for ly in layers:
                if ly["merge"] is not None:
                    mark("merge", km, 0)
                    layernorm(fqvit, ly["merge"])
                    mark("merge", km, 1)
                    km += 1
                mark("ln", k, 0)
                layernorm(fqvit, ly)
                mark("ln", k, 1)
                mark("attn", k, 0)
                attention(fqvit, ly, args.out8)
                mark("attn", k, 1)
                k += 1

    # each kernel kind alone, its launches of ev_steps steps back to back between one pair of events
    # (programmatic dependent launch overlaps each launch's set-up with the previous one's tail, as in
    # the step; no event between two launches)
    grp = {k: (torch.cuda.Event(**ev_kw), torch.cuda.Event(**ev_kw)) for k in ("ln", "attn")}

    def enqueue_groups():
        grp["ln"][0].record()
        for _ in range(ev_steps):
            for ly in layers:
                layernorm(fqvit, ly)
        grp["ln"][1].record()
        grp["attn"][0].record()
        for _ in range(ev_steps):
            for ly in layers:
                attention(fqvit, ly, args.out8)
        grp["attn"][1].record()

    graph = ev_graph = grp_graph = None
    if use_graph:
        try:
            graph = torch.cuda.CUDAGraph()
            with torch.cuda.graph(graph):
                enqueue_steps(steps, False)
            ev_graph = torch.cuda.CUDAGraph()
            with torch.cuda.graph(ev_graph):
                enqueue_steps(ev_steps, True)
            grp_graph = torch.cuda.CUDAGraph()
            with torch.cuda.graph(grp_graph):
                enqueue_groups()
            graph.replay()  # upload and one untimed pass
            torch.cuda.synchronize()
        except Exception as exc:  # noqa: BLE001 - any capture failure falls back to eager launches
            print(f"bench: CUDA graph unavailable ({type(exc).__name__}: {exc}); eager launches", file=sys.stderr)
            graph = ev_graph = grp_graph = None
            torch.cuda.synchronize()
            new_events(dict(enable_timing=True))
            grp = {k: (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for k in grp}
    clocks = ClockSampler(torch.cuda.current_device()) if sample_clocks else None
    if ws > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    if clocks:
        clocks.start()
        time.sleep(0.3)  # let the sampler start before the timed region
    start.record()
    if graph is not None:
        graph.replay()
    else:
        enqueue_steps(steps, False)
    end.record()
    torch.cuda.synchronize()
    clk = clocks.stop() if clocks else None
    elapsed_ms = start.elapsed_time(end)
    if ws > 1:
        t = torch.tensor([elapsed_ms], device=dev)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        elapsed_ms = float(t.item())
        torch.distributed.barrier()

    # per-kernel durations: a separate pass of the same launches with timing events around each
    if ev_graph is not None:
        ev_graph.replay()
    else:
        enqueue_steps(ev_steps, True)
    torch.cuda.synchronize()
    if grp_graph is not None:
        grp_graph.replay()
    else:
        enqueue_groups()
    torch.cuda.synchronize()
    fqvit.sync_status()
    n_launch = ev_steps * len(layers)
    grp_ms = {k: grp[k][0].elapsed_time(grp[k][1]) / n_launch for k in grp}
    attn_ms = [a.elapsed_time(b) for a, b in ev["attn"]]
    ln_ms = [a.elapsed_time(b) for a, b in ev["ln"]]
    merge_ms = [a.elapsed_time(b) for a, b in ev["merge"]]
    ab = [attn_bytes(ly["BH"], ly["L"], ly["d"], 1 if args.out8 else 4, qk=args.qk) for ly in layers]
    lb = [ln_bytes(ly["rows"], ly["C"]) for ly in layers]
    mb = [ln_bytes(m["rows"], m["C"]) for m in merges]
    return dict(elapsed_ms=elapsed_ms, ms_per_step=elapsed_ms / steps, graph=graph is not None, clocks=clk,
                ev_steps=ev_steps, attn_ms=attn_ms, ln_ms=ln_ms, merge_ms=merge_ms, grp_ms=grp_ms, ab=ab, lb=lb, mb=mb,
                merges=merges, step_bytes=sum(ab) + sum(lb) + sum(mb))


def kernel_stats(t, peak, ev_steps):
    """Per-kernel byte rates (algorithmic bytes over CUDA-event durations) of a time_config result.

    The duration of a launch is the time of the step's launches of that kernel back to back,
    between one pair of events, over their number (as in the step, each launch's set-up overlaps
    the previous one's tail).  `event_pair` is the other measure: an event pair around every
    launch, which serialises the kernels and adds the events' own gaps (for short kernels the sum
    of those durations exceeds the step time)."""
    def rates(ms, nbytes):
        gbs = sum(nbytes) / len(nbytes) / (ms / 1e3) / 1e9
        return {"gbs": round(gbs, 1), "frac": round(gbs / peak, 4), "ms_per_launch": round(ms, 5),
                "bytes_per_launch": round(sum(nbytes) / len(nbytes))}, gbs

    attn, attn_gbs = rates(t["grp_ms"]["attn"], t["ab"])
    ln, ln_gbs = rates(t["grp_ms"]["ln"], t["lb"])
    attn["event_pair"] = rates(sum(t["attn_ms"]) / len(t["attn_ms"]), t["ab"])[0]
    ln["event_pair"] = rates(sum(t["ln_ms"]) / len(t["ln_ms"]), t["lb"])[0]
    out = {"attention": attn, "layernorm": ln}
    if t["merges"]:
        mg, _ = rates(sum(t["merge_ms"]) / len(t["merge_ms"]), t["mb"])
        mg["how"] = "event pair around every launch"
        out["patch_merge_layernorm"] = mg
    return out, attn_gbs, ln_gbs


def other_configs(fqvit, args, dev, ws, peak):
    """The other four configs of the workload list, each timed like the headline step (fewer steps,
    no host-copy or CPU legs): tokens/s, HBM GB/s and the fraction of the measured peak."""
    out = {}
    for name in ("deit_t", "deit_s", "vit_b", "swin_s"):
        if name == args.config:
            continue
        cfg = synth.CONFIGS[name]
        try:
            layers = make_layers(cfg, dev, sigma=args.sigma, qk=args.qk)
            steps = max(3, min(args.steps, 10))
            t = time_config(fqvit, cfg, layers, args, steps, 3, dev, ws)
            ks, _, _ = kernel_stats(t, peak, t["ev_steps"])
            gbs = t["step_bytes"] / (t["ms_per_step"] / 1e3) / 1e9
            out[name] = {"value": round(cfg.first_tokens * ws * steps / (t["elapsed_ms"] / 1e3), 1),
                         "unit": "tokens/s", "ms_per_step": round(t["ms_per_step"], 5), "steps": steps,
                         "layers": len(layers), "hbm_gbs": round(gbs, 1), "hbm_frac": round(gbs / peak, 4),
                         "kernels": ks, "workload": f"{cfg.name}: {cfg.note}"}
            del layers
            torch.cuda.empty_cache()
        except Exception as e:  # noqa: BLE001 - one config failing is reported, not fatal to the line
            out[name] = {"error": f"{type(e).__name__}: {e}"[:300]}
    return out


def bench_gpu(args):
    from paper_2111_13824_gb300 import build as fbuild
    from paper_2111_13824_gb300 import fqvit

    ws, rank, local = _dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    if rank == 0 or not os.path.exists(fbuild.LIB):
        fbuild.build()
    if ws > 1:
        torch.distributed.barrier()
    fqvit.load()
    cfg = synth.CONFIGS[args.config]
    if args.qk and args.out8:
        raise SystemExit("--qk and --out8 together are not a bench mode")
    layers = make_layers(cfg, dev, sigma=args.sigma, limit=args.layers, qk=args.qk)
    tokens_per_step = cfg.first_tokens
    peak, peak_kind = peaks()

    t = time_config(fqvit, cfg, layers, args, args.steps, args.warmup, dev, ws, sample_clocks=True)
    elapsed_ms, ms_per_step = t["elapsed_ms"], t["ms_per_step"]
    value = tokens_per_step * ws * args.steps / (elapsed_ms / 1e3)
    ks, attn_gbs, ln_gbs = kernel_stats(t, peak, t["ev_steps"])
    step_bytes = t["step_bytes"]
    stack_gbs = step_bytes / (ms_per_step / 1e3) / 1e9
    dominant = "attention" if t["grp_ms"]["attn"] >= t["grp_ms"]["ln"] else "layernorm"
    dom_gbs = attn_gbs if dominant == "attention" else ln_gbs
    # the records are of the int32 output from logits, or (key "<config>:qk") of the --qk step
    traffic = None if args.out8 else recorded_traffic(args.config + (":qk" if args.qk else ""), dominant)
    if args.traffic:
        traffic = json.loads(args.traffic).get(dominant)

    if args.qk:  # the Q K^T kernel alone on layer 0, all heads in one launch, outside the step
        ly = layers[0]
        full = torch.empty(ly["BH"] * ly["L"], synth.ld_pad(ly["L"]), dtype=torch.int8, device=dev)
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(10)]
        for i in range(13):
            if i >= 3:
                evs[i - 3][0].record()
            fqvit.qk_logits(ly["q"], ly["k"], 0, 0, ly["s_q"], ly["s_k"], ly["s_logit"], ly["zp_logit"], out=full)
            if i >= 3:
                evs[i - 3][1].record()
        torch.cuda.synchronize()
        qk_ms = statistics.mean(a.elapsed_time(b) for a, b in evs)
        qk_b = ly["BH"] * (2 * ly["L"] * ly["d"] + ly["L"] * full.shape[1])
        ks["qk_logits"] = {"gbs": round(qk_b / (qk_ms / 1e3) / 1e9, 1), "ms_per_launch": round(qk_ms, 5),
                           "bytes_per_launch": qk_b, "frac": round(qk_b / (qk_ms / 1e3) / 1e9 / peak, 4),
                           "how": "fqvit_qk_logits on layer 0, all heads in one launch (Q, K read, logits written "
                                  "to HBM), 10 launches after 3, outside the timed step"}
        del full

    if args.linear:  # outside the timed step; a failure here is reported, not fatal to the line
        try:
            ks["linear"] = bench_linear(fqvit, cfg, dev)
        except Exception as e:  # noqa: BLE001
            ks["linear"] = {"error": f"{type(e).__name__}: {e}"[:300]}

    e2e = None
    if not args.no_e2e:
        e2e = bench_e2e(fqvit, layers, tokens_per_step, args, dev, ws)

    cpu = parity = None
    if rank == 0 and ws == 1 and not args.no_cpu:
        cpu, parity = cpu_baseline(cfg, layers, args)

    line = {
        "metric": metric_name(args),
        "value": round(value, 1),
        "unit": "tokens/s",
        "n_gpus": ws,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(ms_per_step, 4),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "int8",
        "data": "synthetic (seeded generator of the paper's layer shapes and statistics)",
        "config": {
            "workload": f"{cfg.name}: {cfg.note}, {cfg.layers} layers of PTF LayerNorm + "
                        f"{'Q K^T + ' if args.qk else ''}fused LIS attention",
            "tokens_per_step_per_gpu": tokens_per_step,
            "layers": len(layers),
            "step_bytes": step_bytes,
            "l2": f"inputs {step_bytes / 1e9:.2f} GB per step, larger than the 129 MB L2 (no flush)",
            "logit_sigma": args.sigma,
            "parallelism": f"replicas x{ws} (independent batches, no collective)",
            "launch": "cuda_graph" if t["graph"] else "eager",
            "attention_output": "uint8 (requantized)" if args.out8 else "int32 accumulators",
            "attention_input": (f"int8 Q, K, V: fqvit_qk_lis_attention, head groups of {qk_group(layers[0])}"
                                if args.qk else "int8 logits, int8 V"),
            "shifted_window_layers": sum(ly["region"] is not None for ly in layers),
            "patch_merges": len(t["merges"]),
        },
        "hbm_gbs": round(stack_gbs, 1),
        "hbm_frac": round(stack_gbs / peak, 4),
        "kernels": ks,
        "roofline": {"kernel": dominant, "bound": "hbm", "achieved": round(dom_gbs, 1), "peak": peak,
                     "unit": "GB/s", "frac": round(dom_gbs / peak, 4), "traffic": traffic,
                     "duration": "the step's launches of the kernel back to back between one event pair, "
                                 "per launch (kernels.<name>.event_pair: an event pair around every launch)",
                     "peak_source": f"{peak_kind} (MEASURED_PEAKS.json hbm_gbs)" if peak_kind == "measured"
                     else "fallback"},
        "clocks": t["clocks"],
        "gpu_launches": (sum(1 + (2 * -(-ly["BH"] // qk_group(ly)) if args.qk else 1) for ly in layers)
                         + len(t["merges"])) * args.steps,
    }
    if e2e is not None:
        line["e2e"] = e2e
    if cpu is not None:
        line["cpu_baseline"] = cpu
        line["parity"] = parity
    if args.all_configs and ws == 1 and args.layers <= 0:
        del layers
        torch.cuda.empty_cache()
        line["configs"] = other_configs(fqvit, args, dev, ws, peak)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()


def bench_e2e(fqvit, layers, tokens_per_step, args, dev, ws):
    """Same metric through the public API with host buffers: every step copies each
    layer's inputs from pinned host memory to the device and its outputs back."""
    host = []
    for ly in layers:
        ins = ("xq", "q", "k", "v") if ly["qk"] else ("xq", "logits", "v")
        h = {k: ly[k].cpu().pin_memory() for k in ins}
        h["yq"] = torch.empty_like(ly["yq"], device="cpu").pin_memory()
        h["acc"] = torch.empty_like(ly["acc"], device="cpu").pin_memory()
        if ly["merge"] is not None:  # the patch merging's LayerNorm input and output
            h["mxq"] = ly["merge"]["xq"].cpu().pin_memory()
            h["myq"] = torch.empty_like(ly["merge"]["yq"], device="cpu").pin_memory()
        host.append(h)
    h2d = sum(h[k].numel() * h[k].element_size() for h in host for k in ("xq", "logits", "q", "k", "v", "mxq")
              if k in h)
    d2h = sum(h[k].numel() * h[k].element_size() for h in host for k in ("yq", "acc", "myq") if k in h)
    steps = max(1, min(args.steps, args.e2e_steps))

    # Three streams, layers pipelined: the inputs of layer l+1 go up while layer l computes and
    # the outputs of layer l-1 come down.  Per layer: upload -> compute -> download (events);
    # across steps a layer's upload waits for its previous compute (inputs read) and its
    # compute for its previous download (outputs read).
    s_in, s_cmp, s_out = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
    main = torch.cuda.current_stream()
    n = len(layers)
    ev_in = [torch.cuda.Event() for _ in range(n)]
    ev_cmp = [torch.cuda.Event() for _ in range(n)]
    ev_out = [torch.cuda.Event() for _ in range(n)]
    started = [False] * n

    def step():
        for st_ in (s_in, s_cmp, s_out):  # nothing of the step starts before the timing event
            st_.wait_stream(main)
        for i, (ly, h) in enumerate(zip(layers, host)):
            with torch.cuda.stream(s_in):
                if started[i]:
                    s_in.wait_event(ev_cmp[i])
                ly["xq"].copy_(h["xq"], non_blocking=True)
                for key in ("logits", "q", "k", "v"):
                    if key in h:
                        ly[key].copy_(h[key], non_blocking=True)
                if "mxq" in h:
                    ly["merge"]["xq"].copy_(h["mxq"], non_blocking=True)
                ev_in[i].record(s_in)
            with torch.cuda.stream(s_cmp):
                s_cmp.wait_event(ev_in[i])
                if started[i]:
                    s_cmp.wait_event(ev_out[i])
                run_layer(fqvit, ly)
                ev_cmp[i].record(s_cmp)
            with torch.cuda.stream(s_out):
                s_out.wait_event(ev_cmp[i])
                h["yq"].copy_(ly["yq"], non_blocking=True)
                h["acc"].copy_(ly["acc"], non_blocking=True)
                if "myq" in h:
                    h["myq"].copy_(ly["merge"]["yq"], non_blocking=True)
                ev_out[i].record(s_out)
            started[i] = True
        # the step ends when its last download has landed
        main.wait_stream(s_out)

    for _ in range(max(3, args.warmup)):  # warm-up, as for the device-resident timing
        step()
    torch.cuda.synchronize()
    if ws > 1:
        torch.distributed.barrier()
    s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s.record()
    for _ in range(steps):
        step()
    e.record()
    torch.cuda.synchronize()
    ms = s.elapsed_time(e)
    if ws > 1:
        t = torch.tensor([ms], device=dev)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        ms = float(t.item())
    return {"value": round(tokens_per_step * ws * steps / (ms / 1e3), 1), "unit": "tokens/s",
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": steps,
            "how": "per layer: pinned H2D of xq, logits (--qk: Q and K), V (and a patch merging's xq); "
                   "LayerNorm(s) + fused "
                   "attention; D2H of yq and acc (and the merging's yq); "
                   "three streams (upload, compute, download), layers pipelined"}


def cpu_baseline(cfg, layers, args):
    """The oracle, as it stands, on this host's cores (OracleLeg): the time of all of layer 0 on all
    cores and of a bounded part of it on one core, each scaled to the whole step, and the parity
    verdict of the same outputs and of sampled rows and heads of every other layer."""
    import oracle

    oracle.build()
    leg = OracleLeg(cfg, layers, args)
    ln_s, at_s = leg.layer0_all_cores()
    ln1_s, at1_s = leg.layer0_one_core()
    leg.other_layers()
    ln_el, logits = step_elements(cfg)
    ly = layers[0]
    ln0, lg0 = ly["rows"] * ly["C"], ly["BH"] * ly["L"] * ly["L"]
    step_all = ln_s * ln_el / ln0 + at_s * logits / lg0
    step_one = ln1_s * ln_el / ln0 + at1_s * logits / lg0
    cores = os.cpu_count() or 1
    cpu = {"value": round(cfg.first_tokens / step_all, 2), "unit": "tokens/s", "cores": cores, "kind": "oracle",
           "single_thread": {"value": round(cfg.first_tokens / step_one, 2), "unit": "tokens/s", "cores": 1},
           "extrapolated_from": "layer 0",
           "sample": (f"all of layer 0 ({ly['rows']} LayerNorm rows, {ly['BH']} attention heads"
                      f"{', logits from Q and K' if args.qk else ''}) on {cores} cores, {ln_s + at_s:.2f} s, and "
                      f"256 rows and 2 {'images' if ly['window'] else 'heads'} of it on one core, each scaled by "
                      f"the step's LayerNorm elements and attention logits to the {cfg.layers}-layer step")}
    return cpu, leg.verdict()


def bench_reference(args):
    """The reference arm: the CPU oracle, as it stands, on the host cores.  Each step is the oracle
    on all of layer 0 of the config (the same sample as the GPU arm's cpu_baseline leg), on the
    inputs the GPU arm generates; ms_per_step is that measured time, and the tokens/s of the whole
    stack is extrapolated from it by LayerNorm elements and attention logits."""
    ws, rank, local = _dist_env()
    if rank != 0:
        return
    cfg = synth.CONFIGS[args.config]
    import oracle

    oracle.build()
    cores = os.cpu_count() or 1
    oracle.set_num_threads(cores)
    layer = make_host_layer0(cfg, args)
    leg = OracleLeg(cfg, [layer], args)

    def one():
        t0 = time.perf_counter()
        leg._ln(layer, slice(None))
        t1 = time.perf_counter()
        leg._attn(layer, 0, layer["BH"])
        return t1 - t0, time.perf_counter() - t1

    for _ in range(min(args.warmup, 1)):
        one()
    times = []
    t0 = time.perf_counter()
    for _ in range(args.steps):
        times.append(one())
    wall = time.perf_counter() - t0
    ln_s = statistics.mean(a for a, _ in times)
    at_s = statistics.mean(b for _, b in times)
    ln_el, logits = step_elements(cfg)
    ln0, lg0 = layer["rows"] * layer["C"], layer["BH"] * layer["L"] * layer["L"]
    step_est = ln_s * ln_el / ln0 + at_s * logits / lg0
    value = cfg.first_tokens / step_est
    sample = (f"per step: all of layer 0 ({layer['rows']} LayerNorm rows, {layer['BH']} attention heads) on "
              f"{cores} cores; tokens/s extrapolated by LayerNorm elements and attention logits to the "
              f"{cfg.layers}-layer step ({step_est * 1e3:.1f} ms)")
    line = {
        "impl": "reference",
        "metric": metric_name(args),
        "value": round(value, 3), "unit": "tokens/s", "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round((ln_s + at_s) * 1e3, 3), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "int8",
        "data": "synthetic (seeded generator of the paper's layer shapes and statistics)",
        "config": {"workload": f"{cfg.name}: {cfg.note}, {cfg.layers} layers of PTF LayerNorm + "
                               f"{'Q K^T + ' if args.qk else ''}LIS attention",
                   "tokens_per_step_per_gpu": cfg.first_tokens, "layers": cfg.layers},
        "extrapolated_from": "layer 0",
        "step_extrapolated_ms": round(step_est * 1e3, 3),
        "cpu_baseline": {"value": round(value, 3), "unit": "tokens/s", "cores": cores, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": round(value, 3), "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "wall_s": round(wall, 2),
    }
    print(json.dumps(line), flush=True)


def make_host_layer0(cfg, args):
    """Layer 0 of a config generated on the host: the GPU arm's shapes and statistics (its device
    generator draws other values), calibrated and quantized by the oracle."""
    import oracle

    st = synth.layer_stage(cfg, 0)
    d = synth.ln_inputs(cfg, 0)
    s, zp, alpha, _ = oracle.calibrate_ptf(d["x_calib"].numpy(), K=cfg.K)
    xq = oracle.ptf_quantize(d["x"].numpy(), s, zp, alpha)
    a = synth.attn_inputs(cfg, 0, sigma=args.sigma)
    return dict(qk=args.qk, q=a["q"], k=a["k"], s_q=a["s_q"], s_k=a["s_k"], zp_logit=a["zp_logit"],
                xq=torch.from_numpy(xq), zp=int(zp), alpha=torch.from_numpy(alpha), gamma=d["gamma"], beta=d["beta"],
                s_out=d["s_out"], zp_out=d["zp_out"], logits=a["logits"], s_logit=a["s_logit"], v=a["v"],
                bias=a["bias"], heads=a["heads"], window=a["window"],
                region=synth.layer_window_mask(cfg, 0), mask_value=synth.swin_mask_value(a["s_logit"]),
                rows=st.rows, C=st.C, BH=st.BH, L=st.L, d=st.d, merge=None)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--config", default="vit_l384", choices=sorted(synth.CONFIGS))
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--sigma", type=float, default=1.0, help="logit spread: 1 literal, 2 peaked")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--traffic", default=None, help="JSON {kernel: dram bytes per launch} from an ncu capture")
    ap.add_argument("--layers", type=int, default=0, help="time only the first N layers (profiling cases)")
    ap.add_argument("--no-graph", action="store_true", help="launch the timed steps eagerly instead of as one CUDA graph")
    ap.add_argument("--qk", action="store_true",
                    help="attention from int8 Q, K, V (fqvit_qk_lis_attention) instead of int8 logits")
    ap.add_argument("--out8", action="store_true",
                    help="the attention output requantized to 8 bits (fqvit_lis_attention_q) instead of int32")
    ap.add_argument("--no-configs", dest="all_configs", action="store_false",
                    help="skip the timing of the other four configs (reported under configs)")
    ap.add_argument("--no-linear", dest="linear", action="store_false",
                    help="skip the separate timing of the block's MinMax Linear layers (fqvit_linear_q), "
                         "which runs after the timed step and is reported under kernels.linear")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        bench_reference(args)
    else:
        bench_gpu(args)


if __name__ == "__main__":
    main()
