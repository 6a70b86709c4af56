"""Benchmark of the FGQ hot path on GB300: ResNet-50 convolution stack, batch 64, 224x224.

One step = one pass of the whole hot path over one batch of synthetic input:
  * FGQ ternarization of every conv layer's fp32 weights at G = 4 and at G = 64
    (the first layer instead gets per-filter 8-bit weights: 8w-8a first layer);
  * DFP quantization of every layer's fp32 input activations to uint8 (derived scale);
  * the 53 convolutions as grouped ternary implicit GEMMs at G = 4 and at G = 64
    (the first layer as a dense 8-bit-weight convolution), fp32 NHWC outputs.
Metric: effective TOPS = sum over both G stacks of 2*M*P*Kred per step / step time.

Roofline: each layer's floor is max(algorithmic bytes / measured HBM bandwidth, ops /
measured bf16 tensor peak) (MEASURED_PEAKS.json; the tensor-core paths run fp16 operands at
the bf16 rate); a family's roofline rate is its ops over the sum of its layers' floors, and
its fraction is that sum over its measured time.  Streaming kernels (quantizer, ternarizer)
are HBM-bound: bytes / time against the measured HBM bandwidth.

The same JSON line carries the other workloads, each measured in the same run:
  config 1  the conv2_x 3x3 layer at batch 1, G = 4 (ternarize + quantize + convolution);
  config 2  the same layer at batch 32, G = 64 and G = 4 side by side, and the standalone
            ternarization of the 25.5 M ResNet-50 weights at G = 4, 16 and 64;
  config 4  the ResNet-101 stack at batch 128 with packed uint4 activations, G = 64;
  config 5  the AlexNet convolutions and fully connected layers at batch 256, int8
            activations, G = 4 and 64, and the square FC sweep M = K in {4096, 8192,
            16384} x batch {1, 64, 1024}.

Usage:  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
        python bench.py --layer res3b_branch2b[,...] --G 4 [--batch B] [--path auto|simt|tc] [--iters n]
        (single convolutions, one JSON line each: the calls profiler captures select)
N > 1 runs under torchrun, one rank per GPU, each rank its own batch of 64 (weak scaling,
no data-path collective).  --impl reference times the CPU oracle (the reference statement of
the method) on a bounded sample of the same workload, over all host cores.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

METRIC = "effective TOPS + % roofline, ternary×int8 FGQ conv stack ResNet-50 b64 (N=4,64)"
UNIT = "TOPS"
BATCH = 64
GROUPS = (4, 64)
ACT_BITS = {"u8": 8, "s8": 8, "u4": 4, "s4": 4}


def parse(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--e2e-steps", type=int, default=3)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--cpu-workers", type=int, default=0, help="oracle processes (0: every host core)")
    ap.add_argument("--no-configs", action="store_true", help="skip the other workloads (configs 1, 2, 4, 5)")
    ap.add_argument("--only", default="", help="profiling captures: run only 'step' (the timed steps)")
    ap.add_argument("--layer", default="", help="time single convolutions instead: ResNet-50 layer names, comma "
                                               "separated (per call, L2 flushed before each; for profiler captures)")
    ap.add_argument("--G", type=int, default=4, help="group size of the --layer calls")
    ap.add_argument("--act", default="u8", help="activation type of the --layer calls")
    ap.add_argument("--path", default="auto", choices=["auto", "simt", "tc", "dense"],
                    help="kernel family of the --layer calls")
    ap.add_argument("--iters", type=int, default=5, help="timed calls per --layer layer")
    ap.add_argument("--batch", type=int, default=BATCH,
                    help="images per GPU (the benchmark workload is 64; smaller batches serve profiler "
                         "captures that must stay small)")
    return ap.parse_args(argv)


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"],
                "bf16_tflops_sustained": d.get("bf16_tflops_sustained", d["bf16_tflops"]),
                "sm_max_mhz": d.get("sm_max_mhz", 2070.0), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "sm_max_mhz": 2070.0,
            "source": "fallback"}


def source_digest():
    """Digest of the CUDA sources: counters taken from another build do not describe this one."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_1705_01462_gb300", "csrc")
    for fn in sorted(os.listdir(csrc)):
        with open(os.path.join(csrc, fn), "rb") as f:
            h.update(fn.encode() + b"\0" + f.read())
    return h.hexdigest()[:16]


def load_traffic(digest=None):
    """Per-call DRAM bytes from the committed ncu summaries (profiles/*traffic*.txt): lines
    'family  bytes_per_call  ...' after a line '# sources <digest>'.  With `digest`, a file
    taken from other sources contributes nothing."""
    out = {}
    pdir = os.path.join(ROOT, "profiles")
    if not os.path.isdir(pdir):
        return out
    for fn in sorted(os.listdir(pdir)):
        if "traffic" not in fn or not fn.endswith(".txt"):
            continue
        file_digest, rows = None, {}
        with open(os.path.join(pdir, fn)) as f:
            for line in f:
                parts = line.split()
                if line.startswith("# sources") and len(parts) >= 3:
                    file_digest = parts[2]
                elif len(parts) >= 2 and not line.startswith("#"):
                    try:
                        rows[parts[0]] = float(parts[1])
                    except ValueError:
                        pass
        if digest is None or file_digest == digest:
            out.update(rows)
    return out


class ClockSampler:
    """nvidia-smi clock / throttle sampling during the timed region."""

    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []
        self.t = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, FileNotFoundError):
            self.proc = None
            return
        self.t = threading.Thread(target=self._read, daemon=True)
        self.t.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        if self.t:
            self.t.join(timeout=2)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 8:
                continue
            try:
                sm.append(float(f[0]))
                smax.append(float(f[1]))
            except ValueError:
                continue
            for n, v in zip(names, f[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "samples": len(sm), "reasons": sorted(reasons)}


# ----------------------------------------------------------------------------- workload and rooflines

def workload_layers():
    from paper_1705_01462_gb300 import synth
    return synth.resnet50_convs()


def total_ops(layers, B, groups=GROUPS):
    return sum(l.ops(B) for l in layers) * len(groups)


def algorithmic_bytes(layer, B, G, act_bits=8):
    """Minimum HBM bytes of one contraction launch: activations once, packed weights once,
    fp32 outputs once.  G None: dense 8-bit weights."""
    act = B * layer.H * layer.W * layer.C * act_bits // 8
    if G is None:
        wbytes = layer.M * layer.Kred + 4 * layer.M
    else:
        ng = -(-layer.Kred // G)
        wbytes = layer.M * (-(-ng * G // 16)) * 4 + layer.M * ng * 4
    out = layer.P(B) * layer.M * 4
    return act + wbytes + out


def layer_floor(layer, B, G, peaks, act_bits=8):
    """(seconds, bound) of one contraction at the measured peaks: the larger of its
    algorithmic bytes over the HBM bandwidth and its ops over the bf16 tensor peak."""
    t_mem = algorithmic_bytes(layer, B, G, act_bits) / (peaks["hbm_gbs"] * 1e9)
    t_ops = layer.ops(B) / (peaks["bf16_tflops"] * 1e12)
    return (t_mem, "hbm") if t_mem >= t_ops else (t_ops, "tensor")


def conv_roofline(layers, B, G, peaks, sec, act_bits=8):
    """Roofline entry of a set of contractions that took `sec` seconds: effective TOPS
    achieved, the roofline rate (ops over the sum of per-layer floors), the fraction (sum of
    floors over the time), the bound holding most of the floor time, and the bytes."""
    ops = sum(l.ops(B) for l in layers)
    floor, by_bound = 0.0, {}
    for l in layers:
        t, b = layer_floor(l, B, G, peaks, act_bits)
        floor += t
        by_bound[b] = by_bound.get(b, 0.0) + t
    return {"bound": max(by_bound, key=by_bound.get), "achieved": ops / sec / 1e12, "peak": ops / floor / 1e12,
            "unit": UNIT, "frac": floor / sec, "floor_ms": floor * 1e3, "ms": sec * 1e3,
            "bytes": sum(algorithmic_bytes(l, B, G, act_bits) for l in layers), "ops": ops}


def hbm_roofline(nbytes, sec, peaks):
    achieved = nbytes / sec / 1e9
    return {"bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
            "frac": achieved / peaks["hbm_gbs"], "ms": sec * 1e3, "bytes": nbytes}


def ternarize_bytes(layers, G):
    """fp32 weights in; 2-bit codes (padded rows) and one fp32 alpha per group out."""
    return sum(l.M * l.Kred * 4 + l.M * (-(-l.Kred // G)) * (4 + G // 4) for l in layers)


def family_roofline(fam, layers, B, peaks, sec, act="u8"):
    """Roofline entry of one kernel family over one step of the workload (`layers[0]` is the
    8-bit-weight first layer)."""
    bits = ACT_BITS[act]
    if fam.startswith("conv_g"):
        return conv_roofline(layers[1:], B, int(fam[6:]), peaks, sec, bits)
    if fam == "conv_w8_stem":
        return conv_roofline(layers[:1], B, None, peaks, sec, 8)
    if fam == "quantize_act":  # fp32 in, codes out (the stem's input is 8-bit)
        nbytes = sum(B * l.H * l.W * l.C * (4 * 8 + (8 if i == 0 else bits)) // 8 for i, l in enumerate(layers))
    elif fam.startswith("ternarize_g"):
        nbytes = ternarize_bytes(layers[1:], int(fam[11:]))
    elif fam == "quantize_weights_w8":
        nbytes = layers[0].M * layers[0].Kred * 5 + 4 * layers[0].M
    else:
        raise ValueError(fam)
    return hbm_roofline(nbytes, sec, peaks)


class Workload:
    """Device-resident inputs and outputs of one step: every layer's fp32 weights and fp32
    input, its codes, alphas, quantized input, scale and quantizer workspace, and its fp32
    output per group size.  With first_w8 the first layer keeps 8-bit weights (8w-8a) and
    8-bit activations."""

    def __init__(self, dev, B, layers, seed_offset=0, groups=GROUPS, act="u8", first_w8=True, fcs=()):
        import ctypes

        import torch
        from paper_1705_01462_gb300 import fgq, synth
        self.torch, self.fgq = torch, fgq
        self.dev, self.B, self.layers, self.groups, self.act = dev, B, list(layers) + list(fcs), groups, act
        self.first_w8 = first_w8
        self.nconv = len(layers)
        self.w, self.x, self.q, self.sc, self.types = [], [], [], [], []
        self.codes = {G: [] for G in groups}
        self.alpha = {G: [] for G in groups}
        self.out = {G: [] for G in groups}
        self.paths = {}
        for i, l in enumerate(self.layers):
            w8 = first_w8 and i == 0
            typ = "u8" if (w8 and act in ("u4", "s4")) else act
            self.types.append(typ)
            self.w.append(synth.torch_weights(l, synth.layer_seed(i, seed_offset), dev))
            self.x.append(synth.torch_activations((B, l.H, l.W, l.C), synth.layer_seed(i, seed_offset + 1), dev))
            n = self.x[-1].numel()
            self.q.append(torch.empty(fgq.act_bytes(n, typ), dtype=torch.uint8, device=dev))
            self.sc.append(torch.empty(1, dtype=torch.float32, device=dev))
            for G in groups:
                if w8:
                    self.codes[G].append(torch.empty((l.M, l.Kred), dtype=torch.int8, device=dev))
                    self.alpha[G].append(torch.empty(l.M, dtype=torch.float32, device=dev))
                else:
                    self.codes[G].append(torch.empty((l.M, fgq.codes_words_per_row(l.Kred, G)), dtype=torch.int32,
                                                     device=dev))
                    self.alpha[G].append(torch.empty((l.M, fgq.num_groups(l.Kred, G)), dtype=torch.float32,
                                                     device=dev))
                self.out[G].append(torch.empty((B, l.Ho, l.Wo, l.M), dtype=torch.float32, device=dev))
        # host tables of every layer's input for fgq_quantize_act_batch
        nl = len(self.layers)
        self.qb_n = nl
        self.qb_x = (ctypes.c_void_p * nl)(*[x.data_ptr() for x in self.x])
        self.qb_n_elem = (ctypes.c_size_t * nl)(*[x.numel() for x in self.x])
        self.qb_types = (ctypes.c_int * nl)(*[fgq.ACT_TYPES[t] for t in self.types])
        self.qb_q = (ctypes.c_void_p * nl)(*[q.data_ptr() for q in self.q])
        self.qb_sc = (ctypes.c_void_p * nl)(*[s_.data_ptr() for s_ in self.sc])
        self.qb_ws = torch.empty(max(4, fgq.lib().fgq_quantize_act_batch_workspace_bytes(nl)), dtype=torch.uint8,
                                 device=dev)
        # host tables of the ternary layers for fgq_ternarize_batch (one launch per G)
        self.tl = [i for i in range(len(self.layers)) if not (first_w8 and i == 0)]
        n = len(self.tl)
        self.tern_n = n
        self.tern_w = (ctypes.c_void_p * n)(*[self.w[i].data_ptr() for i in self.tl])
        self.tern_M = (ctypes.c_int * n)(*[self.layers[i].M for i in self.tl])
        self.tern_K = (ctypes.c_int * n)(*[self.layers[i].Kred for i in self.tl])
        self.tern_codes = {G: (ctypes.c_void_p * n)(*[self.codes[G][i].data_ptr() for i in self.tl]) for G in groups}
        self.tern_alpha = {G: (ctypes.c_void_p * n)(*[self.alpha[G][i].data_ptr() for i in self.tl]) for G in groups}
        torch.cuda.synchronize()

    def ops(self):
        return sum(l.ops(self.B) for l in self.layers) * len(self.groups)

    def step(self, stream, timers=None, counts=None):
        """Issue one step on `stream`.  The calls of one kernel family run back to back, and
        with `timers` (dict family -> list of (start, end) events) one event pair brackets
        each contiguous run of a family, so the per-family times cost a handful of events
        per step instead of two per call; `counts` (dict family -> calls) is filled on the
        way."""
        fgq = self.fgq
        L = fgq.lib()
        sh = stream.cuda_stream
        torch = self.torch
        calls = []  # (family, function) in issue order

        def chk(code, what):
            if code != 0:
                raise RuntimeError(f"{what} failed: {L.fgq_status_string(code).decode()}")

        if self.first_w8:
            l = self.layers[0]
            for G in self.groups:  # first layer: 8-bit weights (8w-8a)
                calls.append(("quantize_weights_w8", lambda G=G, l=l: chk(L.fgq_quantize_weights_w8(
                    self.w[0].data_ptr(), l.M, l.Kred, self.codes[G][0].data_ptr(), self.alpha[G][0].data_ptr(), sh),
                    "w8")))
        for G in self.groups:  # every ternary layer of the stack in one launch per G
            calls.append((f"ternarize_g{G}", lambda G=G: chk(L.fgq_ternarize_batch(
                self.tern_n, self.tern_w, self.tern_M, self.tern_K, G, self.tern_codes[G], self.tern_alpha[G], sh),
                "ternarize_batch")))
        # every layer's input quantized with its own derived scale, in one batched call
        calls.append(("quantize_act", lambda: chk(L.fgq_quantize_act_batch(
            self.qb_n, self.qb_x, self.qb_n_elem, self.qb_types, self.qb_q, self.qb_sc, self.qb_ws.data_ptr(),
            self.qb_ws.numel(), sh), "quantize_batch")))
        if self.first_w8:
            l = self.layers[0]
            for G in self.groups:
                calls.append(("conv_w8_stem", lambda G=G, l=l: chk(L.fgq_conv2d_w8(
                    self.q[0].data_ptr(), fgq.ACT_TYPES[self.types[0]], self.sc[0].data_ptr(), self.B, l.H, l.W, l.C,
                    l.R, l.S, l.stride, l.pad, l.groups, self.codes[G][0].data_ptr(), self.alpha[G][0].data_ptr(),
                    l.M, self.out[G][0].data_ptr(), sh), "conv_w8")))
        for G in self.groups:
            for i in self.tl:
                l = self.layers[i]

                def conv(G=G, i=i, l=l):
                    chk(L.fgq_conv2d(self.q[i].data_ptr(), fgq.ACT_TYPES[self.types[i]], self.sc[i].data_ptr(),
                                     self.B, l.H, l.W, l.C, l.R, l.S, l.stride, l.pad, l.groups,
                                     self.codes[G][i].data_ptr(), self.alpha[G][i].data_ptr(), l.M, G,
                                     self.out[G][i].data_ptr(), sh), "conv")
                    self.paths[(G, i)] = L.fgq_last_path()
                calls.append((f"conv_g{G}", conv))

        cur, e0 = None, None
        for fam, fn in calls:
            if timers is not None and fam != cur:
                if cur is not None:
                    e1 = torch.cuda.Event(enable_timing=True)
                    e1.record(stream)
                    timers.setdefault(cur, []).append((e0, e1))
                e0 = torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                cur = fam
            fn()
            if counts is not None:
                counts[fam] = counts.get(fam, 0) + 1
        if timers is not None and cur is not None:
            e1 = torch.cuda.Event(enable_timing=True)
            e1.record(stream)
            timers.setdefault(cur, []).append((e0, e1))


def timed_steps(W, stream, steps, warmup, flush=None):
    """Warm-up, then `steps` steps timed with one event pair around all of them (inputs
    larger than L2) or, with `flush` (a buffer larger than L2 written before each step),
    one event pair per step (median).  Returns (ms per step, family ms per step, counts)."""
    torch = W.torch
    with torch.cuda.stream(stream):
        for _ in range(max(3, warmup)):
            W.step(stream)
    torch.cuda.synchronize()
    timers, counts = {}, {}
    with torch.cuda.stream(stream):
        if flush is None:
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for _ in range(steps):
                W.step(stream, timers, counts)
            e1.record(stream)
            torch.cuda.synchronize()
            ms = e0.elapsed_time(e1) / steps
        else:
            per = []
            for _ in range(steps):
                flush.zero_()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                W.step(stream, timers, counts)
                e1.record(stream)
                torch.cuda.synchronize()
                per.append(e0.elapsed_time(e1))
            ms = statistics.median(per)
    fam = {f: sum(a.elapsed_time(b) for a, b in ev) / steps for f, ev in timers.items()}
    return ms, fam, counts


def check_status(fgq, stream, what):
    st = fgq.fgq_stream_status(stream)
    if st != fgq.FGQ_OK:
        raise RuntimeError(f"device error during {what}: {st}")


# ----------------------------------------------------------------------------- the other configurations

def measure_stack(dev, stream, peaks, name, layers, B, groups, act, first_w8, steps, warmup, fcs=()):
    """One configuration's step (ternarize + quantize + every contraction), its rate and its
    per-family rooflines."""
    import torch
    from paper_1705_01462_gb300 import fgq
    W = Workload(dev, B, layers, groups=groups, act=act, first_w8=first_w8, fcs=fcs)
    ms, fam, _ = timed_steps(W, stream, steps, warmup)
    check_status(fgq, stream, name)
    allc = list(layers) + list(fcs)
    fams = {}
    for f, v in sorted(fam.items()):
        if f.startswith("conv_g"):
            lay = allc[1:] if first_w8 else allc
            fams[f] = conv_roofline(lay, B, int(f[6:]), peaks, v / 1e3, ACT_BITS[act])
        elif f.startswith("ternarize_g"):
            fams[f] = hbm_roofline(ternarize_bytes(allc[1:] if first_w8 else allc, int(f[11:])), v / 1e3, peaks)
        elif f == "quantize_act":
            nb = sum(B * l.H * l.W * l.C * (32 + (8 if (first_w8 and i == 0) else ACT_BITS[act])) // 8
                     for i, l in enumerate(allc))
            fams[f] = hbm_roofline(nb, v / 1e3, peaks)
        else:
            fams[f] = family_roofline(f, allc, B, peaks, v / 1e3, act)
    layer_paths = {}
    for (G, i), p in W.paths.items():
        layer_paths.setdefault(f"conv_g{G}", {}).setdefault(str(p), 0)
        layer_paths[f"conv_g{G}"][str(p)] += 1
    out = {"workload": name, "ms_per_step": ms, "value": W.ops() / (ms / 1e3) / 1e12, "unit": UNIT,
           "families": {f: _round(r) for f, r in fams.items()}, "paths": layer_paths, "steps": steps}
    del W
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    return out


def _round(d):
    return {k: (round(v, 4) if isinstance(v, float) else v) for k, v in d.items()}


def measure_single_layer(dev, stream, peaks, flush, layer, B, groups, act, steps, warmup):
    """A single layer (ternarize + quantize + convolution per G) with the L2 flushed before
    every step: per G its ms, TOPS and roofline."""
    import torch
    from paper_1705_01462_gb300 import fgq
    res = {}
    for G in groups:
        W = Workload(dev, B, [layer], groups=(G,), act=act, first_w8=False)
        ms, fam, _ = timed_steps(W, stream, steps, warmup, flush=flush)
        check_status(fgq, stream, layer.name)
        conv = conv_roofline([layer], B, G, peaks, fam[f"conv_g{G}"] / 1e3, ACT_BITS[act])
        res[f"G{G}"] = {"ms_per_step": ms, "value": W.ops() / (ms / 1e3) / 1e12,
                        "conv_ms": fam[f"conv_g{G}"], "conv": _round(conv),
                        "path": W.paths.get((G, 0)), "family_ms": {k: round(v, 5) for k, v in fam.items()}}
        del W
    torch.cuda.empty_cache()
    return res


def measure_ternarize_set(dev, stream, peaks, flush, steps):
    """Standalone ternarization of the ResNet-50 weight set (53 convolutions and the fc, 25.5 M
    fp32 weights) at G = 4, 16 and 64, one fgq_ternarize_batch launch per G, L2 flushed."""
    import ctypes

    import torch
    from paper_1705_01462_gb300 import fgq, synth
    layers = synth.resnet50_convs() + [synth.resnet50_fc()]
    L = fgq.lib()
    ws = [synth.torch_weights(l, synth.layer_seed(i, 7), dev) for i, l in enumerate(layers)]
    n = len(layers)
    out = {"weights": sum(l.M * l.Kred for l in layers)}
    for G in (4, 16, 64):
        codes = [torch.empty((l.M, fgq.codes_words_per_row(l.Kred, G)), dtype=torch.int32, device=dev) for l in layers]
        alpha = [torch.empty((l.M, fgq.num_groups(l.Kred, G)), dtype=torch.float32, device=dev) for l in layers]
        args = (n, (ctypes.c_void_p * n)(*[w.data_ptr() for w in ws]), (ctypes.c_int * n)(*[l.M for l in layers]),
                (ctypes.c_int * n)(*[l.Kred for l in layers]), G,
                (ctypes.c_void_p * n)(*[c.data_ptr() for c in codes]), (ctypes.c_void_p * n)(*[a.data_ptr() for a in alpha]),
                stream.cuda_stream)
        for _ in range(3):
            assert L.fgq_ternarize_batch(*args) == 0
        per = []
        for _ in range(steps):
            flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            assert L.fgq_ternarize_batch(*args) == 0
            e1.record(stream)
            torch.cuda.synchronize()
            per.append(e0.elapsed_time(e1))
        ms = statistics.median(per)
        out[f"G{G}"] = _round(hbm_roofline(ternarize_bytes(layers, G), ms / 1e3, peaks))
    check_status(fgq, stream, "ternarize set")
    del ws
    torch.cuda.empty_cache()
    return out


def measure_fc_sweep(dev, stream, peaks, flush, steps):
    """Square FC GEMMs M = K in {4096, 8192, 16384} x batch {1, 64, 1024} at G = 4 and 64:
    the contraction alone (weights ternarized and activations quantized beforehand), L2
    flushed before every call."""
    import torch
    from paper_1705_01462_gb300 import fgq, synth
    L = fgq.lib()
    rows = []
    for n in (4096, 8192, 16384):
        layer = synth.ConvLayer(f"fc{n}", n, n, 1, 1, 1, 0, 1, 1)
        w = synth.torch_weights(layer, 11, dev)
        for G in GROUPS:
            codes, alpha = fgq.fgq_ternarize(w, G, stream=stream)
            for P in (1, 64, 1024):
                x = synth.torch_activations((P, n), 12, dev)
                q, sx = fgq.fgq_quantize_act(x, "s8", stream=stream)
                y = torch.empty((P, n), dtype=torch.float32, device=dev)

                def call():
                    st = L.fgq_gemm(q.data_ptr(), fgq.S8, sx.data_ptr(), P, n, codes.data_ptr(), alpha.data_ptr(),
                                    n, G, y.data_ptr(), stream.cuda_stream)
                    assert st == 0, st
                for _ in range(3):
                    call()
                per = []
                for _ in range(steps):
                    flush.zero_()
                    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    e0.record(stream)
                    call()
                    e1.record(stream)
                    torch.cuda.synchronize()
                    per.append(e0.elapsed_time(e1))
                ms = statistics.median(per)
                r = conv_roofline([layer], P, G, peaks, ms / 1e3, 8)
                rows.append({"M": n, "K": n, "P": P, "G": G, "path": L.fgq_last_path(), "us": round(ms * 1e3, 2),
                             "value": round(r["achieved"], 3), "bound": r["bound"], "frac": round(r["frac"], 4)})
        del w
    check_status(fgq, stream, "fc sweep")
    torch.cuda.empty_cache()
    return rows


def measure_configs(dev, stream, peaks, steps=5, warmup=3):
    import torch
    from paper_1705_01462_gb300 import synth
    flush = torch.empty(512 << 20, dtype=torch.uint8, device=dev)  # > 129 MB L2
    c = {}
    layer = synth.conv2x_3x3()
    c["1"] = {"workload": "ResNet-50 conv2_x 3x3 (64 filters, Kred 576, 56x56), batch 1, G=4, uint8; "
                          "ternarize 36,864 weights + quantize + convolution; L2 flushed before each step",
              **measure_single_layer(dev, stream, peaks, flush, layer, 1, (4,), "u8", 10, warmup)}
    c["2"] = {"workload": "the same layer at batch 32, G=64 (tensor cores) and G=4 side by side, uint8; L2 "
                          "flushed before each step; standalone ternarization of the 25.5 M ResNet-50 weights",
              **measure_single_layer(dev, stream, peaks, flush, layer, 32, (64, 4), "u8", 10, warmup),
              "ternarize_resnet50_weights": measure_ternarize_set(dev, stream, peaks, flush, 10)}
    c["4"] = measure_stack(dev, stream, peaks, "ResNet-101 conv stack (104 convs), batch 128, 224x224, packed "
                           "uint4 activations (first layer 8-bit weights and uint8 input), G=64",
                           synth.resnet101_convs(), 128, (64,), "u4", True, steps, warmup)
    c["5"] = measure_stack(dev, stream, peaks, "AlexNet convs + FCs, batch 256, int8 activations, G=4 and 64",
                           synth.alexnet_convs(), 256, GROUPS, "s8", False, steps, warmup, fcs=synth.alexnet_fcs())
    c["5"]["fc_sweep"] = measure_fc_sweep(dev, stream, peaks, flush, 5)
    del flush
    torch.cuda.empty_cache()
    return c


# ----------------------------------------------------------------------------- end to end through the C ABI

def measure_e2e(dev, W, steps, warmup):
    """The step end to end through the host-buffer entry point fgq_conv2d_host: per layer and
    G, one call copies the layer's fp32 weights and fp32 input from page-locked host memory,
    ternarizes (or 8-bit-quantizes) the weights, quantizes the input, runs the convolution and
    copies the fp32 output back.  Calls alternate over two streams, each with a device
    workspace of its own, so one layer's copies overlap the other's kernels."""
    import torch
    from paper_1705_01462_gb300 import fgq
    L = fgq.lib()
    layers, B = W.layers, W.B
    h_w = [w.to("cpu").pin_memory() for w in W.w]
    h_x = [x.to("cpu").pin_memory() for x in W.x]
    h_out = {G: [torch.empty(o.shape, dtype=torch.float32).pin_memory() for o in W.out[G]] for G in W.groups}
    calls = []
    for G in W.groups:
        for i, l in enumerate(layers):
            g_arg = 0 if (W.first_w8 and i == 0) else G
            calls.append((i, G, g_arg, fgq.ACT_TYPES[W.types[i]]))
    wsb = max(L.fgq_conv2d_host_workspace_bytes(t, B, layers[i].H, layers[i].W, layers[i].C, layers[i].R,
                                                 layers[i].S, layers[i].stride, layers[i].pad, layers[i].groups,
                                                 layers[i].M, ga) for i, _, ga, t in calls)
    streams = [torch.cuda.Stream(device=dev) for _ in range(2)]
    ws = [torch.empty(wsb, dtype=torch.uint8, device=dev) for _ in streams]

    def step():
        for k, (i, G, ga, t) in enumerate(calls):
            l = layers[i]
            s = streams[k % 2]
            st = L.fgq_conv2d_host(h_w[i].data_ptr(), h_x[i].data_ptr(), t, B, l.H, l.W, l.C, l.R, l.S, l.stride,
                                   l.pad, l.groups, l.M, ga, h_out[G][i].data_ptr(), ws[k % 2].data_ptr(), wsb,
                                   s.cuda_stream)
            if st != 0:
                raise RuntimeError(f"fgq_conv2d_host: {L.fgq_status_string(st).decode()}")

    for _ in range(max(2, warmup)):  # first DMA use of page-locked memory is slow
        step()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(streams[0])
    streams[1].wait_event(e0)
    for _ in range(steps):
        step()
    streams[0].wait_stream(streams[1])
    e1.record(streams[0])
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / steps
    for s in streams:
        check_status(fgq, s, "the end-to-end region")
    h2d = sum(h_w[i].numel() * 4 + h_x[i].numel() * 4 for i, _, _, _ in calls)
    d2h = sum(h_out[G][i].numel() * 4 for i, G, _, _ in calls)
    return ms, h2d, d2h


# ----------------------------------------------------------------------------- CPU oracle timing

def _oracle_worker(job):
    """One oracle process: prepare its layers' inputs (untimed: weights ternarized by the
    oracle at G = 4 and 64, one image quantized), then visit them in turn computing the
    grouped contraction at `npos` sampled output positions x all filters for both G, until
    `seconds` of compute have passed.  Returns (ops, busy seconds, visits)."""
    idx, seconds, seed, npos = job
    sys.path.insert(0, ROOT)
    import oracle as O
    from paper_1705_01462_gb300 import synth
    layers = synth.resnet50_convs()
    prep = {}
    for i in idx:
        l = layers[i]
        w = synth.weights(l, synth.layer_seed(i))
        x = synth.activations((1, l.H, l.W, l.C), synth.layer_seed(i, 1))
        q, sc, _, _ = O.quantize(x, O.U8)
        prep[i] = (q, sc, {G: O.ternarize(w, G)[:2] for G in GROUPS})
    rng = np.random.default_rng(seed)
    ops, busy, visits = 0, 0.0, 0
    while busy < seconds:
        for i in idx:
            if busy >= seconds:
                break
            l = layers[i]
            q, sc, tern = prep[i]
            pos = rng.choice(l.Ho * l.Wo, size=npos, replace=False)
            t0 = time.perf_counter()
            for G in GROUPS:
                t, al = tern[G]
                O.conv2d(q, sc, l.R, l.S, l.stride, l.pad, l.groups, t, al, G, positions=pos)
            busy += time.perf_counter() - t0
            ops += 2 * l.M * l.Kred * npos * len(GROUPS)
            visits += 1
    return ops, busy, visits


def oracle_sample(seconds, workers=0, seed=5, npos=8):
    """Times the CPU oracle's grouped contraction on a bounded sample of the workload, over
    `workers` processes (default: every host core), each taking its share of the 52 ternary
    ResNet-50 layers.  Returns (effective TOPS: the sum of the processes' rates, description,
    processes)."""
    import multiprocessing as mp

    import oracle as O
    O.lib()  # built once here, not by every process
    nw = workers or os.cpu_count() or 1
    nl = len(workload_layers())
    nw = min(nw, nl - 1)
    jobs = [(list(range(1 + k, nl, nw)), seconds, seed + k, npos) for k in range(nw)]
    with mp.get_context("spawn").Pool(nw) as pool:
        res = pool.map(_oracle_worker, jobs)
    rate = sum(o / b for o, b, _ in res if b > 0) / 1e12
    ops = sum(o for o, _, _ in res)
    visits = sum(v for _, _, v in res)
    desc = (f"{nw} oracle processes on {os.cpu_count()} host cores, each visiting its share of the 52 ternary "
            f"ResNet-50 layers and computing the grouped contraction at {npos} sampled output positions x all "
            f"filters for G=4 and G=64 ({visits} layer visits, {ops / 1e9:.2f} GOP effective, about {seconds:.0f} s "
            "of compute per process); weights ternarized and inputs quantized by the oracle beforehand")
    return rate, desc, nw


# ----------------------------------------------------------------------------- main

def dist_setup(args):
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def rank_seed_offset(rank):
    """Seed offset of a rank's synthetic inputs: every rank works on its own batch."""
    return rank * 7


def max_over_ranks(dist, value, device):
    """The maximum of a per-rank time over all ranks (the job is as slow as its slowest
    rank); dist is torch.distributed with an initialized group, or None for one rank."""
    if dist is None:
        return value
    import torch
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(ops_per_rank, world, ms_per_step):
    """Whole-job throughput in effective TOPS: the units all ranks processed over the
    (max-over-ranks) step time."""
    return ops_per_rank * world / (ms_per_step / 1e3) / 1e12


def run_reference(args, ws, rank):
    if rank != 0:
        return
    layers = workload_layers()
    per_step = max(2.0, min(15.0, 100.0 / max(1, args.steps + args.warmup)))
    workers = getattr(args, "cpu_workers", 0)
    for _ in range(args.warmup):
        oracle_sample(per_step * 0.25, workers)
    vals, descs, cores = [], [], 1
    for _ in range(args.steps):
        v, d, cores = oracle_sample(per_step, workers)
        vals.append(v)
        descs.append(d)
    value = statistics.mean(vals)
    ms_full_step = total_ops(layers, BATCH) / (value * 1e12) * 1e3  # extrapolated from the sampled rate
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_full_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "int64/f64", "data": "synthetic",
            "config": {"workload": "ResNet-50 conv stack (53 convs), batch 64, 224x224, uint8 DFP "
                                   "activations, ternary weights at G=4 and G=64",
                       "sampled": True, "ms_per_step": "extrapolated from the sampled rate to a full step"},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": descs[-1]},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_layers(args):
    """Times single convolutions of the ResNet-50 stack (fgq_conv2d through the C ABI, the
    weights ternarized and the input quantized beforehand), the L2 flushed before each call;
    prints one JSON line per layer."""
    import torch
    from paper_1705_01462_gb300 import fgq, synth
    dev = torch.device("cuda:0")
    torch.cuda.set_device(dev)
    L = fgq.lib()
    peaks = load_peaks()
    layers = {l.name: (i, l) for i, l in enumerate(synth.resnet50_convs())}
    stream = torch.cuda.Stream(device=dev)
    flush = torch.empty(512 << 20, dtype=torch.uint8, device=dev)
    path = {"auto": fgq.PATH_AUTO, "simt": fgq.PATH_SIMT, "tc": fgq.PATH_TC, "dense": fgq.PATH_DENSE}[args.path]
    B, G = args.batch, args.G
    for name in args.layer.split(","):
        i, l = layers[name]
        w = synth.torch_weights(l, synth.layer_seed(i), dev)
        x = synth.torch_activations((B, l.H, l.W, l.C), synth.layer_seed(i, 1), dev)
        with torch.cuda.stream(stream):
            codes, alpha = fgq.fgq_ternarize(w, G, stream=stream)
            q, sx = fgq.fgq_quantize_act(x, args.act, stream=stream)
        out = torch.empty((B, l.Ho, l.Wo, l.M), dtype=torch.float32, device=dev)
        torch.cuda.synchronize()
        fgq.fgq_set_path(path)

        def call():
            st = L.fgq_conv2d(q.data_ptr(), fgq.ACT_TYPES[args.act], sx.data_ptr(), B, l.H, l.W, l.C, l.R, l.S,
                              l.stride, l.pad, l.groups, codes.data_ptr(), alpha.data_ptr(), l.M, G, out.data_ptr(),
                              stream.cuda_stream)
            if st != 0:
                raise RuntimeError(f"fgq_conv2d {name}: {L.fgq_status_string(st).decode()}")
        for _ in range(2):
            call()
        per = []
        for _ in range(args.iters):
            with torch.cuda.stream(stream):
                flush.zero_()  # on the timed stream, ahead of the event
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            call()
            e1.record(stream)
            torch.cuda.synchronize()
            per.append(e0.elapsed_time(e1))
        check_status(fgq, stream, name)
        ms = statistics.median(per)
        r = conv_roofline([l], B, G, peaks, ms / 1e3, ACT_BITS[args.act])
        print(json.dumps({"layer": name, "batch": B, "G": G, "act": args.act, "path": L.fgq_last_path(),
                          "ms": round(ms, 5), "value": round(r["achieved"], 2), "unit": UNIT,
                          "roofline_frac": round(r["frac"], 4), "bound": r["bound"]}), flush=True)
        fgq.fgq_set_path(fgq.PATH_AUTO)


def main():
    args = parse()
    ws, rank, local = dist_setup(args)
    if args.impl == "reference":
        run_reference(args, ws, rank)
        return
    if args.layer:
        run_layers(args)
        return
    import torch
    from paper_1705_01462_gb300 import fgq
    assert torch.cuda.is_available(), "bench.py needs a CUDA GPU"
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    pg = None
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
        pg = dist
    fgq.lib()
    peaks = load_peaks()
    layers = workload_layers()
    B = args.batch
    W = Workload(dev, B, layers, seed_offset=rank_seed_offset(rank))
    stream = torch.cuda.Stream(device=dev)

    with torch.cuda.stream(stream):
        for _ in range(max(3, args.warmup)):
            W.step(stream)
    torch.cuda.synchronize()

    # ---- device-resident timed region
    if pg:
        pg.barrier()
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    timers, counts = {}, {}
    launches0 = fgq.fgq_launch_count()
    e_start = torch.cuda.Event(enable_timing=True)
    e_end = torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e_start.record(stream)
        for _ in range(args.steps):
            W.step(stream, timers, counts)
        e_end.record(stream)
    torch.cuda.synchronize()
    launches = fgq.fgq_launch_count() - launches0
    clk = clocks.stop()
    total_ms = e_start.elapsed_time(e_end)
    check_status(fgq, stream, "the timed region")
    total_ms = max_over_ranks(pg, total_ms, dev)
    ms_per_step = total_ms / args.steps
    ops_rank = total_ops(layers, B)
    value = whole_job_rate(ops_rank, ws, ms_per_step)
    fam_ms = {f: sum(a.elapsed_time(b) for a, b in ev) / args.steps for f, ev in timers.items()}
    if args.only == "step":
        if rank == 0:
            print(json.dumps({"only": "step", "ms_per_step": ms_per_step, "value": value,
                              "family_ms": {f: round(v, 4) for f, v in sorted(fam_ms.items())}}), flush=True)
        return

    fams = {f: family_roofline(f, layers, B, peaks, v / 1e3) for f, v in fam_ms.items()}
    dom = max(fam_ms, key=fam_ms.get)
    digest = source_digest()
    traffic_tab = load_traffic(digest)
    n_calls = counts[dom] / args.steps  # API calls of the family per step
    d = fams[dom]
    traffic = traffic_tab.get(dom)
    roofline = {"kernel": dom, "bound": d["bound"], "achieved": d["achieved"], "peak": d["peak"], "unit": d["unit"],
                "frac": d["frac"],
                "traffic": traffic * B / 64 if (traffic is not None and dom.startswith("conv")) else traffic,
                "peak_source": (f"{peaks['source']}: per-layer max(algorithmic bytes / {peaks['hbm_gbs']} GB/s, "
                                f"ops / {peaks['bf16_tflops']} TFLOP/s bf16) summed over the family"
                                if d["unit"] == UNIT else f"{peaks['source']}: HBM {peaks['hbm_gbs']} GB/s"),
                "algorithmic_bytes_per_launch": d["bytes"] / n_calls, "launches_per_step": n_calls,
                "sources": digest,
                "families": {f: _round(r) for f, r in sorted(fams.items())},
                "conv_layers_on_tc": {f"conv_g{G}": sum(1 for (g, _), p in W.paths.items() if g == G and p == 2)
                                      for G in GROUPS},
                "conv_layers": len(layers) - 1}

    # ---- end to end through the C ABI with host buffers
    e2e_ms, h2d, d2h = measure_e2e(dev, W, max(1, args.e2e_steps), args.warmup)
    e2e_ms = max_over_ranks(pg, e2e_ms, dev)
    e2e_value = whole_job_rate(ops_rank, ws, e2e_ms)
    del W
    torch.cuda.empty_cache()

    configs = None
    if not args.no_configs:
        configs = measure_configs(dev, stream, peaks)

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        v, desc, cores = oracle_sample(args.cpu_seconds, args.cpu_workers)
        cpu = {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": desc}

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "u8xternary->int32->f32", "data": "synthetic",
                "config": {"workload": f"ResNet-50 conv stack (53 convs), batch {B} per GPU, 224x224, uint8 DFP "
                                       "activations, ternary weights at G=4 and G=64, first layer 8-bit weights",
                           "ops_per_step_per_gpu": ops_rank,
                           "l2": "no flush: per-step working set ~9 GB >> 129 MB L2",
                           "parallelism": f"dp{ws} (independent batches, no collective)"},
                "roofline": roofline, "clocks": clk, "gpu_launches": launches,
                "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                        "ms_per_step": e2e_ms, "steps": max(1, args.e2e_steps),
                        "api": "fgq_conv2d_host per layer and G (one cudaMemcpyAsync per buffer, page-locked host "
                               "memory), two streams with a workspace each"},
                "cpu_baseline": cpu, "configs": configs}
        print(json.dumps(line), flush=True)
    if pg:
        pg.barrier()
        pg.destroy_process_group()


if __name__ == "__main__":
    main()
