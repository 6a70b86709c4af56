"""Chained quantized ResNet forward on the FGQ kernels (Section 4: ternary weights, 8-bit DFP
activations between layers, the first layer at 8-bit weights).

    python -m paper_1705_01462_gb300.resnet --batch 64 --G 4 --iters 5

Two forwards over the same graph (the bottleneck stack of synth.resnet50_convs, Caffe
layout: stride on the first 1x1 of a stage's first block and on its projection):

* dynamic: every conv writes fp32, every tensor gets its own DFP scale from
  fgq_quantize_act (dynamic fixed point, Section 4), residual sums are fp32 and then
  quantized;
* fused: the same graph with per-tensor scales fixed beforehand (those a dynamic run on a
  calibration batch found), so every conv requantizes in its epilogue (fgq_conv2d_rq) and
  the residual add writes codes (fgq_add_codes): no fp32 tensor between layers.

Graph (`graph`): conv1 (8-bit weights) -> u8 (ReLU) -> 3x3/2 max pool -> blocks; a block
is 2a (1x1) -> u8 -> 2b (3x3) -> u8 -> 2c (1x1) -> s8, the shortcut is the projection
branch1 -> s8 (first block of a stage) or the block input, and the block output is
u8(2c + shortcut) (the ReLU after the addition).  BN is taken as folded into the weights.
The command line draws random-init weights ~ N(0, 2/fan_in) and prints one JSON line with
the times of both forwards and how far their output codes agree.
"""
from __future__ import annotations

import argparse
import json
import os
import sys
from dataclasses import dataclass
from typing import Dict, List, Optional, Tuple

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))


@dataclass
class Tensor8:
    """8-bit codes (NHWC) with their type and device scale 2^E."""
    q: object
    type: str
    scale: object
    shape: tuple


@dataclass(frozen=True)
class Node:
    """One step of the forward: its output tensor's name, kind ("quant", "conv", "maxpool",
    "add"), input tensor names, conv layer index (or None) and output code type."""
    name: str
    kind: str
    inputs: Tuple[str, ...]
    layer: Optional[int]
    out_type: str


def graph(layers) -> List[Node]:
    """The forward's steps in execution order, for synth.resnet50_convs / resnet101_convs."""
    assert layers[0].name == "conv1"
    nodes = [Node("input", "quant", (), None, "u8"), Node("conv1", "conv", ("input",), 0, "u8"),
             Node("pool", "maxpool", ("conv1",), None, "u8")]
    x, i, bi = "pool", 1, 0
    while i < len(layers):
        assert layers[i].name.endswith("branch2a"), layers[i].name
        a, b, c = f"b{bi}a", f"b{bi}b", f"b{bi}c"
        nodes += [Node(a, "conv", (x,), i, "u8"), Node(b, "conv", (a,), i + 1, "u8"),
                  Node(c, "conv", (b,), i + 2, "s8")]
        i += 3
        short = x
        if i < len(layers) and layers[i].name.endswith("branch1"):
            short = f"b{bi}p"
            nodes.append(Node(short, "conv", (x,), i, "s8"))
            i += 1
        x = f"b{bi}out"
        nodes.append(Node(x, "add", (c, short), None, "u8"))
        bi += 1
    return nodes


def last_uses(nodes: List[Node]) -> Dict[int, List[str]]:
    """Step index -> tensors read for the last time there (freed after that step)."""
    last: Dict[str, int] = {}
    for j, n in enumerate(nodes):
        for k in n.inputs:
            last[k] = j
    out: Dict[int, List[str]] = {}
    for k, j in last.items():
        out.setdefault(j, []).append(k)
    return out


class QuantResNet:
    """params: optional prepared weights (w8 = (wq int8 [M][Kred], wscale fp32 [M]) for conv1,
    tern = [None, (codes, alpha), ...] for the ternary layers), device tensors; drawn from
    synth.torch_weights and quantized on the GPU when absent."""

    def __init__(self, layers, G: int, dev, seed: int = 1, params=None):
        import torch
        from paper_1705_01462_gb300 import fgq, synth
        self.torch, self.fgq, self.layers, self.G, self.dev = torch, fgq, layers, G, dev
        self.nodes = graph(layers)
        self.frees = last_uses(self.nodes)
        if params is None:
            w8 = fgq.fgq_quantize_weights_w8(synth.torch_weights(layers[0], synth.layer_seed(0, seed), dev))
            tern = [None] + [fgq.fgq_ternarize(synth.torch_weights(l, synth.layer_seed(i, seed), dev), G)
                             for i, l in enumerate(layers) if i > 0]
            params = (w8, tern)
        self.w8, self.tern = params
        self.scales: Dict[str, object] = {}  # output scale (device fp32 [1]) per tensor name
        self.input_scale = 0.0

    def set_scales(self, scales: Dict[str, float]):
        """Fix the per-tensor scales 2^E the fused forward requantizes to."""
        self.scales = {k: self.torch.tensor([float(v)], dtype=self.torch.float32, device=self.dev)
                       for k, v in scales.items()}
        self.input_scale = float(scales["input"])

    def calibrate(self, x_fp32):
        """A dynamic forward; its per-tensor scales become the fused forward's."""
        self.forward_dynamic(x_fp32)
        self.input_scale = float(self.scales["input"].item())

    # -------------------------------------------------------------------- steps
    def _conv(self, n: Node, x: Tensor8, fused: bool):
        fgq, l = self.fgq, self.layers[n.layer]
        B, H, W, C = x.shape
        Ho, Wo = fgq.conv_out_hw(H, W, l.R, l.S, l.stride, l.pad)
        geo = (B, H, W, C, l.R, l.S, l.stride, l.pad, l.groups)
        if n.layer == 0:
            wq, ws = self.w8
            if fused:
                out = fgq.fgq_conv2d_w8_rq(x.q, x.type, x.scale, *geo, wq, ws, l.M, n.out_type, self.scales[n.name])
            else:
                out = fgq.fgq_conv2d_w8(x.q, x.type, x.scale, *geo, wq, ws, l.M)
        else:
            codes, alpha = self.tern[n.layer]
            if fused:
                out = fgq.fgq_conv2d_rq(x.q, x.type, x.scale, *geo, codes, alpha, l.M, self.G, n.out_type,
                                        self.scales[n.name])
            else:
                out = fgq.fgq_conv2d(x.q, x.type, x.scale, *geo, codes, alpha, l.M, self.G)
        return out, (B, Ho, Wo, l.M)

    def _quant(self, y, n: Node) -> Tensor8:
        q, s = self.fgq.fgq_quantize_act(y, n.out_type)
        self.scales[n.name] = s
        return Tensor8(q.view(y.shape), n.out_type, s, tuple(y.shape))

    def _forward(self, x_fp32, fused: bool, trace: Optional[dict]):
        fgq = self.fgq
        t: Dict[str, Tensor8] = {}
        for j, n in enumerate(self.nodes):
            if n.kind == "quant":
                if fused:
                    q, _ = fgq.fgq_quantize_act(x_fp32, n.out_type, scale_in=self.input_scale)
                    out = Tensor8(q.view(x_fp32.shape), n.out_type, self.scales[n.name], tuple(x_fp32.shape))
                else:
                    out = self._quant(x_fp32, n)
            elif n.kind == "conv":
                y, shape = self._conv(n, t[n.inputs[0]], fused)
                out = Tensor8(y, n.out_type, self.scales[n.name], shape) if fused else self._quant(y, n)
            elif n.kind == "maxpool":
                x = t[n.inputs[0]]
                B, H, W, C = x.shape
                q = fgq.fgq_maxpool_u8(x.q, B, H, W, C, 3, 2, 1)
                out = Tensor8(q, x.type, x.scale, tuple(q.shape))
            else:  # add
                a, b = t[n.inputs[0]], t[n.inputs[1]]
                if fused:
                    q = fgq.fgq_add_codes(a.q, a.type, a.scale, b.q, b.type, b.scale, n.out_type, self.scales[n.name])
                    out = Tensor8(q, n.out_type, self.scales[n.name], a.shape)
                else:
                    out = self._quant(fgq.fgq_add_codes(a.q, a.type, a.scale, b.q, b.type, b.scale), n)
            t[n.name] = out
            if trace is not None:
                trace[n.name] = out
            for k in self.frees.get(j, ()):
                t.pop(k, None)
        return t[self.nodes[-1].name]

    def forward_dynamic(self, x_fp32, trace: Optional[dict] = None) -> Tensor8:
        """Every tensor quantized with its own DFP scale (and the scales recorded)."""
        return self._forward(x_fp32, False, trace)

    def forward_fused(self, x_fp32, trace: Optional[dict] = None) -> Tensor8:
        """The same graph at the fixed scales: requantizing epilogues, no fp32 tensors between
        layers."""
        assert self.input_scale > 0, "set_scales or calibrate first"
        return self._forward(x_fp32, True, trace)


def main():
    import torch
    from paper_1705_01462_gb300 import fgq, synth

    ap = argparse.ArgumentParser()
    ap.add_argument("--batch", type=int, default=64)
    ap.add_argument("--G", type=int, default=4)
    ap.add_argument("--iters", type=int, default=5)
    ap.add_argument("--hw", type=int, default=224)
    args = ap.parse_args()
    dev = torch.device("cuda:0")
    layers = synth.resnet50_convs()
    net = QuantResNet(layers, args.G, dev)
    x = synth.torch_activations((args.batch, args.hw, args.hw, 3), 7, dev)
    net.calibrate(x)
    out = {"batch": args.batch, "G": args.G, "hw": args.hw, "convs": len(layers)}
    for name, fwd in (("dynamic", net.forward_dynamic), ("fused", net.forward_fused)):
        for _ in range(2):
            fwd(x)
        torch.cuda.synchronize()
        ts = []
        for _ in range(args.iters):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            n0 = fgq.fgq_launch_count()
            e0.record()
            y = fwd(x)
            e1.record()
            torch.cuda.synchronize()
            ts.append(e0.elapsed_time(e1))
            out[f"{name}_launches"] = fgq.fgq_launch_count() - n0
        ts.sort()
        out[f"{name}_ms"] = round(ts[len(ts) // 2], 3)
        out[f"{name}_images_per_s"] = round(args.batch / ts[len(ts) // 2] * 1e3, 1)
    out["fused_speedup"] = round(out["dynamic_ms"] / out["fused_ms"], 3)
    yd = net.forward_dynamic(x)
    net.input_scale = float(net.scales["input"].item())
    yf = net.forward_fused(x)
    torch.cuda.synchronize()
    d = (yd.q.to(torch.int16) - yf.q.to(torch.int16)).abs()
    out["codes_equal_frac"] = float((d == 0).float().mean().item())
    out["out_nonzero_frac"] = float((yf.q != 0).float().mean().item())
    assert fgq.fgq_stream_status() == fgq.FGQ_OK
    print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
