"""Run the FGQ hot path on one convolution layer and time its kernels.

    python -m paper_1705_01462_gb300.run_layer --layer res2a_branch2c --batch 64 --G 4 --iters 3
    python -m paper_1705_01462_gb300.run_layer --shape C,M,R,S,stride,pad,H,W --batch 8 --G 64

Layers are named as in the ResNet-50 stack (synth.resnet50_convs) or given as a shape.
Inputs are seeded synthetic tensors; each iteration quantizes the activations and runs the
grouped ternary convolution once (weights are ternarized once beforehand).  Prints one JSON
line with the per-kernel CUDA-event times.  Useful as a small, single-kernel case for ncu.
"""
from __future__ import annotations

import argparse
import json
import os
import sys

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))


def main():
    import torch
    from paper_1705_01462_gb300 import fgq, synth

    ap = argparse.ArgumentParser()
    ap.add_argument("--layer", default="res2a_branch2b")
    ap.add_argument("--shape", default=None, help="C,M,R,S,stride,pad,H,W[,groups]")
    ap.add_argument("--batch", type=int, default=32)
    ap.add_argument("--G", type=int, default=4)
    ap.add_argument("--act", default="u8")
    ap.add_argument("--iters", type=int, default=3)
    ap.add_argument("--path", default="auto", choices=["auto", "simt", "tc"])
    a = ap.parse_args()
    if a.shape:
        v = [int(t) for t in a.shape.split(",")]
        layer = synth.ConvLayer("custom", *v[:8], groups=v[8] if len(v) > 8 else 1)
    else:
        layer = next(l for l in synth.resnet50_convs() if l.name == a.layer)
    dev = torch.device("cuda:0")
    B, G = a.batch, a.G
    w = synth.torch_weights(layer, 1, dev)
    x = synth.torch_activations((B, layer.H, layer.W, layer.C), 2, dev)
    fgq.fgq_set_path({"auto": fgq.PATH_AUTO, "simt": fgq.PATH_SIMT, "tc": fgq.PATH_TC}[a.path])
    codes, alpha = fgq.fgq_ternarize(w, G)
    n = x.numel()
    q = torch.empty(fgq.act_bytes(n, a.act), dtype=torch.uint8, device=dev)
    sc = torch.empty(1, dtype=torch.float32, device=dev)
    ws = torch.empty(max(4, fgq.quantize_act_workspace_bytes(n)), dtype=torch.uint8, device=dev)
    out = torch.empty((B, layer.Ho, layer.Wo, layer.M), dtype=torch.float32, device=dev)
    tq, tc = [], []
    for _ in range(a.iters):
        e = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
        e[0].record()
        fgq.fgq_quantize_act(x, a.act, q=q, scale_out=sc, workspace=ws)
        e[1].record()
        fgq.fgq_conv2d(q, a.act, sc, B, layer.H, layer.W, layer.C, layer.R, layer.S, layer.stride, layer.pad,
                       layer.groups, codes, alpha, layer.M, G, out=out)
        e[2].record()
        torch.cuda.synchronize()
        tq.append(e[0].elapsed_time(e[1]))
        tc.append(e[1].elapsed_time(e[2]))
    st = fgq.fgq_stream_status()
    ops = layer.ops(B)
    print(json.dumps({"layer": layer.as_dict(), "batch": B, "G": G, "act": a.act, "path": fgq.fgq_last_path(),
                      "status": st, "quantize_ms": tq, "conv_ms": tc,
                      "conv_effective_tops": ops / (min(tc) / 1e3) / 1e12}))
    if st != fgq.FGQ_OK:
        sys.exit(1)


if __name__ == "__main__":
    main()
