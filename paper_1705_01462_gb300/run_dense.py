"""Folding the group scales into the weights: the dense tensor-core path against the
group-sum kernels, over the ternary convolutions of the ResNet-50 stack.

    python -m paper_1705_01462_gb300.run_dense --batch 64 --G 4,64 --iters 5

For each G and each of the 52 ternary layers (inputs quantized to u8 once): the automatic
path with fp32 alphas (fgq_conv2d), the dense path with 8-bit fixed-point alphas
(fgq_conv2d_qa, the automatic choice for them), the dense path with 4-bit alphas, and the
dense path with fp32 alphas split into two fp16 parts (forced).  Each call is timed with
CUDA events (median of --iters after one warm-up), the 129 MB L2 flushed by writing a
256 MB buffer before every timed call; the fold of the weights runs inside each dense call
and is included.  Prints one JSON line per G with the stack totals in effective TOPS
(2 M P Kred summed over the layers / summed medians) and the per-layer times.

--stack instead enqueues the whole stack back to back per variant, every layer's inputs and
outputs resident (3.4 GB at batch 64, far above the L2), and times each pass with one pair
of CUDA events (median of --iters passes after one warm-up pass): host enqueue overlaps the
GPU as in a forward pass, so the figure is the kernels' own throughput.
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
    ap.add_argument("--batch", type=int, default=64)
    ap.add_argument("--G", default="4,64")
    ap.add_argument("--iters", type=int, default=5)
    ap.add_argument("--layers", default="", help="comma-separated layer names (default: all)")
    ap.add_argument("--variants", default="", help="comma-separated variant names (default: all)")
    ap.add_argument("--stack", action="store_true", help="time whole-stack passes instead of single calls")
    args = ap.parse_args()
    only_layers = set(v for v in args.layers.split(",") if v)
    only_variants = set(v for v in args.variants.split(",") if v)
    dev = torch.device("cuda:0")
    B = args.batch
    layers = synth.resnet50_convs()[1:]
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    L = fgq.lib()
    s = torch.cuda.current_stream()
    outs = {}
    if args.stack:
        return stack_mode(args, layers, only_layers, only_variants)
    for G in (int(v) for v in args.G.split(",")):
        totals, per_layer, paths = {}, [], {}
        ops_total = 0
        for i, l in enumerate(layers):
            if only_layers and l.name not in only_layers:
                continue
            w = synth.torch_weights(l, synth.layer_seed(i + 1), dev)
            codes, alpha = fgq.fgq_ternarize(w, G)
            aq8, sc8 = fgq.fgq_quantize_alpha(alpha, 8)
            aq4, sc4 = fgq.fgq_quantize_alpha(alpha, 4)
            x = synth.torch_activations((B, l.H, l.W, l.C), 2 + i, dev)
            q, sx = fgq.fgq_quantize_act(x, "u8")
            del x
            out = torch.empty((B, l.Ho, l.Wo, l.M), dtype=torch.float32, device=dev)
            geo = (B, l.H, l.W, l.C, l.R, l.S, l.stride, l.pad, l.groups)
            ops = 2 * l.M * l.P(B) * l.Kred
            ops_total += ops

            def conv():
                return L.fgq_conv2d(q.data_ptr(), fgq.U8, sx.data_ptr(), *geo, codes.data_ptr(), alpha.data_ptr(),
                                    l.M, G, out.data_ptr(), s.cuda_stream)

            def conv_qa(aq, bits, asc):
                return lambda: L.fgq_conv2d_qa(q.data_ptr(), fgq.U8, sx.data_ptr(), *geo, codes.data_ptr(),
                                               aq.data_ptr(), bits, asc.data_ptr(), l.M, G, out.data_ptr(),
                                               s.cuda_stream)

            variants = [("alpha_fp32", fgq.PATH_AUTO, conv), ("alpha_8bit", fgq.PATH_AUTO, conv_qa(aq8, 8, sc8)),
                        ("alpha_4bit", fgq.PATH_AUTO, conv_qa(aq4, 4, sc4)),
                        ("alpha_fp32_split_fold", fgq.PATH_DENSE, conv)]
            row = {"layer": l.name, "gop": round(ops / 1e9, 3)}
            for name, path, call in variants:
                if only_variants and name not in only_variants:
                    continue
                fgq.fgq_set_path(path)
                st = call()
                if st != fgq.FGQ_OK:  # the dense path does not cover this shape
                    row[name] = None
                    fgq.fgq_set_path(fgq.PATH_AUTO)
                    continue
                paths.setdefault(name, {}).setdefault(L.fgq_last_path(), 0)
                paths[name][L.fgq_last_path()] += 1
                ts = []
                for _ in range(args.iters):
                    flush.zero_()
                    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    e0.record()
                    st = call()
                    e1.record()
                    torch.cuda.synchronize()
                    assert st == fgq.FGQ_OK, st
                    ts.append(e0.elapsed_time(e1))
                ts.sort()
                ms = ts[len(ts) // 2]
                row[name] = round(ms, 4)
                totals[name] = totals.get(name, 0.0) + ms
                fgq.fgq_set_path(fgq.PATH_AUTO)
            per_layer.append(row)
            del q, out
        assert fgq.fgq_stream_status() == fgq.FGQ_OK
        res = {"G": G, "batch": B, "gop": round(ops_total / 1e9, 2),
               "paths": {k: {str(p): n for p, n in v.items()} for k, v in paths.items()},
               "total_ms": {k: round(v, 3) for k, v in totals.items()},
               "effective_tops": {k: round(ops_total / (v * 1e-3) / 1e12, 1) for k, v in totals.items()
                                  if all(r.get(k) is not None for r in per_layer)},
               "layers_timed": len(per_layer),
               "per_layer": per_layer}
        outs[G] = res
        print(json.dumps(res), flush=True)


def stack_mode(args, layers, only_layers, only_variants):
    import torch
    from paper_1705_01462_gb300 import fgq, synth
    dev = torch.device("cuda:0")
    B = args.batch
    L = fgq.lib()
    s = torch.cuda.current_stream()
    sel = [(i, l) for i, l in enumerate(layers) if not only_layers or l.name in only_layers]
    qs, outs = [], []
    for i, l in sel:
        x = synth.torch_activations((B, l.H, l.W, l.C), 2 + i, dev)
        qs.append(fgq.fgq_quantize_act(x, "u8"))
        del x
        outs.append(torch.empty((B, l.Ho, l.Wo, l.M), dtype=torch.float32, device=dev))
    ops_total = sum(2 * l.M * l.P(B) * l.Kred for _, l in sel)
    for G in (int(v) for v in args.G.split(",")):
        wts = []
        for i, l in sel:
            codes, alpha = fgq.fgq_ternarize(synth.torch_weights(l, synth.layer_seed(i + 1), dev), G)
            wts.append((codes, alpha, fgq.fgq_quantize_alpha(alpha, 8), fgq.fgq_quantize_alpha(alpha, 4)))
        res = {"G": G, "batch": B, "mode": "stack", "layers": len(sel), "gop": round(ops_total / 1e9, 2), "ms": {},
               "effective_tops": {}, "paths": {}}
        for name, path in (("alpha_fp32", fgq.PATH_AUTO), ("alpha_8bit", fgq.PATH_AUTO), ("alpha_4bit", fgq.PATH_AUTO),
                           ("alpha_fp32_split_fold", fgq.PATH_DENSE)):
            if only_variants and name not in only_variants:
                continue
            fgq.fgq_set_path(path)
            paths = {}

            def one_pass():
                for (i, l), (q, sx), out, (codes, alpha, (aq8, s8), (aq4, s4)) in zip(sel, qs, outs, wts):
                    geo = (B, l.H, l.W, l.C, l.R, l.S, l.stride, l.pad, l.groups)
                    if name in ("alpha_fp32", "alpha_fp32_split_fold"):
                        st = L.fgq_conv2d(q.data_ptr(), fgq.U8, sx.data_ptr(), *geo, codes.data_ptr(), alpha.data_ptr(),
                                          l.M, G, out.data_ptr(), s.cuda_stream)
                    else:
                        aq, bits, asc = (aq8, 8, s8) if name == "alpha_8bit" else (aq4, 4, s4)
                        st = L.fgq_conv2d_qa(q.data_ptr(), fgq.U8, sx.data_ptr(), *geo, codes.data_ptr(), aq.data_ptr(),
                                             bits, asc.data_ptr(), l.M, G, out.data_ptr(), s.cuda_stream)
                    assert st == fgq.FGQ_OK, (name, l.name, st)
                    paths[str(L.fgq_last_path())] = paths.get(str(L.fgq_last_path()), 0) + 1

            one_pass()
            torch.cuda.synchronize()
            ts = []
            for _ in range(args.iters):
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                one_pass()
                e1.record()
                torch.cuda.synchronize()
                ts.append(e0.elapsed_time(e1))
            ts.sort()
            ms = ts[len(ts) // 2]
            res["ms"][name] = round(ms, 3)
            res["effective_tops"][name] = round(ops_total / (ms * 1e-3) / 1e12, 1)
            res["paths"][name] = {k: v // (args.iters + 1) for k, v in paths.items()}
            fgq.fgq_set_path(fgq.PATH_AUTO)
        assert fgq.fgq_stream_status() == fgq.FGQ_OK
        print(json.dumps(res), flush=True)


if __name__ == "__main__":
    main()
