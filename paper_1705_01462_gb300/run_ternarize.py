"""Time the ternarizers on the ResNet-50 weight set and compare their ternary error.

    python -m paper_1705_01462_gb300.run_ternarize --G 4,16,64 --iters 5

For each G: the exact per-group search (Eq. 5), the two analytical thresholds per group
(Lemma 1's mean |w|, the Gaussian-model z* rms(w)) and the one-threshold-one-alpha-per-layer
baseline of each rule, all 52 ternary conv layers of ResNet-50 (seeded synthetic weights
~ N(0, 2/fan_in)).  Reports, per variant, the CUDA-event time of the whole weight set, its
HBM throughput (fp32 weights in, 2-bit codes and fp32 alphas out) and the ternary error
sum ||w - alpha t||^2 over the set relative to the exact rule's.  One JSON line per (G,
variant).
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
    ap.add_argument("--G", default="4,16,64")
    ap.add_argument("--iters", type=int, default=5)
    args = ap.parse_args()
    dev = torch.device("cuda:0")
    layers = synth.resnet50_convs()[1:]
    ws = [synth.torch_weights(l, synth.layer_seed(i + 1), dev) for i, l in enumerate(layers)]
    variants = [("exact", None, False), ("lemma1_group", fgq.RULE_EXP, False), ("gauss_group", fgq.RULE_GAUSS, False),
                ("lemma1_layer", fgq.RULE_EXP, True), ("gauss_layer", fgq.RULE_GAUSS, True)]
    L = fgq.lib()
    sh = torch.cuda.current_stream().cuda_stream
    wsb = L.fgq_ternarize_threshold_workspace_bytes()
    scratch = torch.empty(wsb, dtype=torch.uint8, device=dev)
    for G in (int(g) for g in args.G.split(",")):
        e_exact = None
        out = [(torch.empty((l.M, fgq.codes_words_per_row(l.Kred, G)), dtype=torch.int32, device=dev),
                torch.empty((l.M, fgq.num_groups(l.Kred, G)), dtype=torch.float32, device=dev)) for l in layers]
        for name, rule, per_layer in variants:
            def run():  # outputs preallocated; the calls go straight to the C ABI
                for l, w, (c, a) in zip(layers, ws, out):
                    if rule is None:
                        st = L.fgq_ternarize(w.data_ptr(), l.M, l.Kred, G, c.data_ptr(), a.data_ptr(), sh)
                    else:
                        st = L.fgq_ternarize_threshold(w.data_ptr(), l.M, l.Kred, G, rule, int(per_layer), c.data_ptr(),
                                                       a.data_ptr(), scratch.data_ptr(), wsb, None, sh)
                    assert st == 0
                return out
            out = run()
            torch.cuda.synchronize()
            ts = []
            for _ in range(args.iters):
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                out = run()
                e1.record()
                torch.cuda.synchronize()
                ts.append(e0.elapsed_time(e1))
            err = sum(float(fgq.fgq_ternary_error(w, c, a, G).sum()) for w, (c, a) in zip(ws, out))
            if e_exact is None:
                e_exact = err
            nbytes = sum(w.numel() * 4 + c.numel() * 4 + a.numel() * 4 for w, (c, a) in zip(ws, out))
            ms = min(ts)
            print(json.dumps({"G": G, "variant": name, "ms": round(ms, 4), "GB_per_s": round(nbytes / ms / 1e6, 1),
                              "ternary_error": err, "error_vs_exact": round(err / e_exact, 4),
                              "weights": int(sum(w.numel() for w in ws))}), flush=True)
    assert fgq.fgq_stream_status() == fgq.FGQ_OK


if __name__ == "__main__":
    main()
