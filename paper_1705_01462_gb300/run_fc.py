"""Fully connected (GEMM) sweep: the grouped ternary contraction at small batch, with fp32
or fixed-point (8-/4-bit) alphas.

    python -m paper_1705_01462_gb300.run_fc --sizes 4096,8192,16384 --batch 1,8 --G 4,64

For each M = K, batch P and G: the few-row path with fp32 alphas, with 8-bit and with
4-bit alphas, and the tiled CUDA-core kernel (forced) with fp32 alphas, timed with CUDA
events after warm-up; the L2 (129 MB) is flushed by writing a 256 MB buffer before every
timed call.  Bytes per call = 2-bit codes + alphas (+ row scales) + activations + fp32
outputs; GB/s is that over the call time.  One JSON line per case.
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
    ap.add_argument("--sizes", default="4096,8192,16384")
    ap.add_argument("--batch", default="1,8")
    ap.add_argument("--G", default="4,64")
    ap.add_argument("--iters", type=int, default=10)
    args = ap.parse_args()
    dev = torch.device("cuda:0")
    L = fgq.lib()
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    s = torch.cuda.current_stream()
    for n in (int(v) for v in args.sizes.split(",")):
        w = synth.torch_weights_matrix(n, n, 1, dev)
        for G in (int(v) for v in args.G.split(",")):
            codes, alpha = fgq.fgq_ternarize(w, G)
            aq8, sc8 = fgq.fgq_quantize_alpha(alpha, 8)
            aq4, sc4 = fgq.fgq_quantize_alpha(alpha, 4)
            for P in (int(v) for v in args.batch.split(",")):
                x = synth.torch_activations((P, n), 2, dev)
                q, sx = fgq.fgq_quantize_act(x, "u8")
                y = torch.empty((P, n), device=dev)
                ng = alpha.shape[1]
                variants = [("gemv_alpha_fp32", fgq.PATH_AUTO, None, 4 * n * ng),
                            ("gemv_alpha_8bit", fgq.PATH_AUTO, (aq8, 8, sc8), n * ng + 4 * n),
                            ("gemv_alpha_4bit", fgq.PATH_AUTO, (aq4, 4, sc4), n * ((ng + 1) // 2) + 4 * n),
                            ("tiled_alpha_fp32", fgq.PATH_SIMT, None, 4 * n * ng)]
                for name, path, qa, abytes in variants:
                    fgq.fgq_set_path(path)

                    def call():
                        if qa is None:
                            st = L.fgq_gemm(q.data_ptr(), fgq.U8, sx.data_ptr(), P, n, codes.data_ptr(),
                                            alpha.data_ptr(), n, G, y.data_ptr(), s.cuda_stream)
                        else:
                            st = L.fgq_gemm_qa(q.data_ptr(), fgq.U8, sx.data_ptr(), P, n, codes.data_ptr(),
                                               qa[0].data_ptr(), qa[1], qa[2].data_ptr(), n, G, y.data_ptr(),
                                               s.cuda_stream)
                        assert st == 0, st
                    for _ in range(3):
                        call()
                    ts = []
                    for _ in range(args.iters):
                        flush.zero_()
                        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                        e0.record()
                        call()
                        e1.record()
                        torch.cuda.synchronize()
                        ts.append(e0.elapsed_time(e1))
                    ts.sort()
                    ms = ts[len(ts) // 2]
                    nbytes = codes.numel() * 4 + abytes + q.numel() + 4 * P * n
                    print(json.dumps({"M": n, "K": n, "P": P, "G": G, "variant": name, "path": L.fgq_last_path(),
                                      "us": round(ms * 1e3, 2), "bytes": nbytes, "GB_per_s": round(nbytes / ms / 1e6, 1),
                                      "effective_TOPS": round(2.0 * n * n * P / ms / 1e9, 2)}), flush=True)
                fgq.fgq_set_path(fgq.PATH_AUTO)
    assert fgq.fgq_stream_status() == fgq.FGQ_OK


if __name__ == "__main__":
    main()
