"""CPU checks of the benchmark's host-side arithmetic: the peaks it derives from unit counts
and clocks, the blended roofline of a family that runs on several kernels, the per-step
operation count and the traffic table it reads."""
import importlib.util
import os

import pytest

from paper_1705_01462_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    spec = importlib.util.spec_from_file_location("bench_module", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_alu_peak(bench):
    # G = 4: one dp4a (FMA-heavy pipe, 64 lanes/clk/SM) and an add + FMA (128 lanes/clk/SM
    # shared) per unit of 8 effective ops -> max(1/64, 3/128) = 3/128 clk per unit per SM
    assert bench.alu_peak_tops(4, 152, 2.07e9) == pytest.approx(152 * 2.07e9 * 8 / (3 / 128) / 1e12)
    assert bench.alu_peak_tops(4, 152, 2.07e9) == pytest.approx(107.4, abs=0.05)
    # G = 64: 16 dp4a per unit dominate -> 16/64 clk for 128 ops
    assert bench.alu_peak_tops(64, 152, 2.07e9) == pytest.approx(152 * 2.07e9 * 128 / (16 / 64) / 1e12)


def test_tc_peak(bench):
    # G = 4: the MMA bound is a quarter of the bf16 peak (3 of 4 products are structural
    # zeros), the epilogue one FMA per 8 effective ops at 128 lanes/clk/SM: the FMA bound wins
    pk, bound = bench.tc_peak_tops(4, 152, 2.07e9, 1933.1)
    assert bound == "alu" and pk == pytest.approx(152 * 2.07e9 * 128 * 8 / 1e12)
    assert pk == pytest.approx(322.2, abs=0.1)
    pk, bound = bench.tc_peak_tops(64, 152, 2.07e9, 1933.1)
    assert bound == "tensor" and pk == pytest.approx(1933.1)


def test_total_ops_resnet50_b64(bench):
    layers = synth.resnet50_convs()
    want = 0
    for l in layers:  # 2 M P Kred per conv, both group sizes
        Ho = (l.H + 2 * l.pad - l.R) // l.stride + 1
        Wo = (l.W + 2 * l.pad - l.S) // l.stride + 1
        want += 2 * l.M * (64 * Ho * Wo) * (l.R * l.S * l.C // l.groups)
    assert bench.total_ops(layers, 64) == 2 * want
    assert bench.total_ops(layers, 64) == 987116863488


def test_family_roofline_blend(bench):
    layers = synth.resnet50_convs()
    peaks = {"sm_max_mhz": 2070.0, "bf16_tflops": 1933.1, "hbm_gbs": 6778.3}
    tc = {(4, i): 2 for i in range(1, len(layers))}
    simt = {(4, i): 1 for i in range(1, len(layers))}
    r_tc = bench.family_roofline("conv_g4", layers, 64, peaks, 152, 1e-3, tc)
    r_simt = bench.family_roofline("conv_g4", layers, 64, peaks, 152, 1e-3, simt)
    assert r_tc["peak"] == pytest.approx(bench.tc_peak_tops(4, 152, 2.07e9, 1933.1)[0])
    assert r_simt["peak"] == pytest.approx(bench.alu_peak_tops(4, 152, 2.07e9))
    # half of the layers on each kernel: the ops-weighted harmonic blend
    mixed = {(4, i): (2 if i % 2 else 1) for i in range(1, len(layers))}
    r = bench.family_roofline("conv_g4", layers, 64, peaks, 152, 1e-3, mixed)
    ops = [l.ops(64) for l in layers[1:]]
    pk = [r_tc["peak"] if i % 2 else r_simt["peak"] for i in range(1, len(layers))]
    assert r["peak"] == pytest.approx(sum(ops) / sum(o / p for o, p in zip(ops, pk)))
    assert r["achieved"] == pytest.approx(sum(ops) / 1e-3 / 1e12)


def test_traffic_table(bench):
    t = bench.load_traffic()
    assert {"conv_g4", "conv_g64", "quantize_act", "conv_w8_stem"} <= set(t)
    assert all(v > 0 for v in t.values())
