"""CPU checks of the benchmark's host-side arithmetic: per-layer roofline floors at the
measured peaks, a family's roofline over its layers, the streaming kernels' byte counts,
the per-step operation count and the traffic table it reads (ignored when taken from other
sources)."""
import importlib.util
import os

import pytest

from paper_1705_01462_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PEAKS = {"sm_max_mhz": 2070.0, "bf16_tflops": 1933.1, "hbm_gbs": 6778.3}


@pytest.fixture(scope="module")
def bench():
    spec = importlib.util.spec_from_file_location("bench_module", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_total_ops_resnet50_b64(bench):
    layers = synth.resnet50_convs()
    want = 0
    for l in layers:  # 2 M P Kred per conv, both group sizes
        Ho = (l.H + 2 * l.pad - l.R) // l.stride + 1
        Wo = (l.W + 2 * l.pad - l.S) // l.stride + 1
        want += 2 * l.M * (64 * Ho * Wo) * (l.R * l.S * l.C // l.groups)
    assert bench.total_ops(layers, 64) == 2 * want
    assert bench.total_ops(layers, 64) == 987116863488


def test_algorithmic_bytes_by_hand(bench):
    l = synth.conv2x_3x3()  # 64 -> 64, 3x3, 56x56
    B = 32
    act = B * 56 * 56 * 64                        # uint8 input
    codes = 64 * (576 // 16) * 4                  # 2-bit codes, 36 words per row
    alpha = 64 * (576 // 4) * 4                   # one fp32 alpha per group of 4
    out = B * 56 * 56 * 64 * 4                    # fp32 output
    assert bench.algorithmic_bytes(l, B, 4) == act + codes + alpha + out
    assert bench.algorithmic_bytes(l, B, 4, act_bits=4) == act // 2 + codes + alpha + out
    assert bench.algorithmic_bytes(l, B, None) == act + 64 * 576 + 4 * 64 + out


def test_layer_floor_picks_the_larger_bound(bench):
    l = synth.conv2x_3x3()
    t, b = bench.layer_floor(l, 32, 64, PEAKS)
    t_mem = bench.algorithmic_bytes(l, 32, 64) / (PEAKS["hbm_gbs"] * 1e9)
    t_ops = l.ops(32) / (PEAKS["bf16_tflops"] * 1e12)
    assert t == max(t_mem, t_ops) and b == ("hbm" if t_mem >= t_ops else "tensor")
    # a square FC at batch 1024 is tensor-bound, at batch 1 memory-bound
    fc = synth.ConvLayer("fc", 16384, 16384, 1, 1, 1, 0, 1, 1)
    assert bench.layer_floor(fc, 1024, 64, PEAKS)[1] == "tensor"
    assert bench.layer_floor(fc, 1, 64, PEAKS)[1] == "hbm"


def test_conv_roofline_is_sum_of_floors(bench):
    layers = synth.resnet50_convs()[1:]
    sec = 3e-3
    r = bench.conv_roofline(layers, 64, 64, PEAKS, sec)
    floors = [bench.layer_floor(l, 64, 64, PEAKS)[0] for l in layers]
    ops = sum(l.ops(64) for l in layers)
    assert r["frac"] == pytest.approx(sum(floors) / sec)
    assert r["achieved"] == pytest.approx(ops / sec / 1e12)
    assert r["peak"] == pytest.approx(ops / sum(floors) / 1e12)
    assert r["achieved"] / r["peak"] == pytest.approx(r["frac"])
    assert r["bound"] == "hbm"  # fp32 outputs: the stack is memory-bound overall
    # the ResNet-50 stack's floor at G = 64 is about half a millisecond
    assert 0.4 < r["floor_ms"] < 0.7


def test_streaming_family_bytes(bench):
    layers = synth.resnet50_convs()
    B = 64
    q = bench.family_roofline("quantize_act", layers, B, PEAKS, 1e-3)
    want = sum(B * l.H * l.W * l.C * 5 for l in layers)  # 4 B in, 1 B out per element
    assert q["bytes"] == want and q["unit"] == "GB/s" and q["peak"] == PEAKS["hbm_gbs"]
    q4 = bench.family_roofline("quantize_act", layers, B, PEAKS, 1e-3, act="u4")
    first = B * 224 * 224 * 3
    assert q4["bytes"] == first * 5 + sum(B * l.H * l.W * l.C * 9 // 2 for l in layers[1:])
    t = bench.family_roofline("ternarize_g64", layers, B, PEAKS, 1e-3)
    assert t["bytes"] == sum(l.M * l.Kred * 4 + l.M * (-(-l.Kred // 64)) * 20 for l in layers[1:])


def test_traffic_table_needs_matching_sources(bench, tmp_path, monkeypatch):
    assert bench.load_traffic("no-such-digest") == {}
    d = bench.source_digest()
    assert len(d) == 16 and d == bench.source_digest()
    prof = tmp_path / "profiles"
    prof.mkdir()
    (prof / "conv_traffic_x.txt").write_text(f"# sources {d}\nconv_g4 123.0 note\n")
    (prof / "old_traffic_y.txt").write_text("# sources 0000000000000000\nconv_g64 456.0\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.load_traffic(d) == {"conv_g4": 123.0}
    assert bench.load_traffic() == {"conv_g4": 123.0, "conv_g64": 456.0}
