"""GPU parity: the CUDA kernels (called through the C ABI) against the CPU oracle.

Integer outputs (codes, packed activations, group sums) must match bit for bit; fp32
alphas bit for bit (both sides round the exact mean to nearest); fp32 contraction outputs
within 1e-5 * act_scale * sum_g |alpha_g * s_g| per element.
"""
import zlib

import numpy as np
import pytest
import torch

import oracle as O
from paper_1705_01462_gb300 import fgq, synth
from _gpu import (dev, to_dev, codes_u32, check_within, make_codes, quantize_oracle, random_acts,
                  ORACLE_TYPE)

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _clean_status():
    fgq.fgq_set_path(fgq.PATH_AUTO)
    yield
    fgq.fgq_set_path(fgq.PATH_AUTO)
    assert fgq.fgq_stream_status() == fgq.FGQ_OK


# ----------------------------------------------------------------------------- ternarize

def _adversarial_weights(M, K, seed):
    rng = np.random.default_rng(seed)
    w = rng.standard_normal((M, K)).astype(np.float32)
    w[0::7] = rng.choice([-0.5, 0.25, 0.5, 0.125], (len(w[0::7]), K))               # ties
    w[1::7] *= (rng.random((len(w[1::7]), K)) < 0.3)                                 # zeros
    w[2::7] *= np.float32(2.0 ** -140)                                               # subnormal
    w[3::7] *= (2.0 ** rng.integers(-30, 4, (len(w[3::7]), K))).astype(np.float32)    # wide range
    w[4::7] = 0.0                                                                    # all zero
    w[5::7] = (rng.exponential(1.0, (len(w[5::7]), K)) * rng.choice([-1, 1], (len(w[5::7]), K)))
    return w.astype(np.float32)


@pytest.mark.parametrize("G", [1, 2, 4, 8, 16, 32, 64, 128])
@pytest.mark.parametrize("K", [7, 64, 147, 576, 1000])
def test_ternarize_bit_exact(G, K):
    w = _adversarial_weights(37, K, seed=G * 1000 + K)
    t, al, codes = make_codes(w, G)
    gc, ga = fgq.fgq_ternarize(to_dev(w), G)
    assert np.array_equal(codes_u32(gc), codes)
    assert np.array_equal(ga.cpu().numpy().view(np.uint32), al.view(np.uint32))


@pytest.mark.parametrize("G", [4, 16, 64])
def test_ternarize_resnet50_weight_set(G):
    """Full ResNet-50 weight set (53 convs + fc, 25,502,912 weights), every group bit-exact."""
    layers = synth.resnet50_convs() + [synth.resnet50_fc()]
    for i, layer in enumerate(layers):
        w = synth.weights(layer, synth.layer_seed(i))
        t, al, codes = make_codes(w, G)
        gc, ga = fgq.fgq_ternarize(to_dev(w), G)
        assert np.array_equal(codes_u32(gc), codes), layer.name
        assert np.array_equal(ga.cpu().numpy(), al), layer.name


@pytest.mark.parametrize("G", [1, 2, 4, 8, 16, 32, 64, 128])
def test_ternarize_batch_bit_exact(G):
    """fgq_ternarize_batch over several layers in one launch: every set bit-exact against the
    oracle (ResNet-50 layers, a row length not a multiple of 4, an empty set, one filter)."""
    rng = np.random.default_rng(G)
    ws = [synth.weights(l, synth.layer_seed(i)) for i, l in enumerate(synth.resnet50_convs()[1:6], start=1)]
    ws += [rng.standard_normal((3, 7)).astype(np.float32), np.zeros((0, 10), np.float32),
           rng.standard_normal((1, 1001)).astype(np.float32), rng.standard_normal((40, 130)).astype(np.float32)]
    outs = fgq.fgq_ternarize_batch([to_dev(w) for w in ws], G)
    for w, (codes, alpha) in zip(ws, outs):
        if w.size == 0:
            continue
        t, al, _ = O.ternarize(w, G)
        assert np.array_equal(codes.cpu().numpy().view(np.uint32), O.pack_codes(t)), (G, w.shape)
        assert np.array_equal(alpha.cpu().numpy(), al), (G, w.shape)


def test_ternarize_batch_args():
    w = torch.zeros((4, 16), dtype=torch.float32, device=dev())
    with pytest.raises(fgq.FGQError) as e:  # more sets than one call takes
        fgq.fgq_ternarize_batch([w] * 129, 4)
    assert e.value.code == fgq.FGQ_ERR_ARG
    with pytest.raises(fgq.FGQError) as e:  # bad group size
        fgq.fgq_ternarize_batch([w], 5)
    assert e.value.code == fgq.FGQ_ERR_ARG
    assert fgq.fgq_ternarize_batch([], 4) == []


def test_ternarize_nonfinite_status():
    w = np.ones((4, 64), np.float32)
    w[1, 5] = np.nan
    gc, ga = fgq.fgq_ternarize(to_dev(w), 4)
    assert fgq.fgq_stream_status() == fgq.FGQ_ERR_NONFINITE
    a = ga.cpu().numpy()
    assert a[1, 1] == 0 and a[1, 0] == 1.0 and codes_u32(gc)[1, 0] & 0xff00 == 0


def test_quantize_weights_w8():
    rng = np.random.default_rng(5)
    w = (rng.standard_normal((64, 147)) * 0.1).astype(np.float32)
    wq, ws = fgq.fgq_quantize_weights_w8(to_dev(w))
    owq, ows = O.quantize_weights_w8(w)
    assert np.array_equal(wq.cpu().numpy(), owq) and np.array_equal(ws.cpu().numpy(), ows)


# ----------------------------------------------------------------------------- quantize

@pytest.mark.parametrize("act_type", ["u8", "s8", "u4", "s4"])
@pytest.mark.parametrize("n", [1, 15, 16, 17, 4096 + 7, 1 << 20])
def test_quantize_bit_exact(act_type, n):
    rng = np.random.default_rng(n)
    x = (rng.standard_normal(n) * 3).astype(np.float32)
    q, sc, packed = quantize_oracle(x, act_type)
    gq, gs = fgq.fgq_quantize_act(to_dev(x), act_type)
    assert np.array_equal(gq.cpu().numpy(), packed)
    assert gs.item() == sc


@pytest.mark.parametrize("scale_exp", [-149, -140, -60, 0, 20, 120])
def test_quantize_extreme_scales(scale_exp):
    rng = np.random.default_rng(scale_exp + 200)
    x = (rng.standard_normal(1000) * 2.0 ** scale_exp).astype(np.float32)
    for act_type in ("u8", "s4"):
        q, sc, packed = quantize_oracle(x, act_type)
        gq, gs = fgq.fgq_quantize_act(to_dev(x), act_type)
        assert np.array_equal(gq.cpu().numpy(), packed) and gs.item() == sc
        # given power-of-two scale, including ones that saturate
        for e in (scale_exp - 9, scale_exp + 3):
            if -149 <= e <= 127:
                s_in = float(np.float32(2.0 ** e))
                oq, _, _, _ = O.quantize(x, ORACLE_TYPE[act_type], s_in)
                gq, _ = fgq.fgq_quantize_act(to_dev(x), act_type, scale_in=s_in)
                assert np.array_equal(gq.cpu().numpy(), O.pack_act(oq, ORACLE_TYPE[act_type]))


def test_quantize_zero_and_nonfinite():
    gq, gs = fgq.fgq_quantize_act(to_dev(np.zeros(100, np.float32)), "u8")
    assert gs.item() == 1.0 and not gq.cpu().numpy().any()
    x = np.ones(64, np.float32)
    x[3] = np.inf
    fgq.fgq_quantize_act(to_dev(x), "u8")
    assert fgq.fgq_stream_status() == fgq.FGQ_ERR_NONFINITE


# ----------------------------------------------------------------------------- contraction

CONV_CASES = [
    # B, H, W, C, M, R, S, stride, pad, groups, G, act
    (1, 56, 56, 64, 64, 3, 3, 1, 1, 1, 4, "u8"),     # ResNet-50 conv2_x 3x3 at batch 1
    (2, 9, 11, 64, 70, 3, 3, 1, 1, 1, 4, "u8"),      # ragged M and P tiles
    (1, 13, 13, 64, 96, 3, 3, 2, 1, 1, 8, "s8"),
    (2, 8, 8, 32, 40, 1, 1, 1, 0, 1, 16, "u8"),
    (1, 7, 7, 64, 33, 3, 3, 1, 1, 1, 32, "u8"),
    (2, 7, 7, 128, 130, 3, 3, 1, 1, 1, 64, "u8"),
    (1, 6, 6, 256, 64, 1, 1, 1, 0, 1, 128, "s8"),
    (1, 14, 14, 64, 64, 1, 1, 2, 0, 1, 64, "u8"),    # strided 1x1
    (1, 27, 27, 48, 64, 5, 5, 1, 2, 2, 4, "u8"),     # conv groups = 2 (AlexNet towers)
    (1, 23, 23, 3, 16, 11, 11, 4, 0, 1, 4, "u8"),    # C = 3: groups straddle taps
    (1, 9, 9, 16, 8, 3, 3, 1, 1, 1, 1, "u8"),        # G = 1
    (1, 9, 9, 16, 8, 3, 3, 1, 1, 1, 2, "s8"),        # G = 2
    (2, 10, 10, 64, 64, 3, 3, 1, 1, 1, 4, "u4"),     # packed 4-bit activations
    (1, 10, 10, 128, 64, 3, 3, 1, 1, 1, 64, "u4"),
    (1, 8, 8, 64, 32, 3, 3, 1, 1, 1, 4, "s4"),
    (1, 9, 9, 6, 8, 3, 3, 1, 1, 1, 4, "u4"),         # 4-bit with C % 4 != 0
    # G >= 64 tensor-core im2col boxes: H != W, R != S, strides, conv groups, packed 4-bit
    (2, 9, 13, 64, 64, 3, 3, 1, 1, 1, 64, "u8"),
    (1, 9, 12, 64, 64, 1, 3, 1, 1, 1, 64, "u8"),
    (2, 11, 10, 128, 72, 3, 1, 2, 1, 1, 64, "s8"),
    (2, 12, 12, 128, 64, 3, 3, 2, 1, 1, 128, "u4"),
    (1, 8, 8, 256, 128, 3, 3, 1, 1, 2, 64, "u8"),
    (1, 15, 15, 64, 64, 5, 5, 3, 2, 1, 64, "s4"),
    (2, 14, 14, 128, 64, 1, 1, 2, 0, 1, 64, "s4"),    # strided 1x1, 4-bit: gathered e4m3 rows
    (2, 9, 9, 192, 96, 1, 1, 1, 0, 1, 64, "u4"),      # 1x1 stride 1, 4-bit: 2D e4m3 boxes
]


@pytest.mark.parametrize("case", CONV_CASES, ids=lambda c: "x".join(map(str, c)))
def test_conv2d_parity(case):
    B, H, W, C, M, R, S, stride, pad, groups, G, act = case
    rng = np.random.default_rng(zlib.crc32(repr(case).encode()))
    Cg = C // groups
    w = (rng.standard_normal((M, R * S * Cg)) * np.sqrt(2.0 / (R * S * Cg))).astype(np.float32)
    t, al, codes = make_codes(w, G)
    x = random_acts((B, H, W, C), act, rng)
    q, sc, packed = quantize_oracle(x, act)
    y, ym = O.conv2d(q, sc, R, S, stride, pad, groups, t, al, G)
    gout = fgq.fgq_conv2d(to_dev(packed), act, to_dev(np.array([sc], np.float32)), B, H, W, C, R, S, stride,
                          pad, groups, to_dev(codes.view(np.int32)), to_dev(al), M, G)
    check_within(gout.cpu().numpy(), y, ym, f"conv2d {case}")


GEMM_CASES = [(1, 9216, 64, 4, "u8"), (37, 576, 70, 4, "s8"), (129, 200, 65, 8, "u8"), (64, 4096, 128, 64, "u8"),
              (5, 130, 17, 64, "s8"), (300, 256, 64, 128, "u8"), (16, 96, 24, 32, "u4"), (3, 22, 5, 2, "u8")]


@pytest.mark.parametrize("case", GEMM_CASES, ids=lambda c: "x".join(map(str, c)))
def test_gemm_and_group_sums(case):
    P, K, M, G, act = case
    rng = np.random.default_rng(P * 31 + K)
    w = rng.standard_normal((M, K)).astype(np.float32)
    t, al, codes = make_codes(w, G)
    x = random_acts((P, K), act, rng)
    q, sc, packed = quantize_oracle(x, act)
    y, ym = O.gemm(q, sc, t, al, G)
    gy = fgq.fgq_gemm(to_dev(packed), act, to_dev(np.array([sc], np.float32)), P, K, to_dev(codes.view(np.int32)),
                      to_dev(al), M, G)
    check_within(gy.cpu().numpy(), y, ym, f"gemm {case}")
    s = O.group_sums(q, t, G)
    gs = fgq.fgq_group_sums(to_dev(packed), act, P, K, to_dev(codes.view(np.int32)), M, G)
    assert np.array_equal(gs.cpu().numpy().astype(np.int64), s)


def test_conv2d_w8_first_layer():
    """ResNet stem shape (7x7/2, C = 3) with 8-bit weights, at a reduced image size."""
    rng = np.random.default_rng(9)
    B, H, W, C, M, R, stride, pad = 2, 40, 36, 3, 64, 7, 2, 3
    w = (rng.standard_normal((M, R * R * C)) * np.sqrt(2.0 / 147)).astype(np.float32)
    x = np.abs(rng.standard_normal((B, H, W, C))).astype(np.float32)
    q, sc, packed = quantize_oracle(x, "u8")
    wq, ws = fgq.fgq_quantize_weights_w8(to_dev(w))
    owq, ows = O.quantize_weights_w8(w)
    y, ym = O.conv2d_w8(q, sc, R, R, stride, pad, 1, owq, ows)
    g = fgq.fgq_conv2d_w8(to_dev(packed), "u8", to_dev(np.array([sc], np.float32)), B, H, W, C, R, R, stride, pad, 1,
                          wq, ws, M)
    check_within(g.cpu().numpy(), y, ym, "conv2d_w8")


def test_chain_quantize_ternarize_conv_on_device():
    """The whole hot path on device buffers: fp32 weights and activations in, fp32 out."""
    layer = synth.conv2x_3x3()
    B, G = 1, 4
    w = synth.weights(layer, 11)
    x = synth.activations((B, layer.H, layer.W, layer.C), 12)
    t, al, _ = make_codes(w, G)
    q, sc, _ = quantize_oracle(x, "u8")
    y, ym = O.conv2d(q, sc, 3, 3, 1, 1, 1, t, al, G)
    codes, alpha = fgq.fgq_ternarize(to_dev(w), G)
    gq, gs = fgq.fgq_quantize_act(to_dev(x), "u8")
    out = fgq.fgq_conv2d(gq, "u8", gs, B, layer.H, layer.W, layer.C, 3, 3, 1, 1, 1, codes, alpha, layer.M, G)
    check_within(out.cpu().numpy(), y, ym, "chain")


@pytest.mark.parametrize("G", [4, 64])
def test_config2_batch32_sampled(G):
    """ResNet-50 conv2_x 3x3 at batch 32 (100,352 positions): sampled positions, all filters."""
    layer = synth.conv2x_3x3()
    B = 32
    w = synth.weights(layer, 21)
    x = synth.activations((B, layer.H, layer.W, layer.C), 22)
    t, al, codes = make_codes(w, G)
    q, sc, packed = quantize_oracle(x, "u8")
    out = fgq.fgq_conv2d(to_dev(packed), "u8", to_dev(np.array([sc], np.float32)), B, layer.H, layer.W, layer.C,
                         3, 3, 1, 1, 1, to_dev(codes.view(np.int32)), to_dev(al), layer.M, G)
    rng = np.random.default_rng(G)
    P = layer.P(B)
    pos = np.unique(np.r_[rng.choice(P, 600, replace=False), [0, P - 1, 55, 56, 3135, 3136]])
    y, ym = O.conv2d(q, sc, 3, 3, 1, 1, 1, t, al, G, positions=pos)
    check_within(out.reshape(P, layer.M).cpu().numpy()[pos], y, ym, "config2")


def test_wait_timeout_selftest():
    assert fgq.fgq_selftest_wait_timeout(4) == fgq.FGQ_ERR_TIMEOUT
    assert fgq.fgq_stream_status() == fgq.FGQ_OK  # cleared by the read


def test_launch_counter_counts():
    n0 = fgq.fgq_launch_count()
    fgq.fgq_quantize_act(to_dev(np.ones(100, np.float32)), "u8")
    assert fgq.fgq_launch_count() == n0 + 2


# ----------------------------------------------------------------------------- tensor-core path

TC_CASES = [
    # B, H, W, C, M, R, S, stride, pad, groups, G, act
    (1, 7, 9, 64, 128, 1, 1, 1, 0, 1, 64, "u8"),     # single tile, 1x1
    (2, 9, 11, 64, 64, 3, 3, 1, 1, 1, 64, "u8"),     # M = 64 (half tile), ragged P
    (1, 12, 12, 128, 200, 3, 3, 1, 1, 1, 64, "s8"),  # ragged M tile
    (2, 14, 14, 128, 256, 1, 1, 2, 0, 1, 64, "u8"),  # strided 1x1, two M tiles
    (1, 8, 8, 256, 96, 3, 3, 1, 1, 1, 128, "u8"),    # G = 128: two K-tiles per group
    (1, 13, 13, 384, 384, 3, 3, 1, 1, 2, 64, "u8"),  # conv groups = 2, Mg = 192
    (2, 10, 10, 128, 64, 3, 3, 1, 1, 1, 64, "u4"),
    (1, 9, 9, 64, 70, 3, 3, 1, 1, 1, 64, "s4"),
    (3, 28, 28, 64, 64, 3, 3, 1, 1, 1, 64, "u8"),    # many tiles per CTA (persistent loop)
]


# every tensor-core case also at G = 4 (the block-diagonal G = 4 kernel)
TC_CASES = TC_CASES + [c[:10] + (4,) + c[11:] for c in TC_CASES]


@pytest.mark.parametrize("case", TC_CASES, ids=lambda c: "x".join(map(str, c)))
def test_tc_conv2d_parity(case):
    B, H, W, C, M, R, S, stride, pad, groups, G, act = case
    rng = np.random.default_rng(zlib.crc32(repr(case).encode()) + 1)
    Cg = C // groups
    w = (rng.standard_normal((M, R * S * Cg)) * np.sqrt(2.0 / (R * S * Cg))).astype(np.float32)
    t, al, codes = make_codes(w, G)
    x = random_acts((B, H, W, C), act, rng)
    q, sc, packed = quantize_oracle(x, act)
    y, ym = O.conv2d(q, sc, R, S, stride, pad, groups, t, al, G)
    fgq.fgq_set_path(fgq.PATH_TC)
    gout = fgq.fgq_conv2d(to_dev(packed), act, to_dev(np.array([sc], np.float32)), B, H, W, C, R, S, stride,
                          pad, groups, to_dev(codes.view(np.int32)), to_dev(al), M, G)
    assert fgq.fgq_last_path() == fgq.PATH_TC
    check_within(gout.cpu().numpy(), y, ym, f"tc conv2d {case}")


@pytest.mark.parametrize("case", [(128, 64, 128, 64, "u8"), (1, 9216, 4096, 64, "u8"), (300, 256, 64, 128, "s8"),
                                  (257, 1024, 1000, 64, "u8"), (64, 512, 130, 64, "u4"), (128, 64, 128, 4, "u8"),
                                  (1, 9216, 4096, 4, "u8"), (257, 1024, 1000, 4, "s8"), (64, 512, 130, 4, "u4")],
                         ids=lambda c: "x".join(map(str, c)))
def test_tc_gemm_parity(case):
    P, K, M, G, act = case
    rng = np.random.default_rng(P * 7 + K)
    w = rng.standard_normal((M, K)).astype(np.float32)
    t, al, codes = make_codes(w, G)
    x = random_acts((P, K), act, rng)
    q, sc, packed = quantize_oracle(x, act)
    y, ym = O.gemm(q, sc, t, al, G)
    fgq.fgq_set_path(fgq.PATH_TC)
    gy = fgq.fgq_gemm(to_dev(packed), act, to_dev(np.array([sc], np.float32)), P, K, to_dev(codes.view(np.int32)),
                      to_dev(al), M, G)
    assert fgq.fgq_last_path() == fgq.PATH_TC
    check_within(gy.cpu().numpy(), y, ym, f"tc gemm {case}")


KSPLIT_CASES = [
    # B, H, W, C, M, R, S, stride, pad, groups, G, act: fewer tiles than SMs, at least 4096
    # products per output
    (2, 9, 9, 512, 200, 3, 3, 1, 1, 1, 64, "u8"),     # im2col boxes, ragged P and M tiles
    (1, 14, 14, 4096, 256, 1, 1, 1, 0, 1, 64, "s8"),  # 1x1: 2D boxes
    (2, 14, 14, 4096, 128, 1, 1, 2, 0, 1, 64, "u8"),  # strided 1x1: gathered rows
    (1, 8, 8, 1024, 128, 3, 3, 1, 1, 2, 64, "u8"),    # conv groups = 2: fp32 atomics, no output map
    (1, 9, 9, 512, 66, 3, 3, 1, 1, 1, 64, "u8"),      # M % 4 != 0: fp32 atomics
    (2, 7, 7, 512, 128, 3, 3, 1, 1, 1, 128, "u4"),    # e4m3 operands, two K-tiles per group
    (1, 7, 7, 576, 64, 3, 3, 1, 1, 1, 64, "s4"),      # ng = 81: ranges of unequal length
]


@pytest.mark.parametrize("case", KSPLIT_CASES, ids=lambda c: "x".join(map(str, c)))
def test_tc_group_range_split(case):
    """A few-tile layer split into group ranges whose partial sums are added into the output:
    within the contraction tolerance of the oracle, and of the whole-tile result (the same
    sum in another fp32 order)."""
    B, H, W, C, M, R, S, stride, pad, groups, G, act = case
    rng = np.random.default_rng(zlib.crc32(repr(case).encode()) + 2)
    Cg = C // groups
    w = (rng.standard_normal((M, R * S * Cg)) * np.sqrt(2.0 / (R * S * Cg))).astype(np.float32)
    t, al, codes = make_codes(w, G)
    x = random_acts((B, H, W, C), act, rng)
    q, sc, packed = quantize_oracle(x, act)
    y, ym = O.conv2d(q, sc, R, S, stride, pad, groups, t, al, G)
    args = (to_dev(packed), act, to_dev(np.array([sc], np.float32)), B, H, W, C, R, S, stride, pad, groups,
            to_dev(codes.view(np.int32)), to_dev(al), M, G)
    fgq.fgq_set_path(fgq.PATH_TC)
    split = fgq.fgq_conv2d(*args).cpu().numpy()
    assert fgq.fgq_last_path() == fgq.PATH_TC and fgq.fgq_debug_last_ksplit() > 1
    prev = fgq.fgq_debug_max_ksplit(1)
    try:
        whole = fgq.fgq_conv2d(*args).cpu().numpy()
        assert fgq.fgq_debug_last_ksplit() == 1
    finally:
        fgq.fgq_debug_max_ksplit(prev)
    check_within(split, y, ym, f"tc conv2d split {case}")
    check_within(whole, y, ym, f"tc conv2d whole {case}")
    check_within(split, whole.astype(np.float64), ym, f"split vs whole {case}")


def test_tc_gemm_group_range_split():
    """One-tile GEMM (a fully connected layer at small batch) over 8 group ranges."""
    P, K, M, G, act = 60, 4096, 128, 64, "u8"
    rng = np.random.default_rng(4096)
    w = rng.standard_normal((M, K)).astype(np.float32)
    t, al, codes = make_codes(w, G)
    x = random_acts((P, K), act, rng)
    q, sc, packed = quantize_oracle(x, act)
    y, ym = O.gemm(q, sc, t, al, G)
    fgq.fgq_set_path(fgq.PATH_TC)
    gy = fgq.fgq_gemm(to_dev(packed), act, to_dev(np.array([sc], np.float32)), P, K, to_dev(codes.view(np.int32)),
                      to_dev(al), M, G)
    assert fgq.fgq_last_path() == fgq.PATH_TC and fgq.fgq_debug_last_ksplit() == 8
    check_within(gy.cpu().numpy(), y, ym, "tc gemm split")


def test_tc_forced_on_unsupported_shape():
    """A forced tensor-core path on a shape it cannot run returns FGQ_ERR_UNSUPPORTED."""
    fgq.fgq_set_path(fgq.PATH_TC)
    q = torch.zeros(64 * 48, dtype=torch.uint8, device=dev())
    codes = torch.zeros((8, 4), dtype=torch.int32, device=dev())
    al = torch.zeros((8, 1), dtype=torch.float32, device=dev())
    with pytest.raises(fgq.FGQError) as e:
        fgq.fgq_gemm(q, "u8", torch.ones(1, device=dev()), 64, 48, codes, al, 8, 64)
    assert e.value.code == fgq.FGQ_ERR_UNSUPPORTED


@pytest.mark.parametrize("path", ["simt", "tc", "tc_cta_pairs"])
@pytest.mark.parametrize("case", [(1, 56, 56, 64, 64, 3, 3, 1, 1, 1, 4, "u8"), (2, 28, 28, 128, 96, 1, 1, 1, 0, 1, 4, "u8"),
                                  (2, 14, 14, 256, 64, 1, 1, 2, 0, 1, 4, "s8"), (1, 9, 13, 128, 160, 3, 3, 1, 1, 2, 4, "u4"),
                                  (3, 7, 7, 64, 96, 3, 3, 2, 1, 1, 4, "s8")],
                         ids=lambda c: "x".join(map(str, c)))
def test_g4_both_kernel_families(case, path):
    """G = 4 through the dp4a kernel and through the block-diagonal tensor-core kernel, the
    latter on single CTAs (the default) and on CTA pairs."""
    B, H, W, C, M, R, S, stride, pad, groups, G, act = case
    rng = np.random.default_rng(zlib.crc32(repr(case).encode()) + 2)
    Kred = R * S * (C // groups)
    w = (rng.standard_normal((M, Kred)) * np.sqrt(2.0 / Kred)).astype(np.float32)
    t, al, codes = make_codes(w, G)
    x = random_acts((B, H, W, C), act, rng)
    q, sc, packed = quantize_oracle(x, act)
    y, ym = O.conv2d(q, sc, R, S, stride, pad, groups, t, al, G)
    fgq.fgq_set_path(fgq.PATH_SIMT if path == "simt" else fgq.PATH_TC)
    prev = fgq.fgq_debug_cta_pairs(path == "tc_cta_pairs")
    try:
        gout = fgq.fgq_conv2d(to_dev(packed), act, to_dev(np.array([sc], np.float32)), B, H, W, C, R, S, stride,
                              pad, groups, to_dev(codes.view(np.int32)), to_dev(al), M, G)
    finally:
        fgq.fgq_debug_cta_pairs(bool(prev))
    assert fgq.fgq_last_path() == (fgq.PATH_SIMT if path == "simt" else fgq.PATH_TC)
    check_within(gout.cpu().numpy(), y, ym, f"G=4 {path} {case}")
