"""Pins of the oracle's chained-forward steps (max pooling of codes, residual add with
requantization) and of the ResNet graph the forward walks, against library routines,
brute force and hand-worked values."""
import itertools

import numpy as np
import pytest

import oracle as O
from paper_1705_01462_gb300 import resnet, synth


def _pool_brute(q, R, stride, pad):
    """Every (output, input) pair tested for window membership: a second formulation."""
    B, H, W, C = q.shape
    Ho, Wo = (H + 2 * pad - R) // stride + 1, (W + 2 * pad - R) // stride + 1
    out = np.full((B, Ho, Wo, C), np.iinfo(np.int64).min, dtype=np.int64)
    for ho, wo, h, w in itertools.product(range(Ho), range(Wo), range(H), range(W)):
        if 0 <= h - (ho * stride - pad) < R and 0 <= w - (wo * stride - pad) < R:
            out[:, ho, wo, :] = np.maximum(out[:, ho, wo, :], q[:, h, w, :])
    return out


@pytest.mark.parametrize("shape,R,stride,pad", [((2, 7, 9, 3), 3, 2, 1), ((1, 6, 6, 2), 2, 2, 0),
                                                ((1, 8, 5, 4), 3, 1, 1), ((1, 9, 9, 1), 5, 2, 2),
                                                ((1, 4, 4, 2), 3, 3, 0)])
def test_maxpool_brute_force(shape, R, stride, pad):
    rng = np.random.default_rng(R * 100 + stride * 10 + pad)
    for lo, hi in ((0, 256), (-128, 128), (-128, -1)):  # signed codes: padding must not win
        q = rng.integers(lo, hi, size=shape)
        assert np.array_equal(O.maxpool_codes(q, R, stride, pad), _pool_brute(q, R, stride, pad))


def test_maxpool_scipy_maximum_filter():
    """For non-negative codes and pad = R // 2 the pooling is scipy's centred maximum filter
    with zero fill, sampled at the stride."""
    ndimage = pytest.importorskip("scipy.ndimage")
    rng = np.random.default_rng(3)
    q = rng.integers(0, 256, size=(2, 23, 17, 5))
    for R, stride in ((3, 2), (3, 1), (5, 2)):
        ref = ndimage.maximum_filter(q, size=(1, R, R, 1), mode="constant", cval=0)
        got = O.maxpool_codes(q, R, stride, R // 2)
        Ho, Wo = got.shape[1:3]
        assert np.array_equal(got, ref[:, ::stride, ::stride, :][:, :Ho, :Wo, :])


def test_maxpool_resnet_shape():
    q = np.zeros((1, 112, 112, 4), dtype=np.int32)
    assert O.maxpool_codes(q, 3, 2, 1).shape == (1, 56, 56, 4)


def test_add_codes_exact_and_rounding():
    e = np.array
    # one term zero: the other product, exact
    assert O.add_codes(e([255]), 2.0 ** -7, e([0]), 2.0 ** 3)[0] == np.float32(255 * 2.0 ** -7)
    # equal scales: (a + b) * s, exact
    assert O.add_codes(e([200]), 0.25, e([-100]), 0.25)[0] == np.float32(25.0)
    # 2^24 + 1 is a tie between 2^24 and 2^24 + 2: to even, 2^24
    assert O.add_codes(e([128]), 2.0 ** 17, e([1]), 1.0)[0] == np.float32(2.0 ** 24)
    # 2^24 + 3 is a tie between 2^24 + 2 and 2^24 + 4: to even, 2^24 + 4
    assert O.add_codes(e([128]), 2.0 ** 17, e([3]), 1.0)[0] == np.float32(2.0 ** 24 + 4)
    # 2^24 + 5: nearest is 2^24 + 4 (not a tie)
    assert O.add_codes(e([128]), 2.0 ** 17, e([5]), 1.0)[0] == np.float32(2.0 ** 24 + 4)
    # a far smaller term vanishes in the rounding
    assert O.add_codes(e([255]), 1.0, e([1]), 2.0 ** -30)[0] == np.float32(255.0)
    # commutative
    rng = np.random.default_rng(0)
    a, b = rng.integers(-128, 128, 1000), rng.integers(0, 256, 1000)
    assert np.array_equal(O.add_codes(a, 2.0 ** -5, b, 2.0 ** -9), O.add_codes(b, 2.0 ** -9, a, 2.0 ** -5))


def test_add_codes_against_exact_fraction():
    """fp32 sum = the exact rational sum rounded to nearest (checked with integers scaled by
    2^20 and Python's exact int arithmetic)."""
    rng = np.random.default_rng(1)
    a, b = rng.integers(-128, 128, 500), rng.integers(-128, 128, 500)
    got = O.add_codes(a, 2.0 ** -3, b, 2.0 ** -20)
    for ai, bi, g in zip(a, b, got):
        exact = int(ai) * 2 ** 17 + int(bi)  # (a*2^-3 + b*2^-20) * 2^20
        assert float(g) * 2 ** 20 == float(np.float32(exact))  # |exact| < 2^24: representable
    assert np.all(got.astype(np.float64) * 2 ** 20 == a * 2 ** 17 + b)


def test_add_requant_hand_values():
    e = np.array
    # 100 * 1 + (-30) * 0.5 = 85 -> code 85 at scale 1
    assert O.add_requant(e([100]), 1.0, e([-30]), 0.5, O.U8, 1.0)[0] == 85
    # 100 - 128 = -28: u8 -> 0 (the ReLU after the addition), s8 -> -28
    assert O.add_requant(e([100]), 1.0, e([-128]), 1.0, O.U8, 1.0)[0] == 0
    assert O.add_requant(e([100]), 1.0, e([-128]), 1.0, O.S8, 1.0)[0] == -28
    # 255 + 127 = 382 saturates: u8 255, s8 127; at scale 2: 191
    assert O.add_requant(e([255]), 1.0, e([127]), 1.0, O.U8, 1.0)[0] == 255
    assert O.add_requant(e([255]), 1.0, e([127]), 1.0, O.S8, 1.0)[0] == 127
    assert O.add_requant(e([255]), 1.0, e([127]), 1.0, O.U8, 2.0)[0] == 191
    # 2 * 2^-2 + 3 * 2^-4 = 0.6875 at scale 2^-3: 5.5 -> a tie, rounded as the quantizer does
    q55, _, _, _ = O.quantize(np.array([5.5 * 2.0 ** -3], np.float32), O.U8, scale_in=2.0 ** -3)
    assert O.add_requant(e([2]), 2.0 ** -2, e([3]), 2.0 ** -4, O.U8, 2.0 ** -3)[0] == q55[0]


def test_resnet_graph():
    layers = synth.resnet50_convs()
    nodes = resnet.graph(layers)
    convs = [n for n in nodes if n.kind == "conv"]
    assert sorted(n.layer for n in convs) == list(range(len(layers)))  # every conv once
    adds = [n for n in nodes if n.kind == "add"]
    assert len(adds) == 16 and sum(n.inputs[1].endswith("p") for n in adds) == 4
    shape = {"input": (3, 224)}
    for n in nodes:  # channels and spatial size chain through the graph
        if n.kind == "quant":
            continue
        ins = [shape[k] for k in n.inputs]
        if n.kind == "conv":
            l = layers[n.layer]
            assert ins[0] == (l.C, l.H), n
            shape[n.name] = (l.M, l.Ho)
        elif n.kind == "maxpool":
            shape[n.name] = (ins[0][0], (ins[0][1] + 2 - 3) // 2 + 1)
        else:
            assert ins[0] == ins[1], n
            shape[n.name] = ins[0]
    assert shape[nodes[-1].name] == (2048, 7)
    assert [n.name for n in nodes].index("pool") < [n.name for n in nodes].index("b0a")
    # every tensor is freed after its last reader
    last = resnet.last_uses(nodes)
    freed = [k for ks in last.values() for k in ks]
    assert sorted(freed) == sorted({k for n in nodes for k in n.inputs})
    assert len(resnet.graph(synth.resnet101_convs())) == len(nodes) + 17 * 4
