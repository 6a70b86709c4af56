"""Pins of the oracle's fixed-point alphas (Section 4: alphas quantized to 8/4-bit fixed
point; one DFP exponent per filter row): round-trip bounds, minimality of the exponent,
lossless cases, and the contraction with the dequantized alphas."""
import numpy as np
import pytest

import oracle as O


@pytest.mark.parametrize("bits", [8, 4])
def test_roundtrip_bound_and_minimal_exponent(bits):
    rng = np.random.default_rng(bits)
    alpha = np.abs(rng.standard_normal((40, 37))).astype(np.float32) * (2.0 ** rng.integers(-20, 5, (40, 1)))
    alpha = alpha.astype(np.float32)
    alpha[3] = 0.0
    a, sc, _ = O.quantize_alpha(alpha, bits)
    qmax = 2 ** bits - 1
    assert a.min() >= 0 and a.max() <= qmax
    for m in range(40):
        if not alpha[m].any():
            assert sc[m] == 1.0 and not a[m].any()
            continue
        E = int(np.log2(sc[m]))
        assert sc[m] == 2.0 ** E
        mx = float(alpha[m].max())
        assert mx * 2.0 ** -E <= qmax and mx * 2.0 ** -(E - 1) > qmax  # smallest such E
        err = np.abs(alpha[m].astype(np.float64) - a[m] * sc[m].astype(np.float64))
        assert np.all(err <= 2.0 ** (E - 1))  # round to nearest, nothing saturates below max


def test_lossless_when_representable():
    rng = np.random.default_rng(3)
    k = rng.integers(0, 256, (8, 20))
    k[:, 0] = 255  # the row maximum fixes E
    alpha = (k * 2.0 ** -12).astype(np.float32)
    a, sc, _ = O.quantize_alpha(alpha, 8)
    assert np.array_equal(a, k) and np.all(sc == np.float32(2.0 ** -12))
    assert np.array_equal(O.dequantize_alpha(a, sc), alpha)


def test_ties_round_to_even():
    # row max 255 * 2^-4 fixes E = -4; 2.5 * 2^-4 and 3.5 * 2^-4 are ties
    alpha = np.array([[255 / 16, 2.5 / 16, 3.5 / 16, 0.5 / 16]], np.float32)
    a, sc, _ = O.quantize_alpha(alpha, 8)
    assert a.tolist() == [[255, 2, 4, 0]] and sc[0] == 1 / 16


def test_contraction_with_dequantized_alpha():
    """With representable alphas the fixed-point contraction equals the fp32-alpha one."""
    rng = np.random.default_rng(9)
    w = rng.standard_normal((16, 64)).astype(np.float32)
    t, al, _ = O.ternarize(w, 4)
    a, sc, _ = O.quantize_alpha(al, 8)
    ald = O.dequantize_alpha(a, sc)
    x = np.abs(rng.standard_normal((5, 64))).astype(np.float32)
    q, s, _, _ = O.quantize(x, O.U8)
    y1, _ = O.gemm(q, s, t, ald, 4)
    y2, _ = O.gemm(q, s, t, al, 4)
    # each alpha moves by at most half an lsb, 2^(E_m - 1): |dy| <= s_x 2^(E_m - 1) sum_g |s_g|
    sums = O.group_sums(q, t, 4)  # [M][ng][P]
    bound = s * (sc[:, None] / 2.0) * np.abs(sums).sum(axis=1)  # [M][P]
    assert np.all(np.abs(y1 - y2).T <= bound * (1 + 1e-9))
    assert np.max(np.abs(y1 - y2)) > 0  # the quantization did change something
    a2, sc2, _ = O.quantize_alpha(ald, 8)  # quantizing quantized alphas is the identity
    assert np.array_equal(a2, a) and np.array_equal(sc2, sc)


def test_pack4():
    a = np.array([[1, 2, 3], [15, 0, 7]], np.int32)
    assert O.pack_alpha4(a).tolist() == [[0x21, 0x03], [0x0f, 0x07]]
