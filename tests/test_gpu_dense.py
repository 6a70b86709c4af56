"""GPU parity of the dense tensor-core path (alphas folded into fp16 weights), through the
C ABI.

* Fixed-point alphas (Section 4: 8/4-bit codes, one exponent per filter row): the folded
  weights a * t are integers and every product a t q is exact, so the output is the
  oracle's exact value rounded once to fp32 wherever sum_k |a t q| < 2^24 (which bounds
  every partial sum of the accumulator, in any order); beyond that the fp32 accumulator
  rounds at most once per 16 reduction elements, and the error stays within
  (Kp / 16) 2^-23 s_x 2^E_m sum_k |a t q| -- the bound the header states, checked on
  saturated adversarial inputs at Kred = 4608.
* fp32 alphas split into two fp16 parts (an ablation, only when forced and allowed by the
  test switch fgq_debug_allow_split_fold; refused otherwise): within the bound
  its arithmetic gives, s_x sum_k |alpha t q| (2^-21 + steps 2^-23) with one rounding of
  the accumulator per 16 reduction elements and per part, and most outputs inside the
  contraction tolerance as well."""
import zlib

import numpy as np
import pytest
import torch

import oracle as O
from paper_1705_01462_gb300 import fgq
from _gpu import TOL, check_within, dev, make_codes, quantize_oracle, random_acts, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _clean_status():
    fgq.fgq_set_path(fgq.PATH_AUTO)
    fgq.fgq_debug_allow_split_fold(False)
    yield
    fgq.fgq_set_path(fgq.PATH_AUTO)
    fgq.fgq_debug_allow_split_fold(False)
    assert fgq.fgq_stream_status() == fgq.FGQ_OK


def _qa(al, bits):
    a, asc, _ = O.quantize_alpha(al, bits)
    aq = a.astype(np.uint8) if bits == 8 else O.pack_alpha4(a)
    return O.dequantize_alpha(a, asc), aq, asc


def _check_exact(got, y, ym, absum, row_scale, sc, steps, what):
    """got == fp32(y) where sum_k |a t q| = absum / (s_x 2^E_m) is below 2^24 (no partial sum of
    the accumulator can round there); elsewhere within steps 2^-23 absum (+ the final
    rounding).  absum = s_x 2^E_m sum_k |a t q| per output."""
    d = absum / (np.float64(sc) * row_scale.astype(np.float64))
    small = d < 2.0 ** 24
    exact = got == y.astype(np.float32)
    assert np.all(exact | ~small), f"{what}: {np.sum(~exact & small)} outputs differ from the exact value"
    err = np.abs(got.astype(np.float64) - y)
    assert np.all(err <= steps * 2.0 ** -23 * absum + 2.0 ** -24 * np.abs(y)), f"{what}: beyond the stated bound"
    return small


CONV_CASES = [
    # B, H, W, C, M, R, S, stride, pad, groups, G, act
    (2, 14, 14, 128, 128, 3, 3, 1, 1, 1, 4, "u8"),     # gather path, one full filter tile
    (1, 19, 17, 64, 200, 3, 3, 2, 1, 1, 4, "u8"),      # stride 2, ragged M and P
    (3, 10, 10, 256, 64, 1, 1, 1, 0, 1, 16, "s8"),     # 1x1: TMA activation boxes, M < 128
    (2, 9, 9, 128, 130, 1, 1, 2, 0, 1, 64, "u8"),      # strided 1x1: gathered
    (1, 12, 12, 128, 96, 3, 3, 1, 1, 2, 8, "u8"),      # conv groups (Mg = 48)
    (1, 7, 7, 64, 256, 3, 3, 1, 1, 1, 128, "u8"),      # G = 128: Kred 576, Kp 640 (padding)
]


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("case", CONV_CASES, ids=lambda c: "x".join(map(str, c)))
def test_conv2d_qa_dense_exact(case, bits):
    B, H, W, C, M, R, S, stride, pad, groups, G, act = case
    rng = np.random.default_rng(zlib.crc32(repr((case, bits)).encode()))
    Kred = R * S * (C // groups)
    w = (rng.standard_normal((M, Kred)) * np.sqrt(2.0 / Kred)).astype(np.float32)
    t, al, codes = make_codes(w, G)
    x = random_acts((B, H, W, C), act, rng)
    q, sc, packed = quantize_oracle(x, act)
    ad, aq, asc = _qa(al, bits)
    y, ym = O.conv2d(q, sc, R, S, stride, pad, groups, t, ad, G)
    got = fgq.fgq_conv2d_qa(to_dev(packed), act, to_dev(np.array([sc], np.float32)), B, H, W, C, R, S, stride, pad,
                            groups, to_dev(codes.view(np.int32)), to_dev(aq), bits, to_dev(asc), M, G)
    assert fgq.fgq_last_path() == fgq.PATH_DENSE
    absum = _split_bound(q, sc, t, ad, G, (R, S, stride, pad, groups))
    small = _check_exact(got.cpu().numpy(), y, ym, absum, asc.reshape(1, 1, 1, M), sc, -(-Kred // G) * G // 16,
                         f"conv2d_qa dense {case} bits={bits}")
    assert small.mean() > 0.9  # the exact regime covers these inputs almost everywhere


def test_gemm_qa_dense_many_tiles():
    """470 tiles over 152 CTAs: every CTA cycles its two accumulators; sampled rows checked."""
    P, K, M, G = 60000, 256, 256, 4
    rng = np.random.default_rng(11)
    w = rng.standard_normal((M, K)).astype(np.float32)
    t, al, codes = make_codes(w, G)
    x = random_acts((P, K), "u8", rng)
    q, sc, packed = quantize_oracle(x, "u8")
    ad, aq, asc = _qa(al, 8)
    got = fgq.fgq_gemm_qa(to_dev(packed), "u8", to_dev(np.array([sc], np.float32)), P, K,
                          to_dev(codes.view(np.int32)), to_dev(aq), 8, to_dev(asc), M, G).cpu().numpy()
    assert fgq.fgq_last_path() == fgq.PATH_DENSE
    rows = np.unique(np.concatenate([rng.integers(0, P, 600), np.arange(P - 300, P), np.arange(0, 300)]))
    y, ym = O.gemm(q[rows], sc, t, ad, G)
    absum = _split_bound(q[rows], sc, t, ad, G)
    small = _check_exact(got[rows], y, ym, absum, asc.reshape(1, M), sc, K // 16, "gemm_qa dense many tiles")
    assert small.all()


@pytest.mark.parametrize("Kred,bits", [(4608, 8), (4608, 4), (256, 8)])
def test_gemm_qa_dense_saturated_partial_sums(Kred, bits):
    """Adversarial inputs: all codes +1, alpha codes and activations near their maxima, so
    sum_k |a t q| reaches 255 * 255 * 4608 ~ 2^28 and the fp32 accumulator must round: the
    output stays within the stated (Kp / 16) 2^-23 s_x 2^E sum_k |a t q| of the exact value;
    at Kred = 256 every partial sum is below 2^24 and the output is the exact value rounded once."""
    P, M, G = 192, 128, 4
    rng = np.random.default_rng(Kred + bits)
    amax = 255 if bits == 8 else 15
    t = np.ones((M, Kred), np.int8)
    a = rng.integers(amax - amax // 5, amax + 1, (M, Kred // G)).astype(np.int32)
    asc = (2.0 ** -rng.integers(8, 12, M)).astype(np.float32)
    q = rng.integers(200, 256, (P, Kred)).astype(np.int32)
    sc = np.float32(2.0 ** -8)
    ad = a.astype(np.float32) * asc[:, None]
    y, ym = O.gemm(q, sc, t, ad, G)
    aq = a.astype(np.uint8) if bits == 8 else O.pack_alpha4(a)
    got = fgq.fgq_gemm_qa(to_dev(O.pack_act(q, O.U8)), "u8", to_dev(np.array([sc], np.float32)), P, Kred,
                          to_dev(O.pack_codes(t).view(np.int32)), to_dev(aq), bits, to_dev(asc), M, G).cpu().numpy()
    assert fgq.fgq_last_path() == fgq.PATH_DENSE
    absum = _split_bound(q, sc, t, ad, G)
    small = _check_exact(got, y, ym, absum, asc.reshape(1, M), sc, Kred // 16, f"saturated Kred={Kred} bits={bits}")
    if Kred == 256 and bits == 8:
        assert small.all()


def _split_bound(q, sc, t, al, G, conv_args=None):
    """s_x sum_k |alpha t q| from the oracle on |t| and |q|."""
    if conv_args is None:
        s, _ = O.gemm(np.abs(q), sc, np.abs(t), al, G)
    else:
        s, _ = O.conv2d(np.abs(q), sc, *conv_args, np.abs(t), al, G)
    return s


@pytest.mark.parametrize("case", CONV_CASES[:4], ids=lambda c: "x".join(map(str, c)))
def test_conv2d_split_fold_ablation(case):
    B, H, W, C, M, R, S, stride, pad, groups, G, act = case
    rng = np.random.default_rng(zlib.crc32(repr(case).encode()) + 5)
    Kred = R * S * (C // groups)
    w = (rng.standard_normal((M, Kred)) * np.sqrt(2.0 / Kred)).astype(np.float32)
    t, al, codes = make_codes(w, G)
    x = random_acts((B, H, W, C), act, rng)
    q, sc, packed = quantize_oracle(x, act)
    y, ym = O.conv2d(q, sc, R, S, stride, pad, groups, t, al, G)
    args = (to_dev(packed), act, to_dev(np.array([sc], np.float32)), B, H, W, C, R, S, stride, pad, groups,
            to_dev(codes.view(np.int32)), to_dev(al), M, G)
    fgq.fgq_set_path(fgq.PATH_DENSE)
    with pytest.raises(fgq.FGQError) as e:  # fp32 alphas: refused without the ablation switch
        fgq.fgq_conv2d(*args)
    assert e.value.code == fgq.FGQ_ERR_UNSUPPORTED
    fgq.fgq_debug_allow_split_fold(True)
    got = fgq.fgq_conv2d(*args).cpu().numpy()
    assert fgq.fgq_last_path() == fgq.PATH_DENSE
    mag = _split_bound(q, sc, t, al, G, (R, S, stride, pad, groups))
    steps = 2 * Kred // 16
    err = np.abs(got.astype(np.float64) - y)
    assert np.all(err <= mag * (2.0 ** -21 + steps * 2.0 ** -23) + 1e-30), f"split fold {case}"
    assert np.mean(err <= TOL * ym) > 0.99, f"split fold {case}: {np.mean(err <= TOL * ym):.4f} within TOL"


def test_conv2d_rq_dense_split():
    """Requantizing epilogue on the dense path: the codes equal the quantizer applied to the
    same path's fp32 output."""
    B, H, W, C, M, R, S, stride, pad, groups, G, act = CONV_CASES[0]
    rng = np.random.default_rng(21)
    Kred = R * S * C
    w = (rng.standard_normal((M, Kred)) * np.sqrt(2.0 / Kred)).astype(np.float32)
    t, al, codes = make_codes(w, G)
    x = random_acts((B, H, W, C), act, rng)
    q, sc, packed = quantize_oracle(x, act)
    args = (to_dev(packed), act, to_dev(np.array([sc], np.float32)), B, H, W, C, R, S, stride, pad, groups,
            to_dev(codes.view(np.int32)), to_dev(al), M, G)
    fgq.fgq_set_path(fgq.PATH_DENSE)
    fgq.fgq_debug_allow_split_fold(True)
    y32 = fgq.fgq_conv2d(*args).cpu().numpy()
    for out_type, ot in (("u8", O.U8), ("s8", O.S8)):
        scale = np.float32(2.0 ** O.dfp_exponent(y32.reshape(-1), ot))
        got = fgq.fgq_conv2d_rq(*args, out_type, to_dev(np.array([scale], np.float32))).cpu().numpy()
        assert fgq.fgq_last_path() == fgq.PATH_DENSE
        want, _, _, _ = O.quantize(y32.reshape(-1), ot, scale_in=scale)
        g = got.reshape(-1).astype(np.int64)
        if out_type == "s8":
            g = np.where(g > 127, g - 256, g)
        assert np.array_equal(g, want.astype(np.int64)), out_type


def test_dense_unsupported_shapes():
    fgq.fgq_set_path(fgq.PATH_DENSE)
    codes = torch.zeros((8, 4), dtype=torch.int32, device=dev())
    al = torch.zeros((8, 16), dtype=torch.float32, device=dev())
    with pytest.raises(fgq.FGQError) as e:  # 4-bit activations
        fgq.fgq_gemm(torch.zeros(32 * 32, dtype=torch.uint8, device=dev()), "u4", torch.ones(1, device=dev()), 32, 64,
                     codes, al, 8, 4)
    assert e.value.code == fgq.FGQ_ERR_UNSUPPORTED
    with pytest.raises(fgq.FGQError) as e:  # Kred = 48: not a multiple of 64
        fgq.fgq_gemm(torch.zeros(32 * 48, dtype=torch.uint8, device=dev()), "u8", torch.ones(1, device=dev()), 32, 48,
                     codes[:, :3].contiguous(), al[:, :12].contiguous(), 8, 4)
    assert e.value.code == fgq.FGQ_ERR_UNSUPPORTED


W8_CASES = [(2, 40, 36, 3, 64, 7, 2, 3, "u8"),   # the ResNet stem (7x7/2, C = 3) at a reduced image size
            (1, 17, 15, 16, 70, 3, 1, 1, "s8"),  # ragged M (direct stores), signed activations
            (3, 9, 9, 64, 128, 1, 1, 0, "u8")]   # 1x1, Kred = 64: one K-tile, no padding


@pytest.mark.parametrize("case", W8_CASES, ids=lambda c: "x".join(map(str, c)))
def test_conv2d_w8_dense_exact(case):
    """8-bit weights on the dense path (explicit im2col): integer products and sums below 2^24,
    so the output is the exact value, equal to the dp4a path's, and the requantized codes are
    the quantizer applied to the exact value."""
    B, H, W, C, M, R, stride, pad, act = case
    rng = np.random.default_rng(zlib.crc32(repr(case).encode()))
    Kred = R * R * C
    w = (rng.standard_normal((M, Kred)) * np.sqrt(2.0 / Kred)).astype(np.float32)
    x = random_acts((B, H, W, C), act, rng)
    q, sc, packed = quantize_oracle(x, act)
    owq, ows = O.quantize_weights_w8(w)
    y, _ = O.conv2d_w8(q, sc, R, R, stride, pad, 1, owq, ows)
    args = (to_dev(packed), act, to_dev(np.array([sc], np.float32)), B, H, W, C, R, R, stride, pad, 1, to_dev(owq),
            to_dev(ows), M)
    got = fgq.fgq_conv2d_w8(*args).cpu().numpy()
    assert fgq.fgq_last_path() == fgq.PATH_DENSE
    assert np.array_equal(got, y.astype(np.float32))
    fgq.fgq_set_path(fgq.PATH_SIMT)
    simt = fgq.fgq_conv2d_w8(*args).cpu().numpy()
    assert fgq.fgq_last_path() == fgq.PATH_SIMT
    assert np.array_equal(got, simt)
    fgq.fgq_set_path(fgq.PATH_AUTO)
    y32 = y.astype(np.float32).reshape(-1)
    for out_type, ot in (("u8", O.U8), ("s8", O.S8)):
        scale = np.float32(2.0 ** O.dfp_exponent(y32, ot))
        rq = fgq.fgq_conv2d_w8_rq(*args, out_type, to_dev(np.array([scale], np.float32))).cpu().numpy()
        assert fgq.fgq_last_path() == fgq.PATH_DENSE
        want, _, _, _ = O.quantize(y32, ot, scale_in=scale)
        g = rq.reshape(-1).astype(np.int64)
        if out_type == "s8":
            g = np.where(g > 127, g - 256, g)
        assert np.array_equal(g, want.astype(np.int64)), out_type
