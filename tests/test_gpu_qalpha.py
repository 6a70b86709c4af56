"""GPU parity of the fixed-point alphas (Section 4: alphas quantized to 8/4-bit fixed point)
and of the few-row contraction path, through the C ABI against the oracle."""
import zlib

import numpy as np
import pytest
import torch

import oracle as O
from paper_1705_01462_gb300 import fgq
from _gpu import dev, to_dev, check_within, make_codes, quantize_oracle, random_acts

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _clean_status():
    fgq.fgq_set_path(fgq.PATH_AUTO)
    yield
    fgq.fgq_set_path(fgq.PATH_AUTO)
    assert fgq.fgq_stream_status() == fgq.FGQ_OK


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("ng", [1, 7, 144, 1152])
def test_quantize_alpha_bit_exact(bits, ng):
    rng = np.random.default_rng(ng * 10 + bits)
    alpha = (np.abs(rng.standard_normal((37, ng))) * 2.0 ** rng.integers(-40, 10, (37, 1))).astype(np.float32)
    alpha[5] = 0.0
    alpha[6, ::3] = 0.0
    a, sc, _ = O.quantize_alpha(alpha, bits)
    aq, ascale = fgq.fgq_quantize_alpha(to_dev(alpha), bits)
    want = a.astype(np.uint8) if bits == 8 else O.pack_alpha4(a)
    assert np.array_equal(aq.cpu().numpy(), want)
    assert np.array_equal(ascale.cpu().numpy(), sc)


def _gemm_inputs(P, K, M, G, act, seed):
    rng = np.random.default_rng(seed)
    w = rng.standard_normal((M, K)).astype(np.float32)
    t, al, codes = make_codes(w, G)
    x = random_acts((P, K), act, rng)
    q, sc, packed = quantize_oracle(x, act)
    return t, al, codes, q, sc, packed


GEMV_CASES = [(1, 64, 8, 4, "u8"), (1, 9216, 300, 4, "u8"), (3, 576, 64, 8, "s8"), (8, 4096, 129, 16, "u8"),
              (5, 1024, 64, 32, "s8"), (2, 4096, 70, 64, "u8"), (7, 4112, 33, 128, "u8"), (1, 16384, 40, 64, "s8")]


@pytest.mark.parametrize("case", GEMV_CASES, ids=lambda c: "x".join(map(str, c)))
def test_gemv_path_fp32_alpha(case):
    P, K, M, G, act = case
    t, al, codes, q, sc, packed = _gemm_inputs(P, K, M, G, act, zlib.crc32(repr(case).encode()))
    y, ym = O.gemm(q, sc, t, al, G)
    gy = fgq.fgq_gemm(to_dev(packed), act, to_dev(np.array([sc], np.float32)), P, K, to_dev(codes.view(np.int32)),
                      to_dev(al), M, G)
    assert fgq.fgq_last_path() == fgq.PATH_GEMV
    check_within(gy.cpu().numpy(), y, ym, f"gemv {case}")


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("case", GEMV_CASES, ids=lambda c: "x".join(map(str, c)))
def test_gemv_path_fixed_point_alpha_exact(case, bits):
    """Integer alphas times integer group sums, summed exactly: the result is the exact value
    rounded once to fp32."""
    P, K, M, G, act = case
    t, al, codes, q, sc, packed = _gemm_inputs(P, K, M, G, act, zlib.crc32(repr(case).encode()) + bits)
    a, asc, _ = O.quantize_alpha(al, bits)
    y, _ = O.gemm(q, sc, t, O.dequantize_alpha(a, asc), G)
    aq = a.astype(np.uint8) if bits == 8 else O.pack_alpha4(a)
    gy = fgq.fgq_gemm_qa(to_dev(packed), act, to_dev(np.array([sc], np.float32)), P, K, to_dev(codes.view(np.int32)),
                         to_dev(aq), bits, to_dev(asc), M, G)
    assert fgq.fgq_last_path() == fgq.PATH_GEMV
    assert np.array_equal(gy.cpu().numpy(), y.astype(np.float32))


@pytest.mark.parametrize("case", [(300, 576, 64, 4, "u8"), (129, 200, 65, 8, "s8"), (256, 1024, 128, 64, "u8"),
                                  (64, 512, 130, 4, "u4")], ids=lambda c: "x".join(map(str, c)))
def test_gemm_qa_other_paths(case):
    P, K, M, G, act = case
    t, al, codes, q, sc, packed = _gemm_inputs(P, K, M, G, act, zlib.crc32(repr(case).encode()))
    a, asc, _ = O.quantize_alpha(al, 8)
    y, ym = O.gemm(q, sc, t, O.dequantize_alpha(a, asc), G)
    gy = fgq.fgq_gemm_qa(to_dev(packed), act, to_dev(np.array([sc], np.float32)), P, K, to_dev(codes.view(np.int32)),
                         to_dev(a.astype(np.uint8)), 8, to_dev(asc), M, G)
    assert fgq.fgq_last_path() != fgq.PATH_GEMV
    check_within(gy.cpu().numpy(), y, ym, f"gemm_qa {case}")


@pytest.mark.parametrize("bits", [8, 4])
def test_conv2d_qa(bits):
    B, H, W, C, M, R, S, stride, pad, groups, G = 2, 14, 14, 128, 128, 3, 3, 1, 1, 1, 4
    rng = np.random.default_rng(bits)
    w = (rng.standard_normal((M, R * S * C)) * np.sqrt(2.0 / (R * S * C))).astype(np.float32)
    t, al, codes = make_codes(w, G)
    x = random_acts((B, H, W, C), "u8", rng)
    q, sc, packed = quantize_oracle(x, "u8")
    a, asc, _ = O.quantize_alpha(al, bits)
    y, ym = O.conv2d(q, sc, R, S, stride, pad, groups, t, O.dequantize_alpha(a, asc), G)
    aq = a.astype(np.uint8) if bits == 8 else O.pack_alpha4(a)
    gout = fgq.fgq_conv2d_qa(to_dev(packed), "u8", to_dev(np.array([sc], np.float32)), B, H, W, C, R, S, stride, pad,
                             groups, to_dev(codes.view(np.int32)), to_dev(aq), bits, to_dev(asc), M, G)
    check_within(gout.cpu().numpy(), y, ym, f"conv2d_qa bits={bits}")


def test_forced_gemv_on_unsupported_shape():
    fgq.fgq_set_path(fgq.PATH_GEMV)
    q = torch.zeros(16 * 64, dtype=torch.uint8, device=dev())
    codes = torch.zeros((8, 4), dtype=torch.int32, device=dev())
    al = torch.zeros((8, 16), dtype=torch.float32, device=dev())
    with pytest.raises(fgq.FGQError) as e:  # P = 16 rows is more than the path takes
        fgq.fgq_gemm(q, "u8", torch.ones(1, device=dev()), 16, 64, codes, al, 8, 4)
    assert e.value.code == fgq.FGQ_ERR_UNSUPPORTED
