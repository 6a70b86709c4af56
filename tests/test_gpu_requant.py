"""GPU parity of the fused output requantization (Section 4: 32-bit outputs converted to 8
bits and rounded before the next layer) on every contraction path, through the C ABI.

Two checks per case: the requantized codes equal the oracle's quantizer (fixed scale)
applied to the same kernel's fp32 output, bit for bit; and against the oracle's own
output they differ by at most one code, and only where the exact value lies within the
contraction tolerance of a rounding boundary."""
import zlib

import numpy as np
import pytest

import oracle as O
from paper_1705_01462_gb300 import fgq
from _gpu import TOL, to_dev, make_codes, quantize_oracle, random_acts

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _clean_status():
    fgq.fgq_set_path(fgq.PATH_AUTO)
    # whole tiles on the fp32 calls too: their rounding order is the one the requantizing
    # entries use, so the codes can be compared bit for bit
    prev = fgq.fgq_debug_max_ksplit(1)
    yield
    fgq.fgq_debug_max_ksplit(prev)
    fgq.fgq_set_path(fgq.PATH_AUTO)
    assert fgq.fgq_stream_status() == fgq.FGQ_OK


def _check_codes(got, y32_gpu, y_oracle, ym, out_type, scale, what):
    ot = O.U8 if out_type == "u8" else O.S8
    want_self, _, _, _ = O.quantize(y32_gpu.reshape(-1), ot, scale_in=scale)
    g = got.reshape(-1).astype(np.int64)
    if out_type == "s8":
        g = np.where(g > 127, g - 256, g)
    assert np.array_equal(g, want_self.astype(np.int64)), f"{what}: codes differ from requantizing the fp32 output"
    want_o, _, _, _ = O.quantize(y_oracle.reshape(-1).astype(np.float32), ot, scale_in=scale)
    d = np.abs(g - want_o.astype(np.int64))
    assert d.max(initial=0) <= 1, what
    v = y_oracle.reshape(-1) / scale
    b = TOL * ym.reshape(-1) / scale + 1e-9 * np.abs(v)
    near = np.floor(v + b + 0.5) != np.floor(v - b + 0.5)  # a half-integer lies within +-b
    assert np.all((d == 0) | near), f"{what}: a code differs away from a rounding boundary"


def _out_scale(y, out_type, shrink):
    E = O.dfp_exponent(y.astype(np.float32).reshape(-1), O.U8 if out_type == "u8" else O.S8)
    return np.float32(2.0 ** (E - shrink))


CONV_CASES = [
    # B, H, W, C, M, R, S, stride, pad, groups, G, act, path
    (1, 12, 12, 64, 70, 3, 3, 1, 1, 1, 4, "u8", fgq.PATH_SIMT),
    (2, 9, 11, 64, 128, 3, 3, 1, 1, 1, 4, "u8", fgq.PATH_TC),
    (1, 14, 14, 128, 256, 1, 1, 1, 0, 1, 4, "s8", fgq.PATH_TC),
    (2, 9, 9, 64, 130, 3, 3, 1, 1, 1, 64, "u8", fgq.PATH_TC),
    (1, 10, 10, 128, 64, 1, 1, 1, 0, 1, 64, "u8", fgq.PATH_TC),
    (1, 9, 9, 32, 24, 3, 3, 2, 1, 1, 8, "u8", fgq.PATH_SIMT),
    (1, 9, 9, 16, 8, 3, 3, 1, 1, 1, 2, "s8", fgq.PATH_SIMT),
    (1, 13, 13, 48, 64, 5, 5, 1, 2, 2, 4, "u8", fgq.PATH_SIMT),
    (2, 8, 8, 64, 40, 3, 3, 1, 1, 1, 4, "u4", fgq.PATH_SIMT),
]


@pytest.mark.parametrize("out_type", ["u8", "s8"])
@pytest.mark.parametrize("case", CONV_CASES, ids=lambda c: "x".join(map(str, c)))
def test_conv2d_rq(case, out_type):
    B, H, W, C, M, R, S, stride, pad, groups, G, act, path = case
    rng = np.random.default_rng(zlib.crc32(repr((case, out_type)).encode()))
    Cg = C // groups
    w = (rng.standard_normal((M, R * S * Cg)) * np.sqrt(2.0 / (R * S * Cg))).astype(np.float32)
    t, al, codes = make_codes(w, G)
    x = random_acts((B, H, W, C), act, rng)
    q, sc, packed = quantize_oracle(x, act)
    y, ym = O.conv2d(q, sc, R, S, stride, pad, groups, t, al, G)
    args = (to_dev(packed), act, to_dev(np.array([sc], np.float32)), B, H, W, C, R, S, stride, pad, groups,
            to_dev(codes.view(np.int32)), to_dev(al), M, G)
    fgq.fgq_set_path(path)
    y32 = fgq.fgq_conv2d(*args).cpu().numpy()
    for shrink in (0, 2):  # the DFP scale of the output, and one that saturates
        scale = _out_scale(y, out_type, shrink)
        got = fgq.fgq_conv2d_rq(*args, out_type, to_dev(np.array([scale], np.float32)))
        assert fgq.fgq_last_path() == path
        _check_codes(got.cpu().numpy(), y32, y, ym, out_type, scale, f"conv2d_rq {case} {out_type} {shrink}")


@pytest.mark.parametrize("case", [(1, 4096, 300, 4, "u8", fgq.PATH_GEMV), (5, 1024, 64, 64, "s8", fgq.PATH_GEMV),
                                  (300, 576, 64, 4, "u8", fgq.PATH_SIMT), (256, 1024, 256, 64, "u8", fgq.PATH_TC),
                                  (128, 512, 128, 4, "u8", fgq.PATH_TC)], ids=lambda c: "x".join(map(str, c)))
def test_gemm_rq(case):
    P, K, M, G, act, path = case
    rng = np.random.default_rng(P * 7 + K + M)
    w = rng.standard_normal((M, K)).astype(np.float32)
    t, al, codes = make_codes(w, G)
    x = random_acts((P, K), act, rng)
    q, sc, packed = quantize_oracle(x, act)
    y, ym = O.gemm(q, sc, t, al, G)
    args = (to_dev(packed), act, to_dev(np.array([sc], np.float32)), P, K, to_dev(codes.view(np.int32)), to_dev(al),
            M, G)
    fgq.fgq_set_path(path)
    y32 = fgq.fgq_gemm(*args).cpu().numpy()
    scale = _out_scale(y, "u8", 0)
    got = fgq.fgq_gemm_rq(*args, "u8", to_dev(np.array([scale], np.float32)))
    assert fgq.fgq_last_path() == path
    _check_codes(got.cpu().numpy(), y32, y, ym, "u8", scale, f"gemm_rq {case}")
