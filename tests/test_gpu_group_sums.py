"""GPU parity of the 32-bit group accumulators (Section 4; the inner sums of Eq. 2) on every
kernel family that forms them, through the C ABI, bit for bit against the oracle.

The tensor-core kernels hold a group's sum in TMEM as an fp32 value that must be an exact
integer (fp16 codes and 8/4-bit activations, exact products, |s| <= 128 * 255 < 2^24); the
group-sums entry points store exactly those accumulators as int32, so these tests compare
the integers the fp32-output kernels multiply by alpha.  Codes and activations are drawn
over their whole ranges, with saturated all-ones cases for the largest magnitudes."""
import zlib

import numpy as np
import pytest
import torch

import oracle as O
from paper_1705_01462_gb300 import fgq
from _gpu import ORACLE_TYPE, to_dev

pytestmark = pytest.mark.gpu

QRANGE = {"u8": (0, 255), "s8": (-128, 127), "u4": (0, 15), "s4": (-8, 7)}


@pytest.fixture(autouse=True)
def _clean_status():
    fgq.fgq_set_path(fgq.PATH_AUTO)
    yield
    fgq.fgq_set_path(fgq.PATH_AUTO)
    assert fgq.fgq_stream_status() == fgq.FGQ_OK


def _codes(shape, act, rng, saturate=False):
    lo, hi = QRANGE[act]
    if saturate:
        return np.full(shape, lo if act.startswith("s") else hi, np.int32)
    return rng.integers(lo, hi + 1, shape).astype(np.int32)


def _ternary(M, Kred, G, rng, saturate=False):
    ng = O.num_groups(Kred, G)
    t = np.ones((M, ng * G), np.int8) if saturate else rng.integers(-1, 2, (M, ng * G)).astype(np.int8)
    t[:, Kred:] = 0
    return t


def _paths(G, Mg, Kg):
    """(forced path, expected family) pairs to run: the dp4a kernel, the tensor-core kernel
    where it covers the shape, and the automatic choice."""
    out = [(fgq.PATH_SIMT, fgq.PATH_SIMT)]
    tc_ok = G in (4, 64, 128) and Kg % 64 == 0
    if tc_ok:
        out.append((fgq.PATH_TC, fgq.PATH_TC))
    auto = fgq.PATH_TC if tc_ok and not (G == 4 and Mg < 64) else fgq.PATH_SIMT
    out.append((fgq.PATH_AUTO, auto))
    return out


GEMM_CASES = [
    # P, Kred, M, G, act, saturate
    (200, 4608, 200, 4, "u8", False),   # Kred = 3*3*512, ragged P and M tiles
    (130, 4608, 136, 64, "u8", False),
    (129, 4608, 130, 128, "s8", False),
    (96, 1024, 128, 4, "s8", False),
    (70, 512, 256, 4, "u4", False),
    (257, 512, 130, 64, "s4", False),
    (64, 256, 128, 128, "u4", False),
    (100, 4608, 128, 4, "u8", True),    # |s| = 4 * 255 in every group
    (100, 4608, 130, 128, "u8", True),  # |s| = 128 * 255, the largest group sum
    (65, 1024, 128, 64, "s8", True),    # -128 * 64 per group
    (33, 580, 64, 4, "u8", False),      # Kred not a multiple of 64: the dp4a kernel only
]


@pytest.mark.parametrize("case", GEMM_CASES, ids=lambda c: "x".join(map(str, c)))
def test_gemm_group_sums_bit_exact(case):
    P, Kred, M, G, act, sat = case
    rng = np.random.default_rng(zlib.crc32(repr(case).encode()))
    q = _codes((P, Kred), act, rng, sat)
    t = _ternary(M, Kred, G, rng, sat)
    want = O.group_sums(q, t, G)
    qd = to_dev(O.pack_act(q, ORACLE_TYPE[act]))
    cd = to_dev(O.pack_codes(t).view(np.int32))
    for forced, family in _paths(G, M, Kred):
        fgq.fgq_set_path(forced)
        got = fgq.fgq_group_sums(qd, act, P, Kred, cd, M, G).cpu().numpy()
        assert fgq.fgq_last_path() == family, (forced, fgq.fgq_last_path())
        assert np.array_equal(got.astype(np.int64), want), f"{case} path {family}: " \
            f"{int((got != want).sum())} of {want.size} group sums differ"


CONV_CASES = [
    # B, H, W, C, M, R, stride, pad, groups, G, act, saturate
    (2, 9, 9, 512, 128, 3, 1, 1, 1, 4, "u8", False),    # Kred = 4608, gathered rows with padding
    (2, 9, 9, 512, 136, 3, 1, 1, 1, 64, "u8", False),   # ragged M tile
    (3, 11, 10, 128, 256, 3, 2, 1, 2, 4, "s8", False),  # two conv groups (Cg = 64), stride 2
    (3, 11, 10, 128, 256, 3, 2, 1, 2, 64, "u4", False),
    (2, 7, 9, 256, 192, 1, 1, 0, 1, 4, "u8", False),    # 1x1 stride 1: activation rows by TMA
    (2, 7, 9, 256, 130, 1, 1, 0, 1, 128, "s4", False),
    (1, 14, 14, 256, 128, 1, 2, 0, 1, 64, "s8", False), # strided 1x1 (a projection)
    (1, 8, 8, 256, 128, 3, 1, 1, 1, 128, "u8", True),   # saturated: |s| = 128 * 255 inside the image
]


@pytest.mark.parametrize("case", CONV_CASES, ids=lambda c: "x".join(map(str, c)))
def test_conv2d_group_sums_bit_exact(case):
    B, H, W, C, M, R, stride, pad, groups, G, act, sat = case
    rng = np.random.default_rng(zlib.crc32(repr(case).encode()))
    Cg = C // groups
    Kred = R * R * Cg
    q = _codes((B, H, W, C), act, rng, sat)
    t = _ternary(M, Kred, G, rng, sat)
    Ho, Wo = O.conv_out_hw(H, W, R, R, stride, pad)
    P = B * Ho * Wo
    pos = np.unique(np.concatenate([[0, P - 1], rng.choice(P, size=min(P, 48), replace=False)]))
    want = O.conv2d_group_sums(q, R, R, stride, pad, groups, t, G, positions=pos)
    qd = to_dev(O.pack_act(q, ORACLE_TYPE[act]))
    cd = to_dev(O.pack_codes(t).view(np.int32))
    for forced, family in _paths(G, M // groups, Cg):
        fgq.fgq_set_path(forced)
        got = fgq.fgq_conv2d_group_sums(qd, act, B, H, W, C, R, R, stride, pad, groups, cd, M, G).cpu().numpy()
        assert fgq.fgq_last_path() == family, (forced, fgq.fgq_last_path())
        assert got.shape == (M, O.num_groups(Kred, G), P)
        g = got[:, :, pos].astype(np.int64)
        assert np.array_equal(g, want), f"{case} path {family}: {int((g != want).sum())} of {want.size} differ"


def test_group_sums_agree_with_fp32_output():
    """The fp32 output of the tensor-core kernels is s_x * sum_g alpha_g * s_g over the very
    group sums the group-sums call returns (same kernel family, same shape): recombined in
    fp64, the two agree within the contraction tolerance."""
    rng = np.random.default_rng(7)
    B, H, W, C, M, R, stride, pad = 2, 9, 9, 256, 128, 3, 1, 1
    Kred = R * R * C
    q = _codes((B, H, W, C), "u8", rng)
    qd = to_dev(O.pack_act(q, O.U8))
    sc = np.float32(2.0 ** -6)
    for G in (4, 64):
        w = rng.standard_normal((M, Kred)).astype(np.float32)
        t, al, _ = O.ternarize(w, G)
        cd = to_dev(O.pack_codes(t).view(np.int32))
        fgq.fgq_set_path(fgq.PATH_TC)
        s = fgq.fgq_conv2d_group_sums(qd, "u8", B, H, W, C, R, R, stride, pad, 1, cd, M, G).cpu().numpy()
        y = fgq.fgq_conv2d(qd, "u8", to_dev(np.array([sc], np.float32)), B, H, W, C, R, R, stride, pad, 1, cd,
                           to_dev(al), M, G).cpu().numpy().reshape(-1, M)
        assert fgq.fgq_last_path() == fgq.PATH_TC
        s64 = s.astype(np.float64)
        ref = float(sc) * np.einsum("mgp,mg->pm", s64, al.astype(np.float64))
        mag = float(sc) * np.einsum("mgp,mg->pm", np.abs(s64), al.astype(np.float64))
        assert np.all(np.abs(y.astype(np.float64) - ref) <= 1e-5 * mag), f"G={G}"
