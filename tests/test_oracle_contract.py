"""Pins for the oracle's grouped ternary contraction (Eq. 2 applied to convolution and
fully connected layers; 32-bit group accumulators of Section 4; 8-bit first layer)."""
import numpy as np
import pytest
import torch

import oracle as O
from conftest import read_golden, parse_ints


def _dense_weights(t, alpha, G, M, R, S, Cg):
    """alpha_g * t as a dense fp64 torch weight [M][Cg][R][S] (Kred order (r, s, c))."""
    Kp = t.shape[1]
    Kred = R * S * Cg
    wd = (t.astype(np.float64).reshape(M, -1, G) * alpha.astype(np.float64)[:, :, None]).reshape(M, Kp)
    wd = wd[:, :Kred].reshape(M, R, S, Cg).transpose(0, 3, 1, 2)
    return torch.from_numpy(np.ascontiguousarray(wd))


CASES = [
    # B, H, W, C, M, R, S, stride, pad, groups, G
    (1, 6, 7, 8, 5, 3, 3, 1, 1, 1, 4),
    (2, 5, 5, 6, 4, 3, 3, 2, 1, 1, 4),       # Kred = 54, ragged last group
    (1, 9, 9, 3, 6, 7, 7, 2, 3, 1, 8),       # C = 3 stem-like, groups straddle taps
    (2, 7, 6, 8, 6, 5, 5, 1, 2, 2, 16),      # conv groups = 2 (AlexNet towers)
    (1, 4, 4, 64, 3, 1, 1, 1, 0, 1, 64),
    (1, 5, 5, 16, 4, 3, 3, 1, 1, 1, 1),
    (1, 4, 6, 12, 4, 1, 1, 2, 0, 1, 2),      # strided 1x1
]


@pytest.mark.parametrize("case", CASES)
def test_conv2d_matches_torch_conv(case):
    """With alpha_g * t expanded to a dense kernel the contraction is a plain convolution:
    compare against torch.nn.functional.conv2d in fp64 on the CPU."""
    B, H, W, C, M, R, S, stride, pad, groups, G = case
    rng = np.random.default_rng(sum(case))
    Cg = C // groups
    w = rng.standard_normal((M, R * S * Cg)).astype(np.float32)
    t, al, _ = O.ternarize(w, G)
    q = rng.integers(0, 256, (B, H, W, C)).astype(np.int32)
    sx = 2.0 ** -5
    y, ym = O.conv2d(q, sx, R, S, stride, pad, groups, t, al, G)
    ref = torch.nn.functional.conv2d(torch.from_numpy(q.transpose(0, 3, 1, 2).astype(np.float64)),
                                     _dense_weights(t, al, G, M, R, S, Cg), stride=stride, padding=pad,
                                     groups=groups).numpy().transpose(0, 2, 3, 1) * sx
    assert y.shape == ref.shape
    np.testing.assert_allclose(y, ref, rtol=1e-12, atol=1e-12 * np.abs(ref).max())
    assert np.all(ym >= np.abs(y) * (1 - 1e-12))
    # sampled positions give the same values
    Ho, Wo = y.shape[1:3]
    pos = rng.choice(B * Ho * Wo, size=min(7, B * Ho * Wo), replace=False)
    ys, yms = O.conv2d(q, sx, R, S, stride, pad, groups, t, al, G, positions=pos)
    np.testing.assert_array_equal(ys, y.reshape(-1, M)[pos])
    np.testing.assert_array_equal(yms, ym.reshape(-1, M)[pos])


def test_gemm_matches_matmul():
    rng = np.random.default_rng(1)
    for P, K, M, G in [(7, 64, 5, 4), (3, 130, 9, 64), (1, 17, 3, 4), (4, 256, 2, 128)]:
        w = rng.standard_normal((M, K)).astype(np.float32)
        t, al, _ = O.ternarize(w, G)
        q = rng.integers(-128, 128, (P, K)).astype(np.int32)
        y, ym = O.gemm(q, 0.5, t, al, G)
        wd = (t.astype(np.float64).reshape(M, -1, G) * al.astype(np.float64)[:, :, None]).reshape(M, -1)[:, :K]
        np.testing.assert_allclose(y, 0.5 * q.astype(np.float64) @ wd.T, rtol=1e-12, atol=1e-9)


def test_group_sums_direct_enumeration():
    """s[m][g][p] by explicit Python loops, element by element."""
    rng = np.random.default_rng(2)
    P, K, M, G = 5, 22, 3, 4
    t = rng.integers(-1, 2, (M, 24)).astype(np.int8)
    t[:, 22:] = 0
    q = rng.integers(0, 256, (P, K)).astype(np.int32)
    s = O.group_sums(q, t, G)
    for m in range(M):
        for g in range(6):
            for p in range(P):
                acc = 0
                for j in range(g * G, min((g + 1) * G, K)):
                    acc += int(t[m, j]) * int(q[p, j])
                assert s[m, g, p] == acc
    # and the fp64 output is sx * sum_g alpha_g * s_g
    al = rng.random((M, 6)).astype(np.float32)
    y, _ = O.gemm(q, 1.0, t, al, G)
    np.testing.assert_allclose(y, np.einsum("mgp,mg->pm", s.astype(np.float64), al.astype(np.float64)),
                               rtol=1e-13)


def test_box_filter_closed_form():
    """G = Kred, all codes +1, alpha = 1: the output is sx * (sum of the receptive field)."""
    rng = np.random.default_rng(3)
    B, H, W, C, R = 1, 6, 6, 4, 3
    Kred = R * R * C
    t = np.ones((1, Kred), np.int8)
    al = np.ones((1, 1), np.float32)
    q = rng.integers(0, 256, (B, H, W, C)).astype(np.int32)
    y, _ = O.conv2d(q, 0.25, R, R, 1, 0, 1, t, al, Kred)
    for ho in range(H - R + 1):
        for wo in range(W - R + 1):
            assert y[0, ho, wo, 0] == 0.25 * q[0, ho:ho + R, wo:wo + R, :].sum()


def test_w8_first_layer_matches_torch_conv():
    rng = np.random.default_rng(4)
    B, H, W, C, M, R, stride, pad = 2, 11, 11, 3, 8, 7, 2, 3
    w = (rng.standard_normal((M, R * R * C)) * 0.1).astype(np.float32)
    wq, ws = O.quantize_weights_w8(w)
    for m in range(M):
        assert np.abs(wq[m]).max() <= 127 and np.abs(wq[m]).max() >= 64
    q = rng.integers(0, 256, (B, H, W, C)).astype(np.int32)
    y, _ = O.conv2d_w8(q, 2.0 ** -3, R, R, stride, pad, 1, wq, ws)
    wd = (wq.astype(np.float64) * ws.astype(np.float64)[:, None]).reshape(M, R, R, C).transpose(0, 3, 1, 2)
    ref = torch.nn.functional.conv2d(torch.from_numpy(q.transpose(0, 3, 1, 2).astype(np.float64)),
                                     torch.from_numpy(np.ascontiguousarray(wd)), stride=stride,
                                     padding=pad).numpy().transpose(0, 2, 3, 1) * 2.0 ** -3
    np.testing.assert_allclose(y, ref, rtol=1e-13)


def test_codes_worked_examples():
    for ts, ws, why in read_golden("codes_worked.txt", 3):
        t = np.array([parse_ints(ts)], np.int8)
        assert list(O.pack_codes(t)[0]) == parse_ints(ws), why


@pytest.mark.parametrize("B,H,W,C,M,R,stride,pad,groups,G", [
    (2, 6, 5, 8, 6, 3, 1, 1, 1, 4),     # groups of 4 channels at one tap
    (1, 7, 7, 3, 4, 3, 2, 1, 1, 4),     # C = 3: groups straddle taps
    (2, 9, 8, 16, 6, 3, 2, 0, 2, 8),    # two conv groups, stride 2, no padding
    (1, 5, 5, 64, 3, 3, 1, 1, 1, 64),   # G = 64: one group per tap
    (1, 4, 4, 6, 2, 1, 1, 0, 1, 128),   # one group longer than Kred (zero padding)
])
def test_conv_group_sums_match_torch_conv(B, H, W, C, M, R, stride, pad, groups, G):
    """oracle.conv2d_group_sums[m][g] equals a float64 torch convolution whose weights keep
    only group g's codes of filter m (every other code zeroed): the group decomposition of
    Eq. 2 read off a library convolution, including the (r, s, c) order, padding, stride and
    conv groups."""
    rng = np.random.default_rng(11)
    Cg = C // groups
    Kred = R * R * Cg
    ng = O.num_groups(Kred, G)
    Kp = ng * G
    t = rng.integers(-1, 2, (M, Kp)).astype(np.int8)
    t[:, Kred:] = 0
    q = rng.integers(0, 256, (B, H, W, C)).astype(np.int32)
    s = O.conv2d_group_sums(q, R, R, stride, pad, groups, t, G)
    Ho, Wo = O.conv_out_hw(H, W, R, R, stride, pad)
    x = torch.from_numpy(q.transpose(0, 3, 1, 2).astype(np.float64))
    for g in range(ng):
        tm = np.zeros_like(t)
        tm[:, g * G:(g + 1) * G] = t[:, g * G:(g + 1) * G]
        wt = tm[:, :Kred].astype(np.float64).reshape(M, R, R, Cg).transpose(0, 3, 1, 2)
        ref = torch.nn.functional.conv2d(x, torch.from_numpy(np.ascontiguousarray(wt)), stride=stride,
                                         padding=pad, groups=groups).numpy()
        ref = ref.transpose(1, 0, 2, 3).reshape(M, B * Ho * Wo)
        assert np.array_equal(s[:, g, :], ref.astype(np.int64)), f"group {g}"
    # listed positions return the same columns
    pos = rng.choice(B * Ho * Wo, size=min(5, B * Ho * Wo), replace=False)
    assert np.array_equal(O.conv2d_group_sums(q, R, R, stride, pad, groups, t, G, positions=pos), s[:, :, pos])
    # a 1x1 stride-1 convolution is the GEMM of the group sums
    if R == 1 and stride == 1 and pad == 0 and groups == 1:
        assert np.array_equal(s, O.group_sums(q.reshape(-1, C), t, G))
