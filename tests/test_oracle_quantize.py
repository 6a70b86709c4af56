"""Pins for the oracle's dynamic-fixed-point activation quantiser (Section 4: activations
quantised to 8 or 4 bits with one shared exponent per tensor) and its packing."""
import numpy as np
import pytest

import oracle as O
from conftest import read_golden, parse_floats, parse_ints

TYPES = {"u8": O.U8, "s8": O.S8, "u4": O.U4, "s4": O.S4}


def test_worked_examples():
    rows = read_golden("quantize_worked.txt", 6)
    assert len(rows) >= 6
    for ty, sc, xs, qs, E, why in rows:
        x = np.array(parse_floats(xs), np.float32)
        q, scale, e, st = O.quantize(x, TYPES[ty], float(sc))
        assert st == O.OK
        assert list(q) == parse_ints(qs), why
        assert e == int(E) and scale == np.float32(2.0 ** int(E)), why


def test_pack_worked_examples():
    for ty, qs, bs, why in read_golden("pack_act_worked.txt", 4):
        out = O.pack_act(np.array(parse_ints(qs), np.int32), TYPES[ty])
        assert list(out) == parse_ints(bs), why


@pytest.mark.parametrize("ty", ["u8", "s8", "u4", "s4"])
def test_exponent_is_minimal(ty):
    """E is the smallest integer with max*2^-E <= qmax (checked in fp64 around E)."""
    qmin, qmax = O.QRANGE[TYPES[ty]]
    rng = np.random.default_rng(1)
    for _ in range(400):
        e = int(rng.integers(-120, 100))
        x = (rng.standard_normal(16) * 2.0 ** e).astype(np.float32)
        if ty.startswith("u"):
            x = np.abs(x)
        E = O.dfp_exponent(x, TYPES[ty])
        m = float(np.max(np.maximum(x, 0) if ty.startswith("u") else np.abs(x)))
        assert m * 2.0 ** -E <= qmax
        assert m * 2.0 ** -(E - 1) > qmax


@pytest.mark.parametrize("ty", ["u8", "s8", "u4", "s4"])
def test_codes_match_rint(ty):
    """q = clip(rint(x * 2^-E)) with numpy's round-half-even rint, and the round trip
    error of unsaturated values is at most half a step 2^(E-1)."""
    qmin, qmax = O.QRANGE[TYPES[ty]]
    rng = np.random.default_rng(2)
    for s in (1e-30, 1e-3, 1.0, 37.0, 1e20):
        x = (rng.standard_normal(5000) * s).astype(np.float32)
        if ty.startswith("u"):
            x = np.abs(x) * np.where(rng.random(5000) < 0.1, -1, 1).astype(np.float32)
        q, scale, E, st = O.quantize(x, TYPES[ty])
        ref = np.clip(np.rint(x.astype(np.float64) * 2.0 ** -E), qmin, qmax)
        assert np.array_equal(q, ref.astype(np.int32))
        uns = (ref > qmin) & (ref < qmax)
        err = np.abs(x.astype(np.float64) - q * 2.0 ** E)
        assert np.all(err[uns] <= 2.0 ** (E - 1))
        if ty.startswith("u"):
            assert np.all(q[x < 0] == 0)


def test_ties_round_to_even():
    x = np.array([0.5, 1.5, 2.5, 3.5, 254.5, 255.0], np.float32)
    q, _, E, _ = O.quantize(x, O.U8)
    assert E == 0 and list(q) == [0, 2, 2, 4, 254, 255]


def test_given_scale():
    q, sc, E, st = O.quantize(np.array([3.0, -3.0, 1000.0], np.float32), O.S8, 0.25)
    assert st == O.OK and E == -2 and list(q) == [12, -12, 127]
    _, _, _, st = O.quantize(np.array([1.0], np.float32), O.U8, 0.3, check=False)
    assert st == O.ERR_ARG


def test_nonfinite():
    _, _, _, st = O.quantize(np.array([1.0, np.nan], np.float32), O.U8, check=False)
    assert st == O.ERR_NONFINITE


def test_tiny_and_huge_ranges():
    """Exponent clamped to [-149, 127] so that the scale 2^E is an fp32 number."""
    q, sc, E, _ = O.quantize(np.array([2.0 ** -149, 0.0], np.float32), O.U8)
    assert E == -149 and q[0] == 1 and sc == np.float32(2.0 ** -149)
    big = np.float32(3.0e38)
    q, sc, E, _ = O.quantize(np.array([big, 1.0], np.float32), O.U8)
    assert big * 2.0 ** -E <= 255 and q[0] == np.rint(float(big) * 2.0 ** -E)


def test_pack_roundtrip_nibbles():
    rng = np.random.default_rng(3)
    for ty in (O.U4, O.S4):
        lo, hi = O.QRANGE[ty]
        q = rng.integers(lo, hi + 1, 1001).astype(np.int32)
        b = O.pack_act(q, ty)
        assert b.size == 501
        low = (b & 0xF).astype(np.int32)
        high = (b >> 4).astype(np.int32)
        un = np.empty(1002, np.int32)
        un[0::2], un[1::2] = low, high
        un = un[:1001]
        if ty == O.S4:
            un = np.where(un >= 8, un - 16, un)
        assert np.array_equal(un, q)
        assert high[-1] == 0
