"""Exact-rational helpers used by the oracle pins (independent of the oracle's code)."""
from fractions import Fraction
import itertools
import struct

import numpy as np


def f32_from_fraction(x: Fraction) -> np.float32:
    """Nearest fp32 (ties to even, subnormals included) to a non-negative rational."""
    if x == 0:
        return np.float32(0.0)
    assert x > 0
    # binary exponent e with 2^e <= x < 2^(e+1)
    e = x.numerator.bit_length() - x.denominator.bit_length()
    while Fraction(2) ** e > x:
        e -= 1
    while Fraction(2) ** (e + 1) <= x:
        e += 1
    lsb = max(e - 23, -149)
    scaled = x / (Fraction(2) ** lsb)
    fl = scaled.numerator // scaled.denominator
    rem = scaled - fl
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and fl % 2 == 1):
        fl += 1
    return np.float32(float(Fraction(fl) * Fraction(2) ** lsb))


def bits(x) -> int:
    return struct.unpack("<I", struct.pack("<f", float(np.float32(x))))[0]


def best_alpha_for_code(w, t):
    """Optimal alpha >= 0 for a fixed code t: argmin ||w - alpha t||^2 = max(0, <w,t>/|t|)."""
    nz = sum(abs(v) for v in t)
    if nz == 0:
        return Fraction(0)
    a = sum(Fraction(wi) * ti for wi, ti in zip(w, t)) / nz
    return max(a, Fraction(0))


def error(w, t, alpha):
    return sum((Fraction(wi) - alpha * ti) ** 2 for wi, ti in zip(w, t))


def brute_force(w):
    """All 3^G codes with their exact optimal-alpha error; returns (min_err, list of (err, t))."""
    out = []
    for t in itertools.product((-1, 0, 1), repeat=len(w)):
        a = best_alpha_for_code(w, t)
        out.append((error(w, t, a), t))
    return min(e for e, _ in out), out


def is_threshold_code(w, t):
    """t keeps exactly {i : |w_i| >= tau} for some tau > 0, with t_i = sign(w_i)."""
    kept = [abs(Fraction(wi)) for wi, ti in zip(w, t) if ti != 0]
    if not kept:
        return True
    tau = min(kept)
    for wi, ti in zip(w, t):
        a = abs(Fraction(wi))
        if (a >= tau) != (ti != 0):
            return False
        if ti != 0 and (ti > 0) != (wi > 0):
            return False
    return True
