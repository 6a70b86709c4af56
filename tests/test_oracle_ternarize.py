"""Pins for the oracle's FGQ ternarizer (Section 3.1, Eq. 2, Eq. 4, Eq. 5, Lemma 1).

The oracle is checked against things other than itself: hand-worked examples, exact
brute force over all 3^G codes (rational arithmetic), closed forms, equivariances and
the statistics of Lemma 1.
"""
from fractions import Fraction
import itertools

import numpy as np
import pytest

import oracle as O
from conftest import read_golden, parse_floats, parse_ints
from _exact import f32_from_fraction, bits, brute_force, error, is_threshold_code


def _groups(G, n, seed):
    """Adversarial group mix: Gaussian, exponential, uniform, tied, zero-heavy, subnormal,
    wide dynamic range, power-of-two magnitudes."""
    rng = np.random.default_rng(seed)
    out = []
    for i in range(n):
        kind = i % 9
        if kind == 0:
            w = rng.standard_normal(G)
        elif kind == 1:
            w = rng.exponential(1.0, G) * rng.choice([-1, 1], G)
        elif kind == 2:
            w = rng.uniform(-1, 1, G)
        elif kind == 3:
            w = rng.choice([-0.5, 0.25, 0.5, 0.125], G)
        elif kind == 4:
            w = rng.standard_normal(G) * (rng.random(G) < 0.4)
        elif kind == 5:
            w = rng.standard_normal(G) * 2.0 ** -140
        elif kind == 6:
            w = rng.standard_normal(G) * 2.0 ** rng.integers(-30, 5, G)
        elif kind == 7:
            w = rng.choice([-1, 1], G) * 2.0 ** rng.integers(-4, 1, G)
        else:
            w = rng.standard_normal(G) * 2.0 ** rng.integers(-12, 0, G)
        out.append(np.asarray(w, dtype=np.float32))
    return out


def test_worked_examples():
    rows = read_golden("ternarize_worked.txt", 5)
    assert len(rows) >= 10
    for G, ws, ts, abits, why in rows:
        w = np.array(parse_floats(ws), dtype=np.float32)
        assert w.size == int(G)
        t, a, st = O.ternarize_group(w)
        assert st == O.OK
        assert list(t) == parse_ints(ts), why
        assert bits(a) == int(abits, 16), why


@pytest.mark.parametrize("G,n", [(1, 60), (2, 200), (3, 200), (4, 200), (5, 90), (6, 45)])
def test_bruteforce_exact(G, n):
    """Exact rational brute force: the oracle's code attains the minimum of
    ||w - alpha t||^2 over all 3^G codes and all alpha >= 0 (Eq. 1 per group, Eq. 2), it is
    a threshold code (the paper's |w| > Delta rule), no threshold code with fewer kept
    weights attains the minimum, and alpha is the fp32 nearest the exact mean kept |w|."""
    for w in _groups(G, n, seed=100 + G):
        t, a, st = O.ternarize_group(w)
        assert st == O.OK
        emin, allc = brute_force([float(v) for v in w])
        t = tuple(int(v) for v in t)
        kept = [abs(Fraction(float(wi))) for wi, ti in zip(w, t) if ti]
        exact_alpha = sum(kept, Fraction(0)) / len(kept) if kept else Fraction(0)
        assert error([float(v) for v in w], t, exact_alpha) == emin
        assert is_threshold_code([float(v) for v in w], t)
        nk = sum(1 for v in t if v)
        for e, c in allc:
            if e == emin and is_threshold_code([float(v) for v in w], c):
                assert sum(1 for v in c if v) >= nk
        assert bits(a) == bits(f32_from_fraction(exact_alpha))


def test_bruteforce_fp64_G8():
    """G = 8: fp64 brute force over all 6561 codes on many groups; the oracle's error
    equals the minimum to 1e-12 relative."""
    G = 8
    codes = np.array(list(itertools.product((-1, 0, 1), repeat=G)), dtype=np.float64)
    nz = np.abs(codes).sum(1)
    for w in _groups(G, 900, seed=7):
        wd = w.astype(np.float64) / max(1e-300, float(np.abs(w).max()) or 1.0)
        dots = codes @ wd
        al = np.where(nz > 0, np.maximum(dots, 0) / np.maximum(nz, 1), 0.0)
        err = ((wd[None, :] - al[:, None] * codes) ** 2).sum(1)
        t, a, st = O.ternarize_group(w)
        td = t.astype(np.float64)
        k = np.abs(td).sum()
        ao = (np.abs(wd) * np.abs(td)).sum() / k if k else 0.0
        eo = ((wd - ao * td) ** 2).sum()
        assert eo <= err.min() * (1 + 1e-12) + 1e-300


def test_G1_closed_form():
    rng = np.random.default_rng(3)
    for v in rng.standard_normal(500).astype(np.float32):
        t, a, _ = O.ternarize_group([v])
        assert t[0] == (1 if v > 0 else -1) and a == abs(v)


def test_G2_closed_form():
    """Two weights a1 >= a2 > 0: both kept iff (a1+a2)^2/2 > a1^2, i.e. a2 > (sqrt2 - 1) a1."""
    rng = np.random.default_rng(4)
    c = np.float32(np.sqrt(2) - 1)
    a2s = np.concatenate([rng.uniform(0, 1, 400),
                          np.nextafter(np.float32(c), np.float32(1)) + np.zeros(1),
                          np.nextafter(np.float32(c), np.float32(0)) + np.zeros(1), [c]]).astype(np.float32)
    for a2 in a2s:
        a1 = np.float32(1.0)
        t, a, _ = O.ternarize_group([a1, -a2])
        keep = (Fraction(float(a1)) + Fraction(float(a2))) ** 2 > 2 * Fraction(float(a1)) ** 2
        assert (t[1] != 0) == keep
        assert t[0] == 1 and (t[1] in (0, -1))


def test_equal_magnitudes_scaled_sign():
    """All magnitudes equal: the ternary form is a scaled sign, alpha = |w| (for any G)."""
    rng = np.random.default_rng(5)
    for G in (4, 16, 64, 128):
        for _ in range(20):
            m = np.float32(rng.uniform(0.01, 3))
            w = (rng.choice([-1, 1], G) * m).astype(np.float32)
            t, a, _ = O.ternarize_group(w)
            assert np.array_equal(t, np.sign(w).astype(np.int8)) and a == m


def test_all_zero_and_padding():
    t, a, st = O.ternarize_group(np.zeros(64, np.float32))
    assert st == O.OK and a == 0 and not t.any()
    # zero padding of a ragged row never changes the real groups' result
    rng = np.random.default_rng(6)
    w = rng.standard_normal((5, 13)).astype(np.float32)
    t, al, _ = O.ternarize(w, 4)
    assert t.shape == (5, 16) and al.shape == (5, 4)
    for m in range(5):
        for g in range(3):
            tg, ag, _ = O.ternarize_group(w[m, 4 * g:4 * g + 4])
            assert np.array_equal(t[m, 4 * g:4 * g + 4], tg) and al[m, g] == ag
        tg, ag, _ = O.ternarize_group(np.r_[w[m, 12:], np.zeros(3, np.float32)])
        assert np.array_equal(t[m, 12:], tg) and al[m, 3] == ag


@pytest.mark.parametrize("G", [4, 8, 16, 32, 64, 128])
def test_equivariances(G):
    """Sign flip negates t; scaling by 2^e scales alpha by 2^e exactly; a permutation of a
    group permutes its codes."""
    rng = np.random.default_rng(G)
    for w in _groups(G, 60, seed=G + 50):
        t, a, _ = O.ternarize_group(w)
        tn, an, _ = O.ternarize_group(-w)
        assert np.array_equal(tn, -t) and bits(an) == bits(a)
        e = int(rng.integers(-20, 20))
        ws = (w.astype(np.float64) * 2.0 ** e).astype(np.float32)
        if np.all(ws.astype(np.float64) == w.astype(np.float64) * 2.0 ** e) and \
                (np.abs(w).max() == 0 or (np.abs(ws)[w != 0] >= 2.0 ** -126).all() and (np.abs(w)[w != 0] >= 2.0 ** -126).all()):
            tsc, asc, _ = O.ternarize_group(ws)
            assert np.array_equal(tsc, t)
            if a >= 2.0 ** -126 and a * 2.0 ** e >= 2.0 ** -126:
                assert float(asc) == float(a) * 2.0 ** e
        perm = rng.permutation(G)
        tp, ap, _ = O.ternarize_group(w[perm])
        assert np.array_equal(tp, t[perm]) and bits(ap) == bits(a)


def test_at_most_2k_plus_1_values():
    """Section 3.1: k groups represent at most 2k+1 distinct values {0, +-alpha_g}."""
    rng = np.random.default_rng(8)
    w = rng.standard_normal((1, 256)).astype(np.float32)
    for G in (4, 16, 64):
        t, al, _ = O.ternarize(w, G)
        vals = set((t[0].reshape(-1, G) * al[0][:, None]).ravel().tolist())
        assert len(vals) <= 2 * (256 // G) + 1


def test_nonfinite_rejected():
    for bad in (np.nan, np.inf, -np.inf):
        t, a, st = O.ternarize_group(np.array([1.0, bad, 0.5, 0.1], np.float32))
        assert st == O.ERR_NONFINITE and a == 0 and not t.any()


@pytest.mark.parametrize("G", [32, 64, 128])
def test_fp64_path_agrees(G):
    """The plain fp64 sort-and-scan statement of Eq. 5 picks the same kept count on random
    groups (no near-ties occur at this sample size)."""
    for w in _groups(G, 200, seed=G + 9):
        t, a, _ = O.ternarize_group(w)
        tau, k, al = O.ternarize_group_f64(w.astype(np.float64))
        assert k == int(np.count_nonzero(t))
        if k:
            # fp32 rounding of alpha: half an ulp, absolute 2^-150 in the subnormal range
            assert abs(al - float(a)) <= max(2.0 ** -24 * float(a), 2.0 ** -150) * (1 + 1e-9)


def test_lemma1_exponential():
    """Lemma 1 (Section 3.1 and its appendix proof): for |w| ~ Exp(lambda) the optimal
    threshold of Eq. 5 is about 1/lambda = mean |w|."""
    rng = np.random.default_rng(11)
    for lam in (0.5, 2.0, 30.0):
        n = 1 << 20
        w = rng.exponential(1.0 / lam, n) * rng.choice([-1.0, 1.0], n)
        tau, k, al = O.ternarize_group_f64(w)
        assert abs(tau * lam - 1.0) < 0.1, (lam, tau)
        # the kept fraction is then about e^{-1} (appendix: |I_Delta| ~ n e^{-lambda Delta})
        assert abs(k / n - np.exp(-1.0)) < 0.05


def test_round_ratio_exact():
    """alpha rounding: exact RNE of S*2^u/k against an independent rational rounding."""
    rng = np.random.default_rng(12)
    cases = [(1, 3, 0), (5, 2, -1), (7, 5, 0), (384 * 2, 2, -149), (1, 1, -149), (3, 2, -150),
             ((1 << 39) - 1, 127, 80), (0x1555555, 3, -30)]
    for _ in range(3000):
        S = int(rng.integers(1, 1 << 39))
        k = int(rng.integers(1, 129))
        u = int(rng.integers(-157, 88))
        cases.append((S, k, u))
    for S, k, u in cases:
        want = f32_from_fraction(Fraction(S, k) * Fraction(2) ** u)
        got = O.round_ratio_f32(S, k, u)
        if np.isinf(want):
            continue
        assert bits(got) == bits(want), (S, k, u)


@pytest.mark.parametrize("G", [16, 64, 128])
def test_large_group_exact_boundary(G):
    """One weight 1 and a run of G-1 equal magnitudes x: all are kept iff
    (1 + (G-1)x)^2 / G > 1 (exact rationals), else only the large one.  x is swept over
    the fp32 neighbours of the boundary, so the exact comparison decides."""
    n = G - 1
    xb = np.float32((np.sqrt(G) - 1) / n)
    xs = [xb]
    for _ in range(6):
        xs.append(np.nextafter(xs[-1], np.float32(1)))
    x = xb
    for _ in range(6):
        x = np.nextafter(x, np.float32(0))
        xs.append(x)
    for x in xs:
        w = np.full(G, x, np.float32)
        w[0] = 1.0
        w[1::2] *= -1
        t, a, _ = O.ternarize_group(w)
        fx = Fraction(float(x))
        keep_all = (1 + n * fx) ** 2 > G  # J_G > J_1 = 1 ; equality keeps the single weight
        assert (np.count_nonzero(t) == G) == keep_all
        want = (1 + n * fx) / G if keep_all else Fraction(1)
        assert bits(a) == bits(f32_from_fraction(want))
