"""Pins of the oracle's analytical-threshold ternarizer and ternary error (Section 3,
Lemma 1 and its proof in the appendix).

Pinned by hand-worked groups, closed forms of the error, the Lemma 1 and Gaussian limits
on large samples (checked against the exact optimum of the same objective), the Gaussian
constant re-derived by scipy root finding, and invariances.
"""
import numpy as np
import pytest

import oracle as O


def test_hand_worked_groups():
    # [3, -1, 2, 0.5]: mean |w| = 6.5/4 = 1.625 -> keep 3 and 2, alpha = 2.5.
    #                  rms = sqrt(14.25/4) = 1.8875..., Delta = 0.6120 * 1.8875 = 1.155 -> same support.
    # [1, 1, 1, 1]:    mean = 1: the strict rule |w| > 1 keeps nothing (alpha = 0);
    #                  rms = 1, Delta = 0.612: all kept, alpha = 1.
    # [0, 0, 0, 0]:    nothing kept, alpha = 0 for both rules.
    # [-4, 1, 1, 0]:   mean = 1.5 -> keep -4 only, alpha = 4; rms = sqrt(18/4) = 2.121,
    #                  Delta = 1.298 -> keep -4 only.
    w = np.array([[3, -1, 2, 0.5], [1, 1, 1, 1], [0, 0, 0, 0], [-4, 1, 1, 0]], np.float32)
    t0, a0, d0, _ = O.ternarize_threshold(w, 4, O.RULE_EXP)
    assert t0.tolist() == [[1, 0, 1, 0], [0, 0, 0, 0], [0, 0, 0, 0], [-1, 0, 0, 0]]
    assert a0.ravel().tolist() == [2.5, 0.0, 0.0, 4.0]
    assert d0.ravel().tolist() == [1.625, 1.0, 0.0, 1.5]
    t1, a1, d1, _ = O.ternarize_threshold(w, 4, O.RULE_GAUSS)
    assert t1.tolist() == [[1, 0, 1, 0], [1, 1, 1, 1], [0, 0, 0, 0], [-1, 0, 0, 0]]
    assert a1.ravel().tolist() == [2.5, 1.0, 0.0, 4.0]
    assert d1[0, 0] == pytest.approx(0.6120031809624808 * np.sqrt(14.25 / 4), rel=1e-15)


def test_padding_not_counted_and_layer_rule():
    # Kred = 5, G = 4: the second group holds one real weight; its mean is that weight's
    # magnitude, so the strict rule keeps nothing there
    w = np.array([[2, 2, 0, 0, 3]], np.float32)
    t, a, d, _ = O.ternarize_threshold(w, 4, O.RULE_EXP)
    assert d.ravel().tolist() == [1.0, 3.0]
    assert t.tolist() == [[1, 1, 0, 0, 0, 0, 0, 0]]
    assert a.ravel().tolist() == [2.0, 0.0]
    # one threshold and one alpha for the layer: mean over 5 real weights = 7/5 = 1.4 -> keep 2, 2, 3
    t, a, d, _ = O.ternarize_threshold(w, 4, O.RULE_EXP, per_layer=True)
    assert d.tolist() == [1.4]
    assert t.tolist() == [[1, 1, 0, 0, 1, 0, 0, 0]]
    assert a.ravel().tolist() == [np.float32(7 / 3)] * 2


def test_layer_rule_equals_group_rule_for_one_full_group():
    rng = np.random.default_rng(5)
    w = rng.standard_normal((1, 64)).astype(np.float32)
    for rule in (O.RULE_EXP, O.RULE_GAUSS):
        tg, ag, dg, _ = O.ternarize_threshold(w, 64, rule)
        tl, al, dl, _ = O.ternarize_threshold(w, 64, rule, per_layer=True)
        assert np.array_equal(tg, tl) and np.array_equal(ag, al) and dg.ravel()[0] == dl[0]


def test_error_closed_forms():
    rng = np.random.default_rng(7)
    w = rng.standard_normal((6, 40)).astype(np.float32)
    G = 8
    # for alpha = mean of the kept |w| the error is ||w||^2 - (sum kept |w|)^2 / k
    t, a, _, _ = O.ternarize_threshold(w, G, O.RULE_EXP)
    err = O.ternary_error(w, t, a, G)
    wd = w.astype(np.float64)
    for m in range(6):
        for g in range(5):
            seg = wd[m, 8 * g:8 * g + 8]
            kept = np.abs(seg)[t[m, 8 * g:8 * g + 8] != 0]
            # alpha is the fp32-rounded mean, so the closed form holds to fp32 rounding
            want = np.sum(seg ** 2) - (kept.sum() ** 2 / kept.size if kept.size else 0.0)
            assert err[m, g] == pytest.approx(want, rel=1e-6, abs=1e-9)
    # the exact rule (Eq. 5) never does worse than a threshold rule on any group
    te, ae, _ = O.ternarize(w, G)
    ee = O.ternary_error(w, te, ae, G)
    assert np.all(ee <= err * (1 + 1e-6) + 1e-12)


def test_gaussian_constant_maximises_the_limit_objective():
    stats = pytest.importorskip("scipy.stats")
    opt = pytest.importorskip("scipy.optimize")
    f = lambda z: stats.norm.pdf(z) - 2 * z * stats.norm.sf(z)  # derivative condition of phi^2/(1-Phi)
    z = opt.brentq(f, 0.1, 2.0, xtol=1e-15)
    w = np.ones((1, 4), np.float32)
    _, _, d, _ = O.ternarize_threshold(w, 4, O.RULE_GAUSS)  # rms = 1 -> Delta = z*
    assert d.ravel()[0] == pytest.approx(z, rel=1e-12)
    g = lambda x: stats.norm.pdf(x) ** 2 / stats.norm.sf(x)
    assert g(z) > g(z - 1e-3) and g(z) > g(z + 1e-3)


@pytest.mark.parametrize("dist", ["exp", "gauss"])
def test_large_sample_limits_are_near_the_exact_optimum(dist):
    """Lemma 1 (exponential magnitudes) and its Gaussian counterpart: on a large sample the
    analytical threshold reaches the exact optimum of (sum kept |w|)^2 / k to within the
    flatness of the objective (relative drop about 0.25 delta^2 at relative offset delta)."""
    rng = np.random.default_rng(11)
    n = 1 << 18
    if dist == "exp":
        lam = 3.0
        w = (rng.exponential(1 / lam, n) * rng.choice([-1, 1], n)).astype(np.float32)
        rule = O.RULE_EXP
    else:
        w = (0.05 * rng.standard_normal(n)).astype(np.float32)
        rule = O.RULE_GAUSS
    w = w.reshape(1, n)
    t, a, d, _ = O.ternarize_threshold(w, n, rule, per_layer=True)
    kept = np.abs(w[t != 0].astype(np.float64))
    J = kept.sum() ** 2 / kept.size
    tau, k, alpha = O.ternarize_group_f64(w.ravel().astype(np.float64))
    mags = np.sort(np.abs(w.ravel().astype(np.float64)))[::-1]
    Jopt = mags[:k].sum() ** 2 / k
    assert J <= Jopt * (1 + 1e-12)
    assert J >= Jopt * (1 - 2e-3)
    if dist == "exp":
        assert d[0] == pytest.approx(1 / lam, rel=0.02)  # Delta* ~ 1/lambda = mean |w|


def test_invariances():
    rng = np.random.default_rng(13)
    w = rng.standard_normal((5, 48)).astype(np.float32)
    for rule in (O.RULE_EXP, O.RULE_GAUSS):
        for per_layer in (False, True):
            t, a, d, _ = O.ternarize_threshold(w, 16, rule, per_layer)
            tn, an, _, _ = O.ternarize_threshold(-w, 16, rule, per_layer)
            assert np.array_equal(tn, -t) and np.array_equal(an, a)
            ts, as_, ds, _ = O.ternarize_threshold(w * np.float32(8.0), 16, rule, per_layer)
            assert np.array_equal(ts, t) and np.array_equal(as_, a * np.float32(8.0)) and np.array_equal(ds, 8 * d)


def test_nonfinite_reported():
    w = np.array([[1, np.nan, 2, 3, 1, 1, 1, 1]], np.float32)
    t, a, d, st = O.ternarize_threshold(w, 4, O.RULE_EXP, check=False)
    assert st == 4
    assert t[0, :4].tolist() == [0, 0, 0, 0] and a[0, 0] == 0.0 and a[0, 1] == 0.0  # [1,1,1,1]: none > mean
