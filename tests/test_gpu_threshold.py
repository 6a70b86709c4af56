"""GPU parity of the analytical-threshold ternarizer and the ternary error (Section 3,
Lemma 1) against the oracle, through the C ABI."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_1705_01462_gb300 import fgq, synth
from _gpu import dev, to_dev, codes_u32

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _clean_status():
    yield
    assert fgq.fgq_stream_status() == fgq.FGQ_OK


def _weights(M, K, seed):
    rng = np.random.default_rng(seed)
    w = rng.standard_normal((M, K)).astype(np.float32)
    w[0::6] = rng.choice([-0.5, 0.25, 0.5, 0.125], (len(w[0::6]), K))                 # equal magnitudes
    w[1::6] *= (rng.random((len(w[1::6]), K)) < 0.3)                                   # zeros
    w[2::6] *= (2.0 ** rng.integers(-30, 4, (len(w[2::6]), K))).astype(np.float32)    # wide range
    w[3::6] = 0.0                                                                      # all zero
    w[4::6] = (rng.exponential(1.0, (len(w[4::6]), K)) * rng.choice([-1, 1], (len(w[4::6]), K)))
    return w.astype(np.float32)


@pytest.mark.parametrize("rule", [fgq.RULE_EXP, fgq.RULE_GAUSS])
@pytest.mark.parametrize("G", [1, 2, 4, 8, 16, 32, 64, 128])
@pytest.mark.parametrize("K", [7, 64, 147, 576])
def test_group_rule_bit_exact(rule, G, K):
    w = _weights(37, K, 1000 * G + K + rule)
    t, al, _, _ = O.ternarize_threshold(w, G, rule)
    codes, alpha, _ = fgq.fgq_ternarize_threshold(to_dev(w), G, rule)
    assert np.array_equal(codes_u32(codes), O.pack_codes(t)), "codes"
    assert np.array_equal(alpha.cpu().numpy(), al), "alpha"


@pytest.mark.parametrize("rule", [fgq.RULE_EXP, fgq.RULE_GAUSS])
@pytest.mark.parametrize("G", [4, 64])
def test_group_rule_resnet50_layers(rule, G):
    layers = synth.resnet50_convs()
    for i in (1, 12, 40, 50):
        l = layers[i]
        w = synth.weights(l, synth.layer_seed(i))
        t, al, _, _ = O.ternarize_threshold(w, G, rule)
        codes, alpha, _ = fgq.fgq_ternarize_threshold(to_dev(w), G, rule)
        assert np.array_equal(codes_u32(codes), O.pack_codes(t)), f"codes {l.name}"
        assert np.array_equal(alpha.cpu().numpy(), al), f"alpha {l.name}"


@pytest.mark.parametrize("rule", [fgq.RULE_EXP, fgq.RULE_GAUSS])
@pytest.mark.parametrize("shape", [(64, 576), (1, 7), (257, 1000), (512, 4608)])
def test_layer_rule(rule, shape):
    """One threshold and one alpha per layer: the GPU sums in a fixed tree order, so the
    threshold and alpha agree with the sequential oracle to rounding, and the codes agree
    except where a weight sits within rounding of the threshold."""
    M, K = shape
    rng = np.random.default_rng(M + K + rule)
    w = (0.05 * rng.standard_normal((M, K))).astype(np.float32)
    G = 4
    t, al, d, _ = O.ternarize_threshold(w, G, rule, per_layer=True)
    codes, alpha, delta = fgq.fgq_ternarize_threshold(to_dev(w), G, rule, per_layer=True)
    dg = float(delta.cpu().numpy()[0])
    assert dg == pytest.approx(float(d[0]), rel=1e-12)
    near = np.abs(np.abs(w.astype(np.float64)) - d[0]) <= 1e-9 * d[0]
    tg = np.zeros_like(t)
    cw = codes_u32(codes)
    Kp = t.shape[1]
    for j in range(Kp):
        c = (cw[:, j // 16] >> np.uint32(2 * (j % 16))) & 3
        tg[:, j] = np.where(c == 1, 1, np.where(c == 3, -1, 0))
    diff = tg[:, :K] != t[:, :K]
    assert not np.any(diff & ~near), "codes differ away from the threshold"
    ag = alpha.cpu().numpy()
    assert np.all(ag == ag.flat[0]), "one alpha per layer"
    assert ag.flat[0] == pytest.approx(float(al.flat[0]), rel=2 ** -22)


@pytest.mark.parametrize("G", [1, 4, 16, 64, 128])
def test_ternary_error_bit_exact(G):
    w = _weights(29, 300, G)
    for t, al in (O.ternarize(w, G)[:2], O.ternarize_threshold(w, G, O.RULE_EXP)[:2]):
        e = O.ternary_error(w, t, al, G)
        ge = fgq.fgq_ternary_error(to_dev(w), to_dev(O.pack_codes(t).view(np.int32)), to_dev(al), G)
        assert np.array_equal(ge.cpu().numpy(), e)


def test_exact_rule_error_never_above_threshold_rules():
    l = synth.resnet50_convs()[12]
    w = synth.weights(l, 3)
    G = 4
    ce, ae = fgq.fgq_ternarize(to_dev(w), G)
    e_exact = fgq.fgq_ternary_error(to_dev(w), ce, ae, G).cpu().numpy()
    for rule in (fgq.RULE_EXP, fgq.RULE_GAUSS):
        c, a, _ = fgq.fgq_ternarize_threshold(to_dev(w), G, rule)
        e = fgq.fgq_ternary_error(to_dev(w), c, a, G).cpu().numpy()
        assert np.all(e_exact <= e * (1 + 1e-6) + 1e-12)


def test_nonfinite_and_empty():
    w = np.ones((2, 8), np.float32)
    w[0, 1] = np.inf
    codes, alpha, _ = fgq.fgq_ternarize_threshold(to_dev(w), 4, fgq.RULE_GAUSS)
    assert fgq.fgq_stream_status() == fgq.FGQ_ERR_NONFINITE
    a = alpha.cpu().numpy()
    assert a[0, 0] == 0.0 and a[0, 1] == 1.0 and a[1, 0] == 1.0
    assert codes_u32(codes)[0, 0] & 0xff == 0
    e = torch.empty((0, 4), device=dev())
    L = fgq.lib()
    assert L.fgq_ternarize_threshold(e.data_ptr(), 0, 4, 4, 0, 0, None, None, None, 0, None, None) == fgq.FGQ_OK
    assert L.fgq_ternarize_threshold(None, 1, 4, 4, 7, 0, None, None, None, 0, None, None) == fgq.FGQ_ERR_ARG
    wd = to_dev(np.ones((1, 4), np.float32))
    c = torch.empty((1, 1), dtype=torch.int32, device=dev())
    al = torch.empty((1, 1), device=dev())
    assert L.fgq_ternarize_threshold(wd.data_ptr(), 1, 4, 4, 0, 1, c.data_ptr(), al.data_ptr(), None, 0, None,
                                     None) == fgq.FGQ_ERR_ARG  # per-layer rule without workspace
