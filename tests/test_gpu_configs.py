"""Full-size parity of the benchmark configurations, in the launch configuration the
benchmark times (automatic path, the configurations' shapes, batches and activation types),
checked on sampled outputs the oracle computes one by one.

Per layer: the GPU ternarizes the whole weight set, quantizes the whole input and runs the
whole convolution (or GEMM); the oracle ternarizes sampled filter rows itself (codes and
alphas must match bit for bit), quantizes the whole input itself (scale and codes must
match), and computes the sampled outputs (all positions drawn at random plus the first and
last) for those rows, within the contraction tolerance.  Layers that repeat a shape launch
the same kernels, so each configuration is covered by its distinct layer shapes:
  * ResNet-50 conv stack, batch 64, u8, G = 4 and 64, 8-bit-weight stem;
  * ResNet-101 conv stack, batch 128, packed u4, G = 64;
  * AlexNet convs and FCs at batch 256, int8 activations, G = 4 and 64, and the square FC
    sweep M = K in {4096, 8192, 16384} at batch {1, 64, 1024}."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_1705_01462_gb300 import fgq, synth
from _gpu import ORACLE_TYPE, check_within, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _clean_status():
    fgq.fgq_set_path(fgq.PATH_AUTO)
    yield
    assert fgq.fgq_stream_status() == fgq.FGQ_OK


def _distinct(layers):
    seen, out = set(), []
    for i, l in enumerate(layers):
        key = (l.C, l.M, l.R, l.S, l.stride, l.pad, l.H, l.W, l.groups)
        if key not in seen:
            seen.add(key)
            out.append((i, l))
    return out


def _sample_rows(M, groups, rng, per_group=8):
    """Filter rows in increasing order, the same number from every conv group."""
    Mg = M // groups
    rows = []
    for gi in range(groups):
        r = rng.choice(Mg, size=min(per_group, Mg), replace=False)
        r = np.unique(np.r_[r, [0, Mg - 1]][: max(per_group, 2)])
        rows.append(gi * Mg + np.sort(r))
    n = min(len(r) for r in rows)
    return np.concatenate([r[:n] for r in rows])


def _sample_positions(P, rng, n=40):
    return np.unique(np.r_[rng.choice(P, size=min(n, P), replace=False), [0, P - 1]])


def _quantized_input(x, act):
    """Oracle quantization of the whole input; the GPU's must match it (codes and scale)."""
    qo, so, _, _ = O.quantize(x, ORACLE_TYPE[act])
    gq, gs = fgq.fgq_quantize_act(to_dev(x), act)
    assert float(gs.item()) == float(so)
    assert np.array_equal(gq.cpu().numpy(), O.pack_act(qo, ORACLE_TYPE[act]))
    return qo, so, gq, gs


def _check_conv(l, B, Gs, act, seed, rng):
    x = synth.activations((B, l.H, l.W, l.C), seed + 500)
    qo, so, gq, gs = _quantized_input(x, act)
    del x
    w = synth.weights(l, seed)
    P = l.P(B)
    for G in Gs:
        codes, alpha = fgq.fgq_ternarize(to_dev(w), G)
        out = fgq.fgq_conv2d(gq, act, gs, B, l.H, l.W, l.C, l.R, l.S, l.stride, l.pad, l.groups, codes, alpha, l.M, G)
        rows = _sample_rows(l.M, l.groups, rng)
        t, al, _ = O.ternarize(w[rows], G)
        assert np.array_equal(codes.cpu().numpy().view(np.uint32)[rows], O.pack_codes(t)), (l.name, G)
        assert np.array_equal(alpha.cpu().numpy()[rows], al), (l.name, G)
        pos = _sample_positions(P, rng)
        y, ym = O.conv2d(qo, so, l.R, l.S, l.stride, l.pad, l.groups, t, al, G, positions=pos)
        got = out.reshape(P, l.M)[torch.as_tensor(pos, device=out.device)][:, torch.as_tensor(rows, device=out.device)]
        check_within(got.cpu().numpy(), y, ym, f"{l.name} B={B} G={G} {act} path={fgq.fgq_last_path()}")
        del out, codes, alpha


R50 = _distinct(synth.resnet50_convs())
R101 = _distinct(synth.resnet101_convs())


@pytest.mark.parametrize("i,l", R50[1:], ids=[l.name for _, l in R50[1:]])
def test_resnet50_b64_u8(i, l):
    _check_conv(l, 64, (4, 64), "u8", synth.layer_seed(i), np.random.default_rng(i))


def test_resnet50_b64_stem_w8():
    l = synth.resnet50_convs()[0]
    B = 64
    rng = np.random.default_rng(0)
    x = synth.activations((B, l.H, l.W, l.C), 7)
    qo, so, gq, gs = _quantized_input(x, "u8")
    w = synth.weights(l, synth.layer_seed(0))
    wq, ws = fgq.fgq_quantize_weights_w8(to_dev(w))
    owq, ows = O.quantize_weights_w8(w)
    assert np.array_equal(wq.cpu().numpy(), owq) and np.array_equal(ws.cpu().numpy(), ows)
    out = fgq.fgq_conv2d_w8(gq, "u8", gs, B, l.H, l.W, l.C, l.R, l.S, l.stride, l.pad, 1, wq, ws, l.M)
    assert fgq.fgq_last_path() == fgq.PATH_DENSE
    P = l.P(B)
    pos = _sample_positions(P, rng, 200)
    # the oracle's 8-bit-weight conv at the sampled positions: their receptive fields only
    Ho, Wo = l.Ho, l.Wo
    got = out.reshape(P, l.M)[torch.as_tensor(pos, device=out.device)].cpu().numpy()
    for k, p in enumerate(pos):
        b, rem = divmod(int(p), Ho * Wo)
        ho, wo = divmod(rem, Wo)
        h0, w0 = ho * l.stride - l.pad, wo * l.stride - l.pad
        patch = np.zeros((1, l.R, l.S, l.C), dtype=np.int32)
        hs, ws_ = max(h0, 0), max(w0, 0)
        he, we = min(h0 + l.R, l.H), min(w0 + l.S, l.W)
        patch[0, hs - h0:he - h0, ws_ - w0:we - w0, :] = qo[b, hs:he, ws_:we, :]
        y, _ = O.conv2d_w8(patch, so, l.R, l.S, 1, 0, 1, owq, ows)
        assert np.array_equal(got[k], y.reshape(-1).astype(np.float32)), p  # exact integers, scaled


@pytest.mark.parametrize("i,l", R101[1:], ids=[l.name for _, l in R101[1:]])
def test_resnet101_b128_u4(i, l):
    _check_conv(l, 128, (64,), "u4", synth.layer_seed(i, 101), np.random.default_rng(1000 + i))


@pytest.mark.parametrize("i,l", list(enumerate(synth.alexnet_convs() + synth.alexnet_fcs())),
                         ids=[l.name for l in synth.alexnet_convs() + synth.alexnet_fcs()])
def test_alexnet_b256_s8(i, l):
    _check_conv(l, 256, (4, 64), "s8", synth.layer_seed(i, 5), np.random.default_rng(2000 + i))


@pytest.mark.parametrize("n", [4096, 8192, 16384])
def test_fc_sweep(n):
    rng = np.random.default_rng(n)
    w = synth.weights_matrix(n, n, n)
    rows = np.sort(rng.choice(n, size=8, replace=False))
    for G in (4, 64):
        codes, alpha = fgq.fgq_ternarize(to_dev(w), G)
        t, al, _ = O.ternarize(w[rows], G)
        assert np.array_equal(codes.cpu().numpy().view(np.uint32)[rows], O.pack_codes(t))
        assert np.array_equal(alpha.cpu().numpy()[rows], al)
        for P in (1, 64, 1024):
            x = synth.activations((P, n), n + P)
            qo, so, gq, gs = _quantized_input(x, "u8")
            y_dev = fgq.fgq_gemm(gq, "u8", gs, P, n, codes, alpha, n, G)
            prow = _sample_positions(P, rng, 24)
            y, ym = O.gemm(qo[prow], so, t, al, G)
            got = y_dev[torch.as_tensor(prow, device=y_dev.device)][:, torch.as_tensor(rows, device=y_dev.device)]
            check_within(got.cpu().numpy(), y, ym, f"fc {n} P={P} G={G} path={fgq.fgq_last_path()}")
        del codes, alpha
