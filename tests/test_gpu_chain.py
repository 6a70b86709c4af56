"""GPU parity of the chained quantized ResNet forward (Section 4: 8-bit DFP activations
between layers, ternary weights, 8-bit first layer), through the C ABI.

* max pooling of codes and the residual add: bit-exact against the oracle;
* the whole ResNet-50 graph at a small input: the fused forward (requantizing epilogues at
  fixed scales) equals the dynamic forward (fp32 outputs, then the quantizer) bit for bit
  when the fixed scales are the dynamic run's own;
* the fused forward at the scales of the oracle's own dynamic forward against the oracle's
  chain (weights ternarized by the oracle): while a step's inputs are identical its output
  codes differ by at most one code and only next to a rounding boundary (residual adds:
  identical); once rounding differences have entered, the codes must still agree almost
  everywhere."""
import zlib

import numpy as np
import pytest
import torch

import oracle as O
from paper_1705_01462_gb300 import fgq, resnet, synth
from _gpu import TOL, ORACLE_TYPE, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _clean_status():
    fgq.fgq_set_path(fgq.PATH_AUTO)
    yield
    fgq.fgq_set_path(fgq.PATH_AUTO)
    assert fgq.fgq_stream_status() == fgq.FGQ_OK


def _signed(codes: np.ndarray, t: str) -> np.ndarray:
    c = codes.astype(np.int64)
    return np.where(c > 127, c - 256, c) if t == "s8" else c


@pytest.mark.parametrize("shape,R,stride,pad", [((2, 112, 112, 64), 3, 2, 1), ((1, 7, 9, 4), 3, 2, 1),
                                                ((3, 10, 6, 68), 3, 1, 1), ((1, 9, 9, 8), 2, 2, 0),
                                                ((1, 11, 13, 12), 5, 2, 2), ((1, 3, 3, 4), 3, 3, 0)])
def test_maxpool_u8(shape, R, stride, pad):
    rng = np.random.default_rng(zlib.crc32(repr(shape).encode()))
    q = rng.integers(0, 256, size=shape, dtype=np.uint8)
    got = fgq.fgq_maxpool_u8(to_dev(q), *shape, R, stride, pad).cpu().numpy()
    assert np.array_equal(got, O.maxpool_codes(q, R, stride, pad))


def test_maxpool_u8_empty_and_args():
    out = torch.empty(0, dtype=torch.uint8, device="cuda")
    fgq.fgq_maxpool_u8(torch.zeros(4, dtype=torch.uint8, device="cuda"), 0, 5, 5, 4, 3, 2, 1, out=out)
    with pytest.raises(fgq.FGQError):  # C not a multiple of 4
        fgq.fgq_maxpool_u8(torch.zeros(75, dtype=torch.uint8, device="cuda"), 1, 5, 5, 3, 3, 2, 1)
    with pytest.raises(fgq.FGQError):  # pad >= R
        fgq.fgq_maxpool_u8(torch.zeros(100, dtype=torch.uint8, device="cuda"), 1, 5, 5, 4, 2, 2, 2)


ADD_CASES = [("s8", "u8", -3, -6, 1000), ("s8", "s8", -4, -4, 1), ("u8", "u8", 0, -9, 155_648 + 17),
             ("s8", "u8", -7, -2, 8 * 152 * 256 * 3 + 5)]


@pytest.mark.parametrize("ta,tb,ea,eb,n", ADD_CASES)
def test_add_codes(ta, tb, ea, eb, n):
    rng = np.random.default_rng(zlib.crc32(repr((ta, tb, ea, eb, n)).encode()))
    lo = {"u8": 0, "s8": -128}
    qa = rng.integers(lo[ta], lo[ta] + 256, n)
    qb = rng.integers(lo[tb], lo[tb] + 256, n)
    sa, sb = np.float32(2.0 ** ea), np.float32(2.0 ** eb)
    da, db = to_dev(qa.astype(np.int64).astype(np.uint8)), to_dev(qb.astype(np.int64).astype(np.uint8))
    dsa, dsb = to_dev(np.array([sa])), to_dev(np.array([sb]))
    v = fgq.fgq_add_codes(da, ta, dsa, db, tb, dsb).cpu().numpy()
    want = O.add_codes(qa, sa, qb, sb)
    assert np.array_equal(v.view(np.uint32), want.view(np.uint32))
    for to in ("u8", "s8"):
        for shift in (0, -2, 3):  # the DFP scale of the sum, a saturating and a coarse one
            E = O.dfp_exponent(want, ORACLE_TYPE[to]) - shift
            so = np.float32(2.0 ** E)
            got = fgq.fgq_add_codes(da, ta, dsa, db, tb, dsb, to, to_dev(np.array([so]))).cpu().numpy()
            ref = O.add_requant(qa, sa, qb, sb, ORACLE_TYPE[to], so)
            assert np.array_equal(_signed(got, to), ref.astype(np.int64)), (to, shift)


# ------------------------------------------------------------------------- the whole graph

HW, BATCH = 64, 2


def _oracle_params(layers, G, kind, seed=1):
    """conv1: synth.weights at 8 bits; the rest: synth.weights ("gauss") or
    synth.pow2_ternary_weights ("pow2"), ternarized by the oracle.  Returns the device
    parameters and the oracle's own."""
    w0 = synth.weights(layers[0], synth.layer_seed(0, seed))
    wq, ws = O.quantize_weights_w8(w0)
    draw = synth.weights if kind == "gauss" else synth.pow2_ternary_weights
    tern, ora = [None], [None]
    for i, l in enumerate(layers):
        if i == 0:
            continue
        t, al, _ = O.ternarize(draw(l, synth.layer_seed(i, seed)), G)
        ora.append((t, al))
        tern.append((to_dev(O.pack_codes(t).view(np.int32)), to_dev(al)))
    return ((to_dev(wq), to_dev(ws)), tern), (wq, ws, ora)


def _oracle_forward(nodes, layers, x, ora, G):
    """The oracle's chain, every tensor at its own DFP scale: name -> (codes, scale, extra)
    with extra = (y, ymag) for a conv."""
    wq, ws, tern = ora
    out = {}
    for n in nodes:
        ot = ORACLE_TYPE[n.out_type]
        if n.kind == "quant":
            q, s, _, _ = O.quantize(x, ot)
            out[n.name] = (q, s, None)
        elif n.kind == "conv":
            q, s, _ = out[n.inputs[0]]
            l = layers[n.layer]
            if n.layer == 0:
                y, ym = O.conv2d_w8(q, s, l.R, l.S, l.stride, l.pad, l.groups, wq, ws)
            else:
                y, ym = O.conv2d(q, s, l.R, l.S, l.stride, l.pad, l.groups, tern[n.layer][0], tern[n.layer][1], G)
            qo, so, _, _ = O.quantize(y.astype(np.float32), ot)
            out[n.name] = (qo, so, (y, ym))
        elif n.kind == "maxpool":
            q, s, _ = out[n.inputs[0]]
            out[n.name] = (O.maxpool_codes(q, 3, 2, 1), s, None)
        else:
            (qa, sa, _), (qb, sb, _) = out[n.inputs[0]], out[n.inputs[1]]
            qo, so, _, _ = O.quantize(O.add_codes(qa, sa, qb, sb), ot)
            out[n.name] = (qo, so, None)
    return out


_CACHE = {}


def _setup(G, kind):
    if (G, kind) not in _CACHE:
        layers = synth.resnet50_convs()
        nodes = resnet.graph(layers)
        params, ora = _oracle_params(layers, G, kind)
        x = synth.activations((BATCH, HW, HW, 3), 7)
        ref = _oracle_forward(nodes, layers, x, ora, G)
        _CACHE[(G, kind)] = (layers, nodes, params, x, ref)
    return _CACHE[(G, kind)]


def _codes(t, n, shape):
    return _signed(t.q.cpu().numpy().reshape(shape), n.out_type)


@pytest.mark.parametrize("G", [4, 64])
def test_chain_fused_equals_dynamic(G):
    """Requantizing in the epilogue at the dynamic run's own scales changes no code."""
    layers, nodes, params, x, _ = _setup(G, "gauss")
    net = resnet.QuantResNet(layers, G, torch.device("cuda:0"), params=params)
    xd = to_dev(x)
    td, tf = {}, {}
    net.forward_dynamic(xd, trace=td)
    net.input_scale = float(net.scales["input"].item())
    net.forward_fused(xd, trace=tf)
    for n in nodes:
        a, b = td[n.name], tf[n.name]
        assert a.shape == b.shape and a.type == b.type, n
        assert float(a.scale.item()) == float(b.scale.item()), n
        assert torch.equal(a.q.reshape(-1), b.q.reshape(-1)), f"{n.name}: fused and dynamic codes differ"


@pytest.mark.parametrize("G", [4, 64])
def test_chain_exact_against_oracle(G):
    """Ternary weights of one power-of-two magnitude make every step exact on both sides, so
    the whole 53-conv chain must match the oracle's bit for bit: the dynamic forward (scales
    found on the GPU) and the fused forward at the oracle's scales."""
    layers, nodes, params, x, ref = _setup(G, "pow2")
    net = resnet.QuantResNet(layers, G, torch.device("cuda:0"), params=params)
    td = {}
    net.forward_dynamic(to_dev(x), trace=td)
    for n in nodes:
        want_q, want_s, _ = ref[n.name]
        assert float(td[n.name].scale.item()) == float(want_s), f"{n.name}: scale"
        assert np.array_equal(_codes(td[n.name], n, want_q.shape), want_q), f"{n.name}: dynamic codes"
    net.set_scales({k: v[1] for k, v in ref.items() if k != "pool"})
    tf = {}
    net.forward_fused(to_dev(x), trace=tf)
    for n in nodes:
        want_q = ref[n.name][0]
        assert np.array_equal(_codes(tf[n.name], n, want_q.shape), want_q), f"{n.name}: fused codes"
    assert (ref[nodes[-1].name][0] != 0).mean() > 0.2  # the chain still carries signal at the end


def test_chain_prefix_against_oracle():
    """Gaussian weights: rounding decides codes next to a boundary, and once one differs the
    difference spreads through the following layers (a flip rate p becomes about sqrt(p) a
    layer later), so the fused forward at the oracle's scales is compared step by step only
    while a step's inputs are identical to the oracle's: a conv's codes then differ by at
    most one and only next to a rounding boundary; the input, the pool and the adds match."""
    G = 4
    layers, nodes, params, x, ref = _setup(G, "gauss")
    net = resnet.QuantResNet(layers, G, torch.device("cuda:0"), params=params)
    net.set_scales({k: v[1] for k, v in ref.items() if k != "pool"})
    tr = {}
    net.forward_fused(to_dev(x), trace=tr)
    same, strict = {}, 0
    for n in nodes:
        want = ref[n.name][0].astype(np.int64)
        d = np.abs(_codes(tr[n.name], n, want.shape) - want)
        if all(same[k] for k in n.inputs):
            strict += 1
            if n.kind != "conv":
                assert d.max(initial=0) == 0, f"{n.name}: codes differ with identical inputs"
            else:
                y, ym = ref[n.name][2]
                scale = ref[n.name][1]
                v = y.reshape(-1) / scale
                b = TOL * ym.reshape(-1) / scale + 1e-9 * np.abs(v)
                near = np.floor(v + b + 0.5) != np.floor(v - b + 0.5)
                dd = d.reshape(-1)
                assert dd.max(initial=0) <= 1, n.name
                assert np.all((dd == 0) | near), f"{n.name}: a code differs away from a rounding boundary"
        same[n.name] = bool(d.max(initial=0) == 0)
    assert strict >= 4  # the input, conv1, the pool and res2a_branch2a at least
