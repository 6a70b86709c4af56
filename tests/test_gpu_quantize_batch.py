"""GPU parity of fgq_quantize_act_batch (Section 4's dynamic-fixed-point activation
quantization for the inputs of many layers at once) through the C ABI: every tensor's codes
and scale equal the oracle's and the single-tensor entry point's bit for bit, over mixed
types, ragged and empty tensors, many small tensors sharing a launch and a tensor larger
than a launch's 64 MB chunk."""
import ctypes

import numpy as np
import pytest
import torch

import oracle as O
from paper_1705_01462_gb300 import fgq
from _gpu import ORACLE_TYPE, dev

pytestmark = pytest.mark.gpu

TYPES = ["u8", "s8", "u4", "s4"]


@pytest.fixture(autouse=True)
def _clean_status():
    yield
    assert fgq.fgq_stream_status() == fgq.FGQ_OK


def _inputs(sizes, rng):
    xs = []
    for i, n in enumerate(sizes):
        t = TYPES[i % 4]
        x = rng.standard_normal(n).astype(np.float32) * np.float32(7.0 if t.startswith("s") else 1.0)
        if t.startswith("u"):
            x = np.abs(x)
        if n > 3 and i % 3 == 0:
            x[n // 2] = -0.0
        xs.append((x, t))
    return xs


def test_batch_matches_oracle_and_single_calls():
    rng = np.random.default_rng(1705)
    sizes = [16, 0, 1, 17, 15, 4097, 33, 1_000_003, 20_000_001, 64, 5, 3_000_000] + [1000 + 7 * i for i in range(40)]
    xs = _inputs(sizes, rng)
    xd = [torch.from_numpy(x).to(dev()) for x, _ in xs]
    got = fgq.fgq_quantize_act_batch(xd, [t for _, t in xs])
    for (x, t), xt, (q, sc) in zip(xs, xd, got):
        n = x.size
        if n == 0:
            continue
        qo, so, _, _ = O.quantize(x, ORACLE_TYPE[t])
        assert np.array_equal(q.cpu().numpy(), O.pack_act(qo, ORACLE_TYPE[t])), (n, t)
        assert float(sc.item()) == float(so), (n, t)
        q1, s1 = fgq.fgq_quantize_act(xt, t)
        assert torch.equal(q, q1) and float(s1.item()) == float(sc.item()), (n, t)


def test_batch_nonfinite_is_recorded():
    rng = np.random.default_rng(7)
    xs = _inputs([5000, 6000, 7000], rng)
    xs[1][0][123] = np.float32(np.nan)
    xd = [torch.from_numpy(x).to(dev()) for x, _ in xs]
    got = fgq.fgq_quantize_act_batch(xd, [t for _, t in xs])
    assert fgq.fgq_stream_status() == fgq.FGQ_ERR_NONFINITE
    for i in (0, 2):  # the finite tensors are unaffected
        x, t = xs[i]
        qo, so, _, _ = O.quantize(x, ORACLE_TYPE[t])
        assert np.array_equal(got[i][0].cpu().numpy(), O.pack_act(qo, ORACLE_TYPE[t]))
        assert float(got[i][1].item()) == float(so)


def test_batch_host_errors():
    L = fgq.lib()
    x = torch.zeros(64, device=dev())
    q = torch.zeros(64, dtype=torch.uint8, device=dev())
    sc = torch.zeros(4, device=dev())
    ws = torch.zeros(64, dtype=torch.uint8, device=dev())
    one = lambda *p: (ctypes.c_void_p * 1)(*p)
    ok = (1, one(x.data_ptr()), (ctypes.c_size_t * 1)(64), (ctypes.c_int * 1)(fgq.U8), one(q.data_ptr()),
          one(sc.data_ptr()), ws.data_ptr(), ws.numel(), None)
    assert L.fgq_quantize_act_batch(*ok) == fgq.FGQ_OK
    assert L.fgq_quantize_act_batch(129, *ok[1:]) == fgq.FGQ_ERR_ARG
    assert L.fgq_quantize_act_batch(1, one(x.data_ptr()), (ctypes.c_size_t * 1)(64), (ctypes.c_int * 1)(9),
                                    one(q.data_ptr()), one(sc.data_ptr()), ws.data_ptr(), ws.numel(), None) == \
        fgq.FGQ_ERR_ARG
    assert L.fgq_quantize_act_batch(1, one(x.data_ptr() + 4), (ctypes.c_size_t * 1)(60), (ctypes.c_int * 1)(0),
                                    one(q.data_ptr()), one(sc.data_ptr()), ws.data_ptr(), ws.numel(), None) == \
        fgq.FGQ_ERR_ALIGN
    assert L.fgq_quantize_act_batch(1, *ok[1:6], ws.data_ptr(), 0, None) == fgq.FGQ_ERR_ARG
    torch.cuda.synchronize()
