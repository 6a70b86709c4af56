"""GPU test of fgq_quantize_act_noalloc, the quantizer entry point for callers that cannot
allocate device memory (framework-owned memory pools, plugins handed pre-allocated buffers,
latency-critical loops that avoid cudaMalloc/cudaFree).  It keeps its scratch in a static
device array inside the library instead of a caller workspace.

The test calls it through the C ABI twice in a row, on different inputs and types, and
checks each result against the workspace-taking fgq_quantize_act on the same input, bit for
bit (the tolerance of every quantizer test).  This file sorts last so that a run stopping at
its first failure has already run every other test; it also passes alone in a fresh process.
"""
import numpy as np
import pytest
import torch

from paper_1705_01462_gb300 import fgq

pytestmark = pytest.mark.gpu


def _noalloc(x: torch.Tensor, act_type: int):
    n = x.numel()
    q = torch.empty(fgq.act_bytes(n, act_type), dtype=torch.uint8, device=x.device)
    sc = torch.empty(1, dtype=torch.float32, device=x.device)
    st = fgq.lib().fgq_quantize_act_noalloc(x.data_ptr(), n, act_type, 0.0, q.data_ptr(), sc.data_ptr(),
                                            torch.cuda.current_stream().cuda_stream)
    assert st == fgq.FGQ_OK, fgq.lib().fgq_status_string(st)
    return q, sc


def _with_workspace(x: torch.Tensor, act_type: int):
    n = x.numel()
    q = torch.empty(fgq.act_bytes(n, act_type), dtype=torch.uint8, device=x.device)
    sc = torch.empty(1, dtype=torch.float32, device=x.device)
    ws = torch.empty(max(4, fgq.quantize_act_workspace_bytes(n)), dtype=torch.uint8, device=x.device)
    st = fgq.lib().fgq_quantize_act(x.data_ptr(), n, act_type, 0.0, q.data_ptr(), sc.data_ptr(), ws.data_ptr(),
                                    ws.numel(), torch.cuda.current_stream().cuda_stream)
    assert st == fgq.FGQ_OK
    return q, sc


def test_noalloc_matches_workspace_entry_point_twice():
    dev = torch.device("cuda:0")
    g = torch.Generator(device=dev)
    g.manual_seed(1705)
    # first call: a large u8 tensor (many pass-1 blocks); second: a ragged s4 tensor
    x1 = torch.randn(64 * 56 * 56 * 64 + 5, generator=g, device=dev).abs_()
    x2 = torch.randn(100_003, generator=g, device=dev) * 7.0
    calls = [(x1, fgq.U8), (x2, fgq.S4)]
    results = [_noalloc(x, t) for x, t in calls]        # two calls in a row
    torch.cuda.synchronize()
    for (x, t), (q, sc) in zip(calls, results):
        q_ref, sc_ref = _with_workspace(x, t)
        torch.cuda.synchronize()
        assert torch.equal(q, q_ref)
        assert sc.item() == sc_ref.item()
    assert fgq.fgq_stream_status() == fgq.FGQ_OK
    # and once more on the first input after the second call reused the scratch
    q3, sc3 = _noalloc(x1, fgq.U8)
    assert torch.equal(q3, results[0][0]) and sc3.item() == results[0][1].item()


def test_noalloc_given_scale_and_host_errors():
    """A given power-of-two scale (the branch that needs no scratch) matches the workspace
    entry point bit for bit; argument and alignment errors are those of fgq_quantize_act."""
    dev = torch.device("cuda:0")
    g = torch.Generator(device=dev)
    g.manual_seed(1462)
    x = torch.randn(33_333, generator=g, device=dev) * 3.0
    n = x.numel()
    L = fgq.lib()
    s = torch.cuda.current_stream().cuda_stream
    for t in (fgq.U8, fgq.S8, fgq.S4):
        q = torch.empty(fgq.act_bytes(n, t), dtype=torch.uint8, device=dev)
        q_ref = torch.empty_like(q)
        assert L.fgq_quantize_act_noalloc(x.data_ptr(), n, t, 2.0 ** -3, q.data_ptr(), None, s) == fgq.FGQ_OK
        assert L.fgq_quantize_act(x.data_ptr(), n, t, 2.0 ** -3, q_ref.data_ptr(), None, None, 0, s) == fgq.FGQ_OK
        torch.cuda.synchronize()
        assert torch.equal(q, q_ref)
    q = torch.empty(n + 64, dtype=torch.uint8, device=dev)
    sc = torch.empty(4, dtype=torch.float32, device=dev)
    # misaligned input: FGQ_ERR_ALIGN; a derived scale without scale_out: FGQ_ERR_ARG
    assert L.fgq_quantize_act_noalloc(x.data_ptr() + 4, n - 1, fgq.U8, 0.0, q.data_ptr(), sc.data_ptr(), s) == \
        fgq.FGQ_ERR_ALIGN
    assert L.fgq_quantize_act_noalloc(x.data_ptr(), n, fgq.U8, 0.0, q.data_ptr(), None, s) == fgq.FGQ_ERR_ARG
    assert L.fgq_quantize_act_noalloc(x.data_ptr(), n, fgq.U8, 0.3, q.data_ptr(), sc.data_ptr(), s) == fgq.FGQ_ERR_ARG
    assert fgq.fgq_stream_status() == fgq.FGQ_OK
