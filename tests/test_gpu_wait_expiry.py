"""Failure detection in the tensor-core contraction kernels themselves: every mbarrier wait
is bounded, and on expiry the kernel records FGQ_ERR_TIMEOUT, every role leaves its loop,
the copies and MMAs already issued are waited for, and the tensor memory is freed.

A test control (fgq_debug_set_wait_limit_us) shortens the waits of this thread's launches
to nothing, so waits that the kernel's own pipeline would satisfy a few microseconds later
run out: no flag is left unset on purpose and nothing faults, traps or hangs.  The next
call with the normal limits, on the same stream, must then be correct against the oracle,
which it could not be if an aborted CTA had kept its tensor memory (its allocation would
never be granted) or left a copy in flight."""
import numpy as np
import pytest

import oracle as O
from paper_1705_01462_gb300 import fgq
from _gpu import check_within, make_codes, quantize_oracle, random_acts, to_dev

pytestmark = pytest.mark.gpu

TRIES = 12  # calls with the shortened limit until one of them times out


@pytest.fixture(autouse=True)
def _restore():
    fgq.fgq_set_path(fgq.PATH_AUTO)
    fgq.fgq_debug_set_wait_limit_us(-1)
    yield
    fgq.fgq_debug_set_wait_limit_us(-1)
    fgq.fgq_set_path(fgq.PATH_AUTO)
    assert fgq.fgq_stream_status() == fgq.FGQ_OK


@pytest.mark.parametrize("family,G,R", [("tc4", 4, 3), ("tc4", 4, 1), ("tc", 64, 3), ("tc", 64, 1),
                                        ("dense", 4, 3), ("dense", 64, 1)])
def test_forced_wait_expiry_then_exact(family, G, R):
    rng = np.random.default_rng(31 + G + R)
    B, H, W, C, M = 8, 14, 14, 256, 256
    pad = R // 2
    Kred = R * R * C
    w = (rng.standard_normal((M, Kred)) * np.sqrt(2.0 / Kred)).astype(np.float32)
    t, al, codes = make_codes(w, G)
    x = random_acts((B, H, W, C), "u8", rng)
    q, sc, packed = quantize_oracle(x, "u8")
    geo = (B, H, W, C, R, R, 1, pad, 1)
    qd, sd, cd = to_dev(packed), to_dev(np.array([sc], np.float32)), to_dev(codes.view(np.int32))
    if family == "dense":  # 8-bit fixed-point alphas: the dense path is the automatic choice
        a8, asc, _ = O.quantize_alpha(al, 8)
        ad, ascd = to_dev(a8.astype(np.uint8)), to_dev(asc)

        def call():
            return fgq.fgq_conv2d_qa(qd, "u8", sd, *geo, cd, ad, 8, ascd, M, G)
        al_eff = O.dequantize_alpha(a8, asc)
        want_path = fgq.PATH_DENSE
    else:
        fgq.fgq_set_path(fgq.PATH_TC)

        def call():
            return fgq.fgq_conv2d(qd, "u8", sd, *geo, cd, to_dev(al), M, G)
        al_eff = al
        want_path = fgq.PATH_TC
    y, ym = O.conv2d(q, sc, R, R, 1, pad, 1, t, al_eff, G)

    timed_out = 0
    fgq.fgq_debug_set_wait_limit_us(0)
    for _ in range(TRIES):
        out = call()
        assert fgq.fgq_last_path() == want_path
        st = fgq.fgq_stream_status()
        assert st in (fgq.FGQ_OK, fgq.FGQ_ERR_TIMEOUT), st
        if st == fgq.FGQ_OK:  # every wait happened to be satisfied in time: the result stands
            check_within(out.cpu().numpy(), y, ym, f"{family} unexpired call")
        else:
            timed_out += 1
            break
    fgq.fgq_debug_set_wait_limit_us(-1)
    assert timed_out, f"no wait of {family} ran out in {TRIES} calls"
    # the same stream, normal limits: the kernel runs whole and exact
    for _ in range(2):
        out = call().cpu().numpy()
        assert fgq.fgq_stream_status() == fgq.FGQ_OK
        check_within(out, y, ym, f"{family} after an expired call")
