"""CPU checks of the C ABI: the library builds for sm_103a, loads, exports every function
declared in include/fgq.h, and rejects bad arguments on the host (no kernel launches)."""
import ctypes
import os
import re
import shutil

import pytest

from conftest import ROOT

INCLUDE = os.path.join(ROOT, "include")


def header_functions():
    """Every function declared in include/*.h."""
    names = []
    for fn in sorted(os.listdir(INCLUDE)):
        if not fn.endswith(".h"):
            continue
        src = open(os.path.join(INCLUDE, fn)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        names += re.findall(r"^\s*(?:const\s+)?[A-Za-z_][A-Za-z0-9_]*\s*\*?\s*(fgq_[a-z0-9_]+)\s*\(", src, flags=re.M)
    return sorted(set(names))


@pytest.fixture(scope="module")
def L():
    if shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("nvcc not available")
    from paper_1705_01462_gb300 import build, fgq
    build.build()
    return fgq.load()


def test_header_declares_the_boundary():
    names = header_functions()
    for required in ("fgq_ternarize", "fgq_quantize_act", "fgq_gemm", "fgq_conv2d", "fgq_conv2d_w8",
                     "fgq_group_sums", "fgq_stream_status", "fgq_quantize_weights_w8"):
        assert required in names


def test_every_declared_symbol_is_exported(L):
    from paper_1705_01462_gb300 import fgq
    bound = {n for n, _, _ in fgq.SIGNATURES}
    for name in header_functions():
        assert hasattr(L, name), f"{name} declared in include/*.h but not exported"
        assert name in bound, f"{name} has no Python binding"


def test_size_helpers(L):
    assert L.fgq_version() == 1
    assert L.fgq_num_groups(576, 4) == 144 and L.fgq_codes_words_per_row(576, 4) == 36
    assert L.fgq_num_groups(147, 4) == 37 and L.fgq_codes_words_per_row(147, 4) == 10
    assert L.fgq_num_groups(363, 64) == 6 and L.fgq_codes_words_per_row(363, 64) == 24
    assert L.fgq_num_groups(10, 3) == 0  # G must be a power of two <= 128
    assert L.fgq_quantize_act_workspace_bytes(0) == 0


def test_host_argument_errors(L):
    from paper_1705_01462_gb300 import fgq
    p = ctypes.c_void_p(256)
    assert L.fgq_ternarize(p, 4, 16, 3, p, p, None) == fgq.FGQ_ERR_ARG
    assert L.fgq_ternarize(p, -1, 16, 4, p, p, None) == fgq.FGQ_ERR_ARG
    assert L.fgq_ternarize(None, 4, 16, 4, p, p, None) == fgq.FGQ_ERR_ARG
    assert L.fgq_ternarize(ctypes.c_void_p(258), 4, 16, 4, p, p, None) == fgq.FGQ_ERR_ALIGN
    assert L.fgq_ternarize(None, 0, 16, 4, None, None, None) == fgq.FGQ_OK  # empty: nothing launched
    # quantize: non-power-of-two scale, bad type, empty input
    assert L.fgq_quantize_act(p, 16, 0, ctypes.c_float(0.3), p, None, None, 0, None) == fgq.FGQ_ERR_ARG
    assert L.fgq_quantize_act(p, 16, 7, ctypes.c_float(0.0), p, p, p, 1 << 20, None) == fgq.FGQ_ERR_ARG
    assert L.fgq_quantize_act(None, 0, 0, ctypes.c_float(0.0), None, None, None, 0, None) == fgq.FGQ_OK
    assert L.fgq_quantize_act(p, 1000, 0, ctypes.c_float(0.0), p, p, p, 0, None) == fgq.FGQ_ERR_ARG
    # contraction: bad G, odd K for 4-bit, misaligned output, groups not dividing C
    assert L.fgq_gemm(p, 0, p, 8, 64, p, p, 8, 5, p, None) == fgq.FGQ_ERR_ARG
    assert L.fgq_gemm(p, fgq.U4, p, 8, 63, p, p, 8, 4, p, None) == fgq.FGQ_ERR_ARG
    assert L.fgq_gemm(p, 0, p, 8, 64, p, p, 8, 4, ctypes.c_void_p(260), None) == fgq.FGQ_ERR_ALIGN
    assert L.fgq_conv2d(p, 0, p, 1, 8, 8, 6, 3, 3, 1, 1, 4, p, p, 8, 4, p, None) == fgq.FGQ_ERR_ARG
    assert L.fgq_conv2d(p, 0, p, 0, 8, 8, 8, 3, 3, 1, 1, 1, p, p, 8, 4, p, None) == fgq.FGQ_OK  # B = 0
    assert L.fgq_conv2d(p, 0, p, 1, 2, 2, 8, 3, 3, 1, 0, 1, p, p, 8, 4, p, None) == fgq.FGQ_ERR_ARG  # no output
    assert L.fgq_set_path(9) == -1
    prev = L.fgq_set_path(fgq.PATH_SIMT)
    assert L.fgq_set_path(prev) == fgq.PATH_SIMT
    # conv group sums: bad G, groups not dividing C; forced dense / few-row paths form no sums
    assert L.fgq_conv2d_group_sums(p, 0, 1, 8, 8, 8, 3, 3, 1, 1, 1, p, 8, 3, p, None) == fgq.FGQ_ERR_ARG
    assert L.fgq_conv2d_group_sums(p, 0, 1, 8, 8, 6, 3, 3, 1, 1, 4, p, 8, 4, p, None) == fgq.FGQ_ERR_ARG
    assert L.fgq_conv2d_group_sums(p, 0, 0, 8, 8, 8, 3, 3, 1, 1, 1, p, 8, 4, p, None) == fgq.FGQ_OK  # B = 0
    for path in (fgq.PATH_DENSE, fgq.PATH_GEMV):
        prev = L.fgq_set_path(path)
        try:
            assert L.fgq_group_sums(p, 0, 8, 64, p, 8, 4, p, None) == fgq.FGQ_ERR_UNSUPPORTED
        finally:
            L.fgq_set_path(prev)


def test_debug_controls_are_per_thread(L):
    """The test controls of fgq_debug.h set on one host thread leave another's alone."""
    import threading
    from paper_1705_01462_gb300 import fgq
    prev = L.fgq_set_path(fgq.PATH_TC)
    prev_w = L.fgq_debug_set_wait_limit_us(5)
    prev_s = L.fgq_debug_allow_split_fold(1)
    seen = {}

    def other():
        seen["path"] = L.fgq_set_path(fgq.PATH_AUTO)
        seen["wait"] = L.fgq_debug_set_wait_limit_us(-1)
        seen["split"] = L.fgq_debug_allow_split_fold(0)

    th = threading.Thread(target=other)
    th.start()
    th.join()
    try:
        assert seen == {"path": fgq.PATH_AUTO, "wait": -1, "split": 0}
        assert L.fgq_set_path(prev) == fgq.PATH_TC
        assert L.fgq_debug_set_wait_limit_us(prev_w) == 5
        assert L.fgq_debug_allow_split_fold(prev_s) == 1
    finally:
        L.fgq_set_path(prev)
        L.fgq_debug_set_wait_limit_us(prev_w)
        L.fgq_debug_allow_split_fold(prev_s)

