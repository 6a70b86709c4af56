"""CPU oracle for FGQ (arXiv 1705.01462) -- TEST INFRASTRUCTURE ONLY.

Thin ctypes/numpy wrapper around ``fgq_oracle.c``: a plain, single-threaded, exact-integer
and fp64 statement of the FGQ hot path (Eq. 2, Eq. 4/5, the dynamic-fixed-point
activations and the 32-bit group accumulators of Section 4).

Only the test-suite, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline leg
may import this package.  It shares no code with the CUDA library.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import Optional, Tuple

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "fgq_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")

OK, ERR_ARG, ERR_NONFINITE = 0, 1, 4
U8, S8, U4, S4 = 0, 1, 2, 3
QRANGE = {U8: (0, 255), S8: (-128, 127), U4: (0, 15), S4: (-8, 7)}

_lib: Optional[ctypes.CDLL] = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (plain C11, portable, no CPU-specific flags)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-std=gnu11", "-O2", "-fPIC", "-shared", "-fno-fast-math",
                               "-ffp-contract=off", _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def _P(t):
    return ctypes.POINTER(t)


def lib() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        build()
        L = ctypes.CDLL(_LIB)
        c_f, c_d, c_i, c_i64, c_u32, c_u64, c_sz = (ctypes.c_float, ctypes.c_double, ctypes.c_int,
                                                     ctypes.c_int64, ctypes.c_uint32, ctypes.c_uint64,
                                                     ctypes.c_size_t)
        L.oracle_round_ratio_f32.argtypes = [c_u64, c_u32, c_i]
        L.oracle_round_ratio_f32.restype = c_f
        L.oracle_ternarize_group.argtypes = [_P(c_f), c_i, _P(ctypes.c_int8), _P(c_f)]
        L.oracle_ternarize_group_f64.argtypes = [_P(c_d), c_i64, _P(c_d), _P(c_i64), _P(c_d)]
        L.oracle_ternarize.argtypes = [_P(c_f), c_i, c_i, c_i, _P(ctypes.c_int8), _P(c_f)]
        L.oracle_pack_codes.argtypes = [_P(ctypes.c_int8), c_i, c_i, _P(c_u32)]
        L.oracle_pack_codes.restype = None
        L.oracle_dfp_exponent.argtypes = [_P(c_f), c_sz, c_i, _P(c_i)]
        L.oracle_quantize.argtypes = [_P(c_f), c_sz, c_i, c_f, _P(ctypes.c_int32), _P(c_f), _P(c_i)]
        L.oracle_pack_act.argtypes = [_P(ctypes.c_int32), c_sz, c_i, _P(ctypes.c_uint8)]
        L.oracle_pack_act.restype = None
        conv_args = [_P(ctypes.c_int32), c_d] + [c_i] * 9
        L.oracle_conv2d.argtypes = conv_args + [_P(ctypes.c_int8), _P(c_f), c_i, c_i, _P(c_d), _P(c_d)]
        L.oracle_conv2d_at.argtypes = conv_args + [_P(ctypes.c_int8), _P(c_f), c_i, c_i, _P(c_i64),
                                                   c_i64, _P(c_d), _P(c_d)]
        L.oracle_conv2d_w8.argtypes = conv_args + [_P(ctypes.c_int8), _P(c_f), c_i, _P(c_d), _P(c_d)]
        L.oracle_gemm.argtypes = [_P(ctypes.c_int32), c_d, c_i, c_i, _P(ctypes.c_int8), _P(c_f), c_i, c_i,
                                  _P(c_d), _P(c_d)]
        L.oracle_ternarize_threshold.argtypes = [_P(c_f), c_i, c_i, c_i, c_i, c_i, _P(ctypes.c_int8), _P(c_f),
                                                 ctypes.c_void_p]
        L.oracle_ternary_error.argtypes = [_P(c_f), c_i, c_i, c_i, _P(ctypes.c_int8), _P(c_f), _P(c_d)]
        L.oracle_quantize_alpha.argtypes = [_P(c_f), c_i, c_i, c_i, _P(ctypes.c_int32), _P(c_f)]
        L.oracle_group_sums.argtypes = [_P(ctypes.c_int32), c_i, c_i, _P(ctypes.c_int8), c_i, c_i,
                                        _P(ctypes.c_int64)]
        L.oracle_conv2d_group_sums.argtypes = [_P(ctypes.c_int32)] + [c_i] * 9 + [_P(ctypes.c_int8), c_i, c_i,
                                                                               _P(c_i64), c_i64, _P(c_i64)]
        _lib = L
    return _lib


def _ptr(a: np.ndarray, ct):
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.POINTER(ct))


class OracleError(RuntimeError):
    def __init__(self, code: int, what: str):
        super().__init__(f"oracle {what}: status {code}")
        self.code = code


def _check(code: int, what: str):
    if code != OK:
        raise OracleError(code, what)


# --------------------------------------------------------------------------- ternarize

def num_groups(Kred: int, G: int) -> int:
    return (Kred + G - 1) // G


def round_ratio_f32(S: int, k: int, u: int) -> np.float32:
    return np.float32(lib().oracle_round_ratio_f32(S, k, u))


def ternarize_group(w, check: bool = True) -> Tuple[np.ndarray, np.float32, int]:
    w = np.ascontiguousarray(w, dtype=np.float32)
    t = np.zeros(w.size, dtype=np.int8)
    a = np.zeros(1, dtype=np.float32)
    st = lib().oracle_ternarize_group(_ptr(w, ctypes.c_float), w.size, _ptr(t, ctypes.c_int8),
                                      _ptr(a, ctypes.c_float))
    if check and st not in (OK, ERR_NONFINITE):
        _check(st, "ternarize_group")
    return t, a[0], st


def ternarize_group_f64(w) -> Tuple[float, int, float]:
    w = np.ascontiguousarray(w, dtype=np.float64)
    tau = ctypes.c_double()
    k = ctypes.c_int64()
    al = ctypes.c_double()
    _check(lib().oracle_ternarize_group_f64(_ptr(w, ctypes.c_double), w.size, ctypes.byref(tau),
                                            ctypes.byref(k), ctypes.byref(al)), "ternarize_group_f64")
    return tau.value, k.value, al.value


def ternarize(w: np.ndarray, G: int, check: bool = True):
    """w fp32 [M][Kred] -> (t int8 [M][Kp], alpha fp32 [M][Kp/G], status)."""
    w = np.ascontiguousarray(w, dtype=np.float32)
    M, Kred = w.shape
    ng = num_groups(Kred, G)
    t = np.zeros((M, ng * G), dtype=np.int8)
    alpha = np.zeros((M, ng), dtype=np.float32)
    st = lib().oracle_ternarize(_ptr(w, ctypes.c_float), M, Kred, G, _ptr(t, ctypes.c_int8),
                                _ptr(alpha, ctypes.c_float))
    if check:
        _check(st, "ternarize")
    return t, alpha, st


RULE_EXP, RULE_GAUSS = 0, 1


def ternarize_threshold(w: np.ndarray, G: int, rule: int, per_layer: bool = False, check: bool = True):
    """Analytical-threshold ternarization (Section 3, Lemma 1; see the C file):
    w fp32 [M][Kred] -> (t int8 [M][Kp], alpha fp32 [M][Kp/G], delta fp64 [M][Kp/G] or [1], status)."""
    w = np.ascontiguousarray(w, dtype=np.float32)
    M, Kred = w.shape
    ng = num_groups(Kred, G)
    t = np.zeros((M, ng * G), dtype=np.int8)
    alpha = np.zeros((M, ng), dtype=np.float32)
    delta = np.zeros(1 if per_layer else (M, ng), dtype=np.float64)
    st = lib().oracle_ternarize_threshold(_ptr(w, ctypes.c_float), M, Kred, G, rule, int(per_layer),
                                          _ptr(t, ctypes.c_int8), _ptr(alpha, ctypes.c_float),
                                          delta.ctypes.data_as(ctypes.c_void_p))
    if check:
        _check(st, "ternarize_threshold")
    return t, alpha, delta, st


def ternary_error(w: np.ndarray, t: np.ndarray, alpha: np.ndarray, G: int) -> np.ndarray:
    """Per-group ||w - alpha t||^2 (fp64 [M][Kp/G])."""
    w = np.ascontiguousarray(w, dtype=np.float32)
    t = np.ascontiguousarray(t, dtype=np.int8)
    alpha = np.ascontiguousarray(alpha, dtype=np.float32)
    M, Kred = w.shape
    err = np.zeros((M, num_groups(Kred, G)), dtype=np.float64)
    _check(lib().oracle_ternary_error(_ptr(w, ctypes.c_float), M, Kred, G, _ptr(t, ctypes.c_int8),
                                      _ptr(alpha, ctypes.c_float), _ptr(err, ctypes.c_double)), "ternary_error")
    return err


def quantize_alpha(alpha: np.ndarray, bits: int, check: bool = True):
    """Fixed-point alphas (Section 4): alpha fp32 [M][ng] -> (a int32 [M][ng], scale fp32 [M], status)."""
    alpha = np.ascontiguousarray(alpha, dtype=np.float32)
    M, ng = alpha.shape
    a = np.zeros((M, ng), dtype=np.int32)
    scale = np.zeros(M, dtype=np.float32)
    st = lib().oracle_quantize_alpha(_ptr(alpha, ctypes.c_float), M, ng, bits, _ptr(a, ctypes.c_int32),
                                     _ptr(scale, ctypes.c_float))
    if check:
        _check(st, "quantize_alpha")
    return a, scale, st


def dequantize_alpha(a: np.ndarray, scale: np.ndarray) -> np.ndarray:
    """alpha' = a * 2^E per row (exact in fp32)."""
    return (a.astype(np.float32) * scale.astype(np.float32)[:, None]).astype(np.float32)


def pack_alpha4(a: np.ndarray) -> np.ndarray:
    """4-bit alphas two per byte along each row (element 2i in the low nibble)."""
    M, ng = a.shape
    out = np.zeros((M, (ng + 1) // 2), dtype=np.uint8)
    for g in range(ng):
        out[:, g // 2] |= (a[:, g].astype(np.uint8) & 0xf) << (4 * (g % 2))
    return out


def pack_codes(t: np.ndarray) -> np.ndarray:
    """t int8 [M][Kp] -> uint32 [M][ceil(Kp/16)]."""
    t = np.ascontiguousarray(t, dtype=np.int8)
    M, Kp = t.shape
    out = np.zeros((M, (Kp + 15) // 16), dtype=np.uint32)
    lib().oracle_pack_codes(_ptr(t, ctypes.c_int8), M, Kp, _ptr(out, ctypes.c_uint32))
    return out


# --------------------------------------------------------------------------- activations

def dfp_exponent(x: np.ndarray, act_type: int) -> int:
    x = np.ascontiguousarray(x, dtype=np.float32).reshape(-1)
    E = ctypes.c_int()
    _check(lib().oracle_dfp_exponent(_ptr(x, ctypes.c_float), x.size, act_type, ctypes.byref(E)),
           "dfp_exponent")
    return E.value


def quantize(x: np.ndarray, act_type: int, scale_in: float = 0.0, check: bool = True):
    """fp32 array -> (int32 codes of the same shape, scale 2^E (fp32), E, status)."""
    xs = np.ascontiguousarray(x, dtype=np.float32)
    flat = xs.reshape(-1)
    q = np.zeros(flat.size, dtype=np.int32)
    sc = np.zeros(1, dtype=np.float32)
    E = ctypes.c_int(0)
    st = lib().oracle_quantize(_ptr(flat, ctypes.c_float), flat.size, act_type, float(scale_in),
                               _ptr(q, ctypes.c_int32), _ptr(sc, ctypes.c_float), ctypes.byref(E))
    if check:
        _check(st, "quantize")
    return q.reshape(xs.shape), sc[0], E.value, st


def pack_act(q: np.ndarray, act_type: int) -> np.ndarray:
    q = np.ascontiguousarray(q, dtype=np.int32).reshape(-1)
    n = q.size
    nbytes = n if act_type in (U8, S8) else (n + 1) // 2
    out = np.zeros(nbytes, dtype=np.uint8)
    lib().oracle_pack_act(_ptr(q, ctypes.c_int32), n, act_type, _ptr(out, ctypes.c_uint8))
    return out


# --------------------------------------------------------------------------- contraction

def conv_out_hw(H, W, R, S, stride, pad):
    return (H + 2 * pad - R) // stride + 1, (W + 2 * pad - S) // stride + 1


def conv2d(q, act_scale, R, S, stride, pad, groups, t, alpha, G, positions=None):
    """q int32 NHWC codes [B][H][W][C]; t [M][Kp]; alpha [M][ng].

    Returns (y, ymag) fp64 [B][Ho][Wo][M], or [npos][M] when positions (flat output
    indices) are given.
    """
    q = np.ascontiguousarray(q, dtype=np.int32)
    t = np.ascontiguousarray(t, dtype=np.int8)
    alpha = np.ascontiguousarray(alpha, dtype=np.float32)
    B, H, W, C = q.shape
    M = t.shape[0]
    Ho, Wo = conv_out_hw(H, W, R, S, stride, pad)
    args = [_ptr(q, ctypes.c_int32), float(act_scale), B, H, W, C, R, S, stride, pad, groups,
            _ptr(t, ctypes.c_int8), _ptr(alpha, ctypes.c_float), M, G]
    if positions is None:
        y = np.zeros((B, Ho, Wo, M), dtype=np.float64)
        ym = np.zeros_like(y)
        _check(lib().oracle_conv2d(*args, _ptr(y, ctypes.c_double), _ptr(ym, ctypes.c_double)), "conv2d")
    else:
        pos = np.ascontiguousarray(positions, dtype=np.int64)
        y = np.zeros((pos.size, M), dtype=np.float64)
        ym = np.zeros_like(y)
        _check(lib().oracle_conv2d_at(*args, _ptr(pos, ctypes.c_int64), pos.size, _ptr(y, ctypes.c_double),
                                      _ptr(ym, ctypes.c_double)), "conv2d_at")
    return y, ym


def conv2d_w8(q, act_scale, R, S, stride, pad, groups, wq, wscale):
    q = np.ascontiguousarray(q, dtype=np.int32)
    wq = np.ascontiguousarray(wq, dtype=np.int8)
    wscale = np.ascontiguousarray(wscale, dtype=np.float32)
    B, H, W, C = q.shape
    M = wq.shape[0]
    Ho, Wo = conv_out_hw(H, W, R, S, stride, pad)
    y = np.zeros((B, Ho, Wo, M), dtype=np.float64)
    ym = np.zeros_like(y)
    _check(lib().oracle_conv2d_w8(_ptr(q, ctypes.c_int32), float(act_scale), B, H, W, C, R, S, stride, pad,
                                  groups, _ptr(wq, ctypes.c_int8), _ptr(wscale, ctypes.c_float), M,
                                  _ptr(y, ctypes.c_double), _ptr(ym, ctypes.c_double)), "conv2d_w8")
    return y, ym


def gemm(q, act_scale, t, alpha, G):
    """q int32 [P][Kred]; returns (y, ymag) fp64 [P][M]."""
    q = np.ascontiguousarray(q, dtype=np.int32)
    t = np.ascontiguousarray(t, dtype=np.int8)
    alpha = np.ascontiguousarray(alpha, dtype=np.float32)
    P, Kred = q.shape
    M = t.shape[0]
    y = np.zeros((P, M), dtype=np.float64)
    ym = np.zeros_like(y)
    _check(lib().oracle_gemm(_ptr(q, ctypes.c_int32), float(act_scale), P, Kred, _ptr(t, ctypes.c_int8),
                             _ptr(alpha, ctypes.c_float), M, G, _ptr(y, ctypes.c_double),
                             _ptr(ym, ctypes.c_double)), "gemm")
    return y, ym


def group_sums(q, t, G):
    """q int32 [P][Kred], t [M][Kp] -> int64 [M][ng][P]."""
    q = np.ascontiguousarray(q, dtype=np.int32)
    t = np.ascontiguousarray(t, dtype=np.int8)
    P, Kred = q.shape
    M = t.shape[0]
    ng = num_groups(Kred, G)
    s = np.zeros((M, ng, P), dtype=np.int64)
    _check(lib().oracle_group_sums(_ptr(q, ctypes.c_int32), P, Kred, _ptr(t, ctypes.c_int8), M, G,
                                   _ptr(s, ctypes.c_int64)), "group_sums")
    return s


def conv2d_group_sums(q, R, S, stride, pad, groups, t, G, positions=None):
    """Group sums of a convolution: q int32 NHWC codes [B][H][W][C]; t [M][Kp]; positions
    (flat output indices, default all) -> int64 [M][ng][npos]."""
    q = np.ascontiguousarray(q, dtype=np.int32)
    t = np.ascontiguousarray(t, dtype=np.int8)
    B, H, W, C = q.shape
    M = t.shape[0]
    Ho, Wo = conv_out_hw(H, W, R, S, stride, pad)
    if positions is None:
        positions = np.arange(B * Ho * Wo)
    pos = np.ascontiguousarray(positions, dtype=np.int64)
    ng = num_groups(R * S * (C // groups), G)
    s = np.zeros((M, ng, pos.size), dtype=np.int64)
    _check(lib().oracle_conv2d_group_sums(_ptr(q, ctypes.c_int32), B, H, W, C, R, S, stride, pad, groups,
                                          _ptr(t, ctypes.c_int8), M, G, _ptr(pos, ctypes.c_int64), pos.size,
                                          _ptr(s, ctypes.c_int64)), "conv2d_group_sums")
    return s


def quantize_weights_w8(w: np.ndarray):
    """Per-filter DFP int8 weights for the 8-bit first layer: (wq int8 [M][Kred], scale [M])."""
    w = np.ascontiguousarray(w, dtype=np.float32)
    M = w.shape[0]
    wq = np.zeros(w.shape, dtype=np.int8)
    sc = np.zeros(M, dtype=np.float32)
    for m in range(M):
        q, s, _, _ = quantize(w[m], S8)
        wq[m] = q.astype(np.int8)
        sc[m] = s
    return wq, sc


# --------------------------------------------------------------------------- chained forward steps
# The steps between the contractions of a quantized ResNet forward (Section 4 keeps the
# activations between layers as 8-bit dynamic fixed point).  The paper states no rule for
# them; these are the plain definitions this library follows.

def maxpool_codes(q: np.ndarray, R: int, stride: int, pad: int) -> np.ndarray:
    """Max pooling of integer codes, NHWC: out[b][ho][wo][c] = max of q[b][h][w][c] over the
    R x R window at (ho*stride - pad, wo*stride - pad), positions outside the map not taking
    part.  Written as a loop over the output pixels; each window is a numpy slice."""
    q = np.asarray(q)
    B, H, W, C = q.shape
    Ho, Wo = conv_out_hw(H, W, R, R, stride, pad)
    out = np.zeros((B, Ho, Wo, C), dtype=q.dtype)
    for ho in range(Ho):
        h0, h1 = max(ho * stride - pad, 0), min(ho * stride - pad + R, H)
        for wo in range(Wo):
            w0, w1 = max(wo * stride - pad, 0), min(wo * stride - pad + R, W)
            out[:, ho, wo, :] = q[:, h0:h1, w0:w1, :].max(axis=(1, 2))
    return out


def add_codes(qa: np.ndarray, sa: float, qb: np.ndarray, sb: float) -> np.ndarray:
    """Residual sum of two code tensors at scales sa, sb as fp32: the exact value
    qa*sa + qb*sb (fp64 holds it exactly for 8-bit codes and power-of-two scales whose
    exponents differ by less than 40) rounded once to fp32, to nearest even."""
    sa, sb = float(sa), float(sb)
    fa, fb = np.frexp(sa)[1], np.frexp(sb)[1]
    assert abs(int(fa) - int(fb)) < 40, "scales too far apart for an exact fp64 sum"
    v = np.asarray(qa, dtype=np.float64) * sa + np.asarray(qb, dtype=np.float64) * sb
    return v.astype(np.float32)


def add_requant(qa, sa, qb, sb, out_type: int, scale_out: float) -> np.ndarray:
    """add_codes followed by the activation quantizer at the fixed scale scale_out (U8: a
    negative sum becomes 0, the ReLU after the addition)."""
    q, _, _, _ = quantize(add_codes(qa, sa, qb, sb), out_type, scale_in=scale_out)
    return q
