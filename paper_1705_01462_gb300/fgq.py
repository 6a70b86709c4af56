"""Python binding of libfgq (the FGQ CUDA library): argument marshalling only.

Every function here checks tensor dtypes/devices, passes raw device pointers, sizes and
the current CUDA stream to the C ABI of ``include/fgq.h`` and raises on a non-OK status.
All computation happens in the library's CUDA kernels; there is no CPU fallback, and
loading fails loudly if the library is missing or CUDA is unavailable.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Tuple

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libfgq.so")

FGQ_OK, FGQ_ERR_ARG, FGQ_ERR_ALIGN, FGQ_ERR_UNSUPPORTED, FGQ_ERR_NONFINITE, FGQ_ERR_TIMEOUT, FGQ_ERR_CUDA = range(7)
U8, S8, U4, S4 = 0, 1, 2, 3
PATH_AUTO, PATH_SIMT, PATH_TC, PATH_GEMV, PATH_DENSE = 0, 1, 2, 3, 4
ACT_TYPES = {"u8": U8, "s8": S8, "u4": U4, "s4": S4}

_lib: Optional[ctypes.CDLL] = None

# (name, restype, argtypes) of every exported symbol of include/fgq.h and include/fgq_debug.h
_vp, _i, _i64, _u32, _u64, _f, _sz = (ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_uint32,
                                      ctypes.c_uint64, ctypes.c_float, ctypes.c_size_t)
SIGNATURES = [
    ("fgq_version", _i, []),
    ("fgq_status_string", ctypes.c_char_p, [_i]),
    ("fgq_codes_words_per_row", _i64, [_i, _i]),
    ("fgq_num_groups", _i64, [_i, _i]),
    ("fgq_ternarize", _i, [_vp, _i, _i, _i, _vp, _vp, _vp]),
    ("fgq_ternarize_batch", _i, [_i, _vp, _vp, _vp, _i, _vp, _vp, _vp]),
    ("fgq_ternarize_threshold_workspace_bytes", _sz, []),
    ("fgq_ternarize_threshold", _i, [_vp, _i, _i, _i, _i, _i, _vp, _vp, _vp, _sz, _vp, _vp]),
    ("fgq_ternary_error", _i, [_vp, _i, _i, _i, _vp, _vp, _vp, _vp]),
    ("fgq_quantize_act_workspace_bytes", _sz, [_sz]),
    ("fgq_quantize_act", _i, [_vp, _sz, _i, _f, _vp, _vp, _vp, _sz, _vp]),
    ("fgq_quantize_act_noalloc", _i, [_vp, _sz, _i, _f, _vp, _vp, _vp]),
    ("fgq_quantize_act_batch_workspace_bytes", _sz, [_i]),
    ("fgq_quantize_act_batch", _i, [_i, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    ("fgq_quantize_weights_w8", _i, [_vp, _i, _i, _vp, _vp, _vp]),
    ("fgq_gemm", _i, [_vp, _i, _vp, _i, _i, _vp, _vp, _i, _i, _vp, _vp]),
    ("fgq_conv2d", _i, [_vp, _i, _vp] + [_i] * 9 + [_vp, _vp, _i, _i, _vp, _vp]),
    ("fgq_conv2d_w8", _i, [_vp, _i, _vp] + [_i] * 9 + [_vp, _vp, _i, _vp, _vp]),
    ("fgq_quantize_alpha", _i, [_vp, _i, _i, _i, _vp, _vp, _vp]),
    ("fgq_conv2d_w8_rq", _i, [_vp, _i, _vp] + [_i] * 9 + [_vp, _vp, _i, _i, _vp, _vp, _vp]),
    ("fgq_maxpool_u8", _i, [_vp] + [_i] * 7 + [_vp, _vp]),
    ("fgq_add_codes", _i, [_vp, _i, _vp, _vp, _i, _vp, _sz, _vp, _i, _vp, _vp, _vp]),
    ("fgq_gemm_rq", _i, [_vp, _i, _vp, _i, _i, _vp, _vp, _i, _i, _i, _vp, _vp, _vp]),
    ("fgq_conv2d_rq", _i, [_vp, _i, _vp] + [_i] * 9 + [_vp, _vp, _i, _i, _i, _vp, _vp, _vp]),
    ("fgq_gemm_qa", _i, [_vp, _i, _vp, _i, _i, _vp, _vp, _i, _vp, _i, _i, _vp, _vp]),
    ("fgq_conv2d_qa", _i, [_vp, _i, _vp] + [_i] * 9 + [_vp, _vp, _i, _vp, _i, _i, _vp, _vp]),
    ("fgq_group_sums", _i, [_vp, _i, _i, _i, _vp, _i, _i, _vp, _vp]),
    ("fgq_conv2d_group_sums", _i, [_vp, _i] + [_i] * 9 + [_vp, _i, _i, _vp, _vp]),
    ("fgq_conv2d_host_workspace_bytes", _sz, [_i] * 12),
    ("fgq_conv2d_host", _i, [_vp, _vp, _i] + [_i] * 11 + [_vp, _vp, _sz, _vp]),
    ("fgq_stream_status", _i, [_vp]),
    ("fgq_set_path", _i, [_i]),
    ("fgq_last_path", _i, []),
    ("fgq_launch_count", _u64, []),
    ("fgq_selftest_wait_timeout", _i, [_u32, _vp]),
    ("fgq_debug_set_wait_limit_us", _i64, [_i64]),
    ("fgq_debug_allow_split_fold", _i, [_i]),
    ("fgq_debug_last_cuda_error", _i, [_vp, _sz]),
    ("fgq_debug_cta_pairs", _i, [_i]),
    ("fgq_debug_max_ksplit", _i, [_i]),
    ("fgq_debug_last_ksplit", _i, []),
]


class FGQError(RuntimeError):
    def __init__(self, code: int, what: str):
        name = lib().fgq_status_string(code).decode() if _lib is not None else str(code)
        super().__init__(f"{what}: {name}")
        self.code = code


def load(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libfgq.so (built by paper_1705_01462_gb300.build) and declare its signatures."""
    if not os.path.exists(path):
        raise RuntimeError(f"libfgq.so not found at {path}: build it with "
                           "`python -c 'import __graft_entry__ as g; g.build()'` (no CPU fallback exists)")
    L = ctypes.CDLL(path)
    for name, res, args in SIGNATURES:
        fn = getattr(L, name)
        fn.restype = res
        fn.argtypes = args
    return L


def lib() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        _lib = load()
    return _lib


def _require_cuda():
    if not torch.cuda.is_available():
        raise RuntimeError("libfgq needs a CUDA GPU; there is no CPU fallback")


def _check(code: int, what: str):
    if code != FGQ_OK:
        raise FGQError(code, what)


def _stream(stream=None) -> int:
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def _dev(t: torch.Tensor, dtype, name: str) -> int:
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t.data_ptr()


def _act_type(t) -> int:
    return ACT_TYPES[t] if isinstance(t, str) else int(t)


# --------------------------------------------------------------------------- sizes

def codes_words_per_row(Kred: int, G: int) -> int:
    return int(lib().fgq_codes_words_per_row(Kred, G))


def num_groups(Kred: int, G: int) -> int:
    return int(lib().fgq_num_groups(Kred, G))


def quantize_act_workspace_bytes(n: int) -> int:
    return int(lib().fgq_quantize_act_workspace_bytes(n))


def act_bytes(n: int, act_type) -> int:
    return n if _act_type(act_type) in (U8, S8) else (n + 1) // 2


# --------------------------------------------------------------------------- calls

def fgq_ternarize(w: torch.Tensor, G: int, codes: Optional[torch.Tensor] = None,
                  alpha: Optional[torch.Tensor] = None, stream=None) -> Tuple[torch.Tensor, torch.Tensor]:
    """w fp32 [M][Kred] -> (codes int32-view of uint32 [M][words], alpha fp32 [M][ng])."""
    _require_cuda()
    M, Kred = w.shape
    if codes is None:
        codes = torch.empty((M, codes_words_per_row(Kred, G)), dtype=torch.int32, device=w.device)
    if alpha is None:
        alpha = torch.empty((M, num_groups(Kred, G)), dtype=torch.float32, device=w.device)
    _check(lib().fgq_ternarize(_dev(w, torch.float32, "w"), M, Kred, G, _dev(codes, torch.int32, "codes"),
                               _dev(alpha, torch.float32, "alpha"), _stream(stream)), "fgq_ternarize")
    return codes, alpha


RULE_EXP, RULE_GAUSS = 0, 1


def fgq_ternarize_batch(ws, G: int, stream=None):
    """fgq_ternarize of every fp32 [M][Kred] tensor in ws (one group size, one launch) ->
    list of (codes, alpha)."""
    _require_cuda()
    n = len(ws)
    outs = []
    for w in ws:
        M, Kred = w.shape
        codes = torch.empty((M, codes_words_per_row(Kred, G)), dtype=torch.int32, device=w.device)
        alpha = torch.empty((M, num_groups(Kred, G)), dtype=torch.float32, device=w.device)
        outs.append((codes, alpha))
    VP, I = ctypes.c_void_p * max(n, 1), ctypes.c_int * max(n, 1)
    tw = VP(*[_dev(w, torch.float32, "w") for w in ws])
    tm = I(*[int(w.shape[0]) for w in ws])
    tk = I(*[int(w.shape[1]) for w in ws])
    tc = VP(*[c.data_ptr() for c, _ in outs])
    ta = VP(*[a.data_ptr() for _, a in outs])
    _check(lib().fgq_ternarize_batch(n, tw, tm, tk, G, tc, ta, _stream(stream)), "fgq_ternarize_batch")
    return outs


def fgq_ternarize_threshold(w: torch.Tensor, G: int, rule: int, per_layer: bool = False, stream=None):
    """Analytical-threshold ternarization: w fp32 [M][Kred] -> (codes, alpha, delta); delta is a
    device fp64 [1] tensor for per_layer, else None."""
    _require_cuda()
    M, Kred = w.shape
    codes = torch.empty((M, codes_words_per_row(Kred, G)), dtype=torch.int32, device=w.device)
    alpha = torch.empty((M, num_groups(Kred, G)), dtype=torch.float32, device=w.device)
    ws, wsb, delta = None, 0, None
    if per_layer:
        wsb = lib().fgq_ternarize_threshold_workspace_bytes()
        ws = torch.empty(wsb, dtype=torch.uint8, device=w.device)
        delta = torch.empty(1, dtype=torch.float64, device=w.device)
    _check(lib().fgq_ternarize_threshold(_dev(w, torch.float32, "w"), M, Kred, G, rule, int(per_layer),
                                         _dev(codes, torch.int32, "codes"), _dev(alpha, torch.float32, "alpha"),
                                         ws.data_ptr() if ws is not None else None, wsb,
                                         delta.data_ptr() if delta is not None else None, _stream(stream)),
           "fgq_ternarize_threshold")
    return codes, alpha, delta


def fgq_ternary_error(w: torch.Tensor, codes: torch.Tensor, alpha: torch.Tensor, G: int, stream=None) -> torch.Tensor:
    """Per-group ||w - alpha t||^2, device fp64 [M][ng]."""
    _require_cuda()
    M, Kred = w.shape
    err = torch.empty((M, num_groups(Kred, G)), dtype=torch.float64, device=w.device)
    _check(lib().fgq_ternary_error(_dev(w, torch.float32, "w"), M, Kred, G, _dev(codes, torch.int32, "codes"),
                                   _dev(alpha, torch.float32, "alpha"), err.data_ptr(), _stream(stream)),
           "fgq_ternary_error")
    return err


def fgq_quantize_act(x: torch.Tensor, act_type="u8", scale_in: float = 0.0, q: Optional[torch.Tensor] = None,
                     scale_out: Optional[torch.Tensor] = None, workspace: Optional[torch.Tensor] = None,
                     stream=None) -> Tuple[torch.Tensor, torch.Tensor]:
    """fp32 tensor -> (codes uint8 [n or ceil(n/2)], scale fp32 [1] = 2^E)."""
    _require_cuda()
    ty = _act_type(act_type)
    n = x.numel()
    if q is None:
        q = torch.empty(act_bytes(n, ty), dtype=torch.uint8, device=x.device)
    if scale_out is None:
        scale_out = torch.empty(1, dtype=torch.float32, device=x.device)
        if scale_in > 0:
            scale_out.fill_(scale_in)
    wsb = quantize_act_workspace_bytes(n)
    if workspace is None and scale_in <= 0:
        workspace = torch.empty(max(wsb, 4), dtype=torch.uint8, device=x.device)
    ws_ptr = workspace.data_ptr() if workspace is not None else None
    ws_len = workspace.numel() * workspace.element_size() if workspace is not None else 0
    _check(lib().fgq_quantize_act(_dev(x, torch.float32, "x"), n, ty, float(scale_in), _dev(q, torch.uint8, "q"),
                                  _dev(scale_out, torch.float32, "scale_out") if scale_in <= 0 else None,
                                  ws_ptr, ws_len, _stream(stream)), "fgq_quantize_act")
    return q, scale_out


def fgq_quantize_act_batch(xs, act_types, stream=None):
    """fgq_quantize_act_batch over a list of fp32 device tensors with derived scales: returns
    [(q, scale)] in the same order (q packed as fgq_quantize_act's)."""
    _require_cuda()
    n = len(xs)
    types = [_act_type(t) for t in act_types]
    qs = [torch.empty(act_bytes(x.numel(), t), dtype=torch.uint8, device=x.device) for x, t in zip(xs, types)]
    scs = [torch.empty(1, dtype=torch.float32, device=x.device) for x in xs]
    ws = torch.empty(max(4, int(lib().fgq_quantize_act_batch_workspace_bytes(n))), dtype=torch.uint8,
                     device=xs[0].device if n else "cuda")
    arr = lambda ts: (ctypes.c_void_p * n)(*[_dev(t, t.dtype, "tensor") for t in ts])
    _check(lib().fgq_quantize_act_batch(n, arr(xs), (ctypes.c_size_t * n)(*[x.numel() for x in xs]),
                                        (ctypes.c_int * n)(*types), arr(qs), arr(scs), ws.data_ptr(), ws.numel(),
                                        _stream(stream)), "fgq_quantize_act_batch")
    return list(zip(qs, scs))


def fgq_quantize_weights_w8(w: torch.Tensor, stream=None) -> Tuple[torch.Tensor, torch.Tensor]:
    _require_cuda()
    M, Kred = w.shape
    wq = torch.empty((M, Kred), dtype=torch.int8, device=w.device)
    ws = torch.empty(M, dtype=torch.float32, device=w.device)
    _check(lib().fgq_quantize_weights_w8(_dev(w, torch.float32, "w"), M, Kred, wq.data_ptr(), ws.data_ptr(),
                                         _stream(stream)), "fgq_quantize_weights_w8")
    return wq, ws


def fgq_gemm(q: torch.Tensor, act_type, act_scale: torch.Tensor, P: int, Kred: int, codes: torch.Tensor,
             alpha: torch.Tensor, M: int, G: int, y: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    _require_cuda()
    if y is None:
        y = torch.empty((P, M), dtype=torch.float32, device=q.device)
    _check(lib().fgq_gemm(_dev(q, torch.uint8, "q"), _act_type(act_type), _dev(act_scale, torch.float32, "act_scale"),
                          P, Kred, _dev(codes, torch.int32, "codes"), _dev(alpha, torch.float32, "alpha"), M, G,
                          _dev(y, torch.float32, "y"), _stream(stream)), "fgq_gemm")
    return y


def fgq_gemm_rq(q: torch.Tensor, act_type, act_scale: torch.Tensor, P: int, Kred: int, codes: torch.Tensor,
                alpha: torch.Tensor, M: int, G: int, out_type, out_scale: torch.Tensor,
                out_q: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """fgq_gemm with the output requantized in the kernel: uint8 [P][M] codes at out_scale."""
    _require_cuda()
    if out_q is None:
        out_q = torch.empty((P, M), dtype=torch.uint8, device=q.device)
    _check(lib().fgq_gemm_rq(_dev(q, torch.uint8, "q"), _act_type(act_type), _dev(act_scale, torch.float32, "act_scale"),
                             P, Kred, _dev(codes, torch.int32, "codes"), _dev(alpha, torch.float32, "alpha"), M, G,
                             _act_type(out_type), _dev(out_scale, torch.float32, "out_scale"),
                             _dev(out_q, torch.uint8, "out_q"), _stream(stream)), "fgq_gemm_rq")
    return out_q


def fgq_conv2d_rq(act: torch.Tensor, act_type, act_scale: torch.Tensor, B: int, H: int, W: int, C: int, R: int,
                  S: int, stride: int, pad: int, groups: int, codes: torch.Tensor, alpha: torch.Tensor, M: int, G: int,
                  out_type, out_scale: torch.Tensor, out_q: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """fgq_conv2d with the output requantized in the kernel: uint8 NHWC [B][Ho][Wo][M] codes."""
    _require_cuda()
    Ho, Wo = conv_out_hw(H, W, R, S, stride, pad)
    if out_q is None:
        out_q = torch.empty((B, Ho, Wo, M), dtype=torch.uint8, device=act.device)
    _check(lib().fgq_conv2d_rq(_dev(act, torch.uint8, "act"), _act_type(act_type),
                               _dev(act_scale, torch.float32, "act_scale"), B, H, W, C, R, S, stride, pad, groups,
                               _dev(codes, torch.int32, "codes"), _dev(alpha, torch.float32, "alpha"), M, G,
                               _act_type(out_type), _dev(out_scale, torch.float32, "out_scale"),
                               _dev(out_q, torch.uint8, "out_q"), _stream(stream)), "fgq_conv2d_rq")
    return out_q


def fgq_quantize_alpha(alpha: torch.Tensor, bits: int, stream=None) -> Tuple[torch.Tensor, torch.Tensor]:
    """Fixed-point alphas: fp32 [M][ng] -> (aq uint8 [M][ng] or [M][ceil(ng/2)], ascale fp32 [M])."""
    _require_cuda()
    M, ng = alpha.shape
    aq = torch.empty((M, ng if bits == 8 else (ng + 1) // 2), dtype=torch.uint8, device=alpha.device)
    ascale = torch.empty(M, dtype=torch.float32, device=alpha.device)
    _check(lib().fgq_quantize_alpha(_dev(alpha, torch.float32, "alpha"), M, ng, bits, _dev(aq, torch.uint8, "aq"),
                                    _dev(ascale, torch.float32, "ascale"), _stream(stream)), "fgq_quantize_alpha")
    return aq, ascale


def fgq_gemm_qa(q: torch.Tensor, act_type, act_scale: torch.Tensor, P: int, Kred: int, codes: torch.Tensor,
                aq: torch.Tensor, abits: int, ascale: torch.Tensor, M: int, G: int, y: Optional[torch.Tensor] = None,
                stream=None) -> torch.Tensor:
    _require_cuda()
    if y is None:
        y = torch.empty((P, M), dtype=torch.float32, device=q.device)
    _check(lib().fgq_gemm_qa(_dev(q, torch.uint8, "q"), _act_type(act_type), _dev(act_scale, torch.float32, "act_scale"),
                             P, Kred, _dev(codes, torch.int32, "codes"), _dev(aq, torch.uint8, "aq"), abits,
                             _dev(ascale, torch.float32, "ascale"), M, G, _dev(y, torch.float32, "y"), _stream(stream)),
           "fgq_gemm_qa")
    return y


def fgq_conv2d_qa(act: torch.Tensor, act_type, act_scale: torch.Tensor, B: int, H: int, W: int, C: int, R: int,
                  S: int, stride: int, pad: int, groups: int, codes: torch.Tensor, aq: torch.Tensor, abits: int,
                  ascale: torch.Tensor, M: int, G: int, out: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    _require_cuda()
    Ho, Wo = conv_out_hw(H, W, R, S, stride, pad)
    if out is None:
        out = torch.empty((B, Ho, Wo, M), dtype=torch.float32, device=act.device)
    _check(lib().fgq_conv2d_qa(_dev(act, torch.uint8, "act"), _act_type(act_type),
                               _dev(act_scale, torch.float32, "act_scale"), B, H, W, C, R, S, stride, pad, groups,
                               _dev(codes, torch.int32, "codes"), _dev(aq, torch.uint8, "aq"), abits,
                               _dev(ascale, torch.float32, "ascale"), M, G, _dev(out, torch.float32, "out"),
                               _stream(stream)), "fgq_conv2d_qa")
    return out


def conv_out_hw(H, W, R, S, stride, pad):
    return (H + 2 * pad - R) // stride + 1, (W + 2 * pad - S) // stride + 1


def fgq_conv2d(act: torch.Tensor, act_type, act_scale: torch.Tensor, B: int, H: int, W: int, C: int, R: int, S: int,
               stride: int, pad: int, groups: int, codes: torch.Tensor, alpha: torch.Tensor, M: int, G: int,
               out: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    _require_cuda()
    Ho, Wo = conv_out_hw(H, W, R, S, stride, pad)
    if out is None:
        out = torch.empty((B, Ho, Wo, M), dtype=torch.float32, device=act.device)
    _check(lib().fgq_conv2d(_dev(act, torch.uint8, "act"), _act_type(act_type),
                            _dev(act_scale, torch.float32, "act_scale"), B, H, W, C, R, S, stride, pad, groups,
                            _dev(codes, torch.int32, "codes"), _dev(alpha, torch.float32, "alpha"), M, G,
                            _dev(out, torch.float32, "out"), _stream(stream)), "fgq_conv2d")
    return out


def fgq_conv2d_w8(act: torch.Tensor, act_type, act_scale: torch.Tensor, B: int, H: int, W: int, C: int, R: int,
                  S: int, stride: int, pad: int, groups: int, wq: torch.Tensor, wscale: torch.Tensor, M: int,
                  out: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    _require_cuda()
    Ho, Wo = conv_out_hw(H, W, R, S, stride, pad)
    if out is None:
        out = torch.empty((B, Ho, Wo, M), dtype=torch.float32, device=act.device)
    _check(lib().fgq_conv2d_w8(_dev(act, torch.uint8, "act"), _act_type(act_type),
                               _dev(act_scale, torch.float32, "act_scale"), B, H, W, C, R, S, stride, pad, groups,
                               _dev(wq, torch.int8, "wq"), _dev(wscale, torch.float32, "wscale"), M,
                               _dev(out, torch.float32, "out"), _stream(stream)), "fgq_conv2d_w8")
    return out


def fgq_conv2d_w8_rq(act: torch.Tensor, act_type, act_scale: torch.Tensor, B: int, H: int, W: int, C: int, R: int,
                     S: int, stride: int, pad: int, groups: int, wq: torch.Tensor, wscale: torch.Tensor, M: int,
                     out_type, out_scale: torch.Tensor, out_q: Optional[torch.Tensor] = None,
                     stream=None) -> torch.Tensor:
    """fgq_conv2d_w8 with the output requantized in the kernel: uint8 NHWC [B][Ho][Wo][M] codes."""
    _require_cuda()
    Ho, Wo = conv_out_hw(H, W, R, S, stride, pad)
    if out_q is None:
        out_q = torch.empty((B, Ho, Wo, M), dtype=torch.uint8, device=act.device)
    _check(lib().fgq_conv2d_w8_rq(_dev(act, torch.uint8, "act"), _act_type(act_type),
                                  _dev(act_scale, torch.float32, "act_scale"), B, H, W, C, R, S, stride, pad, groups,
                                  _dev(wq, torch.int8, "wq"), _dev(wscale, torch.float32, "wscale"), M,
                                  _act_type(out_type), _dev(out_scale, torch.float32, "out_scale"),
                                  _dev(out_q, torch.uint8, "out_q"), _stream(stream)), "fgq_conv2d_w8_rq")
    return out_q


def fgq_maxpool_u8(x: torch.Tensor, B: int, H: int, W: int, C: int, R: int, stride: int, pad: int,
                   out: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """R x R max pooling of unsigned codes, NHWC -> uint8 [B][Ho][Wo][C]."""
    _require_cuda()
    Ho, Wo = conv_out_hw(H, W, R, R, stride, pad)
    if out is None:
        out = torch.empty((B, Ho, Wo, C), dtype=torch.uint8, device=x.device)
    _check(lib().fgq_maxpool_u8(_dev(x, torch.uint8, "x"), B, H, W, C, R, stride, pad, _dev(out, torch.uint8, "out"),
                                _stream(stream)), "fgq_maxpool_u8")
    return out


def fgq_add_codes(a: torch.Tensor, a_type, a_scale: torch.Tensor, b: torch.Tensor, b_type, b_scale: torch.Tensor,
                  out_type=None, out_scale: Optional[torch.Tensor] = None, out: Optional[torch.Tensor] = None,
                  stream=None) -> torch.Tensor:
    """a * a_scale + b * b_scale: fp32 (out_type None) or codes requantized at out_scale."""
    _require_cuda()
    n = a.numel()
    if b.numel() != n:
        raise ValueError("fgq_add_codes: a and b differ in size")
    if out_type is None:
        if out is None:
            out = torch.empty(a.shape, dtype=torch.float32, device=a.device)
        st = lib().fgq_add_codes(_dev(a, torch.uint8, "a"), _act_type(a_type), _dev(a_scale, torch.float32, "a_scale"),
                                 _dev(b, torch.uint8, "b"), _act_type(b_type), _dev(b_scale, torch.float32, "b_scale"),
                                 n, _dev(out, torch.float32, "out"), 0, None, None, _stream(stream))
    else:
        if out is None:
            out = torch.empty(a.shape, dtype=torch.uint8, device=a.device)
        st = lib().fgq_add_codes(_dev(a, torch.uint8, "a"), _act_type(a_type), _dev(a_scale, torch.float32, "a_scale"),
                                 _dev(b, torch.uint8, "b"), _act_type(b_type), _dev(b_scale, torch.float32, "b_scale"),
                                 n, None, _act_type(out_type), _dev(out_scale, torch.float32, "out_scale"),
                                 _dev(out, torch.uint8, "out"), _stream(stream))
    _check(st, "fgq_add_codes")
    return out


def fgq_group_sums(q: torch.Tensor, act_type, P: int, Kred: int, codes: torch.Tensor, M: int, G: int,
                   stream=None) -> torch.Tensor:
    _require_cuda()
    s = torch.empty((M, num_groups(Kred, G), P), dtype=torch.int32, device=q.device)
    _check(lib().fgq_group_sums(_dev(q, torch.uint8, "q"), _act_type(act_type), P, Kred,
                                _dev(codes, torch.int32, "codes"), M, G, s.data_ptr(), _stream(stream)),
           "fgq_group_sums")
    return s


def fgq_conv2d_group_sums(act: torch.Tensor, act_type, B: int, H: int, W: int, C: int, R: int, S: int, stride: int,
                          pad: int, groups: int, codes: torch.Tensor, M: int, G: int, stream=None) -> torch.Tensor:
    _require_cuda()
    Ho, Wo = conv_out_hw(H, W, R, S, stride, pad)
    s = torch.empty((M, num_groups(R * S * (C // groups), G), B * Ho * Wo), dtype=torch.int32, device=act.device)
    _check(lib().fgq_conv2d_group_sums(_dev(act, torch.uint8, "act"), _act_type(act_type), B, H, W, C, R, S, stride,
                                       pad, groups, _dev(codes, torch.int32, "codes"), M, G, s.data_ptr(),
                                       _stream(stream)), "fgq_conv2d_group_sums")
    return s


def conv2d_host_workspace_bytes(act_type, B: int, H: int, W: int, C: int, R: int, S: int, stride: int, pad: int,
                                groups: int, M: int, G: int) -> int:
    return int(lib().fgq_conv2d_host_workspace_bytes(_act_type(act_type), B, H, W, C, R, S, stride, pad, groups, M, G))


def fgq_conv2d_host(h_w: torch.Tensor, h_x: torch.Tensor, act_type, B: int, H: int, W: int, C: int, R: int, S: int,
                    stride: int, pad: int, groups: int, M: int, G: int, h_out: torch.Tensor, workspace: torch.Tensor,
                    stream=None) -> None:
    """One layer end to end from host fp32 tensors (h_w [M][Kred], h_x NHWC) into host fp32
    h_out, through the C ABI; asynchronous on the stream (synchronize before reading h_out)."""
    _require_cuda()
    for t, name in ((h_w, "h_w"), (h_x, "h_x"), (h_out, "h_out")):
        if t.device.type != "cpu" or t.dtype != torch.float32 or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous float32 host tensor")
    if not workspace.is_cuda or not workspace.is_contiguous():
        raise ValueError("workspace must be a contiguous device tensor")
    _check(lib().fgq_conv2d_host(h_w.data_ptr(), h_x.data_ptr(), _act_type(act_type), B, H, W, C, R, S, stride, pad,
                                 groups, M, G, h_out.data_ptr(), workspace.data_ptr(),
                                 workspace.numel() * workspace.element_size(), _stream(stream)), "fgq_conv2d_host")


def fgq_stream_status(stream=None) -> int:
    return int(lib().fgq_stream_status(_stream(stream)))


def fgq_set_path(path: int) -> int:
    """Kernel family of this thread's contraction calls (test and benchmark control)."""
    return int(lib().fgq_set_path(path))


def fgq_debug_set_wait_limit_us(us: int) -> int:
    """Wait limit of this thread's tensor-core kernel launches (test control; -1 restores)."""
    return int(lib().fgq_debug_set_wait_limit_us(us))


def fgq_debug_allow_split_fold(allow: bool) -> int:
    """Lets FGQ_PATH_DENSE run fp32 alphas as the split-fp16 ablation on this thread."""
    return int(lib().fgq_debug_allow_split_fold(1 if allow else 0))


def fgq_debug_cta_pairs(on: bool) -> int:
    """G = 4 output kernel on CTA pairs or single CTAs (the default) for this thread's calls."""
    return int(lib().fgq_debug_cta_pairs(1 if on else 0))


def fgq_debug_max_ksplit(k: int) -> int:
    """At most k group ranges per G >= 64 tensor-core tile on this thread (1: whole tiles)."""
    return int(lib().fgq_debug_max_ksplit(int(k)))


def fgq_debug_last_ksplit() -> int:
    """Group ranges per tile of this thread's last G >= 64 tensor-core call."""
    return int(lib().fgq_debug_last_ksplit())


def fgq_debug_last_cuda_error() -> tuple:
    """(cudaError_t value, name) behind this thread's last FGQ_ERR_CUDA from a launch; clears it."""
    buf = ctypes.create_string_buffer(64)
    code = int(lib().fgq_debug_last_cuda_error(buf, 64))
    return code, buf.value.decode()


def fgq_last_path() -> int:
    return int(lib().fgq_last_path())


def fgq_launch_count() -> int:
    return int(lib().fgq_launch_count())


def fgq_selftest_wait_timeout(max_iterations: int, stream=None) -> int:
    _check(lib().fgq_selftest_wait_timeout(max_iterations, _stream(stream)), "fgq_selftest_wait_timeout")
    return fgq_stream_status(stream)
