"""Shared helpers for the GPU parity tests (CUDA path through the C ABI vs the oracle)."""
import numpy as np
import torch

import oracle as O

TOL = 1e-5  # |y_gpu - y_oracle| <= TOL * act_scale * sum_g |alpha_g * s_g| per element

ORACLE_TYPE = {"u8": O.U8, "s8": O.S8, "u4": O.U4, "s4": O.S4}


def dev():
    assert torch.cuda.is_available(), "GPU test needs CUDA"
    return torch.device("cuda:0")


def to_dev(a: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a)).to(dev())


def codes_u32(t: torch.Tensor) -> np.ndarray:
    return t.cpu().numpy().view(np.uint32)


def check_within(got: np.ndarray, want: np.ndarray, mag: np.ndarray, what: str):
    got = got.astype(np.float64)
    err = np.abs(got - want)
    bound = TOL * mag
    bad = err > bound
    if bad.any():
        i = np.argwhere(bad)[0]
        raise AssertionError(f"{what}: {bad.sum()} of {bad.size} outside tolerance; first at {tuple(i)}: "
                             f"gpu {got[tuple(i)]!r} oracle {want[tuple(i)]!r} bound {bound[tuple(i)]!r}")


def make_codes(w: np.ndarray, G: int):
    """Oracle ternarization of w -> (t, alpha, packed codes)."""
    t, al, _ = O.ternarize(w, G)
    return t, al, O.pack_codes(t)


def quantize_oracle(x: np.ndarray, act_type: str):
    """Oracle DFP quantization -> (int32 codes, scale, packed bytes)."""
    q, sc, _, _ = O.quantize(x, ORACLE_TYPE[act_type])
    return q, sc, O.pack_act(q, ORACLE_TYPE[act_type])


def random_acts(shape, act_type: str, rng) -> np.ndarray:
    """fp32 activations: half-normal for unsigned types, normal for signed types."""
    x = rng.standard_normal(shape).astype(np.float32)
    return np.abs(x) if act_type.startswith("u") else x
