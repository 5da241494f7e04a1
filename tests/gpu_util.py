"""Helpers for the GPU parity tests: move seeded numpy inputs to the device,
call the C ABI through the binding, bring results back."""
from __future__ import annotations

import numpy as np


def torch_cuda():
    import pytest

    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return torch


def to_dev(torch, x: np.ndarray, dtype: str = "f32"):
    t = torch.from_numpy(np.ascontiguousarray(x)).cuda()
    if dtype == "bf16":
        t = t.to(torch.bfloat16)
    return t


def widen(torch, t) -> np.ndarray:
    """Exact FP32 values of a device FP32/BF16 tensor (the oracle's input)."""
    return t.float().cpu().numpy()


def new_status(torch):
    return torch.zeros(1, dtype=torch.int32, device="cuda")


def status_bits(status) -> int:
    return int(status.item()) & 0xFFFFFFFF


FP32_UNDERFLOW = 2.0 ** -149  # an FP32 output cannot resolve anything finer


def normalised_error(c_gpu: np.ndarray, c_ref: np.ndarray, na: np.ndarray, nb: np.ndarray) -> float:
    """max (|C_gpu - C_ref| - 2^-149)_+ / (||a_i|| ||b_j||) over outputs with a
    nonzero norm: the 1e-5 bound is relative to the operand norms, on top of
    the FP32 output's own underflow granularity."""
    den = np.outer(na, nb)
    err = np.maximum(np.abs(c_gpu.astype(np.float64) - c_ref) - FP32_UNDERFLOW, 0.0)
    mask = den > 0
    assert np.all(err[~mask] == 0)
    return float((err[mask] / den[mask]).max()) if mask.any() else 0.0
