"""Helpers shared by the GPU parity tests: host arrays -> CUDA tensors and back."""
from __future__ import annotations

import numpy as np
import torch

from paper_2609_36314_gb300 import synth

BF16_TOL = 1e-2
F32_TOL = 1e-5


def to_dev(a: np.ndarray) -> torch.Tensor:
    """uint16 arrays are bf16 bit patterns; float32 stays float32."""
    if a.dtype == np.uint16:
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda().view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def to_host64(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy().astype(np.float64)


def dev_inputs(d: dict) -> dict:
    return {k: to_dev(v) for k, v in d.items()}


def f64_inputs(d: dict) -> dict:
    return {k: synth.to_f64(v) for k, v in d.items()}


def tol(dtype: str) -> float:
    return F32_TOL if dtype == "f32" else BF16_TOL


def assert_close(name, got, ref, tolerance):
    err = synth.rel_l2(got, ref)
    assert np.all(np.isfinite(got)), f"{name}: non-finite values"
    assert err <= tolerance, f"{name}: rel-L2 {err:.3e} > {tolerance:.1e}"
    return err
