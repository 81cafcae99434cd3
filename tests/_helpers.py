"""Shared plumbing for the GPU parity tests: tensor <-> numpy conversion and
tolerances.  No method arithmetic lives here."""
import numpy as np
import torch

# Tolerances on floats (max-abs against the fp64 oracle): 2e-2 for bf16, 1e-5 for fp32.
TOL = {"bf16": 2e-2, "f32": 1e-5}


def f64(t: torch.Tensor) -> np.ndarray:
    """Exact fp64 values of a bf16 / fp32 tensor."""
    return t.detach().float().cpu().numpy().astype(np.float64)


def bits16(t: torch.Tensor) -> np.ndarray:
    """uint16 bit patterns of a bf16 tensor."""
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def cuda(x, dtype=None):
    t = torch.as_tensor(x)
    if dtype is not None:
        t = t.to(dtype)
    return t.cuda()
