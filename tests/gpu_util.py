"""Helpers for the GPU parity tests: torch is used only to hold device memory."""
import numpy as np

try:
    import torch
except ImportError:  # pragma: no cover
    torch = None


def to_dev(a):
    """numpy -> CUDA tensor; bf16 bit patterns (uint16) travel as int16."""
    if a.dtype == np.uint16:
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda()
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def empty_bf16(*shape):
    return torch.empty(*shape, dtype=torch.int16, device="cuda")


def from_dev_bf16(t):
    """CUDA int16 tensor holding bf16 bits -> float64 numpy (exact widening)."""
    u = t.cpu().numpy().view(np.uint16).astype(np.uint32) << np.uint32(16)
    return u.view(np.float32).astype(np.float64)


def rel_err(got, ref):
    """Normwise max-relative error max|got - ref| / max|ref|."""
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    return float(np.max(np.abs(got - ref)) / max(float(np.max(np.abs(ref))), 1e-30))
