"""Shared helpers of the test suite (no method arithmetic)."""
import numpy as np
import torch


def gpu_available() -> bool:
    return torch.cuda.is_available()


def ulp_diff(a, b):
    """Distance in float32 ulps between two float32 arrays of equal sign."""
    ai = np.asarray(a, np.float32).view(np.int32).astype(np.int64)
    bi = np.asarray(b, np.float32).view(np.int32).astype(np.int64)
    return np.abs(ai - bi)


def rel_err(a, b):
    a = float(a)
    b = float(b)
    return abs(a - b) / max(abs(b), 1e-300)
