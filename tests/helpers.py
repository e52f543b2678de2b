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


def record(kind: str, **fields):
    """Parity evidence: prints one JSON line and appends it to the file named
    by TERMEZO_PARITY_LOG when that variable is set."""
    import json
    import os

    line = json.dumps(dict(kind=kind, **fields), default=float)
    print(line)
    path = os.environ.get("TERMEZO_PARITY_LOG")
    if path:
        with open(path, "a") as f:
            f.write(line + "\n")
