"""The allocation-free absmean entry point (for callers that cannot
allocate device memory, such as code inside a framework that owns all of
the GPU's memory) against the existing path: termezo_build_mask computes
the same exact gamma and tau per projection.  Two calls in a row on
different tensors -- a large one, then a smaller one -- so that partial
sums left in the shared scratch by the first call would show up in the
second.  Collected last."""
import numpy as np
import pytest
import torch

from paper_2609_33548_gb300 import synth
from paper_2609_33548_gb300 import termezo as tz

pytestmark = pytest.mark.gpu


def _existing_tau(w_dev, N, K):
    ctx = tz.Context(tz.op_cfg(N, K, 128), 0.01)
    ctx.termezo_load_params(w_dev)
    ctx.termezo_build_mask(0.01)
    return ctx.termezo_export_state(packed=False)["tau_cur"][0]


def test_absmean_noalloc_matches_build_mask_twice():
    shapes = [(6912, 2560), (640, 2560)]
    for i, (N, K) in enumerate(shapes):
        w = synth.op_latents(N, K, seed=20 + i).reshape(-1).cuda()
        out = torch.full((3,), float("nan"), dtype=torch.float32, device="cuda")
        tz.termezo_absmean_noalloc(w, out)
        torch.cuda.synchronize()
        gamma, tau, sw = out.cpu().numpy()
        ref = _existing_tau(w, N, K)
        assert np.float32(tau).view(np.uint32) == np.float32(ref).view(np.uint32)
        assert np.float32(sw) == np.float32(2.0) * np.float32(tau)
        assert abs(float(gamma) - float(w.abs().double().mean())) <= 1e-6 * float(gamma)


def test_absmean_noalloc_rejects_oversize():
    out = torch.zeros(3, dtype=torch.float32, device="cuda")
    w = torch.zeros(16, dtype=torch.float32, device="cuda")
    lib = tz.load()
    import ctypes
    st = lib.termezo_absmean_noalloc(ctypes.c_void_p(w.data_ptr()), (1 << 28) + 1,
                                     ctypes.c_void_p(out.data_ptr()), None)
    assert st == tz.EINVAL
