"""Exactness of the BitLinear GEMM's e4m3 tensor-core accumulation at the
extremes of the int8 x ternary range (the GEMM of Sec. 3's BitLinear: int8
activations times ternary weights with an exact int32 accumulator).

The kernel carries each int8 code q as the e4m3 pair hi = 16 floor(q / 16),
lo = q - hi and issues two kind::f8f6f4 MMAs into one fp32 accumulator.  The
result is the exact integer dot product only if the tensor core keeps every
bit of partial sums up to 127 K (877,824 at K = 6912, below 2^24).  These
inputs drive the accumulator to those extremes, then add small products to a
large partial sum:

* all activation codes +127 (or -127) against all-+1 weights: acc = +-127 K;
* codes +127 on the first half of K and +1 on the second half: every
  partial sum of the second half is a large value plus a small one;
* codes +-127 with random signs against random +-1 weights;
* codes +127 against random +-1 weights with a bias towards +1.

Every shape runs a different kernel configuration: output tile widths 256,
192, 160 and 128, the K-split tail (the last wave's tiles split along K and
their partial accumulators added) and the narrow-column tail.  Accumulators
are compared bit for bit with int64 sums (float64 BLAS of integers below
2^53), on every row or on 64 sampled rows of the large shapes."""
import numpy as np
import pytest
import torch

from paper_2609_33548_gb300 import termezo as tz

pytestmark = pytest.mark.gpu

# (N, K, M) of the BitLinear GEMM tests: tile widths 256, 128, 128, 160, 192,
# the K-split tail (640 tiles, K 6912) and the narrow tail (640 tiles, K 2560)
SHAPES = [(6912, 2560, 2048), (688, 688, 200), (256, 2560, 130), (2560, 1536, 1000), (1536, 768, 4096),
          (2560, 6912, 8192), (2560, 2560, 8192)]
PATTERNS = ["all+127", "all-127", "big-then-small", "random-signs", "biased"]


def _inputs(pattern, N, K, M, rng):
    """Latents w [N, K] (fp32) whose ternary codes are the pattern's weights,
    and bf16 activations x [M, K] whose per-row absmax int8 codes are the
    pattern's codes (1.0 -> 127, 1/127 -> 1)."""
    if pattern in ("random-signs",):
        wsgn = rng.choice([-1.0, 1.0], size=(N, K))
    elif pattern == "biased":
        wsgn = np.where(rng.random((N, K)) < 0.9, 1.0, -1.0)
    else:
        wsgn = np.ones((N, K))
    w = (0.05 * wsgn).astype(np.float32)          # gamma = 0.05, tau ~ 0.025: codes = signs
    x = np.ones((M, K), dtype=np.float32)
    if pattern == "all-127":
        x = -x
    elif pattern == "big-then-small":
        x[:, K // 2:] = 1.0 / 127.0
    elif pattern == "random-signs":
        x = rng.choice([-1.0, 1.0], size=(M, K)).astype(np.float32)
    xb = torch.from_numpy(x).to(torch.bfloat16)
    return w, xb, wsgn


@pytest.mark.parametrize("shape", SHAPES, ids=[f"{n}x{k}x{m}" for n, k, m in SHAPES])
def test_e4m3_accumulation_exact_at_extremes(shape):
    N, K, M = shape
    rng = np.random.default_rng(N + K + M)
    for pattern in PATTERNS:
        w, xb, wsgn = _inputs(pattern, N, K, M, rng)
        ctx = tz.Context(tz.op_cfg(N, K, max(M, 128)), 0.01)
        wd = torch.from_numpy(w.reshape(-1)).cuda()
        ctx.termezo_load_params(wd)
        ctx.termezo_build_mask(0.01)
        acc = torch.zeros(M, N, dtype=torch.int32, device="cuda")
        ctx.termezo_bitlinear(0, xb.cuda(), acc, None)
        torch.cuda.synchronize()
        got = acc.cpu().numpy()
        rows = np.arange(M) if M <= 1024 else np.sort(rng.choice(M, 64, replace=False))
        xs = xb.float().numpy()[rows]
        q = np.clip(np.rint(xs * (np.float32(127.0) / np.abs(xs).max(axis=1, keepdims=True))), -128, 127)
        want = np.rint(q.astype(np.float64) @ wsgn.T).astype(np.int64)
        np.testing.assert_array_equal(got[rows].astype(np.int64), want, err_msg=f"{shape} {pattern}")
        if pattern == "all+127":
            assert np.all(got == 127 * K)
        if pattern == "big-then-small":
            assert np.all(got == 127 * (K // 2) + (K - K // 2))
        del ctx
