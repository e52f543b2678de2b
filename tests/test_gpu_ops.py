"""GPU parity of the single-projection ("BitLinear op") workload against the
oracle: z generation, exact absmean and mask selection (Eqs. 2-4),
perturb/requantise (Alg. 1), restore/update, and the int8 x ternary GEMM.
Calls go through the C ABI."""
import numpy as np
import pytest
import torch

from oracle import bitnet, philox, ternary, termezo as otz
from paper_2609_33548_gb300 import synth
from paper_2609_33548_gb300 import termezo as tz

from helpers import ulp_diff

pytestmark = pytest.mark.gpu

N, K, M = synth.BITLINEAR_OP["N"], synth.BITLINEAR_OP["K"], synth.BITLINEAR_OP["M"]


@pytest.fixture(scope="module")
def op_latents():
    return synth.op_latents(N, K).numpy().reshape(-1)


def _ctx(w, density, n=N, k=K, m=M):
    ctx = tz.Context(tz.op_cfg(n, k, m), density)
    wd = torch.from_numpy(w).cuda()
    ctx.termezo_load_params(wd)
    return ctx, wd


def test_normal_matches_oracle():
    rng = np.random.default_rng(0)
    idx = np.concatenate([np.arange(4096), rng.integers(0, 2**32 - 1, 100000, dtype=np.uint64)]).astype(np.uint32)
    for seed in (0, 1001, 2**40 + 7):
        z_gpu = torch.empty(idx.size, dtype=torch.float32, device="cuda")
        tz.termezo_normal(seed, torch.from_numpy(idx.astype(np.int32)).cuda(), z_gpu)
        z = z_gpu.cpu().numpy()
        zo = philox.normal(seed, idx.astype(np.uint64))
        err = np.abs(z.astype(np.float64) - zo)
        assert np.all(err <= 4e-7 * np.maximum(1.0, np.abs(zo)) + 1e-7), err.max()
        assert np.median(ulp_diff(z, zo)) <= 1


@pytest.mark.parametrize("density", synth.BITLINEAR_OP["densities"])
def test_mask_build_bit_exact(op_latents, density):
    w = op_latents
    ctx, _ = _ctx(w, density)
    k0, xi0 = ctx.termezo_build_mask(density)
    st = ctx.termezo_export_state()
    reg = otz.single_registry(N, K)
    sel, xi0_o, k0_o, tau_o = otz.initial_mask(w, reg, density)
    assert k0 == k0_o == int(np.floor(density * N * K))
    assert np.float32(xi0).view(np.uint32) == np.float32(xi0_o).view(np.uint32)
    assert st["tau_cur"][0].view(np.uint32) == tau_o[0].view(np.uint32)
    np.testing.assert_array_equal(st["idx"], sel.astype(np.uint32))
    np.testing.assert_array_equal(st["latents"], w[sel])
    np.testing.assert_array_equal(st["packed"], ternary.pack_codes(ternary.quantize(w, tau_o[0])))


@pytest.mark.parametrize("zbuf", [False, True], ids=["regenerate-z", "z-buffer"])
def test_perturb_requantize_update(op_latents, zbuf):
    density, seed, eps, lr, g = 0.01, 1000, np.float32(1e-3), np.float32(1e-3), -5.25
    w = op_latents
    ctx = tz.Context(tz.op_cfg(N, K, M, zbuf), density)
    ctx.termezo_load_params(torch.from_numpy(w).cuda())
    ctx.termezo_build_mask(density)
    reg = otz.single_registry(N, K)
    state = otz.build(w, reg, density)
    act = state.active
    z = philox.normal(seed, act)
    e = (eps * z).astype(np.float32)

    def check(sign, wp):
        st = ctx.termezo_export_state()
        codes, tau, sw = otz.requantize(wp, reg)
        key = "tau_plus" if sign > 0 else "tau_minus"
        assert st[key][0].view(np.uint32) == tau[0].view(np.uint32)
        got = ternary.unpack_codes(st["packed"])
        near = otz.near_threshold(wp[act], tau[np.zeros(act.size, int)], sw[np.zeros(act.size, int)])
        bad = np.nonzero(got != codes)[0]
        frozen_bad = np.setdiff1d(bad, act)
        assert frozen_bad.size == 0
        act_bad = np.isin(act, bad)
        assert np.all(near[act_bad]), (act_bad.sum(), near.sum())
        return near.sum()

    ctx.termezo_requantize(seed, float(eps), +1)
    w_plus = w.copy()
    w_plus[act] = (w[act] + e).astype(np.float32)
    check(+1, w_plus)
    ctx.termezo_requantize(seed, float(eps), -1)
    w_minus = w_plus.copy()
    w_minus[act] = (w_plus[act] - np.float32(2) * e).astype(np.float32)
    check(-1, w_minus)
    ctx.termezo_update(seed, float(eps), float(lr), g)
    st = ctx.termezo_export_state(packed=False)
    w_rest = (w_minus[act] + e).astype(np.float32)
    c = np.float32(float(lr) * g)
    expect = (w_rest - (c * z).astype(np.float32)).astype(np.float32)
    np.testing.assert_array_equal(st["idx"], act.astype(np.uint32))
    # z agrees to a few ulp; the restore ((w+e)-2e)+e rounds at the scale of
    # |w| + 2|e|, so the tolerance is relative to that scale
    tol = 1e-5 * (np.abs(expect).astype(np.float64) + 2 * np.abs(e))
    assert np.all(np.abs(st["latents"].astype(np.float64) - expect) <= tol)


# (N, K, M): the GEMM picks its output tile width per shape to fill the last
# wave of the persistent grid; these shapes take widths 256, 128, 128, 160
# (ragged M) and 192 on a 152-SM GB300.
# (2560, 6912, 8192): 640 tiles on 152 CTAs; the 32 of the last wave are
# split along K into four partial accumulators summed by the last finisher.
# (2560, 2560, 8192): the same 640 tiles with a short K; the last wave's 32
# tiles become 128 units of 64 columns.  (1536, 768, 4096): 192 tiles, the
# last 40 split into 80 units of 128 columns.
@pytest.mark.parametrize("shape", [(N, K, M), (688, 688, 200), (256, 2560, 130), (2560, 1536, 1000),
                                   (1536, 768, 4096), (2560, 6912, 8192), (2560, 2560, 8192)])
def test_bitlinear_int32_accumulators_bit_exact(shape):
    n, k, m = shape
    w = synth.op_latents(n, k, seed=11).numpy().reshape(-1)
    ctx, _ = _ctx(w, 0.01, n, k, max(m, 128))
    ctx.termezo_build_mask(0.01)
    x = synth.op_activations(m, k, seed=12)
    acc = torch.zeros(m, n, dtype=torch.int32, device="cuda")
    y = torch.zeros(m, n, dtype=torch.float32, device="cuda")
    ctx.termezo_bitlinear(0, x.cuda(), acc, y)
    torch.cuda.synchronize()
    reg = otz.single_registry(n, k)
    _, tau, sw = otz.thresholds(w, reg)
    codes = ternary.quantize(w, tau[0]).reshape(n, k)
    q, a = bitnet.act_quant(x.float().numpy())
    acc_o = bitnet.int_matmul(q, codes)
    np.testing.assert_array_equal(acc.cpu().numpy(), acc_o)
    y_o = acc_o.astype(np.float64) * (a.astype(np.float64)[:, None] / 127.0) * float(sw[0])
    np.testing.assert_allclose(y.cpu().numpy(), y_o, rtol=2e-6, atol=1e-30)


PER_TENSOR_DENSITIES = (0.003, 0.02, 0.1)


@pytest.mark.parametrize("density", PER_TENSOR_DENSITIES)
def test_per_tensor_mask_bit_exact(density):
    """The per-tensor quantile on the 14 projections of the tiny decoder:
    the sorted index list, latents, every projection's xi_0 and every
    packed code equal the oracle's bit for bit."""
    cfg = synth.TINY
    w = synth.latents(cfg)
    ctx = tz.Context(tz.make_cfg(cfg), density)
    emb, gains, head = synth.theta(cfg)
    ctx.termezo_load_params(w.cuda(), emb.cuda(), gains.cuda(), head.cuda())
    k0, xi0 = ctx.termezo_build_mask_rule(density, tz.MASK_PER_TENSOR)
    reg = otz.registry(cfg)
    wn = w.numpy()
    sel, xi_o, k0_o, tau = otz.initial_mask_per_tensor(wn, reg, density)
    assert k0 == k0_o
    np.testing.assert_array_equal(xi0.view(np.uint32), xi_o.view(np.uint32))
    st = ctx.termezo_export_state()
    np.testing.assert_array_equal(st["idx"], sel.astype(np.uint32))
    np.testing.assert_array_equal(st["latents"], wn[sel])
    np.testing.assert_array_equal(st["tau_cur"].view(np.uint32), tau.view(np.uint32))
    codes = np.concatenate([ternary.quantize(wn[p.base:p.base + p.n], tau[j]) for j, p in enumerate(reg)])
    np.testing.assert_array_equal(st["packed"], ternary.pack_codes(codes))
