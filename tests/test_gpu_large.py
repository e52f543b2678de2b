"""GPU parity at the full model-shaped workloads (0.7B-, 2B- and 2B-long-
shaped: 24-30 layers, d 1536-2560, 0.68-2.08 G latents) in the launch
configuration bench.py times.

* Mask (Eqs. 2-4) at full size: S_0, xi_0 and tau_0 of every projection
  bit-exact against the oracle's global selection, and the packed codes of
  every weight bit for bit.
* Perturb / requantise (Eq. 2, Algorithm 1) after one full step, on sampled
  projections: tau+ and tau- bit-exact, codes of the - pass bit-exact except
  latents within 1e-5 s_w of a threshold.
* BitLinear GEMM at the 2B shapes (M 8192 tokens): int32 accumulators of
  sampled rows bit-exact.
* One step on the 0.7B and 2B models (2B at densities 1 % and 0.1 %): the loss
  of each sequence depends only on that sequence, so sampled sequences are
  evaluated by the oracle at +eps z and -eps z, next to 8 valid fp32
  re-roundings of the oracle (oracle/rounding.py).  At 24-30 layers these
  move a sequence's F by several percent and its g by tens of percent: one
  flipped activation code changes every later layer, so the loss of such a
  random-init decoder is determined by its definition only to that spread.
  The comparison is therefore statistical: F+-, g lie within 5 sample
  standard deviations of the mean of the oracle and its re-roundings
  (rounding.agrees / rounding.consistent; a false alarm about once in 1000), and every value is
  recorded.  The exact, per-operation parity of these forwards is
  test_gpu_layerwise.py's (bit-exact given the same inputs).  tau+ and tau- of
  every projection are bit-exact.
Inputs are drawn on the host by the seeded generator (so the oracle can
redraw them anywhere) and copied to the device."""
import numpy as np
import pytest
import torch

from oracle import bitnet, philox, rounding, ternary, termezo as otz
from paper_2609_33548_gb300 import synth
from paper_2609_33548_gb300 import termezo as tz

from helpers import record

pytestmark = pytest.mark.gpu

EPS, LR = 1e-3, 1e-6


def _setup(cfg, density):
    w = synth.latents(cfg)
    emb, gains, head = synth.theta(cfg)
    tok, tgt = synth.batch(cfg)
    ctx = tz.Context(tz.make_cfg(cfg), density)
    dev = [t.cuda() for t in (w, emb, gains, head, tok, tgt)]
    ctx.termezo_load_params(dev[0], dev[1], dev[2], dev[3])
    return ctx, dev, (w.numpy(), emb.numpy(), gains.numpy(), head.float().numpy(), tok.numpy(), tgt.numpy())


def _mask_exact(ctx, w, reg, density):
    k0, xi0 = ctx.termezo_build_mask(density)
    st = ctx.termezo_export_state()
    sel, xi0_o, k0_o, tau = otz.initial_mask(w, reg, density)
    assert k0 == k0_o
    assert np.float32(xi0).view(np.uint32) == np.float32(xi0_o).view(np.uint32)
    np.testing.assert_array_equal(st["tau_cur"].view(np.uint32), tau.view(np.uint32))
    np.testing.assert_array_equal(st["idx"], sel.astype(np.uint32))
    np.testing.assert_array_equal(st["latents"], w[sel])
    for j, p in enumerate(reg):  # packed codes, projection by projection
        np.testing.assert_array_equal(st["packed"][p.base // 16:(p.base + p.n) // 16],
                                      ternary.pack_codes(ternary.quantize(w[p.base:p.base + p.n], tau[j])))
    return sel


def _requant_sampled(ctx, w, reg, act, seed, picks):
    st = ctx.termezo_export_state()
    z_all = philox.normal(seed, act)
    for j in picks:
        p = reg[j]
        lo, hi = np.searchsorted(act, [p.base, p.base + p.n])
        a, z = act[lo:hi], z_all[lo:hi]
        e = (np.float32(EPS) * z).astype(np.float32)
        v = w[p.base:p.base + p.n].copy()
        v[a - p.base] = (v[a - p.base] + e).astype(np.float32)
        gp = ternary.absmean(v)
        tp = ternary.threshold(gp)
        v[a - p.base] = (v[a - p.base] - np.float32(2) * e).astype(np.float32)
        gm = ternary.absmean(v)
        tm, swm = ternary.threshold(gm), ternary.weight_scale(gm)
        assert st["tau_plus"][j].view(np.uint32) == tp.view(np.uint32), (p, st["tau_plus"][j], tp)
        assert st["tau_minus"][j].view(np.uint32) == tm.view(np.uint32), (p, st["tau_minus"][j], tm)
        got = ternary.unpack_codes(st["packed"][p.base // 16:(p.base + p.n) // 16])
        want = ternary.quantize(v, tm)
        bad = np.flatnonzero(got != want) + p.base
        near = a[otz.near_threshold(v[a - p.base], np.full(a.size, tm), np.full(a.size, swm))]
        assert np.all(np.isin(bad, near)), (p, bad.size)


@pytest.mark.parametrize("name", ["2b", "2b-long"])
def test_full_size_mask_requant_and_gemm(name):
    cfg, density = {"2b": (synth.BITNET_2B, 0.01), "2b-long": (synth.BITNET_2B_LONG, 0.05)}[name]
    ctx, dev, (w, *_r) = _setup(cfg, density)
    reg = otz.registry(cfg)
    act = _mask_exact(ctx, w, reg, density)
    seed = synth.step_seed(0)
    out = ctx.termezo_step(seed, EPS, LR, density, dev[4], dev[5])
    assert out["k_active"] == act.size and out["n_jumps"] == 0
    picks = [0, 7 * 14 + 4, len(reg) - 1]          # layer 0 q, layer 14 gate, last down
    _requant_sampled(ctx, w, reg, act, seed, picks)
    if name == "2b":
        # the BitLinear GEMM at the model's token count, on codes at tau_0
        ctx2 = tz.Context(tz.make_cfg(cfg), density)
        ctx2.termezo_load_params(dev[0], dev[1], dev[2], dev[3])
        ctx2.termezo_build_mask(density)
        j = 7 * 14 + 4
        p = reg[j]
        x = synth.op_activations(cfg.tokens, p.K, seed=31)
        acc = torch.zeros(cfg.tokens, p.N, dtype=torch.int32, device="cuda")
        ctx2.termezo_bitlinear(j, x.cuda(), acc, None)
        torch.cuda.synchronize()
        tau = ternary.threshold(ternary.absmean(w[p.base:p.base + p.n]))
        codes = ternary.quantize(w[p.base:p.base + p.n], tau).reshape(p.N, p.K)
        rows = np.random.default_rng(3).choice(cfg.tokens, 64, replace=False)
        q, _ = bitnet.act_quant(x.float().numpy()[rows])
        np.testing.assert_array_equal(acc.cpu().numpy()[rows], bitnet.int_matmul(q, codes))


@pytest.mark.parametrize("planted", ["near", "far"])
def test_mask_build_when_the_sampled_histogram_misleads(planted):
    """A projection of 16384 x 16384 latents has 65536 dense blocks of 4096,
    so the mask build takes its superset bound from the distance histogram
    of one block in 16 (blocks 16 j + 8).  Those blocks are planted here:
    with latents at about tau_0 ("near") the sample overstates the weights
    close to the threshold 16-fold and the superset holds fewer than k0
    weights; with latents at 10 tau_0 ("far") it understates them and the
    superset outgrows its buffer.  Either way the build falls back to the
    six-pass selection, and S_0, xi_0, tau_0 and every packed code are
    bit-exact against the oracle."""
    n, k, density = 16384, 16384, 0.01
    w = synth.op_latents(n, k, seed=21).numpy().reshape(-1)
    reg = otz.single_registry(n, k)
    sampled = w.reshape(-1, 4096)[8::16]           # a view: the sampled blocks
    rng = np.random.default_rng(5)
    sign = np.where(rng.random(sampled.shape) < 0.5, -1.0, 1.0)
    jitter = rng.standard_normal(sampled.shape)
    for _ in range(2):                             # tau_0 moves a little with the planted values
        _, tau, _ = otz.thresholds(w, reg)
        mag = tau[0] * (1.0 + 1e-3 * jitter) if planted == "near" else 10.0 * tau[0] * (1.0 + 0.1 * np.abs(jitter))
        sampled[...] = (sign * mag).astype(np.float32)
    ctx = tz.Context(tz.op_cfg(n, k, 128), density)
    ctx.termezo_load_params(torch.from_numpy(w).cuda())
    _mask_exact(ctx, w, reg, density)


def test_full_size_per_tensor_mask():
    """The per-tensor quantile at the full 2B shape (210 projections, 2.08 G
    latents): k0, every projection's xi_0 and the sorted index list
    bit-exact against the oracle."""
    cfg, density = synth.BITNET_2B, 0.01
    ctx, dev, (w, *_r) = _setup(cfg, density)
    k0, xi0 = ctx.termezo_build_mask_rule(density, tz.MASK_PER_TENSOR)
    sel, xi_o, k0_o, tau = otz.initial_mask_per_tensor(w, otz.registry(cfg), density)
    assert k0 == k0_o
    np.testing.assert_array_equal(xi0.view(np.uint32), xi_o.view(np.uint32))
    st = ctx.termezo_export_state(packed=False)
    np.testing.assert_array_equal(st["idx"], sel.astype(np.uint32))
    np.testing.assert_array_equal(st["latents"], w[sel])


def _step_sampled_sequences(cfg, density, rows, name):
    ctx, dev, (w, emb, gains, head, tok, tgt) = _setup(cfg, density)
    reg = otz.registry(cfg)
    k0, xi0 = ctx.termezo_build_mask(density)
    act, xi0_o, k0_o, _ = otz.initial_mask(w, reg, density)
    assert k0 == k0_o and np.float32(xi0).view(np.uint32) == np.float32(xi0_o).view(np.uint32)
    seed = synth.step_seed(0)
    out = ctx.termezo_step(seed, EPS, LR, density, dev[4], dev[5])
    z = philox.normal(seed, act)
    e = (np.float32(EPS) * z).astype(np.float32)
    del dev[0]
    wp = w.copy()
    wp[act] = (w[act] + e).astype(np.float32)
    cp, tp, swp = otz.requantize(wp, reg)
    wp[act] = (wp[act] - np.float32(2) * e).astype(np.float32)
    wm = wp
    del w
    cm, tm, swm = otz.requantize(wm, reg)
    st = ctx.termezo_export_state(packed=False)
    np.testing.assert_array_equal(st["tau_plus"].view(np.uint32), tp.view(np.uint32))
    np.testing.assert_array_equal(st["tau_minus"].view(np.uint32), tm.view(np.uint32))
    split = lambda c: [c[p.base:p.base + p.n].reshape(p.N, p.K) for p in reg]
    th = (emb, gains, head, tok, tgt)
    per_p, _ = bitnet.batch_loss(cfg, split(cp), swp, *th, rows=rows)
    per_m, _ = bitnet.batch_loss(cfg, split(cm), swm, *th, rows=rows)
    ens_p = rounding.loss_ensemble(cfg, (split(cp), swp), th, n=8, rows=rows)
    ens_m = rounding.loss_ensemble(cfg, (split(cm), swm), th, n=8, rows=rows)
    two_eps = 2 * float(np.float32(EPS))
    for i, b in enumerate(rows):
        g_gpu = (out["per_seq_plus"][b] - out["per_seq_minus"][b]) / two_eps
        g_ref = (per_p[i] - per_m[i]) / two_eps
        g_ens = (ens_p[:, i] - ens_m[:, i]) / two_eps
        record("sampled_step", workload=name, sequence=b, F_plus=rounding.summary(out["per_seq_plus"][b], per_p[i],
                                                                                 ens_p[:, i]),
               F_minus=rounding.summary(out["per_seq_minus"][b], per_m[i], ens_m[:, i]),
               g=rounding.summary(g_gpu, g_ref, g_ens))
        assert rounding.agrees(out["per_seq_plus"][b], per_p[i], ens_p[:, i]), (b, out["per_seq_plus"][b], per_p[i])
        assert rounding.agrees(out["per_seq_minus"][b], per_m[i], ens_m[:, i])
        assert rounding.agrees(g_gpu, g_ref, g_ens), (b, g_gpu, g_ref)
    assert out["n_jumps"] == 0 and out["k_active"] == act.size


def test_step_sampled_sequences_0_7b():
    _step_sampled_sequences(synth.BITNET_07B, 0.01, [0, 1], "0.7b")


@pytest.mark.parametrize("density", [0.01, 0.001])
def test_step_sampled_sequences_2b(density):
    _step_sampled_sequences(synth.BITNET_2B, density, [3], f"2b density {density}")
