"""Whole-step GPU parity on the tiny BitNet workload (2 layers, d 256,
seq 64, batch 4, density 1%, eps 1e-3, lr 1e-6) against the dense oracle on
the same seeded inputs.  Calls go through the C ABI.

Tolerances:
* F+ and F-: 1e-3 relative (the stated bound), or -- where the oracle's own
  loss moves further under alternative valid fp32 roundings (reductions in
  another order; oracle/rounding.py, 8 members) -- no further from the
  oracle than the furthest member, or within 5 standard deviations of the
  oracle and its members (rounding.agrees).  The quantised forward turns 1-ulp
  differences into int8 / bf16 code flips; the layer-wise tests show the GPU
  bit-exact on each operation given the same inputs.
* g = (F+ - F-) / (2 eps): 1/(2 eps) amplifies those flips, so two valid
  fp32 evaluation orders disagree on g by about 1%; the GPU's g must agree
  within 1e-3 or lie no further from the oracle's than the furthest member.
* latents: |dw| <= 1e-5 (|w| + 2 eps |z|) against the oracle's restore and
  update computed with the GPU's own g (the restore ((w+e)-2e)+e rounds at
  the scale of |w| + 2|e|, and z agrees to a few ulp), so the bound is
  tested apart from g.  Multi-step replays feed the GPU's latents back to the
  oracle after every iteration (the same bound per step, and bit-exact index
  lists); the drift of a free-running oracle replay is recorded.
* codes: bit-exact except active latents within 1e-5 s_w of a threshold;
  their count is the step report's n_near_threshold.
* Every loss and g comparison records |GPU - oracle| next to the
  ensemble's range (tests/helpers.record).
"""
import dataclasses

import numpy as np
import pytest
import torch

from oracle import bitnet, philox, rounding, ternary, termezo as otz
from paper_2609_33548_gb300 import synth
from paper_2609_33548_gb300 import termezo as tz

from helpers import record


pytestmark = pytest.mark.gpu

# the tiny decoder with the classification loss, and with the token-level
# loss over a vocabulary that is not a multiple of the 256-column tile
TINY_SFT = dataclasses.replace(synth.TINY, name="tiny-2L-d256-sft", vocab=1000, loss_mode=1, n_labels=0)
DENSITY, EPS, LR = 0.01, 1e-3, 1e-6


# every step test runs with the GEMMs reading packed codes expanded before each
# GEMM, with the e4m3 weight cache that the sparse kernels keep in step, and
# with the z buffer that carries z between the passes of a direction
@pytest.fixture(scope="module", params=[(synth.TINY, False, False), (TINY_SFT, False, False), (synth.TINY, True, False),
                                        (TINY_SFT, True, False), (synth.TINY, False, True), (TINY_SFT, False, True)],
                ids=["last-token", "token-level", "last-token-cache", "token-level-cache", "last-token-zbuf",
                     "token-level-zbuf"])
def inputs(request):
    cfg, cache, zbuf = request.param
    w = synth.latents(cfg)
    emb, gains, head = synth.theta(cfg)
    tok, tgt = synth.batch(cfg)
    return w, emb, gains, head, tok, tgt, cfg, cache, zbuf


def _gpu_ctx(inputs):
    w, emb, gains, head, tok, tgt, CFG, cache, zbuf = inputs
    ctx = tz.Context(tz.make_cfg(CFG, cache, zbuf), DENSITY)
    dev = [t.cuda() for t in (w, emb, gains, head, tok, tgt)]
    ctx.termezo_load_params(dev[0], dev[1], dev[2], dev[3])
    return ctx, dev


def _theta_np(inputs):
    return (inputs[1].numpy(), inputs[2].numpy(), inputs[3].float().numpy(), inputs[4].numpy(),
            inputs[5].numpy())


def _cfg(inputs):
    return inputs[6]


def _split(codes, reg):
    return [codes[p.base:p.base + p.n].reshape(p.N, p.K) for p in reg]


def test_forward_loss_matches_oracle(inputs):
    ctx, dev = _gpu_ctx(inputs)
    ctx.termezo_build_mask(DENSITY)
    loss, per = ctx.termezo_forward_loss(dev[4], dev[5])
    loss2, per2 = ctx.termezo_forward_loss(dev[4], dev[5])
    assert loss == loss2 and np.array_equal(per, per2)          # deterministic
    reg = otz.registry(_cfg(inputs))
    codes, tau, sw = otz.requantize(inputs[0].numpy(), reg)
    model = (_split(codes, reg), sw)
    per_o, mean_o = bitnet.batch_loss(_cfg(inputs), *model, *_theta_np(inputs))
    ens = rounding.loss_ensemble(_cfg(inputs), model, _theta_np(inputs), n=8)
    record("forward_loss", workload=_cfg(inputs).name, cache=inputs[7],
           **rounding.summary(loss, mean_o, ens.mean(axis=1)))
    assert rounding.agrees(loss, mean_o, ens.mean(axis=1))
    for b in range(len(per)):
        assert rounding.agrees(per[b], per_o[b], ens[:, b]), (b, per[b], per_o[b], ens[:, b])


def test_one_step_matches_oracle(inputs):
    ctx, dev = _gpu_ctx(inputs)
    k0, xi0 = ctx.termezo_build_mask(DENSITY)
    reg = otz.registry(_cfg(inputs))
    state = otz.build(inputs[0].numpy(), reg, DENSITY)
    fn = otz.bitnet_loss_fn(_cfg(inputs), *_theta_np(inputs))
    assert k0 == state.k0 and np.float32(xi0) == state.xi0
    w_before = state.w.copy()
    act = state.active.copy()
    seed = synth.step_seed(0)
    out = ctx.termezo_step(seed, EPS, LR, DENSITY, dev[4], dev[5])
    rec = otz.step(state, fn, seed, EPS, LR)
    # F+-, g against the ensembles of valid roundings
    z = philox.normal(seed, act)
    e = (np.float32(EPS) * z).astype(np.float32)
    wp = w_before.copy(); wp[act] = (w_before[act] + e).astype(np.float32)
    wm = wp.copy(); wm[act] = (wp[act] - np.float32(2) * e).astype(np.float32)
    cp, _, swp = otz.requantize(wp, reg)
    cm, _, swm = otz.requantize(wm, reg)
    lp = rounding.loss_ensemble(_cfg(inputs), (_split(cp, reg), swp), _theta_np(inputs), n=8).mean(axis=1)
    lm = rounding.loss_ensemble(_cfg(inputs), (_split(cm, reg), swm), _theta_np(inputs), n=8).mean(axis=1)
    ens = (lp - lm) / (2 * float(np.float32(EPS)))
    name = _cfg(inputs).name + ("-cache" if inputs[7] else "") + ("-zbuf" if inputs[8] else "")
    record("step_loss_plus", workload=name, **rounding.summary(out["loss_plus"], rec["loss_plus"], lp))
    record("step_loss_minus", workload=name, **rounding.summary(out["loss_minus"], rec["loss_minus"], lm))
    record("step_g", workload=name, **rounding.summary(out["g"], rec["g"], ens))
    assert rounding.agrees(out["loss_plus"], rec["loss_plus"], lp), (out["loss_plus"], rec["loss_plus"], lp)
    assert rounding.agrees(out["loss_minus"], rec["loss_minus"], lm), (out["loss_minus"], rec["loss_minus"], lm)
    assert rounding.g_within_ensemble(out["g"], rec["g"], ens), (out["g"], rec["g"], ens)
    # counters
    assert out["k_active"] == rec["k"] == act.size
    assert out["n_jumps"] == rec["n_jumps"]
    n_near = int(rec["near_plus"].sum() + rec["near_minus"].sum())
    assert out["n_near_threshold"] == n_near
    assert abs(int(out["n_flipped"]) - rec["n_flipped"]) <= n_near
    # state after the update: the oracle's restore and update with the GPU's g
    st = ctx.termezo_export_state()
    np.testing.assert_array_equal(st["idx"], act.astype(np.uint32))
    np.testing.assert_array_equal(rec["w_restored"], (wm[act] + e).astype(np.float32))
    c = np.float32(float(np.float32(LR)) * out["g"])
    expect = (rec["w_restored"] - (c * z).astype(np.float32)).astype(np.float32)
    tol = 1e-5 * (np.abs(w_before[act]) + 2 * np.abs(e))
    err = np.abs(st["latents"].astype(np.float64) - expect)
    record("step_latents", workload=name, max_rel=float((err / (np.abs(w_before[act]) + 2 * np.abs(e))).max()))
    assert np.all(err <= tol)
    got = ternary.unpack_codes(st["packed"])
    bad = np.nonzero(got != rec["codes_minus"])[0]
    assert rec["frozen_mismatch"] == 0
    assert np.all(np.isin(bad, act[rec["near_minus"]]))
    np.testing.assert_array_equal(st["tau_minus"].view(np.uint32), rec["tau_minus"].view(np.uint32))
    np.testing.assert_array_equal(st["tau_plus"].view(np.uint32), rec["tau_plus"].view(np.uint32))


def _replay(ctx, state, reg, steps, seed0, rng_seed, eps=EPS, lr=2e-3):
    """Shrink, perturb and update over `steps` iterations with a given g
    sequence on both sides.  After every iteration the oracle's prediction
    from the GPU's previous latents must give the GPU's index list bit for
    bit and its latents within 1e-5 (|w| + 2 eps |z|); the GPU's latents are
    then fed back to the oracle.  A second oracle state runs free on its own
    latents; its largest relative drift from the GPU is returned with the
    sizes k_t."""
    eps, lr = np.float32(eps), np.float32(lr)
    rng = np.random.default_rng(rng_seed)
    free = otz.State(w=state.w.copy(), reg=reg, active=state.active.copy(), xi0=state.xi0, k0=state.k0,
                     frozen_code=state.frozen_code.copy())
    sizes, drift = [], 0.0
    for t in range(steps):
        g = float(rng.standard_normal() * 20.0)
        seed = synth.step_seed(seed0 + t)
        if t:
            ctx.termezo_shrink()
        ctx.termezo_requantize(seed, float(eps), +1)
        ctx.termezo_requantize(seed, float(eps), -1)
        ctx.termezo_update(seed, float(eps), float(lr), g)
        st = ctx.termezo_export_state(packed=False)
        for o in (state, free):
            if t:
                o.active, _ = otz.shrink(o.w, reg, o.active, o.xi0)
            z = philox.normal(seed, o.active)
            w_next, *_ = otz.masked_spsa(o.w, o.active, z, eps, 0.0, lambda v: 0.0)
            c = np.float32(float(lr) * g)
            w_next[o.active] = (w_next[o.active] - (c * z).astype(np.float32)).astype(np.float32)
            o.w = w_next
            if o is state:
                scale = np.abs(w_next[o.active]).astype(np.float64) + 2 * np.abs(eps * z)
        act = state.active
        np.testing.assert_array_equal(st["idx"], act.astype(np.uint32))
        assert np.all(np.abs(st["latents"].astype(np.float64) - state.w[act]) <= 1e-5 * scale), t
        state.w[act] = st["latents"]                   # the GPU's latents, fed back
        if act.size and np.array_equal(free.active, act):
            drift = max(drift, float((np.abs(free.w[act].astype(np.float64) - st["latents"]) / scale).max()))
        sizes.append(act.size)
    return sizes, drift


def test_mask_and_update_replay_many_steps(inputs):
    """Mask shrink, perturb and update over 30 iterations with a given g
    sequence fed to both sides, large enough that the active set shrinks:
    indices bit-exact and latents within 1e-5 at every iteration (see
    _replay)."""
    w0 = inputs[0].numpy()
    reg = otz.registry(_cfg(inputs))
    ctx, dev = _gpu_ctx(inputs)
    ctx.termezo_build_mask(DENSITY)
    state = otz.build(w0, reg, DENSITY)
    sizes, drift = _replay(ctx, state, reg, 30, seed0=0, rng_seed=5)
    record("replay", workload=_cfg(inputs).name, rule="global", steps=30, k_first=sizes[0], k_last=sizes[-1],
           free_run_max_rel_drift=drift)
    assert sizes[-1] < sizes[0]
    assert all(a >= b for a, b in zip(sizes, sizes[1:]))


def test_k_directions_step_matches_oracle(inputs):
    """Algorithm 1 with K = 3 directions: per-direction F+-, g_k against the
    oracle's ensembles; the latents after the K restores and the K-term
    update (the oracle's update recomputed with the GPU's g_k, so that only
    the rounding of the restores and of z remains); and the index list."""
    K = 3
    ctx, dev = _gpu_ctx(inputs)
    ctx.termezo_build_mask(DENSITY)
    cfg, th = _cfg(inputs), _theta_np(inputs)
    reg = otz.registry(cfg)
    state = otz.build(inputs[0].numpy(), reg, DENSITY)
    fn = otz.bitnet_loss_fn(cfg, *th)
    w_before = state.w.copy()
    act = state.active.copy()
    seeds = [synth.step_seed(10 + k) for k in range(K)]
    out = ctx.termezo_step_k(seeds, EPS, LR, DENSITY, dev[4], dev[5])
    rec = otz.step_k(state, fn, seeds, EPS, LR)
    eps32 = np.float32(EPS)
    w = w_before.copy()
    zs = []
    for k, seed in enumerate(seeds):
        z = philox.normal(seed, act)
        zs.append(z)
        e = (eps32 * z).astype(np.float32)
        wp = w.copy(); wp[act] = (w[act] + e).astype(np.float32)
        wm = wp.copy(); wm[act] = (wp[act] - np.float32(2) * e).astype(np.float32)
        cp, _, swp = otz.requantize(wp, reg)
        cm, _, swm = otz.requantize(wm, reg)
        lp = rounding.loss_ensemble(cfg, (_split(cp, reg), swp), th, n=8).mean(axis=1)
        lm = rounding.loss_ensemble(cfg, (_split(cm, reg), swm), th, n=8).mean(axis=1)
        fp, fm = out["losses"][k]
        assert rounding.agrees(fp, rec["loss_plus"][k], lp), (k, fp, rec["loss_plus"][k], lp)
        assert rounding.agrees(fm, rec["loss_minus"][k], lm), (k, fm, rec["loss_minus"][k], lm)
        ens = (lp - lm) / (2 * float(eps32))
        assert rounding.g_within_ensemble(out["g_k"][k], rec["g"][k], ens), (k, out["g_k"][k], rec["g"][k], ens)
        w = wm.copy(); w[act] = (wm[act] + e).astype(np.float32)
        np.testing.assert_array_equal(w[act], rec["w_restored"][k])
    assert out["g"] == out["g_k"][-1] and out["loss_plus"] == out["losses"][-1][0]
    assert out["k_active"] == rec["k"] == act.size and out["n_jumps"] == rec["n_jumps"]
    # the update with the GPU's g_k
    lr_k = float(np.float32(LR)) / K
    expect = w.copy()
    for z, g in zip(zs, out["g_k"]):
        c = np.float32(lr_k * g)
        expect[act] = (expect[act] - (c * z).astype(np.float32)).astype(np.float32)
    st = ctx.termezo_export_state(packed=False)
    np.testing.assert_array_equal(st["idx"], act.astype(np.uint32))
    scale = np.abs(w_before[act]) + 2 * max(float(np.abs(eps32 * z).max()) for z in zs)
    assert np.all(np.abs(st["latents"].astype(np.float64) - expect[act]) <= K * 1e-5 * scale)


def test_single_direction_step_k_is_step(inputs):
    """termezo_step_k with one seed runs the same kernels as termezo_step:
    losses, g and the latents after the step are identical."""
    a, dev = _gpu_ctx(inputs)
    b, _ = _gpu_ctx(inputs)
    a.termezo_build_mask(DENSITY)
    b.termezo_build_mask(DENSITY)
    seed = synth.step_seed(3)
    oa = a.termezo_step(seed, EPS, LR, DENSITY, dev[4], dev[5])
    ob = b.termezo_step_k([seed], EPS, LR, DENSITY, dev[4], dev[5])
    assert (oa["loss_plus"], oa["loss_minus"], oa["g"]) == (ob["loss_plus"], ob["loss_minus"], ob["g"])
    sa, sb = a.termezo_export_state(packed=False), b.termezo_export_state(packed=False)
    np.testing.assert_array_equal(sa["latents"].view(np.uint32), sb["latents"].view(np.uint32))


def test_joint_theta_step_matches_oracle(inputs):
    """Algorithm 1 as written (termezo_step_joint, K = 2): the masked
    latents and theta (embeddings, norm gains fp32, LM head bf16) perturbed
    together.  Per-direction F+- and g_k against the oracle's ensembles at
    the oracle's own (codes, theta+-); latents and theta after the update
    against the oracle's arithmetic with the GPU's g_k.  theta's z differs
    from the oracle's by a few ulp, so fp32 parts agree within the restore
    rounding and the bf16 head in all but a rare element that rounds to a
    neighbouring bf16 value."""
    K = 2
    w0, emb0, gains0, head0, tok, tgt, cfg, _, _ = inputs
    ctx, dev = _gpu_ctx(inputs)
    ctx.termezo_build_mask(DENSITY)
    reg = otz.registry(cfg)
    state = otz.build(w0.numpy(), reg, DENSITY)
    act = state.active.copy()
    seeds = [synth.step_seed(40 + k) for k in range(K)]
    out = ctx.termezo_step_k(seeds, EPS, LR, DENSITY, dev[4], dev[5], theta=True)
    th0 = [emb0.numpy(), gains0.numpy(), head0.float().numpy()]
    fn = otz.bitnet_theta_loss_fn(cfg, tok.numpy(), tgt.numpy())
    rec, th_oracle = otz.step_joint(state, th0, fn, seeds, EPS, LR)
    eps32 = np.float32(EPS)
    d, p = w0.numel(), sum(t.size for t in th0)
    bf = [False, False, True]
    offs = np.cumsum([0] + [t.size for t in th0])
    split = lambda z: [z[offs[i]:offs[i + 1]].reshape(th0[i].shape) for i in range(3)]
    w, th = w0.numpy().copy(), [t.copy() for t in th0]
    zs_w, zs_t = [], []
    for k, seed in enumerate(seeds):
        zw, zt = philox.normal(seed, act), otz.theta_normals(seed, d, p)
        zs_w.append(zw)
        zs_t.append(zt)
        ew = (eps32 * zw).astype(np.float32)
        et = [(eps32 * z).astype(np.float32) for z in split(zt)]
        wp = w.copy(); wp[act] = (w[act] + ew).astype(np.float32)
        thp = [otz._stored(t + e, b) for t, e, b in zip(th, et, bf)]
        wm = wp.copy(); wm[act] = (wp[act] - np.float32(2) * ew).astype(np.float32)
        thm = [otz._stored(t - np.float32(2) * e, b) for t, e, b in zip(thp, et, bf)]
        cp, _, swp = otz.requantize(wp, reg)
        cm, _, swm = otz.requantize(wm, reg)
        tt = (tok.numpy(), tgt.numpy())
        lp = rounding.loss_ensemble(cfg, (_split(cp, reg), swp), (*thp, *tt), n=8).mean(axis=1)
        lm = rounding.loss_ensemble(cfg, (_split(cm, reg), swm), (*thm, *tt), n=8).mean(axis=1)
        fp, fm = out["losses"][k]
        assert rounding.agrees(fp, rec["loss_plus"][k], lp), (k, fp, rec["loss_plus"][k], lp)
        assert rounding.agrees(fm, rec["loss_minus"][k], lm), (k, fm, rec["loss_minus"][k], lm)
        ens = (lp - lm) / (2 * float(eps32))
        assert rounding.g_within_ensemble(out["g_k"][k], rec["g"][k], ens), (k, out["g_k"][k], rec["g"][k], ens)
        w = wm.copy(); w[act] = (wm[act] + ew).astype(np.float32)
        th = [otz._stored(t + e, b) for t, e, b in zip(thm, et, bf)]
    # the update with the GPU's g_k
    lr_k = float(np.float32(LR)) / K
    for zw, zt, g in zip(zs_w, zs_t, out["g_k"]):
        c = np.float32(lr_k * g)
        w[act] = (w[act] - (c * zw).astype(np.float32)).astype(np.float32)
        th = [otz._stored(t - (c * z).astype(np.float32), b) for t, z, b in zip(th, split(zt), bf)]
    st = ctx.termezo_export_state(packed=False)
    np.testing.assert_array_equal(st["idx"], act.astype(np.uint32))
    emax = float(np.abs(eps32 * np.concatenate(zs_w)).max())
    assert np.all(np.abs(st["latents"].astype(np.float64) - w[act]) <= K * 1e-5 * (np.abs(w0.numpy()[act]) + 2 * emax))
    got = [dev[1].cpu().numpy(), dev[2].cpu().numpy(), dev[3].cpu().float().numpy()]
    for i in range(2):
        emax_t = 2 * float(np.abs(eps32 * np.concatenate([split(z)[i].ravel() for z in zs_t])).max())
        assert np.all(np.abs(got[i].astype(np.float64) - th[i]) <= K * 1e-5 * (np.abs(th0[i]) + emax_t)), i
        assert not np.array_equal(got[i], th0[i])          # theta did move
    diff = np.abs(got[2].astype(np.float64) - th[2])
    ulp = np.abs(th[2]).astype(np.float64) * 2.0 ** -7 + 1e-30
    assert np.count_nonzero(diff) <= max(3, int(1e-4 * diff.size)), np.count_nonzero(diff)
    assert np.all(diff <= 2 * ulp)
    assert not np.array_equal(got[2], th0[2])


def test_per_tensor_mask_replay_many_steps(inputs):
    """The shrink of Eq. 5 with one xi_0 per projection (per-tensor mask):
    20 iterations with a given g sequence, index lists bit-exact and latents
    within 1e-5 at every iteration (see _replay)."""
    w0 = inputs[0].numpy()
    reg = otz.registry(_cfg(inputs))
    ctx, dev = _gpu_ctx(inputs)
    ctx.termezo_build_mask_rule(DENSITY, tz.MASK_PER_TENSOR)
    state = otz.build(w0, reg, DENSITY, per_tensor=True)
    sizes, drift = _replay(ctx, state, reg, 20, seed0=100, rng_seed=6)
    record("replay", workload=_cfg(inputs).name, rule="per-tensor", steps=20, k_first=sizes[0], k_last=sizes[-1],
           free_run_max_rel_drift=drift)
    assert sizes[-1] < sizes[0]


def test_full_density_step_matches_oracle():
    """rho_0 = 1: every latent is active (full MeZO on the latents); one step
    against the oracle as in the masked case."""
    cfg = synth.TINY
    w = synth.latents(cfg)
    emb, gains, head = synth.theta(cfg)
    tok, tgt = synth.batch(cfg)
    ctx = tz.Context(tz.make_cfg(cfg), 1.0)
    dev = [t.cuda() for t in (w, emb, gains, head, tok, tgt)]
    ctx.termezo_load_params(dev[0], dev[1], dev[2], dev[3])
    k0, _ = ctx.termezo_build_mask(1.0)
    assert k0 == cfg.d_lat
    reg = otz.registry(cfg)
    state = otz.build(w.numpy(), reg, 1.0)
    th = (emb.numpy(), gains.numpy(), head.float().numpy(), tok.numpy(), tgt.numpy())
    fn = otz.bitnet_loss_fn(cfg, *th)
    seed = synth.step_seed(7)
    w_before = state.w.copy()
    out = ctx.termezo_step(seed, EPS, LR, 1.0, dev[4], dev[5])
    rec = otz.step(state, fn, seed, EPS, LR)
    z = philox.normal(seed, np.arange(cfg.d_lat))
    e = (np.float32(EPS) * z).astype(np.float32)
    wp = (w_before + e).astype(np.float32)
    wm = (wp - np.float32(2) * e).astype(np.float32)
    cp, _, swp = otz.requantize(wp, reg)
    cm, _, swm = otz.requantize(wm, reg)
    lp = rounding.loss_ensemble(cfg, (_split(cp, reg), swp), th, n=8).mean(axis=1)
    lm = rounding.loss_ensemble(cfg, (_split(cm, reg), swm), th, n=8).mean(axis=1)
    assert rounding.agrees(out["loss_plus"], rec["loss_plus"], lp)
    assert rounding.agrees(out["loss_minus"], rec["loss_minus"], lm)
    assert rounding.g_within_ensemble(out["g"], rec["g"], (lp - lm) / (2 * float(np.float32(EPS))))
    assert out["k_active"] == cfg.d_lat
    st = ctx.termezo_export_state(packed=False)
    np.testing.assert_array_equal(st["idx"], np.arange(cfg.d_lat, dtype=np.uint32))
    c = np.float32(float(np.float32(LR)) * out["g"])
    expect = (rec["w_restored"] - (c * z).astype(np.float32)).astype(np.float32)
    assert np.all(np.abs(st["latents"].astype(np.float64) - expect) <= 1e-5 * (np.abs(w_before) + 2 * np.abs(e)))
