"""100 consecutive TerMeZO steps on the 2B-long-shaped workload: 30 layers,
d 2560, 20 / 5 heads, FFN 6912, sequences of 2048 tokens x batch 4,
token-level cross-entropy over the 128,256-token vocabulary, mask density
5 %, perturbation seed 1000 + t and a new minibatch at every step t.

Every step (Algorithm 1's loop body; Eq. 5's shrink from t = 1):
* the GPU's g_t drives a replay of shrink, perturb and update in the oracle
  over three projections (layer 0 q, layer 14 k, layer 29 o; each
  projection's mask, thresholds and latents depend only on itself and g);
  the replay starts every step from the GPU's latents of the step before;
* the active index list of each of them equals the oracle's shrink bit for
  bit, their tau+ and tau- equal the oracle's, and their latents agree with
  the oracle's restore and update within 1e-5 (|w| + 2 eps |z|);
* the active set only shrinks, and a second, free-running oracle replay
  reports its drift from the GPU.

At t in {0, 1, 50, 99} the forward at the step's - codes is traced: its loss
equals the step's F- bit for bit, layers 0 and 29 pass the layer-wise checks
(tests/layerwise.py) on one sequence, the loss from the GPU's last residual
stream agrees with the GPU's to 1e-5, and the - codes of the three
projections equal the oracle's except latents within 1e-5 s_w of tau."""
import numpy as np
import pytest
import torch

from oracle import philox, ternary, termezo as otz
from paper_2609_33548_gb300 import synth
from paper_2609_33548_gb300 import termezo as tz

import layerwise as lw
from helpers import record

pytestmark = pytest.mark.gpu

EPS, LR, STEPS = 1e-3, 1e-6, 100
CHECK_T = (0, 1, 50, 99)
SUBSET = (0, 7 * 14 + 1, 7 * 29 + 3)       # layer 0 q, layer 14 k, layer 29 o


class _Proj:
    """Oracle state of one projection: its dense latents, active set (local
    indices) and the xi_0 of the mask."""

    def __init__(self, p, w, act_local, xi0):
        self.p, self.w, self.act, self.xi0 = p, w, act_local, xi0
        self.reg = otz.single_registry(p.N, p.K)

    def step(self, t, seed, g, shrink=True):
        """The oracle's iteration t with the GPU's g: returns (kept, tau+,
        tau-, codes-, latents after the update, scale of the restore)."""
        if t and shrink:
            self.act, _ = otz.shrink(self.w, self.reg, self.act, self.xi0)
        a = self.act
        z = philox.normal(seed, a + self.p.base)
        e = (np.float32(EPS) * z).astype(np.float32)
        wp = self.w.copy()
        wp[a] = (self.w[a] + e).astype(np.float32)
        tp = ternary.threshold(ternary.absmean(wp))
        wm = wp.copy()
        wm[a] = (wp[a] - np.float32(2) * e).astype(np.float32)
        gm = ternary.absmean(wm)
        tm = ternary.threshold(gm)
        codes_m = ternary.quantize(wm, tm)
        near_m = otz.near_threshold(wm[a], np.full(a.size, tm), np.full(a.size, ternary.weight_scale(gm)))
        rest = (wm[a] + e).astype(np.float32)
        c = np.float32(float(np.float32(LR)) * g)
        new = (rest - (c * z).astype(np.float32)).astype(np.float32)
        scale = np.abs(self.w[a]).astype(np.float64) + 2 * np.abs(e)
        self.w[a] = new
        return a, tp, tm, codes_m, near_m, scale


def test_100_steps_2b_long():
    cfg, density = synth.BITNET_2B_LONG, 0.05
    w = synth.latents(cfg)
    emb, gains, head = synth.theta(cfg)
    ctx = tz.Context(tz.make_cfg(cfg), density)
    dev = [t.cuda() for t in (w, emb, gains, head)]
    ctx.termezo_load_params(*dev)
    k0, xi0 = ctx.termezo_build_mask(density)
    del dev[0]
    reg = otz.registry(cfg)
    st = ctx.termezo_export_state(packed=False)
    wn = w.numpy()
    teach, free = [], []
    for j in SUBSET:
        p = reg[j]
        lo, hi = np.searchsorted(st["idx"], [p.base, p.base + p.n])
        a = st["idx"][lo:hi].astype(np.int64) - p.base
        np.testing.assert_array_equal(st["latents"][lo:hi], wn[p.base:p.base + p.n][a])
        teach.append(_Proj(p, wn[p.base:p.base + p.n].copy(), a, xi0))
        free.append(_Proj(p, wn[p.base:p.base + p.n].copy(), a.copy(), xi0))
    del w, wn
    gains_np, head_np = gains.numpy(), head.float().numpy()
    ks, gs, max_rel, drift = [], [], 0.0, 0.0
    k_prev = k0
    for t in range(STEPS):
        tok, tgt = synth.batch(cfg, step=t)
        tok_d, tgt_d = tok.cuda(), tgt.cuda()
        seed = synth.step_seed(t)
        out = ctx.termezo_step(seed, EPS, LR, density, tok_d, tgt_d)
        assert out["k_active"] <= k_prev and out["n_jumps"] == 0
        k_prev = out["k_active"]
        ks.append(int(out["k_active"]))
        gs.append(float(out["g"]))
        check = t in CHECK_T
        st = ctx.termezo_export_state(packed=check)
        for j, pt, pf in zip(SUBSET, teach, free):
            p = reg[j]
            lo, hi = np.searchsorted(st["idx"], [p.base, p.base + p.n])
            a_gpu = st["idx"][lo:hi].astype(np.int64) - p.base
            a, tp, tm, codes_m, near_m, scale = pt.step(t, seed, out["g"])
            np.testing.assert_array_equal(a_gpu, a, err_msg=f"t {t} proj {j} index list")
            assert st["tau_plus"][j].view(np.uint32) == tp.view(np.uint32), (t, j)
            assert st["tau_minus"][j].view(np.uint32) == tm.view(np.uint32), (t, j)
            err = np.abs(st["latents"][lo:hi].astype(np.float64) - pt.w[a]) / scale
            assert np.all(err <= 1e-5), (t, j, err.max())
            max_rel = max(max_rel, float(err.max()))
            pt.w[a] = st["latents"][lo:hi]                      # the GPU's latents, fed back
            af, *_ = pf.step(t, seed, out["g"])
            if np.array_equal(af, a):
                drift = max(drift, float((np.abs(pf.w[a].astype(np.float64) - st["latents"][lo:hi]) / scale).max()))
            if check:
                got = ternary.unpack_codes(st["packed"][p.base // 16:(p.base + p.n) // 16])
                bad = np.flatnonzero(got != codes_m)
                assert np.all(np.isin(bad, a[near_m])), (t, j, bad.size)
        if check:
            stats = {}
            _, per, tr = ctx.termezo_forward_trace(tok_d, tgt_d, 0)
            np.testing.assert_array_equal(per, out["per_seq_minus"])        # the step's F-, bit for bit
            sw = (np.float32(2.0) * st["tau_minus"]).astype(np.float32)
            for l in (0, cfg.layers - 1):
                if l:
                    _, _, tr = ctx.termezo_forward_trace(tok_d, tgt_d, l)
                tn = {n: v.cpu().numpy() for n, v in tr.items()}
                del tr
                lw.check_layer(cfg, l, tn, [0], lw.layer_codes(st["packed"], reg, l), sw[7 * l:7 * l + 7],
                               gains_np, stats, f"2b-long t {t}")
            _, per, tr = ctx.termezo_forward_trace(tok_d, tgt_d, cfg.layers)
            stats["head_rel_err"] = lw.check_head(cfg, tr["x_in"].cpu().numpy(), per, [0], gains_np, head_np,
                                                  tgt.numpy())
            record("long_run_check", t=t, g=out["g"], loss_minus=out["loss_minus"], k=out["k_active"], **stats)
    assert ks[-1] <= ks[0]
    record("long_run", workload=cfg.name, steps=STEPS, k0=k0, k_last=ks[-1], g_first=gs[0], g_last=gs[-1],
           max_rel_latent_err=max_rel, free_run_max_rel_drift=drift)
