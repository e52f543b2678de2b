"""Pins of the oracle's mask rules (Eqs. 4-5, Algorithm 1): cardinality,
quantile order, index tie-break, global selection across projections,
nesting S_t within S_{t-1}, frozen weights keeping their code.  CPU only."""
import math

import numpy as np
import pytest

from oracle import ternary, termezo
from paper_2609_33548_gb300 import synth


def _reg(sizes):
    out, base = [], 0
    for j, (N, K) in enumerate(sizes):
        out.append(termezo.Proj(0, f"t{j}", N, K, base))
        base += N * K
    return out


def test_initial_mask_cardinality_and_quantile_order():
    reg = _reg([(32, 64), (48, 16), (16, 128)])
    n = sum(p.n for p in reg)
    rng = np.random.default_rng(0)
    w = (rng.standard_normal(n) * 0.02).astype(np.float32)
    for rho in (1e-4, 0.01, 0.05, 0.5, 1.0):
        sel, xi0, k0, tau = termezo.initial_mask(w, reg, rho)
        assert k0 == int(np.floor(rho * n)) and sel.size == k0
        assert np.all(np.diff(sel) > 0)
        if k0 == 0:
            continue
        d = np.concatenate([ternary.distance(w[p.base:p.base + p.n], tau[j]) for j, p in enumerate(reg)])
        mask = np.zeros(n, bool)
        mask[sel] = True
        assert d[mask].max() == xi0
        assert np.all(d[~mask] >= xi0)
        # the brute-force definition: the k0 smallest (d, i) pairs
        brute = sorted(range(n), key=lambda i: (float(d[i]), i))[:k0]
        assert np.array_equal(np.sort(brute), sel)


def test_ties_broken_towards_lower_index():
    reg = _reg([(4, 16)])
    w = np.full(64, 0.05, np.float32)          # every distance equal
    sel, xi0, k0, _ = termezo.initial_mask(w, reg, 10 / 64)
    assert k0 == 10 and np.array_equal(sel, np.arange(10))


def test_selection_is_global_across_projections():
    reg = _reg([(16, 16), (16, 16)])
    rng = np.random.default_rng(2)
    a = (rng.standard_normal(256) * 0.02).astype(np.float32)
    tau_a = ternary.threshold(ternary.absmean(a))
    # second projection: every weight sits far from its boundary (|w| = gamma)
    b = np.where(rng.random(256) < 0.5, 1.0, -1.0).astype(np.float32) * np.float32(0.04)
    w = np.concatenate([a, b])
    sel, xi0, k0, tau = termezo.initial_mask(w, reg, 0.25)
    assert tau[0] == tau_a
    assert k0 == 128 and np.all(sel < 256)      # all from the first projection


def test_rho_bounds():
    reg = _reg([(4, 16)])
    w = np.zeros(64, np.float32)
    with pytest.raises(ValueError):
        termezo.initial_mask(w, reg, 0.0)
    with pytest.raises(ValueError):
        termezo.initial_mask(w, reg, 1.5)
    sel, _, k0, _ = termezo.initial_mask(w, reg, 1.0)
    assert k0 == 64 and sel.size == 64


def test_shrink_nesting_over_many_steps():
    reg = _reg([(64, 64), (32, 64)])
    n = sum(p.n for p in reg)
    rng = np.random.default_rng(3)
    w = (rng.standard_normal(n) * 0.02).astype(np.float32)
    active, xi0, k0, _ = termezo.initial_mask(w, reg, 0.05)
    sizes = [active.size]
    for t in range(40):
        w[active] += (rng.standard_normal(active.size) * 3e-5).astype(np.float32)
        new, tau = termezo.shrink(w, reg, active, xi0)
        assert np.all(np.isin(new, active))
        d = np.concatenate([ternary.distance(w[p.base:p.base + p.n], tau[j]) for j, p in enumerate(reg)])
        assert np.all(d[new] <= xi0)
        assert np.all(d[np.setdiff1d(active, new)] > xi0)
        active = new
        sizes.append(active.size)
    assert all(a >= b for a, b in zip(sizes, sizes[1:]))
    assert sizes[-1] < sizes[0] <= k0


def test_step_keeps_frozen_weights_and_codes():
    """Frozen latents never move, and their dense requantisation at every
    perturbed tau equals the code they froze with."""
    reg = _reg([(32, 64), (64, 32)])
    n = sum(p.n for p in reg)
    rng = np.random.default_rng(4)
    w0 = (rng.standard_normal(n) * 0.02).astype(np.float32)
    st = termezo.build(w0, reg, 0.02)
    target = rng.standard_normal(n)

    def loss(codes, sw):
        flat = np.concatenate([c.reshape(-1) for c in codes]).astype(np.float64)
        return float(np.mean((flat - np.sign(target)) ** 2))

    prev = st.active
    for t in range(20):
        w_before = st.w.copy()
        rec = termezo.step(st, loss, 1000 + t, 1e-3, 1e-3)
        frozen = np.setdiff1d(np.arange(n), st.active)
        assert np.array_equal(st.w[frozen], w_before[frozen])
        never = np.setdiff1d(np.arange(n), termezo.build(w0, reg, 0.02).active)
        assert np.array_equal(st.w[never], w0[never])
        assert rec["frozen_mismatch"] == 0
        assert rec["n_jumps"] == 0
        assert rec["k"] == st.active.size <= prev.size
        prev = st.active


def test_per_tensor_mask_cardinality_and_order_within_each_projection():
    """Per-tensor variant of Eq. 4: projection l keeps floor(rho_0 n_l) of its
    own smallest (d, i); within it every kept distance <= xi_0^l <= every
    dropped one, ties to the lower index; one projection is the global rule."""
    cfg = synth.TINY
    reg = termezo.registry(cfg)
    w = synth.latents(cfg).numpy()
    rho = 0.013
    sel, xi, k0, tau = termezo.initial_mask_per_tensor(w, reg, rho)
    d = termezo.all_distances(w, reg, tau)
    assert xi.shape == (len(reg),) and np.all(np.diff(sel) > 0)
    total = 0
    for j, p in enumerate(reg):
        inside = sel[(sel >= p.base) & (sel < p.base + p.n)]
        assert inside.size == math.floor(rho * p.n)
        total += inside.size
        dp = d[p.base:p.base + p.n]
        mask = np.zeros(p.n, bool)
        mask[inside - p.base] = True
        assert dp[mask].max() == xi[j] and np.all(dp[~mask] >= xi[j])
        ties = np.flatnonzero(dp == xi[j])
        assert np.all(np.flatnonzero(mask & (dp == xi[j])) == ties[:np.count_nonzero(mask & (dp == xi[j]))])
    assert total == k0
    one = termezo.single_registry(688, 256)
    w1 = w[:688 * 256]
    a = termezo.initial_mask(w1, one, rho)
    b = termezo.initial_mask_per_tensor(w1, one, rho)
    assert np.array_equal(a[0], b[0]) and a[1] == b[1][0] and a[2] == b[2]


def test_per_tensor_shrink_uses_each_projections_xi():
    """Eq. 5 with the per-tensor xi_0^l: a weight is kept iff its distance is
    within its own projection's xi_0^l; the sets nest."""
    cfg = synth.TINY
    reg = termezo.registry(cfg)
    w = synth.latents(cfg).numpy()
    state = termezo.build(w, reg, 0.02, per_tensor=True)
    rng = np.random.default_rng(3)
    w2 = (w + rng.standard_normal(w.size).astype(np.float32) * np.float32(2e-4)).astype(np.float32)
    kept, tau = termezo.shrink(w2, reg, state.active, state.xi0)
    d = termezo.all_distances(w2, reg, tau)
    tj = termezo._tensor_of(reg, state.active)
    expect = state.active[d[state.active] <= state.xi0[tj]]
    assert np.array_equal(kept, expect) and kept.size < state.active.size
    assert np.all(np.isin(kept, state.active))
