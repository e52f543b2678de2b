"""Pins of the oracle's masked two-sided SPSA step (Eq. 1, Algorithm 1,
App. E) against closed forms: the exact two-point quotient of a quadratic,
the expectation identity of the Gaussian-smoothed objective, and the
restore/update arithmetic.  CPU only."""
import math

import numpy as np

from oracle import philox, ternary, termezo


def _quadratic(n, seed=0):
    rng = np.random.default_rng(seed)
    M = rng.standard_normal((n, n))
    A = M @ M.T / n + np.eye(n)
    b = rng.standard_normal(n)
    return A, b, lambda w: 0.5 * w.astype(np.float64) @ A @ w.astype(np.float64) + b @ w.astype(np.float64)


def test_quadratic_two_point_quotient_is_exact():
    n = 64
    A, b, F = _quadratic(n)
    rng = np.random.default_rng(1)
    w = (rng.standard_normal(n) * 0.1).astype(np.float32)
    active = np.sort(rng.choice(n, 20, replace=False)).astype(np.int64)
    z = philox.normal(123, active)
    eps, lr = 1e-3, 1e-2
    w_next, fp, fm, g, w_plus, w_minus, _ = termezo.masked_spsa(w, active, z, eps, lr, F)
    # for a quadratic F(w+) - F(w-) = (w+ - w-)^T (A (w+ + w-)/2 + b) exactly
    dp = w_plus.astype(np.float64) - w_minus.astype(np.float64)
    mid = (w_plus.astype(np.float64) + w_minus.astype(np.float64)) / 2
    g_closed = dp @ (A @ mid + b) / (2 * float(np.float32(eps)))
    assert abs(g - g_closed) <= 1e-9 * max(1.0, abs(g_closed))
    # and it approximates z_S^T grad F(w) (perturbation only on S)
    grad = A @ w.astype(np.float64) + b
    assert abs(g - z.astype(np.float64) @ grad[active]) < 1e-2 * max(1.0, abs(g))
    # untouched coordinates never move
    frozen = np.setdiff1d(np.arange(n), active)
    assert np.array_equal(w_next[frozen], w[frozen])
    assert np.array_equal(w_plus[frozen], w[frozen]) and np.array_equal(w_minus[frozen], w[frozen])


def test_spsa_is_unbiased_for_masked_gradient():
    """E[g z_S] = m . grad F for a quadratic (App. E): mean over many seeds."""
    n = 8
    A, b, F = _quadratic(n, seed=4)
    w = np.linspace(-0.5, 0.5, n).astype(np.float32)
    active = np.array([1, 2, 5, 6], dtype=np.int64)
    N = 6000
    acc = np.zeros(n)
    samples = []
    for s in range(N):
        z = philox.normal(10_000 + s, active)
        _, _, _, g, _, _, _ = termezo.masked_spsa(w, active, z, 1e-2, 0.0, F)
        v = np.zeros(n)
        v[active] = g * z
        samples.append(v)
    samples = np.array(samples)
    mean = samples.mean(axis=0)
    se = samples.std(axis=0) / math.sqrt(N) + 1e-12
    grad = A @ w.astype(np.float64) + b
    expect = np.zeros(n)
    expect[active] = grad[active]
    assert np.all(np.abs(mean - expect) < 5 * se + 1e-9)
    assert np.all(mean[np.setdiff1d(np.arange(n), active)] == 0)


def test_ternary_smoothed_gradient_closed_form():
    """One ternary weight, fixed tau: F(w) = Q(w).  The Gaussian-smoothed
    objective is Phi((w - tau)/eps) - Phi((-tau - w)/eps); its derivative is
    (phi((w - tau)/eps) + phi((w + tau)/eps)) / eps (App. E, Eq. smoothed_grad)."""
    tau = np.float32(0.1)
    eps = 0.05
    w = np.array([0.08], np.float32)
    active = np.array([0], dtype=np.int64)
    F = lambda v: float(ternary.quantize(v, tau)[0])
    N = 20000
    vals = np.empty(N)
    for s in range(N):
        z = philox.normal(s, np.array([s], dtype=np.uint64))   # fresh z per draw
        _, _, _, g, _, _, _ = termezo.masked_spsa(w, active, z, eps, 0.0, F)
        vals[s] = g * float(z[0])
    phi = lambda x: math.exp(-0.5 * x * x) / math.sqrt(2 * math.pi)
    expect = (phi((0.08 - 0.1) / eps) + phi((0.08 + 0.1) / eps)) / eps
    se = vals.std() / math.sqrt(N)
    assert abs(vals.mean() - expect) < 5 * se


def test_restore_and_update_arithmetic():
    rng = np.random.default_rng(11)
    n = 100000
    w = (rng.standard_normal(n) * 0.02).astype(np.float32)
    active = np.arange(0, n, 3, dtype=np.int64)
    z = philox.normal(9, active)
    eps, lr = np.float32(1e-3), np.float32(1e-6)
    F = lambda v: float(np.sum(v.astype(np.float64) ** 3))
    w_next, fp, fm, g, w_plus, w_minus, w_rest = termezo.masked_spsa(w, active, z, eps, lr, F)
    e = (eps * z).astype(np.float32)
    # +eps z, -2 eps z, +eps z restores within a few ulp of |w| + 2|e|
    bound = 1.5 * np.spacing(np.abs(w[active]) + 2 * np.abs(e)).astype(np.float64)
    assert np.all(np.abs(w_rest[active].astype(np.float64) - w[active]) <= bound)
    # exact restore where w + e and w + e - 2e are exact (e a multiple of ulp(w))
    exact = (np.float32(w[active] + e) - e == w[active]) & (np.float32(np.float32(w[active] + e) - 2 * e) + e == w[active])
    assert np.all(w_rest[active][exact] == w[active][exact])
    # update regenerates the same z and moves by fl32(fl32(lr g) z)
    c = np.float32(float(lr) * g)
    assert np.array_equal(w_next[active], (w_rest[active] - (c * z).astype(np.float32)).astype(np.float32))
    assert g == (fp - fm) / (2 * float(eps))


def test_k_directions_reduce_to_one_and_apply_every_term():
    """Algorithm 1 with K directions: K = 1 is the single-direction pass bit
    for bit; for K = 3 each g_k is the exact two-point quotient at the
    restored point of direction k, and the update applies the K terms
    (lr / K) g_k z_k in order."""
    n = 48
    A, b, F = _quadratic(n, seed=3)
    rng = np.random.default_rng(4)
    w = (rng.standard_normal(n) * 0.1).astype(np.float32)
    active = np.sort(rng.choice(n, 16, replace=False)).astype(np.int64)
    eps, lr = 1e-3, 5e-3
    z1 = philox.normal(7, active)
    one = termezo.masked_spsa(w, active, z1, eps, lr, F)
    many = termezo.masked_spsa_k(w, active, [z1], eps, lr, F)
    assert np.array_equal(one[0], many[0]) and one[3] == many[3][0]
    zs = [philox.normal(s, active) for s in (11, 12, 13)]
    w_next, fps, fms, gs, rests = termezo.masked_spsa_k(w, active, zs, eps, lr, F)
    e32 = np.float32(eps)
    start = w.copy()
    for k, z in enumerate(zs):
        e = (e32 * z).astype(np.float32)
        wp = start.copy()
        wp[active] = (start[active] + e).astype(np.float32)
        wm = wp.copy()
        wm[active] = (wp[active] - np.float32(2) * e).astype(np.float32)
        dp = wp.astype(np.float64) - wm.astype(np.float64)
        mid = (wp.astype(np.float64) + wm.astype(np.float64)) / 2
        assert abs(gs[k] - dp @ (A @ mid + b) / (2 * float(e32))) <= 1e-9 * max(1.0, abs(gs[k]))
        start = wm.copy()
        start[active] = (wm[active] + e).astype(np.float32)
        assert np.array_equal(start[active], rests[k])
    expect = start.copy()
    for z, g in zip(zs, gs):
        c = np.float32(float(np.float32(lr)) / 3 * g)
        expect[active] = (expect[active] - (c * z).astype(np.float32)).astype(np.float32)
    assert np.array_equal(w_next, expect)
    frozen = np.setdiff1d(np.arange(n), active)
    assert np.array_equal(w_next[frozen], w[frozen])


def test_k_direction_update_averages_to_the_masked_gradient():
    """E[z z^T] = I: over K directions the update -(lr / K) sum_k g_k z_k
    tends to -lr (m * grad F) (App. E), which pins the 1 / K factor."""
    n = 8
    A, b, F = _quadratic(n, seed=5)
    w = np.linspace(-0.5, 0.5, n).astype(np.float32)
    active = np.array([0, 2, 3, 6], dtype=np.int64)
    K, eps, lr = 4000, 1e-2, 1e-3
    zs = [philox.normal(100 + k, active) for k in range(K)]
    w_next, *_ = termezo.masked_spsa_k(w, active, zs, eps, lr, F)
    step = (w_next.astype(np.float64) - w.astype(np.float64)) / -lr
    grad = A @ w.astype(np.float64) + b
    assert np.allclose(step[active], grad[active], atol=6 * np.abs(grad).max() / math.sqrt(K) + 0.05)
    assert np.all(step[np.setdiff1d(np.arange(n), active)] == 0)


def test_joint_theta_loops_reduce_and_are_exact_two_point_quotients():
    """Algorithm 1 over (w, theta): with no theta it is the latent-only
    loops; on a quadratic over the concatenated vector each g_k is the exact
    two-point quotient of that direction's perturbed pair, and theta's
    entries follow the same fp32 arithmetic as the latents."""
    n_w, n_t = 24, 10
    A, b, F = _quadratic(n_w + n_t, seed=8)
    rng = np.random.default_rng(9)
    w = (rng.standard_normal(n_w) * 0.1).astype(np.float32)
    th = [(rng.standard_normal(n_t) * 0.1).astype(np.float32)]
    active = np.sort(rng.choice(n_w, 9, replace=False)).astype(np.int64)
    eps, lr = 1e-3, 5e-3
    zs_w = [philox.normal(s, active) for s in (21, 22)]
    zs_t = [termezo.theta_normals(s, n_w, n_t) for s in (21, 22)]
    # no theta: the latent-only loops bit for bit
    a = termezo.masked_spsa_k(w, active, zs_w, eps, lr, lambda v: F(np.concatenate([v, th[0]])))
    j = termezo.joint_spsa_k(w, active, [], [], zs_w, [np.zeros(0, np.float32)] * 2, eps, lr,
                             lambda v, t: F(np.concatenate([v, th[0]])))
    assert np.array_equal(a[0], j[0]) and a[3] == j[4]
    # joint: exact quotients on the quadratic
    Fj = lambda v, t: F(np.concatenate([v, t[0]]))
    w1, th1, fps, fms, gs = termezo.joint_spsa_k(w, active, th, [False], zs_w, zs_t, eps, lr, Fj)
    e32 = np.float32(eps)
    cw, ct = w.copy(), th[0].copy()
    for k in range(2):
        ew = (e32 * zs_w[k]).astype(np.float32)
        et = (e32 * zs_t[k]).astype(np.float32)
        wp, tp = cw.copy(), (ct + et).astype(np.float32)
        wp[active] = (cw[active] + ew).astype(np.float32)
        wm, tm = wp.copy(), (tp - np.float32(2) * et).astype(np.float32)
        wm[active] = (wp[active] - np.float32(2) * ew).astype(np.float32)
        xp = np.concatenate([wp, tp]).astype(np.float64)
        xm = np.concatenate([wm, tm]).astype(np.float64)
        g = (xp - xm) @ (A @ ((xp + xm) / 2) + b) / (2 * float(e32))
        assert abs(gs[k] - g) <= 1e-9 * max(1.0, abs(g))
        cw = wm.copy()
        cw[active] = (wm[active] + ew).astype(np.float32)
        ct = (tm + et).astype(np.float32)
    lr_k = float(np.float32(lr)) / 2
    for k in range(2):
        c = np.float32(lr_k * gs[k])
        cw[active] = (cw[active] - (c * zs_w[k]).astype(np.float32)).astype(np.float32)
        ct = (ct - (c * zs_t[k]).astype(np.float32)).astype(np.float32)
    assert np.array_equal(w1, cw) and np.array_equal(th1[0], ct)
    assert np.array_equal(w1[np.setdiff1d(np.arange(n_w), active)], w[np.setdiff1d(np.arange(n_w), active)])


def test_joint_theta_update_averages_to_both_gradient_blocks():
    """Over K directions the joint update tends to -lr (m * grad_w F,
    grad_theta F): theta is perturbed densely, the latents on the mask."""
    n_w, n_t = 6, 3
    A, b, F = _quadratic(n_w + n_t, seed=10)
    w = np.linspace(-0.4, 0.4, n_w).astype(np.float32)
    th = [np.array([0.3, -0.2, 0.1], dtype=np.float32)]
    active = np.array([1, 4], dtype=np.int64)
    K, eps, lr = 4000, 1e-2, 1e-3
    seeds = range(300, 300 + K)
    zs_w = [philox.normal(s, active) for s in seeds]
    zs_t = [termezo.theta_normals(s, n_w, n_t) for s in seeds]
    w1, th1, *_ = termezo.joint_spsa_k(w, active, th, [False], zs_w, zs_t, eps, lr,
                                       lambda v, t: F(np.concatenate([v, t[0]])))
    grad = A @ np.concatenate([w, th[0]]).astype(np.float64) + b
    tol = 6 * np.abs(grad).max() / math.sqrt(K) + 0.05
    step_w = (w1.astype(np.float64) - w) / -lr
    step_t = (th1[0].astype(np.float64) - th[0]) / -lr
    assert np.allclose(step_w[active], grad[active], atol=tol)
    assert np.allclose(step_t, grad[n_w:], atol=tol)
    assert np.all(step_w[np.setdiff1d(np.arange(n_w), active)] == 0)


def test_bf16_theta_part_is_rounded_at_every_assignment():
    """A part stored in bfloat16 (the LM head) is rounded to bfloat16 after
    each float32 operation of Algorithm 1, so its restore need not return
    the starting value; each step is checked by hand."""
    from oracle import bitnet
    th = [bitnet.bf16_round(np.array([0.0213, -0.0117, 0.5], dtype=np.float32))]
    zt = [termezo.theta_normals(77, 4, 3)]
    eps, lr, g = np.float32(1e-3), 1e-3, None
    seen = []
    w1, th1, fps, fms, gs = termezo.joint_spsa_k(np.zeros(4, np.float32), np.zeros(0, np.int64), th, [True],
                                                 [np.zeros(0, np.float32)], zt, eps, lr,
                                                 lambda v, t: (seen.append(t[0].copy()), float(t[0].sum()))[1])
    e = (eps * zt[0]).astype(np.float32)
    tp = bitnet.bf16_round((th[0] + e).astype(np.float32))
    tm = bitnet.bf16_round((tp - np.float32(2) * e).astype(np.float32))
    tr = bitnet.bf16_round((tm + e).astype(np.float32))
    assert np.array_equal(seen[0], tp) and np.array_equal(seen[1], tm)
    c = np.float32(float(np.float32(lr)) * gs[0])
    assert np.array_equal(th1[0], bitnet.bf16_round((tr - (c * zt[0]).astype(np.float32)).astype(np.float32)))
