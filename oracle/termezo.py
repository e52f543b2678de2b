"""TerMeZO mask selection and masked two-sided SPSA step -- oracle.

TEST INFRASTRUCTURE ONLY (see the package header).

Dense restatement of Algorithm 1 (App. C) with K = 1 perturbation, acting on
the latent weights w only (theta held fixed):

* ``registry``      -- the global order of the ternary linear projections:
  layer 0..L-1, within a layer q, k, v, o, gate, up, down, each a row-major
  [N_out, K_in] matrix.  w is their concatenation.
* ``initial_mask``  -- Eq. 4 and the first two lines of Algorithm 1: tau_0
  per projection, distances of all weights of all projections, xi_0 the
  lower rho_0-quantile of these distances (global, across layers), S_0 the
  weights with d <= xi_0.  Reading: k0 = floor(rho_0 * d) weights are kept
  exactly, ties at xi_0 broken towards the lower global index, so that
  |S_0| = k0.
* ``shrink``        -- Eq. 5: tau_t recomputed on w_t, S_t keeps the members of
  S_{t-1} with d <= xi_0 (xi_0 fixed).
* ``masked_spsa``   -- the inner loop of Algorithm 1 for any objective F:
  w <- w + eps m.z; F+; w <- w - 2 eps m.z; F-; w <- w + eps m.z (restore);
  g = (F+ - F-) / (2 eps) (Eq. 1 projected onto z); z re-drawn from the seed;
  w <- w - lr g (m.z).  All latent arithmetic is float32 (the stored
  precision of the latents), with e = fl32(eps z) and c = fl32(lr g).
* ``step``          -- one TerMeZO iteration on a BitNet objective: shrink
  (t >= 1), masked SPSA with the dense requantisation of every projection
  (tau recomputed from the perturbed latents, Eq. 2) before each forward,
  and the counters of Eq. 11 (k_t, codes that change between the two
  evaluations) plus the invariant that frozen weights keep their code.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

from . import bitnet, philox, ternary


@dataclass(frozen=True)
class Proj:
    layer: int
    name: str
    N: int
    K: int
    base: int

    @property
    def n(self) -> int:
        return self.N * self.K


def registry(cfg):
    D, F = cfg.hidden, cfg.ffn
    hd = D // cfg.heads
    Hq, Hkv = cfg.heads * hd, cfg.kv_heads * hd
    shapes = [("q", Hq, D), ("k", Hkv, D), ("v", Hkv, D), ("o", D, Hq),
              ("gate", F, D), ("up", F, D), ("down", D, F)]
    out, base = [], 0
    for l in range(cfg.layers):
        for name, N, K in shapes:
            out.append(Proj(l, name, N, K, base))
            base += N * K
    return out


def single_registry(N: int, K: int):
    """Registry of one projection (the BitLinear-op workload)."""
    return [Proj(0, "w", N, K, 0)]


def views(w: np.ndarray, reg):
    return [w[p.base:p.base + p.n] for p in reg]


def thresholds(w: np.ndarray, reg):
    """Per projection (gamma, tau, s_w) on the dense latents w."""
    gam = [ternary.absmean(v) for v in views(w, reg)]
    return (np.array(gam, dtype=np.float32),
            np.array([ternary.threshold(g) for g in gam], dtype=np.float32),
            np.array([ternary.weight_scale(g) for g in gam], dtype=np.float32))


def all_distances(w: np.ndarray, reg, tau) -> np.ndarray:
    return np.concatenate([ternary.distance(v, tau[j]) for j, v in enumerate(views(w, reg))])


def requantize(w: np.ndarray, reg):
    """Dense codes of every projection at its own tau (Eq. 2)."""
    _, tau, sw = thresholds(w, reg)
    codes = np.concatenate([ternary.quantize(v, tau[j]) for j, v in enumerate(views(w, reg))])
    return codes, tau, sw


def keep_count(rho0: float, d: int) -> int:
    if not (0.0 < rho0 <= 1.0):
        raise ValueError("rho_0 must lie in (0, 1]")
    return int(math.floor(float(rho0) * float(d)))


def select_smallest(d: np.ndarray, k0: int):
    """The k0 smallest (d_i, i) pairs: xi = the k0-th smallest distance;
    every i with d_i < xi, then the lowest indices with d_i == xi.
    Returns (sorted indices, xi)."""
    if k0 == 0:
        return np.zeros(0, dtype=np.int64), np.float32(0.0)
    xi = np.float32(np.partition(d, k0 - 1)[k0 - 1])
    below = np.flatnonzero(d < xi)
    ties = np.flatnonzero(d == xi)[:k0 - below.size]
    return np.sort(np.concatenate([below, ties])).astype(np.int64), xi


def initial_mask(w: np.ndarray, reg, rho0: float):
    """Returns (S_0 as sorted int64 global indices, xi_0 float32, k0, tau_0)."""
    _, tau, _ = thresholds(w, reg)
    d = all_distances(w, reg, tau)
    k0 = keep_count(rho0, d.size)
    sel, xi0 = select_smallest(d, k0)
    return sel, xi0, k0, tau


def initial_mask_per_tensor(w: np.ndarray, reg, rho0: float):
    """The per-tensor variant of Eq. 4: every projection l keeps its own
    floor(rho_0 n_l) smallest (d_i, i) pairs (ties to the lower index), and
    xi_0^l is that projection's quantile.  Returns (S_0 sorted, xi_0 [P]
    float32, k0 = sum of the k_l, tau_0)."""
    _, tau, _ = thresholds(w, reg)
    d = all_distances(w, reg, tau)
    sels, xis = [], []
    for p in reg:
        sel, xi = select_smallest(d[p.base:p.base + p.n], keep_count(rho0, p.n))
        sels.append(sel + p.base)
        xis.append(xi)
    sel = np.concatenate(sels).astype(np.int64) if sels else np.zeros(0, np.int64)
    return sel, np.array(xis, dtype=np.float32), int(sel.size), tau


def shrink(w: np.ndarray, reg, active: np.ndarray, xi0):
    """Eq. 5: members of S_{t-1} whose distance at tau_t is <= xi_0 (a
    scalar, or one xi_0^l per projection for the per-tensor mask)."""
    _, tau, _ = thresholds(w, reg)
    d = all_distances(w, reg, tau)
    xi = np.asarray(xi0, dtype=np.float32)
    thr = xi[_tensor_of(reg, active)] if xi.ndim else xi
    keep = d[active] <= thr
    return active[keep], tau


def masked_spsa(w: np.ndarray, active: np.ndarray, z: np.ndarray, eps, lr, objective):
    """One K = 1 pass of Algorithm 1's inner loops for objective(w) -> float.

    Returns (w_next, F+, F-, g, w_plus, w_minus, w_restored)."""
    eps = np.float32(eps)
    e = (eps * z.astype(np.float32)).astype(np.float32)
    w_plus = w.copy()
    w_plus[active] = (w[active] + e).astype(np.float32)
    f_plus = float(objective(w_plus))
    w_minus = w_plus.copy()
    w_minus[active] = (w_plus[active] - (np.float32(2.0) * e)).astype(np.float32)
    f_minus = float(objective(w_minus))
    w_rest = w_minus.copy()
    w_rest[active] = (w_minus[active] + e).astype(np.float32)
    g = (f_plus - f_minus) / (2.0 * float(eps))
    c = np.float32(float(np.float32(lr)) * g)
    w_next = w_rest.copy()
    w_next[active] = (w_rest[active] - (c * z.astype(np.float32)).astype(np.float32)).astype(np.float32)
    return w_next, f_plus, f_minus, g, w_plus, w_minus, w_rest


def masked_spsa_k(w: np.ndarray, active: np.ndarray, zs, eps, lr, objective):
    """Algorithm 1's two inner loops with K = len(zs) directions.

    Loop 1, for each direction k in order: w+ = w + e_k, F+; w- = w+ - 2 e_k,
    F-; restore w = w- + e_k (the next direction starts from this restored
    w); g_k = (F+ - F-) / (2 eps).  Loop 2, for each k in order with z_k
    drawn again: w = w - (lr / K) g_k z_k, the coefficient (lr / K) g_k
    formed in float64 and rounded to float32, every latent operation in
    float32.  With K = 1 this is ``masked_spsa``.

    Returns (w_next, [F+], [F-], [g], [w_restored after direction k])."""
    eps = np.float32(eps)
    K = len(zs)
    w = w.copy()
    fps, fms, gs, rests = [], [], [], []
    for z in zs:
        e = (eps * np.asarray(z, dtype=np.float32)).astype(np.float32)
        w_plus = w.copy()
        w_plus[active] = (w[active] + e).astype(np.float32)
        fp = float(objective(w_plus))
        w_minus = w_plus.copy()
        w_minus[active] = (w_plus[active] - (np.float32(2.0) * e)).astype(np.float32)
        fm = float(objective(w_minus))
        w = w_minus.copy()
        w[active] = (w_minus[active] + e).astype(np.float32)
        fps.append(fp)
        fms.append(fm)
        gs.append((fp - fm) / (2.0 * float(eps)))
        rests.append(w[active].copy())
    lr_k = float(np.float32(lr)) / K
    for z, g in zip(zs, gs):
        c = np.float32(lr_k * g)
        w[active] = (w[active] - (c * np.asarray(z, dtype=np.float32)).astype(np.float32)).astype(np.float32)
    return w, fps, fms, gs, rests


def _stored(x, bf16: bool) -> np.ndarray:
    """x rounded to a part's stored precision: float32, then bfloat16 for a
    bf16 part (round to nearest even)."""
    x = np.asarray(x, dtype=np.float32)
    return bitnet.bf16_round(x) if bf16 else x


def joint_spsa_k(w: np.ndarray, active: np.ndarray, theta, bf16, zs_w, zs_t, eps, lr, objective):
    """Algorithm 1's two inner loops over the masked latents w[active] and
    the full-precision parameters theta together (both perturbed with the
    seed of each direction).

    theta: list of float32 arrays (embeddings, norm gains, LM head); bf16[i]
    marks a part stored in bfloat16.  zs_t[k]: z of theta for direction k,
    the parts concatenated in order.  Every assignment of Algorithm 1 is
    rounded to the stored precision of what it assigns (float32; bfloat16
    after the float32 operation for a bf16 part).  objective(w, theta) ->
    float.  Returns (w, theta, [F+], [F-], [g])."""
    eps = np.float32(eps)
    K = len(zs_w)
    w = w.copy()
    th = [np.asarray(t, dtype=np.float32).copy() for t in theta]
    offs = np.cumsum([0] + [t.size for t in th])

    def split(z):
        return [np.asarray(z[offs[i]:offs[i + 1]], dtype=np.float32).reshape(th[i].shape) for i in range(len(th))]

    fps, fms, gs = [], [], []
    for zw, zt in zip(zs_w, zs_t):
        ew = (eps * np.asarray(zw, dtype=np.float32)).astype(np.float32)
        et = [(eps * z).astype(np.float32) for z in split(zt)]
        w[active] = (w[active] + ew).astype(np.float32)
        th = [_stored(t + e, b) for t, e, b in zip(th, et, bf16)]
        fp = float(objective(w, th))
        w[active] = (w[active] - np.float32(2.0) * ew).astype(np.float32)
        th = [_stored(t - np.float32(2.0) * e, b) for t, e, b in zip(th, et, bf16)]
        fm = float(objective(w, th))
        w[active] = (w[active] + ew).astype(np.float32)
        th = [_stored(t + e, b) for t, e, b in zip(th, et, bf16)]
        fps.append(fp)
        fms.append(fm)
        gs.append((fp - fm) / (2.0 * float(eps)))
    lr_k = float(np.float32(lr)) / K
    for zw, zt, g in zip(zs_w, zs_t, gs):
        c = np.float32(lr_k * g)
        w[active] = (w[active] - (c * np.asarray(zw, dtype=np.float32)).astype(np.float32)).astype(np.float32)
        th = [_stored(t - (c * z).astype(np.float32), b) for t, z, b in zip(th, split(zt), bf16)]
    return w, th, fps, fms, gs


def theta_normals(seed: int, d: int, p: int) -> np.ndarray:
    """z of the full-precision parameters for one direction: the Philox
    stream of the seed at global indices d .. d + p - 1 (after the d
    latents), so that it never shares a value with the latents' z."""
    return philox.normal(seed, np.arange(d, d + p, dtype=np.uint64))


@dataclass
class State:
    """Dense oracle state of a TerMeZO run."""
    w: np.ndarray                 # dense fp32 latents w_t
    reg: list
    active: np.ndarray            # S_t, sorted global indices
    xi0: np.float32
    k0: int
    frozen_code: np.ndarray       # code each weight had when it froze (int8)
    t: int = 0
    log: list = field(default_factory=list)


def build(w0: np.ndarray, reg, rho0: float, per_tensor: bool = False) -> State:
    """Oracle state after the initial mask: the global quantile of Eq. 4, or
    its per-tensor variant (xi_0 then holds one value per projection)."""
    active, xi0, k0, tau0 = (initial_mask_per_tensor if per_tensor else initial_mask)(w0, reg, rho0)
    codes0 = np.concatenate([ternary.quantize(v, tau0[j]) for j, v in enumerate(views(w0, reg))])
    return State(w=w0.astype(np.float32).copy(), reg=reg, active=active, xi0=xi0,
                 k0=k0, frozen_code=codes0)


def near_threshold(w_act: np.ndarray, tau_act: np.ndarray, sw_act: np.ndarray) -> np.ndarray:
    """Active latents within 1e-5 * s_w of +-tau (codes excluded from
    bit-exact comparison)."""
    dist = np.abs(np.abs(w_act.astype(np.float64)) - tau_act.astype(np.float64))
    return dist < 1e-5 * sw_act.astype(np.float64)


def _tensor_of(reg, idx):
    bases = np.array([p.base for p in reg], dtype=np.int64)
    return np.searchsorted(bases, idx, side="right") - 1


def step(state: State, loss_fn, seed: int, eps, lr):
    """One TerMeZO iteration (Algorithm 1, K = 1) on loss_fn(codes, s_w) ->
    float, where codes are the dense per-projection int8 arrays."""
    reg = state.reg
    if state.t >= 1:
        kept, tau_t = shrink(state.w, reg, state.active, state.xi0)
        dropped = np.setdiff1d(state.active, kept)
        if dropped.size:
            tj = _tensor_of(reg, dropped)
            state.frozen_code[dropped] = ternary.quantize(state.w[dropped], tau_t[tj])
        state.active = kept
    active = state.active
    z = philox.normal(seed, active) if active.size else np.zeros(0, np.float32)
    passes = {}

    def objective(wp):
        codes, tau, sw = requantize(wp, reg)
        frozen = np.ones(wp.size, dtype=bool)
        frozen[active] = False
        mism = int(np.count_nonzero(codes[frozen] != state.frozen_code[frozen]))
        split = [codes[p.base:p.base + p.n].reshape(p.N, p.K) for p in reg]
        key = "plus" if "plus" not in passes else "minus"
        tj = _tensor_of(reg, active)
        passes[key] = dict(codes=codes, tau=tau, sw=sw, frozen_mismatch=mism,
                           near=near_threshold(wp[active], tau[tj], sw[tj]))
        return loss_fn(split, sw)

    w_next, fp, fm, g, w_plus, w_minus, w_rest = masked_spsa(state.w, active, z, eps, lr, objective)
    cp = passes["plus"]["codes"][active].astype(np.int64)
    cm = passes["minus"]["codes"][active].astype(np.int64)
    rec = dict(t=state.t, seed=seed, loss_plus=fp, loss_minus=fm, g=g, k=int(active.size),
               n_flipped=int(np.count_nonzero(cp != cm)),
               n_jumps=int(np.count_nonzero(np.abs(cp - cm) == 2)),
               frozen_mismatch=passes["plus"]["frozen_mismatch"] + passes["minus"]["frozen_mismatch"],
               tau_plus=passes["plus"]["tau"], tau_minus=passes["minus"]["tau"],
               codes_minus=passes["minus"]["codes"],
               near_plus=passes["plus"]["near"], near_minus=passes["minus"]["near"],
               w_restored=w_rest[active].copy())
    state.w = w_next
    state.t += 1
    state.log.append(rec)
    return rec


def step_k(state: State, loss_fn, seeds, eps, lr):
    """One TerMeZO iteration of Algorithm 1 with K = len(seeds) directions:
    the mask shrinks once (Eq. 5), then ``masked_spsa_k`` with z_k drawn
    from seeds[k] at the active indices.  Returns per-direction losses,
    g and counters (codes compared between the + and - pass of each
    direction)."""
    reg = state.reg
    if state.t >= 1:
        kept, tau_t = shrink(state.w, reg, state.active, state.xi0)
        dropped = np.setdiff1d(state.active, kept)
        if dropped.size:
            tj = _tensor_of(reg, dropped)
            state.frozen_code[dropped] = ternary.quantize(state.w[dropped], tau_t[tj])
        state.active = kept
    active = state.active
    zs = [philox.normal(s, active) if active.size else np.zeros(0, np.float32) for s in seeds]
    passes = []

    def objective(wp):
        codes, tau, sw = requantize(wp, reg)
        frozen = np.ones(wp.size, dtype=bool)
        frozen[active] = False
        mism = int(np.count_nonzero(codes[frozen] != state.frozen_code[frozen]))
        split = [codes[p.base:p.base + p.n].reshape(p.N, p.K) for p in reg]
        passes.append(dict(codes=codes[active].astype(np.int64), tau=tau, sw=sw, frozen_mismatch=mism))
        return loss_fn(split, sw)

    w_next, fps, fms, gs, rests = masked_spsa_k(state.w, active, zs, eps, lr, objective)
    flips = sum(int(np.count_nonzero(passes[2 * k]["codes"] != passes[2 * k + 1]["codes"])) for k in range(len(seeds)))
    jumps = sum(int(np.count_nonzero(np.abs(passes[2 * k]["codes"] - passes[2 * k + 1]["codes"]) == 2))
                for k in range(len(seeds)))
    rec = dict(t=state.t, seeds=list(seeds), loss_plus=fps, loss_minus=fms, g=gs, k=int(active.size),
               n_flipped=flips, n_jumps=jumps, frozen_mismatch=sum(p["frozen_mismatch"] for p in passes),
               tau_plus=[passes[2 * k]["tau"] for k in range(len(seeds))],
               tau_minus=[passes[2 * k + 1]["tau"] for k in range(len(seeds))], w_restored=rests)
    state.w = w_next
    state.t += 1
    state.log.append(rec)
    return rec


def step_joint(state: State, theta, loss_fn, seeds, eps, lr):
    """One iteration of Algorithm 1 as written: K = len(seeds) directions
    over the masked latents and theta = [embeddings fp32, norm gains fp32,
    LM head bf16] together.  loss_fn(codes, s_w, theta) -> float.  Returns
    the record and the new theta."""
    reg = state.reg
    if state.t >= 1:
        kept, tau_t = shrink(state.w, reg, state.active, state.xi0)
        dropped = np.setdiff1d(state.active, kept)
        if dropped.size:
            tj = _tensor_of(reg, dropped)
            state.frozen_code[dropped] = ternary.quantize(state.w[dropped], tau_t[tj])
        state.active = kept
    active = state.active
    d = state.w.size
    p = sum(np.asarray(t).size for t in theta)
    zs_w = [philox.normal(s, active) if active.size else np.zeros(0, np.float32) for s in seeds]
    zs_t = [theta_normals(s, d, p) for s in seeds]

    def objective(wp, th):
        codes, tau, sw = requantize(wp, reg)
        split = [codes[q.base:q.base + q.n].reshape(q.N, q.K) for q in reg]
        return loss_fn(split, sw, th)

    w_next, th_next, fps, fms, gs = joint_spsa_k(state.w, active, theta, [False, False, True], zs_w, zs_t, eps,
                                                 lr, objective)
    rec = dict(t=state.t, seeds=list(seeds), loss_plus=fps, loss_minus=fms, g=gs, k=int(active.size))
    state.w = w_next
    state.t += 1
    state.log.append(rec)
    return rec, th_next


def bitnet_theta_loss_fn(cfg, tokens, targets, rows=None):
    """loss_fn for ``step_joint``: minibatch loss of Eq. 7 with theta =
    [embeddings, norm gains, LM head] passed per call."""
    def fn(codes, sw, th):
        per, mean = bitnet.batch_loss(cfg, codes, sw, th[0], th[1], th[2], tokens, targets, rows)
        fn.per_sequence.append(per)
        return mean

    fn.per_sequence = []
    return fn


def bitnet_loss_fn(cfg, embed, gains, head, tokens, targets, rows=None):
    """loss_fn for ``step``: minibatch loss of Eq. 7 of the BitNet forward."""
    embed = np.asarray(embed, dtype=np.float32)
    gains = np.asarray(gains, dtype=np.float32)
    head = np.asarray(head, dtype=np.float32)

    def fn(codes, sw):
        per, mean = bitnet.batch_loss(cfg, codes, sw, embed, gains, head, tokens, targets, rows)
        fn.per_sequence.append(per)
        return mean

    fn.per_sequence = []
    return fn
