"""Pins of the oracle's BitNet forward building blocks against brute-force
integer arithmetic, library routines (float64 torch ops) and closed forms.
CPU only."""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import bitnet, termezo
from paper_2609_33548_gb300 import synth


def test_int8_ternary_dot_brute_force():
    rng = np.random.default_rng(0)
    q = rng.integers(-128, 128, size=(5, 48))
    c = rng.integers(-1, 2, size=(7, 48)).astype(np.int8)
    acc = bitnet.int_matmul(q, c)
    for m in range(5):
        for n in range(7):
            assert acc[m, n] == sum(int(q[m, k]) * int(c[n, k]) for k in range(48))
    # extreme magnitudes stay exact
    q = np.full((2, 6912), -128)
    c = np.ones((3, 6912), np.int8)
    assert np.all(bitnet.int_matmul(q, c) == -128 * 6912)
    # large partial sums followed by small terms, random signs: int64 sums
    q = np.concatenate([rng.choice([-127, 127], size=(4, 3456)), rng.integers(-3, 4, size=(4, 3456))], axis=1)
    c = rng.integers(-1, 2, size=(6, 6912)).astype(np.int8)
    c[0] = 1
    want = q.astype(np.int64) @ c.astype(np.int64).T
    np.testing.assert_array_equal(bitnet.int_matmul(q, c), want)
    # beyond K = 2^17 the float64 path is taken
    q = np.full((1, 1 << 17), 127)
    assert bitnet.int_matmul(q, np.ones((1, 1 << 17), np.int8))[0, 0] == 127 << 17


def test_act_quant_properties():
    rng = np.random.default_rng(1)
    x = (rng.standard_normal((64, 300)) * rng.uniform(0.01, 10, (64, 1))).astype(np.float32)
    q, a = bitnet.act_quant(x)
    assert q.min() >= -128 and q.max() <= 127
    np.testing.assert_array_equal(a, np.abs(x).max(axis=1))
    assert np.all(np.abs(q).max(axis=1) == 127)
    err = np.abs(q * (a[:, None].astype(np.float64) / 127) - x)
    assert np.all(err <= a[:, None] / 254 * (1 + 1e-5))
    q0, a0 = bitnet.act_quant(np.zeros((2, 8), np.float32))
    assert np.all(q0 == 0) and np.all(a0 == np.float32(1e-5))


def test_bf16_round_matches_torch():
    rng = np.random.default_rng(2)
    x = (rng.standard_normal(100000) * 10 ** rng.uniform(-8, 8, 100000)).astype(np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).float().numpy()
    np.testing.assert_array_equal(bitnet.bf16_round(x), ref)


def test_rmsnorm_matches_torch():
    rng = np.random.default_rng(3)
    x = rng.standard_normal((16, 256)).astype(np.float32)
    g = rng.uniform(0.5, 1.5, 256).astype(np.float32)
    ref = F.rms_norm(torch.from_numpy(x).double(), (256,), torch.from_numpy(g).double(), eps=1e-5)
    np.testing.assert_allclose(bitnet.rmsnorm(x, g), ref.float().numpy(), rtol=1e-6, atol=1e-7)


def test_gated_hidden_is_squared_relu_times_up():
    """relu(g)^2 u (the MLP's gate): against float64 torch within the two
    float32 roundings, exactly 0 wherever g <= 0, and exact on values whose
    square and product are representable."""
    rng = np.random.default_rng(7)
    g = rng.standard_normal((8, 688)).astype(np.float32)
    u = rng.standard_normal((8, 688)).astype(np.float32)
    h = bitnet.gated_hidden(g, u)
    ref = (F.relu(torch.from_numpy(g).double()) ** 2 * torch.from_numpy(u).double()).numpy()
    assert np.all(h[g <= 0] == 0)
    pos = g > 0
    assert np.all(np.abs(h[pos] - ref[pos]) <= 2.0 ** -23 * np.abs(ref[pos]))
    exact = bitnet.gated_hidden(np.array([0.5, 3.0, -2.0], np.float32), np.array([3.0, -0.25, 5.0], np.float32))
    np.testing.assert_array_equal(exact, np.array([0.75, -2.25, 0.0], np.float32))


def test_rope_is_complex_rotation():
    rng = np.random.default_rng(4)
    S, nh, hd = 33, 3, 16
    x = rng.standard_normal((S, nh, hd)).astype(np.float32)
    y = bitnet.rope(x, hd)
    half = hd // 2
    zc = x[..., :half].astype(np.float64) + 1j * x[..., half:]
    theta = np.arange(S)[:, None] * (10000.0 ** (-np.arange(half) / half))[None, :]
    rot = zc * np.exp(1j * theta)[:, None, :]
    np.testing.assert_allclose(y[..., :half], rot.real, rtol=1e-5, atol=1e-6)
    np.testing.assert_allclose(y[..., half:], rot.imag, rtol=1e-5, atol=1e-6)
    np.testing.assert_allclose(np.linalg.norm(y, axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-5)


def test_attention_matches_sdpa_within_bf16():
    rng = np.random.default_rng(5)
    S, H, KV, hd = 40, 4, 2, 16
    q = rng.standard_normal((S, H, hd)).astype(np.float32)
    k = rng.standard_normal((S, KV, hd)).astype(np.float32)
    v = rng.standard_normal((S, KV, hd)).astype(np.float32)
    out = bitnet.attention(q, k, v).reshape(S, H, hd)
    qt = torch.from_numpy(bitnet.bf16_round(q)).double().permute(1, 0, 2)
    kt = torch.from_numpy(bitnet.bf16_round(k)).double().permute(1, 0, 2).repeat_interleave(H // KV, 0)
    vt = torch.from_numpy(bitnet.bf16_round(v)).double().permute(1, 0, 2).repeat_interleave(H // KV, 0)
    ref = F.scaled_dot_product_attention(qt, kt, vt, is_causal=True).permute(1, 0, 2).numpy()
    np.testing.assert_allclose(out, ref, rtol=0, atol=2e-2)
    assert np.abs(out - ref).mean() < 2e-3
    # the first position attends only to itself
    np.testing.assert_array_equal(out[0], bitnet.bf16_round(v)[0].repeat(H // KV, axis=0))


def test_attention_equal_scores_average_values():
    S, H, hd = 9, 2, 8
    q = np.zeros((S, H, hd), np.float32)
    k = np.ones((S, 1, hd), np.float32)
    v = np.arange(S * hd, dtype=np.float32).reshape(S, 1, hd)
    out = bitnet.attention(q, k, v).reshape(S, H, hd)
    for i in range(S):
        np.testing.assert_allclose(out[i, 0], v[:i + 1, 0].mean(axis=0), rtol=1e-6)


def test_cross_entropy_matches_torch():
    rng = np.random.default_rng(6)
    z = rng.standard_normal((12, 50)) * 3
    t = rng.integers(0, 50, 12)
    ref = F.cross_entropy(torch.from_numpy(z), torch.from_numpy(t), reduction="none").numpy()
    np.testing.assert_allclose(bitnet.cross_entropy(z, t), ref, rtol=1e-12)


def test_random_init_loss_is_near_uniform():
    cfg = synth.TINY
    w = synth.latents(cfg).numpy()
    emb, gains, head = synth.theta(cfg)
    tok, tgt = synth.batch(cfg)
    reg = termezo.registry(cfg)
    codes, tau, sw = termezo.requantize(w, reg)
    split = [codes[p.base:p.base + p.n].reshape(p.N, p.K) for p in reg]
    per, mean = bitnet.batch_loss(cfg, split, sw, emb.numpy(), gains.numpy(), head.float().numpy(),
                                  tok.numpy(), tgt.numpy())
    assert per.shape == (cfg.batch,)
    assert abs(mean - math.log(cfg.n_labels)) < 0.5
    assert reg[-1].base + reg[-1].n == cfg.d_lat == 1581056
