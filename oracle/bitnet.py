"""BitNet forward and minibatch loss (Sec. 3, Eqs. 6-7) -- oracle.

TEST INFRASTRUCTURE ONLY (see the package header).

The paper states that BitNet ternarises every linear projection of the
transformer blocks (q, k, v, o and all MLP linears) with 8-bit activations,
keeping embeddings, normalisation layers and the LM head in full precision
(Sec. 3, first paragraph), and that the loss is the minibatch average of
the per-example loss (Eq. 7).  It prints no further architecture detail, so
the following reading of a BitNet-b1.58 decoder is used (parity of these
details is unpinned by the paper; each building block is pinned against a
library routine or brute force in tests/test_oracle_bitnet.py):

* embedding lookup, fp32;
* per layer: x += o(Attn(RoPE(q(n1(x))), RoPE(k(n1(x))), v(n1(x))));
             x += down(relu(gate(n2(x)))^2 * up(n2(x)));
  n1, n2 are RMSNorm (eps 1e-5, fp32 gain); no bias anywhere;
* final RMSNorm, then the LM head in bf16;
* BitLinear(x) with ternary codes C (N x K) and weight scale s_w: per row
  a = max(max_k |x_k|, 1e-5), s = fl32(127 / a),
  q_k = clamp(rint(fl32(x_k * s)), -128, 127)  (the int8 code is decided in
  float32, as in the kernel), acc = q C^T as an exact integer,
  y = acc * (a / 127) * s_w;
* RoPE base 10000, rotate-half pairing (j, j + hd/2);
* causal softmax attention with grouped KV heads (head h reads KV head
  h // (H / KV)), scores scaled by 1/sqrt(hd): Q, K, V are rounded to bf16,
  P = exp(S - max_j S) is rounded to bf16, O = (P V) / sum_j P;
* loss mode 0: cross-entropy of the last position over the label tokens
  vocab-C .. vocab-1 (logits = bf16(h) . W_head[label]); loss mode 1:
  token-level cross-entropy over the full vocabulary at every position;
* precision: every value that is stored between kernels and feeds a
  quantizer (the residual stream, RMSNorm output, BitLinear outputs, RoPE,
  attention scores / probabilities / output, the MLP hidden) is computed in
  float32, the kernels' precision, with plain numpy float32 operations in
  the order the definition writes them (reductions in numpy's own order):
  an int8 or bf16 code is decided on a float32 value on both sides.  The
  LM-head logits of the last position and every cross-entropy are float64.
"""
from __future__ import annotations

import numpy as np

RMS_EPS = 1e-5
ACT_EPS = np.float32(1e-5)
ROPE_BASE = 10000.0


def bf16_round(x) -> np.ndarray:
    """Round float32 values to bfloat16 (nearest, ties to even), as float32."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    r = ((u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))) >> np.uint64(16)) << np.uint64(16)
    return (r & np.uint64(0xFFFFFFFF)).astype(np.uint32).view(np.float32)


F32 = np.float32


def rmsnorm(x: np.ndarray, gain: np.ndarray) -> np.ndarray:
    """x * r * g with r = 1 / sqrt(mean(x^2) + 1e-5), float32."""
    x = np.asarray(x, dtype=F32)
    ms = (np.sum(x * x, axis=-1, keepdims=True, dtype=F32) / F32(x.shape[-1])).astype(F32)
    r = (F32(1.0) / np.sqrt(ms + F32(RMS_EPS))).astype(F32)
    return ((x * r).astype(F32) * np.asarray(gain, dtype=F32)).astype(F32)


def act_quant(x: np.ndarray):
    """Per-row absmax int8 quantisation; returns (q int64, a float32)."""
    x = np.asarray(x, dtype=np.float32)
    a = np.maximum(np.max(np.abs(x), axis=-1), ACT_EPS).astype(np.float32)
    s = (np.float32(127.0) / a).astype(np.float32)
    q = np.rint((x * s[:, None]).astype(np.float32))
    return np.clip(q, -128, 127).astype(np.int64), a


def int_matmul(q: np.ndarray, codes: np.ndarray) -> np.ndarray:
    """Exact integer acc[m, n] = sum_k q[m, k] * codes[n, k] for int8 codes q
    (|q| <= 128) and ternary codes, returned as int64.  Every product is an
    integer of magnitude <= 128 and every partial sum of any subset of them
    at most 128 K in magnitude; for 128 K < 2**24 all of these are exact in
    float32, so float32 BLAS returns the exact sums in any summation order.
    Larger K use float64 (exact below 2**53)."""
    K = q.shape[-1]
    dt = np.float32 if 128 * K < (1 << 24) else np.float64
    acc = q.astype(dt) @ codes.astype(dt).T
    return np.rint(acc).astype(np.int64)


def bitlinear_codes(q: np.ndarray, dq: np.ndarray, codes: np.ndarray, s_w) -> np.ndarray:
    """y = (acc * dq) * s_w in float32 for int8 activation codes q [M, K]
    with per-row dq = fl32(a / 127) (acc is an exact integer)."""
    acc = int_matmul(q, codes).astype(F32)          # exact: |acc| < 2^24
    return ((acc * np.asarray(dq, dtype=F32)[:, None]).astype(F32) * F32(s_w)).astype(F32)


def bitlinear(x: np.ndarray, codes: np.ndarray, s_w) -> np.ndarray:
    """y = (acc * (a / 127)) * s_w in float32 (acc is an exact integer)."""
    q, a = act_quant(x)
    return bitlinear_codes(q, (a / F32(127.0)).astype(F32), codes, s_w)


def gated_hidden(g: np.ndarray, u: np.ndarray) -> np.ndarray:
    """The squared-ReLU gated MLP hidden relu(g)^2 * u, float32."""
    g = np.maximum(np.asarray(g, dtype=F32), F32(0.0))
    return ((g * g).astype(F32) * np.asarray(u, dtype=F32)).astype(F32)


def rope(x: np.ndarray, hd: int) -> np.ndarray:
    """x: [S, nh, hd] fp32 at positions 0..S-1 -> rotated fp32.  The angles
    pos * 10000^(-2j/hd) and their cos / sin are float64, rounded to float32;
    the rotation (x1 c - x2 s, x2 c + x1 s) is float32."""
    S = x.shape[0]
    half = hd // 2
    inv = ROPE_BASE ** (-(2.0 * np.arange(half)) / hd)
    ang = np.arange(S, dtype=np.float64)[:, None] * inv[None, :]
    c = np.cos(ang).astype(F32)[:, None, :]
    s = np.sin(ang).astype(F32)[:, None, :]
    x1 = np.asarray(x[..., :half], dtype=F32)
    x2 = np.asarray(x[..., half:], dtype=F32)
    return np.concatenate([((x1 * c).astype(F32) - (x2 * s).astype(F32)).astype(F32),
                           ((x2 * c).astype(F32) + (x1 * s).astype(F32)).astype(F32)], axis=-1)


def attention(q: np.ndarray, k: np.ndarray, v: np.ndarray) -> np.ndarray:
    """Causal GQA attention for one sequence.
    q: [S, H, hd], k, v: [S, KV, hd] (fp32) -> [S, H*hd] fp32."""
    S, H, hd = q.shape
    KV = k.shape[1]
    qb, kb, vb = (bf16_round(t) for t in (q, k, v))
    scale = F32(1.0) / np.sqrt(F32(hd))
    causal = np.tril(np.ones((S, S), dtype=bool))
    out = np.empty((S, H, hd), dtype=F32)
    for h in range(H):
        j = h // (H // KV)
        s = ((qb[:, h, :] @ kb[:, j, :].T).astype(F32) * scale).astype(F32)
        s = np.where(causal, s, F32(-np.inf))
        p = np.exp((s - s.max(axis=1, keepdims=True)).astype(F32)).astype(F32)
        pb = bf16_round(p)
        l = np.sum(pb, axis=1, keepdims=True, dtype=F32)
        out[:, h, :] = ((pb @ vb[:, j, :]).astype(F32) / l).astype(F32)
    return out.reshape(S, H * hd)


def cross_entropy(logits: np.ndarray, target: np.ndarray) -> np.ndarray:
    """Per-row -log softmax(logits)[target], float64."""
    z = logits.astype(np.float64)
    m = z.max(axis=-1, keepdims=True)
    lse = m[:, 0] + np.log(np.exp(z - m).sum(axis=-1))
    return lse - z[np.arange(z.shape[0]), target]


def sequence_loss(cfg, codes, s_w, embed, gains, head, tokens, target) -> float:
    """Loss of one sequence.  codes: per-tensor int8 [N, K] arrays in the
    global order (q, k, v, o, gate, up, down per layer); s_w: per-tensor
    float32 weight scales; gains: [2L+1, D]; head: bf16 values as float32
    [V, D]; tokens: [S]; target: class id (mode 0) or [S] token ids."""
    D, H, KV = cfg.hidden, cfg.heads, cfg.kv_heads
    hd = D // H
    S = tokens.shape[0]
    x = embed[np.asarray(tokens, dtype=np.int64)].astype(np.float32)
    for l in range(cfg.layers):
        t = 7 * l
        cq, ck, cv, co, cg, cu, cd = codes[t:t + 7]
        sq, sk, sv, so, sg, su, sd = s_w[t:t + 7]
        h = rmsnorm(x, gains[2 * l])
        q = bitlinear(h, cq, sq).reshape(S, H, hd)
        k = bitlinear(h, ck, sk).reshape(S, KV, hd)
        v = bitlinear(h, cv, sv).reshape(S, KV, hd)
        a = attention(rope(q, hd), rope(k, hd), v)
        x = (x + bitlinear(a, co, so)).astype(np.float32)
        h = rmsnorm(x, gains[2 * l + 1])
        hid = gated_hidden(bitlinear(h, cg, sg), bitlinear(h, cu, su))
        x = (x + bitlinear(hid, cd, sd)).astype(np.float32)
    return head_loss(cfg, x, gains, head, target)


def head_loss(cfg, x, gains, head, target) -> float:
    """Loss of one sequence from the residual stream x [S, D] after the last
    layer: final RMSNorm, the LM head on bf16(h), cross-entropy (mode 0:
    last position over the label tokens; mode 1: every position over the
    vocabulary, averaged)."""
    S = x.shape[0]
    h = bf16_round(rmsnorm(x, gains[2 * cfg.layers])).astype(np.float64)
    W = np.asarray(head, dtype=np.float64)
    if cfg.loss_mode == 0:
        C = cfg.n_labels
        logits = h[S - 1:S] @ W[cfg.vocab - C:].T
        return float(cross_entropy(logits, np.array([int(target)]))[0])
    logits = (h.astype(F32) @ W.astype(F32).T).astype(F32)   # tensor-core logits: bf16 x bf16, fp32 sums
    return float(cross_entropy(logits, np.asarray(target, dtype=np.int64)).mean())


def batch_loss(cfg, codes, s_w, embed, gains, head, tokens, targets, rows=None):
    """Per-sequence losses (float64) for the rows asked for (default: all)
    and the minibatch mean of Eq. 7 over those rows."""
    tokens = np.asarray(tokens)
    targets = np.asarray(targets)
    rows = range(tokens.shape[0]) if rows is None else rows
    per = np.array([sequence_loss(cfg, codes, s_w, embed, gains, head,
                                  tokens[b], targets[b]) for b in rows])
    return per, float(per.mean())
