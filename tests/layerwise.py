"""The per-layer parity checks of the BitNet forward (Sec. 3 block; Eqs.
6-7 evaluate it) used by the layer-wise tests: the GPU's intermediates of one
layer (termezo_forward_trace) are fed to the oracle's pieces of that layer.
Imported by tests only."""
import numpy as np

from oracle import bitnet, ternary

from helpers import ulp_diff

F32 = np.float32


def _bf16_bits_to_f32(t):
    return (t.astype(np.uint16).astype(np.uint32) << 16).view(np.float32)


def _near_boundary(v, tol_ulps=8):
    """float32 values v = x * (127 / a) within tol_ulps ulp of a rounding
    boundary (an odd multiple of 1/2)."""
    v = np.asarray(v, dtype=np.float64)
    dist = np.abs(v - (np.floor(v) + 0.5))
    return dist <= tol_ulps * np.spacing(np.maximum(np.abs(v), 1.0).astype(np.float32)).astype(np.float64)


def _check_norm_codes(x, gain, codes_gpu, deq_gpu, stats, key):
    h = bitnet.rmsnorm(x, gain)
    q, a = bitnet.act_quant(h)
    dq = (a / F32(127.0)).astype(F32)
    # deq = a / 127 scales with r = 1 / sqrt(mean x^2 + eps): two orders of the
    # float32 mean-square sum of D positive terms differ by at most 2 D u
    # relatively (u = 2^-24), r by half of that, plus the roundings of h, a, deq
    D = x.shape[1]
    rel = np.abs(deq_gpu.astype(np.float64) / dq - 1.0)
    assert np.all(rel <= (D + 8) * 2.0 ** -24), (key, rel.max())
    stats[key + "_deq_max_ulp"] = max(stats.get(key + "_deq_max_ulp", 0), int(ulp_diff(deq_gpu, dq).max()))
    # the code's value x * (127 / a) is invariant to r up to roundings, so a
    # code may differ only where that value lies within a few ulp of x + 1/2
    s = (F32(127.0) / a).astype(F32)
    v = (h * s[:, None]).astype(F32)
    bad = codes_gpu.astype(np.int64) != q
    assert np.all(np.abs(codes_gpu.astype(np.int64) - q)[bad] == 1), key
    assert np.all(_near_boundary(v[bad], 16)), (key, int(bad.sum()))
    stats[key + "_near_mismatch"] = stats.get(key + "_near_mismatch", 0) + int(bad.sum())
    stats[key + "_codes"] = stats.get(key + "_codes", 0) + int(q.size)


def _check_plain_codes(x, codes_gpu, deq_gpu, key):
    q, a = bitnet.act_quant(x)
    np.testing.assert_array_equal(codes_gpu.astype(np.int64), q, err_msg=key)
    np.testing.assert_array_equal(deq_gpu.view(np.uint32), (a / F32(127.0)).astype(F32).view(np.uint32),
                                  err_msg=key)


def _check_attention(q, k, v, out_gpu, stats):
    o = bitnet.attention(q, k, v)
    err = np.abs(out_gpu.astype(np.float64) - o)
    rel_row = err.sum(axis=1) / np.maximum(np.abs(o).sum(axis=1), 1e-30)
    assert np.median(err) < 1e-5 and np.percentile(rel_row, 99) < 2e-4, (np.median(err), rel_row.max())
    stats["attn_max_abs_err"] = max(stats.get("attn_max_abs_err", 0.0), float(err.max()))
    stats["attn_p99_row_rel_l1"] = max(stats.get("attn_p99_row_rel_l1", 0.0), float(np.percentile(rel_row, 99)))


def layer_codes(packed, reg, l):
    """Codes [N, K] of the seven projections of layer l from a packed store."""
    out = []
    for j in range(7):
        p = reg[7 * l + j]
        out.append(ternary.unpack_codes(packed[p.base // 16:(p.base + p.n) // 16]).reshape(p.N, p.K))
    return out


def check_layer(cfg, l, t, seqs, codes, sw, gains_np, stats, name):
    """All checks of layer l on the trace t (numpy arrays over every row) for
    the sequences seqs; codes: the layer's seven [N, K] code matrices, sw: the
    seven weight scales.  Returns the expected x_out rows."""
    S, D, H, KV = cfg.seq, cfg.hidden, cfg.heads, cfg.kv_heads
    hd = D // H
    rows = np.concatenate([np.arange(b * S, (b + 1) * S) for b in seqs])
    cq, ck, cv, co, cg, cu, cd = codes
    sq, sk, sv, so, sg, su, sd = sw
    x_in = t["x_in"][rows]
    _check_norm_codes(x_in, gains_np[2 * l], t["codes_attn"][rows], t["deq_attn"][rows], stats, "attn_in")
    ca, da = t["codes_attn"][rows].astype(np.int64), t["deq_attn"][rows]
    for i, b in enumerate(seqs):
        r = slice(i * S, (i + 1) * S)
        qo = bitnet.rope(bitnet.bitlinear_codes(ca[r], da[r], cq, sq).reshape(S, H, hd), hd)
        ko = bitnet.rope(bitnet.bitlinear_codes(ca[r], da[r], ck, sk).reshape(S, KV, hd), hd)
        vo = bitnet.bitlinear_codes(ca[r], da[r], cv, sv).reshape(S, KV, hd)
        qg = _bf16_bits_to_f32(t["q"][b]).transpose(1, 0, 2)        # [S, H, hd]
        kg = _bf16_bits_to_f32(t["k"][b]).transpose(1, 0, 2)
        vg = _bf16_bits_to_f32(t["vt"][b]).transpose(2, 0, 1)       # [KV, hd, S] -> [S, KV, hd]
        for nm, want, got in (("q", qo, qg), ("k", ko, kg), ("v", vo, vg)):
            np.testing.assert_array_equal(got.view(np.uint32), bitnet.bf16_round(want).view(np.uint32),
                                          err_msg=f"{name} layer {l} {nm}")
        _check_attention(qg, kg, vg, t["attn"][rows][r], stats)
    _check_plain_codes(t["attn"][rows], t["codes_o"][rows], t["deq_o"][rows], f"{name} layer {l} o codes")
    x_mid = (x_in + bitnet.bitlinear_codes(t["codes_o"][rows].astype(np.int64), t["deq_o"][rows], co, so)
             ).astype(F32)
    np.testing.assert_array_equal(t["x_mid"][rows].view(np.uint32), x_mid.view(np.uint32),
                                  err_msg=f"{name} layer {l} x_mid")
    _check_norm_codes(x_mid, gains_np[2 * l + 1], t["codes_mlp"][rows], t["deq_mlp"][rows], stats, "mlp_in")
    cm, dm = t["codes_mlp"][rows].astype(np.int64), t["deq_mlp"][rows]
    hid = bitnet.gated_hidden(bitnet.bitlinear_codes(cm, dm, cg, sg), bitnet.bitlinear_codes(cm, dm, cu, su))
    np.testing.assert_array_equal(t["hid"][rows].view(np.uint32), hid.view(np.uint32),
                                  err_msg=f"{name} layer {l} hid")
    _check_plain_codes(hid, t["codes_down"][rows], t["deq_down"][rows], f"{name} layer {l} down codes")
    x_out = (x_mid + bitnet.bitlinear_codes(t["codes_down"][rows].astype(np.int64), t["deq_down"][rows], cd, sd)
             ).astype(F32)
    np.testing.assert_array_equal(t["x_out"][rows].view(np.uint32), x_out.view(np.uint32),
                                  err_msg=f"{name} layer {l} x_out")
    return x_out


def check_head(cfg, x_final, per_gpu, seqs, gains_np, head_np, targets, rel=1e-5):
    """The loss of each sequence from the GPU's residual stream after the
    last layer (x_final [T, D]) against the GPU's own per-sequence loss.
    Returns the largest relative difference."""
    S = cfg.seq
    err = 0.0
    for b in seqs:
        ref = bitnet.head_loss(cfg, x_final[b * S:(b + 1) * S], gains_np, head_np, targets[b])
        err = max(err, abs(per_gpu[b] - ref) / abs(ref))
    assert err <= rel, err
    return err
