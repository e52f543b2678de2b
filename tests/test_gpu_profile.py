"""Kernel timing through the C ABI: every n-th launch of each kind is timed,
every launch is counted, and the timed subset carries positive times and the
algorithmic work of exactly the launches it timed."""
import pytest
import torch

from paper_2609_33548_gb300 import synth
from paper_2609_33548_gb300 import termezo as tz

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("stride", [1, 3])
def test_sampled_profile_counts(stride):
    cfg = synth.TINY
    w = synth.latents(cfg)
    emb, gains, head = synth.theta(cfg)
    tok, tgt = synth.batch(cfg)
    ctx = tz.Context(tz.make_cfg(cfg), 0.01)
    dev = [t.cuda() for t in (w, emb, gains, head, tok, tgt)]
    ctx.termezo_load_params(dev[0], dev[1], dev[2], dev[3])
    ctx.termezo_build_mask(0.01)
    ctx.termezo_forward_loss(dev[4], dev[5])
    ctx.termezo_profile(stride)
    for _ in range(2):
        ctx.termezo_forward_loss(dev[4], dev[5])
    p = ctx.termezo_profile(0, read=True)
    torch.cuda.synchronize()
    # a forward launches the q,k,v / o / gate,up / down GEMMs and one
    # attention per layer (the classification head is not a GEMM)
    n_gemm, n_attn = 2 * 4 * cfg.layers, 2 * cfg.layers
    assert p["gemm_seen"] == n_gemm and p["attn_seen"] == n_attn
    assert p["gemm_launches"] == -(-n_gemm // stride)
    assert p["attn_launches"] == -(-n_attn // stride)
    assert p["gemm_ms"] > 0 and p["attn_ms"] > 0
    # the timed GEMMs' work: the sampled launches walk the four shapes in turn
    hq, hkv, D, F, T = cfg.heads * cfg.head_dim, cfg.kv_heads * cfg.head_dim, cfg.hidden, cfg.ffn, cfg.tokens
    per_layer = [2.0 * T * (hq + 2 * hkv) * D, 2.0 * T * D * hq, 2.0 * T * (2 * F) * D, 2.0 * T * D * F]
    expect = sum(per_layer[i % 4] for i in range(0, n_gemm, stride))
    assert p["gemm_flops"] == pytest.approx(expect, rel=1e-12)
