"""Forward-loss parity of small decoders chosen to exercise each kernel path
the larger workloads use: several 64-key attention blocks (S > 64), head
dims 64 / 96 / 128, grouped KV heads, and GEMMs whose persistent CTAs walk
several output tiles (T >= 128 * 152 / tiles-per-row) in the store,
residual-add and fused gate/up modes.  Calls go through the C ABI."""
import dataclasses

import numpy as np
import pytest
import torch

from oracle import bitnet, rounding, termezo as otz
from paper_2609_33548_gb300 import synth
from paper_2609_33548_gb300 import termezo as tz

from helpers import record

pytestmark = pytest.mark.gpu

T = synth.TINY
MATRIX = {
    "seq256": dataclasses.replace(T, name="seq256", seq=256, batch=2),
    "many-tiles": dataclasses.replace(T, name="many-tiles", seq=64, batch=80),
    "hd96": dataclasses.replace(T, name="hd96", hidden=384, heads=4, kv_heads=4, ffn=1024, seq=128, batch=2),
    "hd128-gqa": dataclasses.replace(T, name="hd128-gqa", hidden=512, heads=4, kv_heads=2, ffn=1376, seq=192,
                                     batch=2),
    "gqa-long-sft": dataclasses.replace(T, name="gqa-long-sft", hidden=256, heads=4, kv_heads=1, seq=512, batch=1,
                                        vocab=3000, loss_mode=1, n_labels=0),
    # fused-RoPE QKV GEMM of 160 tiles: the 8 of the last wave run as 16
    # units of one 128-column head each
    "narrow-tail": dataclasses.replace(T, name="narrow-tail", hidden=512, heads=4, kv_heads=2, ffn=1376, seq=128,
                                       batch=40),
}


CACHED = ("hd128-gqa", "narrow-tail", "gqa-long-sft")


@pytest.mark.parametrize("name,cache", [(n, False) for n in sorted(MATRIX)] + [(n, True) for n in CACHED])
def test_forward_loss_matrix(name, cache):
    cfg = MATRIX[name]
    w = synth.latents(cfg)
    emb, gains, head = synth.theta(cfg)
    tok, tgt = synth.batch(cfg)
    ctx = tz.Context(tz.make_cfg(cfg, cache), 0.01)
    dev = [t.cuda() for t in (w, emb, gains, head, tok, tgt)]
    ctx.termezo_load_params(dev[0], dev[1], dev[2], dev[3])
    ctx.termezo_build_mask(0.01)
    loss, per = ctx.termezo_forward_loss(dev[4], dev[5])
    reg = otz.registry(cfg)
    codes, tau, sw = otz.requantize(w.numpy(), reg)
    split = [codes[p.base:p.base + p.n].reshape(p.N, p.K) for p in reg]
    rows = list(range(min(cfg.batch, 4)))
    th = (emb.numpy(), gains.numpy(), head.float().numpy(), tok.numpy(), tgt.numpy())
    per_o, _ = bitnet.batch_loss(cfg, split, sw, *th, rows=rows)
    ens = rounding.loss_ensemble(cfg, (split, sw), th, n=8, rows=rows)
    for b in rows:
        # 1e-3, or no further from the oracle than its valid fp32 re-roundings,
        # or within 5 standard deviations of them (rounding.agrees)
        record("forward_matrix", workload=name, cache=cache, sequence=b, **rounding.summary(per[b], per_o[b], ens[:, b]))
        assert rounding.agrees(per[b], per_o[b], ens[:, b]), (name, b, per[b], per_o[b], ens[:, b])
