"""Layer-by-layer parity of the BitNet forward (Sec. 3; the minibatch loss of
Eqs. 6-7) through termezo_forward_trace: the GPU's own intermediates of a
layer are fed to the oracle's pieces of that layer, so every check compares
one operation on identical inputs, with no error carried in from earlier
layers.  Per layer:

* int8 activation codes of RMSNorm(x) (attention and MLP inputs): bit-exact
  except codes whose float32 value x * (127 / a) lies within a few ulp of a
  rounding boundary (x + 1/2), which two valid orders of the mean-square sum
  may round either way; those are counted and recorded.  deq = a / 127 within
  one ulp.
* codes of the attention output and of the MLP hidden (plain absmax
  quantisation of the GPU's own float32 values): bit-exact, deq bit-exact.
* BitLinear outputs from the GPU's codes: RoPE'd bf16 Q and K, bf16 V, the
  residual stream after the o and down projections, and relu(gate)^2 * up:
  bit-exact (exact int32 accumulators, the same float32 operations).
* attention on the GPU's Q, K, V: the attention op tolerance (median |err|
  < 1e-5, 99th percentile of the per-row relative L1 error < 2e-4).
* the loss from the GPU's residual stream after the last layer: 1e-5
  relative.

Shapes: the tiny decoder (both loss modes, every layer), a head-dim-96
decoder (the unfused RoPE path), the 0.7B-shaped model (every layer) and
the 2B- and 2B-long-shaped models (first, middle, last layer), on sampled
sequences.  Codes are the GPU's packed store (bit-exact against the oracle in
the mask and step tests) with s_w = 2 tau."""
import dataclasses

import numpy as np
import pytest
import torch

from oracle import termezo as otz
from paper_2609_33548_gb300 import synth
from paper_2609_33548_gb300 import termezo as tz

import layerwise as lw
from helpers import record

pytestmark = pytest.mark.gpu

DENSITY = 0.01
TINY_SFT = dataclasses.replace(synth.TINY, name="tiny-2L-d256-sft", vocab=1000, loss_mode=1, n_labels=0)
HD96 = dataclasses.replace(synth.TINY, name="hd96", hidden=384, heads=4, kv_heads=4, ffn=1024, seq=128, batch=2)

# name -> (config, layers checked, sequences checked)
CASES = {
    "tiny": (synth.TINY, None, [0, 3]),
    "tiny-sft": (TINY_SFT, None, [1]),
    "hd96": (HD96, None, [0, 1]),
    "0.7b": (synth.BITNET_07B, None, [0, 5]),
    "2b": (synth.BITNET_2B, [0, 14, 29], [0, 9]),
    "2b-long": (synth.BITNET_2B_LONG, [0, 29], [2]),
}


def _run(name):
    cfg, layers, seqs = CASES[name]
    w = synth.latents(cfg)
    emb, gains, head = synth.theta(cfg)
    tok, tgt = synth.batch(cfg)
    ctx = tz.Context(tz.make_cfg(cfg), DENSITY)
    dev = [t.cuda() for t in (w, emb, gains, head, tok, tgt)]
    ctx.termezo_load_params(dev[0], dev[1], dev[2], dev[3])
    ctx.termezo_build_mask(DENSITY)
    del w, dev[0]
    reg = otz.registry(cfg)
    st = ctx.termezo_export_state(packed=True)
    sw = (np.float32(2.0) * st["tau_cur"]).astype(np.float32)   # s_w = gamma + delta = 2 tau exactly
    layers = list(range(cfg.layers)) if layers is None else layers
    S = cfg.seq
    rows = np.concatenate([np.arange(b * S, (b + 1) * S) for b in seqs])
    gains_np, head_np = gains.numpy(), head.float().numpy()
    stats = {}
    prev = None
    for l in layers:
        _, per, tr = ctx.termezo_forward_trace(dev[3], dev[4], l)
        t = {n: v.cpu().numpy() for n, v in tr.items()}
        del tr
        if prev is not None and prev[0] == l - 1:     # the forward is deterministic: layers chain bit for bit
            np.testing.assert_array_equal(t["x_in"][rows].view(np.uint32), prev[1].view(np.uint32))
        x_out = lw.check_layer(cfg, l, t, seqs, lw.layer_codes(st["packed"], reg, l), sw[7 * l:7 * l + 7],
                               gains_np, stats, name)
        prev = (l, x_out)
    _, per, tr = ctx.termezo_forward_trace(dev[3], dev[4], cfg.layers)
    stats["head_rel_err"] = lw.check_head(cfg, tr["x_in"].cpu().numpy(), per, seqs, gains_np, head_np, tgt.numpy())
    record("layerwise", workload=name, layers=layers, sequences=seqs, **stats)


@pytest.mark.parametrize("name", list(CASES))
def test_layerwise_forward_parity(name):
    _run(name)
