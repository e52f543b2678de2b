"""Seeded synthetic inputs shaped like the paper's fine-tuning workloads.

This module only draws random numbers and names workload shapes; it holds
none of TerMeZO's arithmetic (no quantizer, mask, perturbation or forward
math).  Both the CUDA path and the CPU oracle consume what it returns, so
that every comparison runs on identical inputs.

Workloads (the paper fine-tunes BitNet-b1.58-2B-4T and Falcon-E models on
GLUE/SuperGLUE with batch 16-32 and on GSM8K / MagiCoder SFT with batch 16,
context 512 and 2048-token truncation, Sec. 5 and App. G).  No dataset is
available here, so uniform random token ids stand in for the text and
random-init latents N(0, 0.02) stand in for the pretrained weights.

Seeds: latents 0, token ids 1, targets 2, embeddings 3, LM head 4,
BitLinear-op activations 5; TerMeZO step t uses perturbation seed 1000 + t.
"""
from __future__ import annotations

from dataclasses import dataclass, replace

import numpy as np
import torch

SEED_LATENTS = 0
SEED_TOKENS = 1
SEED_TARGETS = 2
SEED_EMBED = 3
SEED_HEAD = 4
SEED_ACTS = 5
LATENT_STD = 0.02


def step_seed(t: int) -> int:
    """Perturbation seed s_t of TerMeZO iteration t (K = 1)."""
    return 1000 + int(t)


@dataclass(frozen=True)
class ModelConfig:
    """Shape of a BitNet decoder and of one minibatch.

    loss_mode 0: cross-entropy of the last position over ``n_labels`` label
    tokens (ids vocab-n_labels .. vocab-1), the GLUE-style classification
    loss.  loss_mode 1: token-level cross-entropy over the full vocabulary at
    every position, the SFT loss.
    """

    name: str
    layers: int
    hidden: int
    heads: int
    kv_heads: int
    ffn: int
    vocab: int
    seq: int
    batch: int
    loss_mode: int
    n_labels: int

    @property
    def head_dim(self) -> int:
        return self.hidden // self.heads

    @property
    def tokens(self) -> int:
        return self.batch * self.seq

    @property
    def d_lat(self) -> int:
        """Number of ternary latent weights (all q,k,v,o,gate,up,down)."""
        D, F, hd = self.hidden, self.ffn, self.head_dim
        per_layer = (2 * self.heads * hd * D + 2 * self.kv_heads * hd * D
                     + 3 * F * D)
        return self.layers * per_layer

    def with_batch(self, batch: int) -> "ModelConfig":
        return replace(self, batch=batch)


# The four model-shaped workloads (the BitLinear-op workload is described by
# BITLINEAR_OP below).
TINY = ModelConfig("tiny-2L-d256", layers=2, hidden=256, heads=4, kv_heads=4,
                   ffn=688, vocab=1024, seq=64, batch=4, loss_mode=0,
                   n_labels=2)
BITNET_07B = ModelConfig("bitnet-0.7B-shaped", layers=24, hidden=1536,
                         heads=16, kv_heads=16, ffn=4096, vocab=32000,
                         seq=256, batch=16, loss_mode=0, n_labels=2)
BITNET_2B = ModelConfig("bitnet-b1.58-2B-shaped", layers=30, hidden=2560,
                        heads=20, kv_heads=5, ffn=6912, vocab=128256,
                        seq=512, batch=16, loss_mode=0, n_labels=4)
BITNET_2B_LONG = ModelConfig("bitnet-b1.58-2B-shaped-seq2048", layers=30,
                             hidden=2560, heads=20, kv_heads=5, ffn=6912,
                             vocab=128256, seq=2048, batch=4, loss_mode=1,
                             n_labels=0)

WORKLOADS = {c.name: c for c in (TINY, BITNET_07B, BITNET_2B, BITNET_2B_LONG)}

# BitLinear op alone: M tokens x K features of activations, N x K latents.
BITLINEAR_OP = dict(M=2048, K=2560, N=6912, densities=(0.001, 0.01, 0.05))


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def latents(cfg: ModelConfig, device="cpu", seed: int = SEED_LATENTS,
            std: float = LATENT_STD) -> torch.Tensor:
    """Dense fp32 latents w_0 ~ N(0, std^2), in the global index order."""
    n = cfg.d_lat
    out = torch.empty(n, dtype=torch.float32, device=device)
    g = _gen(seed, device)
    chunk = 1 << 28
    for s in range(0, n, chunk):
        e = min(n, s + chunk)
        out[s:e].normal_(0.0, std, generator=g)
    return out


def theta(cfg: ModelConfig, device="cpu"):
    """Full-precision parameters: embeddings fp32 [V, D] ~ N(0, 0.02^2),
    RMSNorm gains fp32 [2L+1, D] = 1, LM head bf16 [V, D] ~ N(0, 0.02^2)."""
    V, D, L = cfg.vocab, cfg.hidden, cfg.layers
    embed = torch.empty(V, D, dtype=torch.float32, device=device)
    embed.normal_(0.0, LATENT_STD, generator=_gen(SEED_EMBED, device))
    gains = torch.ones(2 * L + 1, D, dtype=torch.float32, device=device)
    head = torch.empty(V, D, dtype=torch.float32, device=device)
    head.normal_(0.0, LATENT_STD, generator=_gen(SEED_HEAD, device))
    return embed, gains, head.to(torch.bfloat16)


def batch(cfg: ModelConfig, device="cpu", step: int = 0):
    """Token ids int32 [B, S] uniform in [0, V); targets int32: class ids
    [B] uniform in [0, n_labels) (loss_mode 0) or token ids [B, S] uniform
    in [0, V) (loss_mode 1).  ``step`` offsets the seeds for new batches."""
    B, S, V = cfg.batch, cfg.seq, cfg.vocab
    tok = torch.randint(0, V, (B, S), generator=_gen(SEED_TOKENS + 7919 * step, device),
                        device=device, dtype=torch.int64).to(torch.int32)
    gt = _gen(SEED_TARGETS + 7919 * step, device)
    if cfg.loss_mode == 0:
        tgt = torch.randint(0, cfg.n_labels, (B,), generator=gt, device=device,
                            dtype=torch.int64).to(torch.int32)
    else:
        tgt = torch.randint(0, V, (B, S), generator=gt, device=device,
                            dtype=torch.int64).to(torch.int32)
    return tok, tgt


def op_activations(M: int, K: int, device="cpu", seed: int = SEED_ACTS):
    """BitLinear-op activations: bf16 [M, K] ~ N(0, 1)."""
    x = torch.empty(M, K, dtype=torch.float32, device=device)
    x.normal_(0.0, 1.0, generator=_gen(seed, device))
    return x.to(torch.bfloat16)


def op_latents(N: int, K: int, device="cpu", seed: int = SEED_LATENTS):
    """BitLinear-op latent weight: fp32 [N, K] ~ N(0, 0.02^2)."""
    w = torch.empty(N, K, dtype=torch.float32, device=device)
    w.normal_(0.0, LATENT_STD, generator=_gen(seed, device))
    return w


def numpy_rng(seed: int) -> np.random.Generator:
    return np.random.default_rng(seed)
