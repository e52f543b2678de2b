"""Memory accounting of a context against the memory equation of Sec. 5:
TerMeZO keeps full-precision copies of the rho_0 d active latents only,
2-bit codes (B_Q = 2/8 byte) of all d latents, and a mask
M_mask = min(ceil(d / 8), ceil(rho_0 d ceil(log2 d) / 8)).  The report is
computed on the host from the same carve as the workspace."""
import math

import pytest

from paper_2609_33548_gb300 import synth
from paper_2609_33548_gb300 import termezo as tz

CASES = [(synth.TINY, 0.01), (synth.BITNET_07B, 0.01), (synth.BITNET_2B, 0.01), (synth.BITNET_2B, 0.001),
         (synth.BITNET_2B_LONG, 0.05)]


def _round_up(n, a=256):
    return (n + a - 1) // a * a


@pytest.mark.parametrize("cfg,density", CASES, ids=[f"{c.name}-{d}" for c, d in CASES])
def test_memory_report_parts(cfg, density):
    m = tz.termezo_memory(tz.make_cfg(cfg), density)
    d = cfg.d_lat
    k0 = math.floor(density * d)
    assert m["d"] == d and m["k_cap"] == k0
    # every part is what the layout says, up to the 256-byte alignment of each buffer
    assert d // 4 <= m["packed"] < d // 4 + 256
    assert 2 * 4 * k0 <= m["sparse_index"] < 2 * 4 * k0 + 2 * 256
    assert 2 * 4 * k0 <= m["sparse_latents"] < 2 * 4 * k0 + 2 * 256
    parts = m["packed"] + m["sparse_index"] + m["sparse_latents"] + m["mask_state"] + m["forward"] + m["weight_cache"]
    assert m["weight_cache"] == 0
    assert m["workspace"] == parts + 256 == tz.termezo_workspace_bytes(tz.make_cfg(cfg), density)
    assert m["theta"] == cfg.vocab * cfg.hidden * (4 + 2) + (2 * cfg.layers + 1) * cfg.hidden * 4
    # the paper's two mask options
    assert m["mask_bitmask"] == math.ceil(d / 8)
    assert m["mask_index_list"] == math.ceil(k0 * math.ceil(math.log2(d)) / 8)


def test_latent_storage_against_the_memory_equation():
    """Latent-related bytes of the equation with this library's precisions
    (B = 4: fp32 latents, B_Q = 1/4, the index list at 32 bits) equal the
    build's packed codes plus one buffer of the sparse store; the second
    buffer (written by the order-preserving shrink) is the only addition."""
    cfg, density = synth.BITNET_2B, 0.01
    m = tz.termezo_memory(tz.make_cfg(cfg), density)
    d, k0 = m["d"], m["k_cap"]
    B, BQ = 4, 0.25
    mask32 = math.ceil(k0 * 32 / 8)
    eq = d * B - math.ceil(d * (1 - density) * (B - BQ)) + math.ceil(density * d * BQ) + mask32
    build = m["packed"] + (m["sparse_index"] + m["sparse_latents"]) // 2
    assert abs(build - eq) <= 4 * 256 + 8
    # at 1 % the index list beats the bit mask, as Sec. 5 expects for small rho_0
    assert m["mask_index_list"] < m["mask_bitmask"]


@pytest.mark.parametrize("cfg,density", CASES, ids=[f"{c.name}-{d}" for c, d in CASES])
def test_weight_cache_part(cfg, density):
    """The e4m3 weight cache is one byte per weight, its own part; the two
    expansion buffers it replaces leave the forward part."""
    m0 = tz.termezo_memory(tz.make_cfg(cfg), density)
    m1 = tz.termezo_memory(tz.make_cfg(cfg, weight_cache=True), density)
    d = cfg.d_lat
    assert d <= m1["weight_cache"] < d + 256
    assert m1["forward"] < m0["forward"]
    assert m1["workspace"] - m0["workspace"] == m1["weight_cache"] - (m0["forward"] - m1["forward"])
    for k in ("packed", "sparse_index", "sparse_latents", "mask_state", "theta"):
        assert m1[k] == m0[k]


@pytest.mark.parametrize("cfg,density", CASES, ids=[f"{c.name}-{d}" for c, d in CASES])
def test_z_cache_part(cfg, density):
    """The optional z buffer is one float per active weight of the store's
    capacity, its own part outside the memory equation."""
    m0 = tz.termezo_memory(tz.make_cfg(cfg), density)
    m1 = tz.termezo_memory(tz.make_cfg(cfg, z_cache=True), density)
    k0 = math.floor(density * cfg.d_lat)
    assert m0["z_cache"] == 0
    assert 4 * k0 <= m1["z_cache"] < 4 * k0 + 256
    assert abs((m1["workspace"] - m0["workspace"]) - m1["z_cache"]) <= 256
    for k in ("packed", "sparse_index", "sparse_latents", "forward", "theta", "weight_cache"):
        assert m1[k] == m0[k]
