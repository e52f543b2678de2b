"""The C ABI library loads without a GPU and exports every function that
include/termezo.h declares; host-side argument checks need no device."""
import ctypes
import os
import re

import pytest

from paper_2609_33548_gb300 import build, termezo
from paper_2609_33548_gb300 import synth

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "termezo.h")


def declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(termezo_\w+)\s*\(", text)))


def test_header_lists_the_binding_exports():
    assert declared() == sorted(termezo.EXPORTS)


def test_library_builds_loads_and_exports_all_symbols():
    lib = termezo.load()
    assert os.path.exists(build.LIB)
    for name in declared():
        assert hasattr(lib, name), name


def test_workspace_bytes_and_validation_on_host():
    cfg = termezo.make_cfg(synth.TINY)
    n = termezo.termezo_workspace_bytes(cfg, 0.01)
    assert n > synth.TINY.d_lat // 4          # holds at least the packed store
    with pytest.raises(termezo.TermezoError):
        termezo.termezo_workspace_bytes(cfg, 0.0)
    with pytest.raises(termezo.TermezoError):
        termezo.termezo_workspace_bytes(cfg, 1.5)
    bad = termezo.make_cfg(synth.TINY)
    bad.heads = 3                              # hidden not divisible by heads
    with pytest.raises(termezo.TermezoError):
        termezo.termezo_workspace_bytes(bad, 0.01)
    bad = termezo.make_cfg(synth.TINY)
    bad.seq = 100                              # attention tiles of 64 positions
    with pytest.raises(termezo.TermezoError):
        termezo.termezo_workspace_bytes(bad, 0.01)
    op = termezo.op_cfg(6912, 2560, 2048)
    assert termezo.termezo_workspace_bytes(op, 0.05) > 6912 * 2560 // 4
    assert termezo.load().termezo_strerror(-3).decode().startswith("workspace")


def test_null_context_is_rejected_without_a_device():
    lib = termezo.load()
    assert lib.termezo_build_mask(None, 0.01, None, None) == termezo.EINVAL
    assert lib.termezo_step(None, 1, 1e-3, 1e-6, 0.01, None, None, None, None, None) == termezo.EINVAL
    assert lib.termezo_create(None, 0.01, None, 0, None, None) == termezo.EINVAL


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    """The binding has no host fallback: without the built library it raises
    rather than computing anything."""
    monkeypatch.setattr(termezo, "_LIB", None)
    monkeypatch.setattr(termezo, "library_path", lambda: str(tmp_path / "libtermezo.so"))
    with pytest.raises(OSError):
        termezo.load(build_if_missing=False)
