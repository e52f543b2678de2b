"""Thin ctypes binding of libtermezo.so (declared in include/termezo.h).

Argument marshalling only: every step of the TerMeZO path runs in the
library's CUDA kernels.  Device buffers are torch tensors (their data_ptr
is passed); the workspace is one torch uint8 tensor on the device.  There
is no CPU fallback: loading fails loudly when the library is missing.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np
import torch

from . import build as _build

OK, WMASKFIXED, EINVAL, ESTATE, ENOMEM, ECUDA, ETIMEOUT = 0, 1, -1, -2, -3, -4, -5

# Every function declared in include/termezo.h.
EXPORTS = (
    "termezo_workspace_bytes", "termezo_memory", "termezo_create", "termezo_load_params", "termezo_build_mask",
    "termezo_build_mask_rule", "termezo_forward_loss", "termezo_forward_trace", "termezo_step", "termezo_step_k", "termezo_step_joint", "termezo_shrink", "termezo_requantize", "termezo_update",
    "termezo_bitlinear", "termezo_state_sizes", "termezo_export_state", "termezo_normal",
    "termezo_absmean_noalloc", "termezo_attention", "termezo_profile", "termezo_destroy", "termezo_strerror",
)


class ModelCfg(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in
                ("layers", "hidden", "heads", "kv_heads", "ffn", "vocab", "seq", "batch",
                 "loss_mode", "n_labels", "weight_cache", "z_cache")]


class StepOut(ctypes.Structure):
    _fields_ = [("loss_plus", ctypes.c_double), ("loss_minus", ctypes.c_double),
                ("g", ctypes.c_double), ("k_active", ctypes.c_uint64),
                ("n_flipped", ctypes.c_uint64), ("n_jumps", ctypes.c_uint64),
                ("n_dropped", ctypes.c_uint64), ("n_near_threshold", ctypes.c_uint64)]

    def as_dict(self):
        return {n: getattr(self, n) for n, _ in self._fields_}


class MemoryOut(ctypes.Structure):
    _fields_ = [(n, ctypes.c_uint64) for n in
                ("d", "k_cap", "packed", "sparse_index", "sparse_latents", "mask_state", "forward", "workspace",
                 "theta", "mask_bitmask", "mask_index_list", "weight_cache", "z_cache")]

    def as_dict(self):
        return {n: getattr(self, n) for n, _ in self._fields_}


class ProfileOut(ctypes.Structure):
    _fields_ = [("launches", ctypes.c_uint64), ("gemm_launches", ctypes.c_uint64),
                ("gemm_ms", ctypes.c_double), ("gemm_flops", ctypes.c_double),
                ("attn_launches", ctypes.c_uint64), ("attn_ms", ctypes.c_double),
                ("attn_flops", ctypes.c_double), ("sparse_launches", ctypes.c_uint64),
                ("sparse_ms", ctypes.c_double), ("sparse_bytes", ctypes.c_double),
                ("gemm_seen", ctypes.c_uint64), ("attn_seen", ctypes.c_uint64), ("sparse_seen", ctypes.c_uint64),
                ("pass_launches", ctypes.c_uint64 * 5), ("pass_seen", ctypes.c_uint64 * 5),
                ("pass_ms", ctypes.c_double * 5), ("pass_bytes", ctypes.c_double * 5)]

    def as_dict(self):
        return {n: (list(getattr(self, n)) if n.startswith("pass_") else getattr(self, n)) for n, _ in self._fields_}


# sparse pass kinds of ProfileOut.pass_* (include/termezo.h)
PASS_KINDS = ("pm_sum", "requant", "update", "shrink", "theta")


TRACE_FIELDS = ("x_in", "codes_attn", "deq_attn", "q", "k", "vt", "attn", "codes_o", "deq_o", "x_mid",
                "codes_mlp", "deq_mlp", "hid", "codes_down", "deq_down", "x_out")


class LayerTrace(ctypes.Structure):
    """termezo_layer_trace: device pointers of the buffers to fill (NULL: skip)."""
    _fields_ = [(n, ctypes.c_void_p) for n in TRACE_FIELDS]

MASK_GLOBAL, MASK_PER_TENSOR = 0, 1


class TermezoError(RuntimeError):
    def __init__(self, fn, status, msg):
        super().__init__(f"{fn} failed: {msg} (status {status})")
        self.status = status


_LIB = None


def library_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = True) -> ctypes.CDLL:
    """Loads libtermezo.so (building it with nvcc first if it is absent)."""
    global _LIB
    if _LIB is not None:
        return _LIB
    path = library_path()
    if not os.path.exists(path):
        if not build_if_missing:
            raise OSError(f"libtermezo.so not built: {path}")
        _build.build()
    lib = ctypes.CDLL(path)
    P, I32, U64, F32, F64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_uint64, ctypes.c_float, ctypes.c_double
    sig = {
        "termezo_workspace_bytes": (I32, [ctypes.POINTER(ModelCfg), F64, ctypes.POINTER(ctypes.c_size_t)]),
        "termezo_memory": (I32, [ctypes.POINTER(ModelCfg), F64, ctypes.POINTER(MemoryOut)]),
        "termezo_create": (I32, [ctypes.POINTER(ModelCfg), F64, P, ctypes.c_size_t, P, ctypes.POINTER(P)]),
        "termezo_load_params": (I32, [P, P, P, P, P]),
        "termezo_build_mask": (I32, [P, F64, ctypes.POINTER(U64), ctypes.POINTER(F32)]),
        "termezo_build_mask_rule": (I32, [P, F64, I32, ctypes.POINTER(U64), P]),
        "termezo_forward_loss": (I32, [P, P, P, ctypes.POINTER(F64), P]),
        "termezo_forward_trace": (I32, [P, P, P, I32, ctypes.POINTER(LayerTrace), ctypes.POINTER(F64), P]),
        "termezo_step": (I32, [P, U64, F32, F32, F64, P, P, ctypes.POINTER(StepOut), P, P]),
        "termezo_step_k": (I32, [P, P, I32, F32, F32, F64, P, P, ctypes.POINTER(StepOut), P, P]),
        "termezo_step_joint": (I32, [P, P, I32, F32, F32, F64, P, P, ctypes.POINTER(StepOut), P, P]),
        "termezo_shrink": (I32, [P, ctypes.POINTER(U64)]),
        "termezo_requantize": (I32, [P, U64, F32, I32]),
        "termezo_update": (I32, [P, U64, F32, F32, F64]),
        "termezo_bitlinear": (I32, [P, I32, P, I32, P, P]),
        "termezo_state_sizes": (I32, [P, ctypes.POINTER(U64), ctypes.POINTER(U64), ctypes.POINTER(I32)]),
        "termezo_export_state": (I32, [P, P, P, P, P]),
        "termezo_normal": (I32, [U64, P, U64, P, P]),
        "termezo_absmean_noalloc": (I32, [P, U64, P, P]),
        "termezo_attention": (I32, [P, P, P, I32, I32, I32, I32, I32, P, P]),
        "termezo_profile": (I32, [P, I32, ctypes.POINTER(ProfileOut)]),
        "termezo_destroy": (None, [P]),
        "termezo_strerror": (ctypes.c_char_p, [I32]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    _LIB = lib
    return lib


def _check(fn, status, allow=(OK,)):
    if status not in allow:
        msg = load().termezo_strerror(status).decode()
        raise TermezoError(fn, status, msg)
    return status


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def make_cfg(cfg, weight_cache: bool = False, z_cache: bool = False) -> ModelCfg:
    """ModelCfg from any object with the ModelConfig attribute names;
    weight_cache keeps an e4m3 byte per weight for the forward's GEMMs,
    z_cache a float per active weight for z between the passes of a step."""
    return ModelCfg(cfg.layers, cfg.hidden, cfg.heads, cfg.kv_heads, cfg.ffn, cfg.vocab, cfg.seq,
                    cfg.batch, cfg.loss_mode, cfg.n_labels, 1 if weight_cache else 0, 1 if z_cache else 0)


def op_cfg(N: int, K: int, M: int, z_cache: bool = False) -> ModelCfg:
    """Single-projection context: one [N, K] ternary projection, M rows."""
    return ModelCfg(0, K, 0, 0, N, 0, M, 1, 0, 0, 0, 1 if z_cache else 0)


def termezo_workspace_bytes(cfg: ModelCfg, density: float) -> int:
    n = ctypes.c_size_t(0)
    _check("termezo_workspace_bytes", load().termezo_workspace_bytes(ctypes.byref(cfg), density, ctypes.byref(n)))
    return n.value


def termezo_memory(cfg: ModelCfg, density: float) -> dict:
    """Device bytes of a context by part (host only)."""
    out = MemoryOut()
    _check("termezo_memory", load().termezo_memory(ctypes.byref(cfg), density, ctypes.byref(out)))
    return out.as_dict()


class Context:
    """Owns the device workspace (a torch tensor) and the library context."""

    def __init__(self, cfg: ModelCfg, density: float, device="cuda", stream=None):
        lib = load()
        self.cfg = cfg
        self.density = density
        nbytes = termezo_workspace_bytes(cfg, density)
        self.workspace = torch.empty(nbytes, dtype=torch.uint8, device=device)
        self.stream = stream
        h = ctypes.c_void_p()
        _check("termezo_create", lib.termezo_create(ctypes.byref(cfg), density, _ptr(self.workspace),
                                                    nbytes, _stream(stream), ctypes.byref(h)))
        self.handle = h
        self._keep = []

    def close(self):
        if getattr(self, "handle", None):
            load().termezo_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- the paper's calls ---------------------------------------------------
    def termezo_load_params(self, latents, embed=None, gains=None, head=None):
        self._keep = [latents, embed, gains, head]
        _check("termezo_load_params", load().termezo_load_params(
            self.handle, _ptr(latents), _ptr(embed), _ptr(gains),
            None if head is None else ctypes.c_void_p(head.data_ptr())))

    def termezo_build_mask(self, density: float):
        k0 = ctypes.c_uint64(0)
        xi0 = ctypes.c_float(0)
        _check("termezo_build_mask", load().termezo_build_mask(self.handle, density, ctypes.byref(k0),
                                                               ctypes.byref(xi0)))
        self._keep[0] = None  # the library no longer reads the dense latents
        return k0.value, np.float32(xi0.value)

    def termezo_build_mask_rule(self, density: float, rule: int):
        """Mask rule MASK_GLOBAL (Eq. 4) or MASK_PER_TENSOR; returns (k0,
        xi0: a float32, or an array with one xi_0 per projection)."""
        k0 = ctypes.c_uint64(0)
        n = self.termezo_state_sizes()[2] if rule == MASK_PER_TENSOR else 1
        xi0 = np.zeros(n, dtype=np.float32)
        _check("termezo_build_mask_rule", load().termezo_build_mask_rule(
            self.handle, density, rule, ctypes.byref(k0), xi0.ctypes.data_as(ctypes.c_void_p)))
        self._keep[0] = None
        return k0.value, (xi0 if rule == MASK_PER_TENSOR else xi0[0])

    def termezo_forward_loss(self, tokens, targets):
        loss = ctypes.c_double(0)
        per = np.zeros(self.cfg.batch, dtype=np.float64)
        _check("termezo_forward_loss", load().termezo_forward_loss(
            self.handle, _ptr(tokens), _ptr(targets), ctypes.byref(loss),
            per.ctypes.data_as(ctypes.c_void_p)))
        return loss.value, per

    def termezo_forward_trace(self, tokens, targets, layer: int, fields=TRACE_FIELDS):
        """Forward at the codes now in the packed store; returns (loss,
        per-sequence losses, dict of device tensors with the intermediates
        of `layer` named in `fields`; layer == layers: only x_in, the
        residual stream after the last layer)."""
        c = self.cfg
        T, D, F = c.seq * c.batch, c.hidden, c.ffn
        hd = c.hidden // c.heads
        shapes = dict(x_in=((T, D), torch.float32), codes_attn=((T, D), torch.int8), deq_attn=((T,), torch.float32),
                      q=((c.batch, c.heads, c.seq, hd), torch.int16), k=((c.batch, c.kv_heads, c.seq, hd), torch.int16),
                      vt=((c.batch, c.kv_heads, hd, c.seq), torch.int16), attn=((T, c.heads * hd), torch.float32),
                      codes_o=((T, c.heads * hd), torch.int8), deq_o=((T,), torch.float32),
                      x_mid=((T, D), torch.float32), codes_mlp=((T, D), torch.int8), deq_mlp=((T,), torch.float32),
                      hid=((T, F), torch.float32), codes_down=((T, F), torch.int8), deq_down=((T,), torch.float32),
                      x_out=((T, D), torch.float32))
        if layer == c.layers:
            fields = ("x_in",)
        bufs = {n: torch.empty(shapes[n][0], dtype=shapes[n][1], device=self.workspace.device) for n in fields}
        tr = LayerTrace(**{n: t.data_ptr() for n, t in bufs.items()})
        loss = ctypes.c_double(0)
        per = np.zeros(c.batch, dtype=np.float64)
        _check("termezo_forward_trace", load().termezo_forward_trace(
            self.handle, _ptr(tokens), _ptr(targets), layer, ctypes.byref(tr), ctypes.byref(loss),
            per.ctypes.data_as(ctypes.c_void_p)))
        return loss.value, per, bufs

    def termezo_step(self, seed: int, eps: float, lr: float, density: float, tokens, targets):
        out = StepOut()
        pp = np.zeros(self.cfg.batch, dtype=np.float64)
        pm = np.zeros(self.cfg.batch, dtype=np.float64)
        st = load().termezo_step(self.handle, seed, eps, lr, density, _ptr(tokens), _ptr(targets),
                                 ctypes.byref(out), pp.ctypes.data_as(ctypes.c_void_p),
                                 pm.ctypes.data_as(ctypes.c_void_p))
        _check("termezo_step", st, allow=(OK, WMASKFIXED))
        d = out.as_dict()
        d["per_seq_plus"], d["per_seq_minus"], d["status"] = pp, pm, st
        return d

    def termezo_step_k(self, seeds, eps: float, lr: float, density: float, tokens, targets, theta=False):
        """Algorithm 1 with K = len(seeds) directions; adds per-direction
        losses [K, 2] (F+, F-) and g [K] to the report.  theta=True also
        perturbs and updates the embeddings, norm gains and LM head in place
        (termezo_step_joint)."""
        K = len(seeds)
        sd = np.asarray(seeds, dtype=np.uint64)
        out = StepOut()
        losses = np.zeros(2 * K, dtype=np.float64)
        g = np.zeros(K, dtype=np.float64)
        fn = "termezo_step_joint" if theta else "termezo_step_k"
        st = getattr(load(), fn)(self.handle, sd.ctypes.data_as(ctypes.c_void_p), K, eps, lr, density,
                                 _ptr(tokens), _ptr(targets), ctypes.byref(out),
                                 losses.ctypes.data_as(ctypes.c_void_p), g.ctypes.data_as(ctypes.c_void_p))
        _check(fn, st, allow=(OK, WMASKFIXED))
        d = out.as_dict()
        d["losses"], d["g_k"], d["status"] = losses.reshape(K, 2), g, st
        return d

    # -- pieces of the step -------------------------------------------------
    def termezo_shrink(self):
        n = ctypes.c_uint64(0)
        _check("termezo_shrink", load().termezo_shrink(self.handle, ctypes.byref(n)))
        return n.value

    def termezo_requantize(self, seed: int, eps: float, sign: int):
        _check("termezo_requantize", load().termezo_requantize(self.handle, seed, eps, sign))

    def termezo_update(self, seed: int, eps: float, lr: float, g: float):
        _check("termezo_update", load().termezo_update(self.handle, seed, eps, lr, g))

    def termezo_bitlinear(self, proj: int, x_bf16, acc=None, y=None):
        M = x_bf16.shape[0]
        _check("termezo_bitlinear", load().termezo_bitlinear(self.handle, proj, _ptr(x_bf16), M, _ptr(acc),
                                                             _ptr(y)))

    def termezo_profile(self, enable: int, read: bool = False):
        out = ProfileOut()
        _check("termezo_profile", load().termezo_profile(self.handle, enable,
                                                         ctypes.byref(out) if read else None))
        return out.as_dict() if read else None

    def termezo_state_sizes(self):
        d, k, p = ctypes.c_uint64(0), ctypes.c_uint64(0), ctypes.c_int32(0)
        _check("termezo_state_sizes", load().termezo_state_sizes(self.handle, ctypes.byref(d), ctypes.byref(k),
                                                                 ctypes.byref(p)))
        return d.value, k.value, p.value

    def termezo_export_state(self, packed=True):
        d, k, P = self.termezo_state_sizes()
        idx = np.zeros(k, dtype=np.uint32)
        lat = np.zeros(k, dtype=np.float32)
        pk = np.zeros(d // 16, dtype=np.uint32) if packed else None
        tau = np.zeros(3 * P, dtype=np.float32)
        vp = lambda a: None if a is None else a.ctypes.data_as(ctypes.c_void_p)
        _check("termezo_export_state", load().termezo_export_state(self.handle, vp(idx), vp(lat), vp(pk), vp(tau)))
        return dict(idx=idx, latents=lat, packed=pk, tau_cur=tau[:P], tau_plus=tau[P:2 * P],
                    tau_minus=tau[2 * P:])


def termezo_normal(seed: int, idx_u32, z_out, stream=None):
    _check("termezo_normal", load().termezo_normal(seed, _ptr(idx_u32), idx_u32.numel(), _ptr(z_out),
                                                   _stream(stream)))


def termezo_absmean_noalloc(w, out, stream=None):
    """gamma, tau, s_w of the fp32 device tensor w into the 3-float device
    tensor out, without any device allocation (for callers that cannot
    allocate: the library's fixed scratch array is used)."""
    _check("termezo_absmean_noalloc", load().termezo_absmean_noalloc(_ptr(w), w.numel(), _ptr(out),
                                                                     _stream(stream)))


def termezo_attention(q, k, vt, out, stream=None):
    """Causal attention op: q bf16 [B, H, S, hd], k bf16 [B, KV, S, hd],
    vt bf16 [B, KV, hd, S] -> out fp32 [B*S, H*hd]."""
    B, H, S, hd = q.shape
    KV = k.shape[1]
    _check("termezo_attention", load().termezo_attention(_ptr(q), _ptr(k), _ptr(vt), B, S, H, KV, hd, _ptr(out),
                                                         _stream(stream)))
