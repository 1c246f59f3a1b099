"""Thin ctypes binding of the C ABI in include/dfs.h (argument marshalling only).

Every function here has the name of the C entry point it calls and does no compute:
pointers are taken from torch tensors (``data_ptr()``), numpy arrays or plain ints, the
stream defaults to torch's current CUDA stream, and a non-zero status raises DfsError
with the library's message.  The library must have been built (``build.build()``);
loading fails loudly otherwise - there is no fallback path.
"""
from __future__ import annotations

import ctypes
import os
from typing import Any, Dict, Optional, Sequence

import numpy as np

from . import build as _build

DFS_OK, DFS_EINVAL, DFS_ENOMEM, DFS_ECUDA, DFS_ETIMEOUT, DFS_EUNSUPPORTED = range(6)
_STATUS = {0: "DFS_OK", 1: "DFS_EINVAL", 2: "DFS_ENOMEM", 3: "DFS_ECUDA", 4: "DFS_ETIMEOUT",
           5: "DFS_EUNSUPPORTED"}

EXPORTED = ("dfs_plan_create", "dfs_block_forward", "dfs_block_forward_layer", "dfs_block_forward_host",
            "dfs_block_forward_host_async", "dfs_block_forward_noalloc",
            "dfs_denoise", "dfs_plan_indices", "dfs_plan_panel", "dfs_plan_union_panel", "dfs_plan_memory",
            "dfs_plan_flops", "dfs_plan_workspace",
            "dfs_plan_sync", "dfs_selftest_wait_timeout", "dfs_plan_profile", "dfs_plan_profile_read", "dfs_gates_from_soft_masks",
            "dfs_model_attach", "dfs_model_forward", "dfs_model_denoise",
            "dfs_plan_destroy", "dfs_last_error")

KERNEL_KINDS = ("modulation", "adaln", "gemm_qkv", "qk_norm_rope", "attention", "gemm_o", "gemm_up",
                "gemm_down", "cross", "other", "gather", "model")

PANELS = {"wqkv": 0, "bqkv": 1, "gq": 2, "gk": 3, "wo": 4, "w_up": 5, "b_up": 6, "w_down": 7,
          "cwq": 8, "cbq": 9, "cwkv": 10, "cbkv": 11, "cgq": 12, "cgk": 13, "cwo": 14}
WORKSPACE = {"xm": 0, "qk": 1, "vt": 2, "attn": 3, "x1": 4, "h": 5, "mod": 6}
UNION_PANELS = {"wqkv": 0, "wo": 1, "w_up": 2, "w_down": 3, "cwq": 4, "cwo": 5}
DFS_ENGINE_COMPACTED, DFS_ENGINE_UNION = 0, 1
ENGINES = {"compacted": DFS_ENGINE_COMPACTED, "union": DFS_ENGINE_UNION}
# dfs_plan_indices kinds
INDEX_KINDS = {"heads": 0, "chunks": 1, "xheads": 2, "union_heads": 3, "union_chunks": 4, "union_xheads": 5,
               "pos_heads": 6, "pos_chunks": 7, "pos_xheads": 8}


class DfsError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__("%s: %s" % (_STATUS.get(status, status), msg))
        self.status = status


class dfs_config(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int) for n in ("dim", "n_heads", "head_dim", "ffn_dim", "ffn_chunk", "n_layers",
                                            "n_steps", "grid_t", "grid_h", "grid_w", "ctx_len", "has_cross")] + \
               [("ln_eps", ctypes.c_float), ("rope_theta", ctypes.c_float), ("qk_norm_mode", ctypes.c_int),
                ("engine", ctypes.c_int)]


LAYER_FIELDS = ("wq", "bq", "wk", "bk", "wv", "bv", "wo", "bo", "gq", "gk", "w_up", "b_up", "w_down", "b_down",
                "e_mod", "cwq", "cbq", "cwk", "cbk", "cwv", "cbv", "cwo", "cbo", "cgq", "cgk", "cln_w", "cln_b")


class dfs_layer_weights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in LAYER_FIELDS]


class dfs_masks(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in ("block_gate", "head_gate", "xhead_gate", "ffn_gate")]


MODEL_FIELDS = ("patch_w", "patch_b", "t_w1", "t_b1", "t_w2", "t_b2", "head_mod", "head_w", "head_b")


class dfs_model_weights(ctypes.Structure):
    _fields_ = [("in_channels", ctypes.c_int), ("freq_dim", ctypes.c_int)] + \
               [(n, ctypes.c_void_p) for n in MODEL_FIELDS]


_lib = None


def lib() -> ctypes.CDLL:
    """Loads libdfs.so (built in-tree); raises if it is missing."""
    global _lib
    if _lib is None:
        path = _build.LIB
        if not os.path.exists(path):
            raise RuntimeError("libdfs.so is not built (%s); run paper_2607_06631_gb300.build.build()" % path)
        L = ctypes.CDLL(path)
        vp, i32, i64p = ctypes.c_void_p, ctypes.c_int, ctypes.POINTER(ctypes.c_int64)
        L.dfs_plan_create.argtypes = [ctypes.POINTER(dfs_config), ctypes.POINTER(dfs_layer_weights), vp, vp,
                                      ctypes.POINTER(dfs_masks), vp, vp, ctypes.POINTER(vp)]
        L.dfs_block_forward.argtypes = [vp, i32, vp, vp, vp, vp]
        L.dfs_block_forward_layer.argtypes = [vp, i32, i32, vp, vp, vp, vp]
        L.dfs_block_forward_host.argtypes = [vp, i32, i32, vp, vp, vp, vp]
        L.dfs_block_forward_host_async.argtypes = [vp, i32, i32, vp, vp, vp, vp]
        L.dfs_block_forward_noalloc.argtypes = [vp, i32, i32, vp, vp, vp, vp]
        L.dfs_denoise.argtypes = [vp, vp, i32, vp, vp]
        L.dfs_plan_indices.argtypes = [vp, i32, i32, i32, ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(i32)]
        L.dfs_plan_panel.argtypes = [vp, i32, i32, i32, ctypes.POINTER(vp), i64p, i64p, i64p]
        L.dfs_plan_union_panel.argtypes = [vp, i32, i32, ctypes.POINTER(vp), i64p, i64p, i64p]
        L.dfs_plan_memory.argtypes = [vp, i64p, i64p]
        L.dfs_plan_flops.argtypes = [vp, i32, i32, ctypes.POINTER(ctypes.c_double)]
        L.dfs_plan_workspace.argtypes = [vp, i32, ctypes.POINTER(vp), i64p, i64p, i64p, ctypes.POINTER(i32)]
        L.dfs_plan_sync.argtypes = [vp, vp]
        L.dfs_selftest_wait_timeout.argtypes = [vp, vp]
        L.dfs_plan_profile.argtypes = [vp, i32]
        L.dfs_plan_profile_read.argtypes = [vp, i32, ctypes.POINTER(ctypes.c_double), i64p]
        L.dfs_gates_from_soft_masks.argtypes = [i32, i32, i32, i32, vp, vp]
        L.dfs_model_attach.argtypes = [vp, ctypes.POINTER(dfs_model_weights), vp]
        L.dfs_model_forward.argtypes = [vp, i32, vp, ctypes.c_float, vp, vp]
        L.dfs_model_denoise.argtypes = [vp, vp, i32, vp, vp]
        L.dfs_plan_destroy.argtypes = [vp]
        L.dfs_plan_destroy.restype = None
        L.dfs_last_error.restype = ctypes.c_char_p
        for n in EXPORTED:
            if n not in ("dfs_plan_destroy", "dfs_last_error"):
                getattr(L, n).restype = ctypes.c_int
        _lib = L
    return _lib


def dfs_last_error() -> str:
    """Message of the calling thread's last failed call (empty if none)."""
    return lib().dfs_last_error().decode()


def _check(status: int):
    if status != DFS_OK:
        raise DfsError(status, dfs_last_error())


def _ptr(x) -> Optional[int]:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    if isinstance(x, np.ndarray):
        return x.ctypes.data
    raise TypeError("cannot take a pointer of %r" % type(x))


def _stream(s) -> Optional[int]:
    if s is None:
        try:
            import torch
            if torch.cuda.is_available():
                return torch.cuda.current_stream().cuda_stream
        except ImportError:
            pass
        return None
    if isinstance(s, int):
        return s
    return s.cuda_stream


def make_config(cfg: Any) -> dfs_config:
    """dfs_config from any object / dict with the dfs_config field names (grid as a tuple)."""
    g = (lambda k: cfg[k]) if isinstance(cfg, dict) else (lambda k: getattr(cfg, k))
    grid = g("grid")
    c = dfs_config()
    c.dim, c.n_heads, c.head_dim, c.ffn_dim = g("dim"), g("n_heads"), g("head_dim"), g("ffn_dim")
    c.ffn_chunk, c.n_layers, c.n_steps = g("ffn_chunk"), g("n_layers"), g("n_steps")
    c.grid_t, c.grid_h, c.grid_w = int(grid[0]), int(grid[1]), int(grid[2])
    c.ctx_len, c.has_cross = g("ctx_len"), g("has_cross")
    c.ln_eps, c.rope_theta, c.qk_norm_mode = g("ln_eps"), g("rope_theta"), g("qk_norm_mode")
    try:
        eng = g("engine")
    except (KeyError, AttributeError):
        eng = DFS_ENGINE_COMPACTED
    c.engine = ENGINES[eng] if isinstance(eng, str) else int(eng)
    return c


class Plan:
    """Owning handle of a dfs_plan (destroyed with dfs_plan_destroy)."""

    def __init__(self, handle: int, keep: Sequence[Any] = ()):
        self.handle = handle
        self._keep = list(keep)

    def __int__(self):
        return self.handle

    def close(self):
        if self.handle:
            lib().dfs_plan_destroy(self.handle)
            self.handle = 0

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def _h(plan) -> int:
    return plan.handle if isinstance(plan, Plan) else int(plan)


def dfs_plan_create(cfg, layers: Sequence[Dict[str, Any]], w_t, b_t, masks: Dict[str, np.ndarray], ctx=None,
                    stream=None) -> Plan:
    """cfg: dfs_config or an object with its fields; layers: per-layer dicts of device
    buffers keyed like dfs_layer_weights; masks: host uint8 arrays (block_gate [T,L],
    head_gate [T,L,H], xhead_gate or None, ffn_gate [T,L,F/C])."""
    c = cfg if isinstance(cfg, dfs_config) else make_config(cfg)
    L = len(layers)
    arr = (dfs_layer_weights * max(L, 1))()
    for i, lw in enumerate(layers):
        for f in LAYER_FIELDS:
            setattr(arr[i], f, _ptr(lw.get(f)))
    keep = []
    m = dfs_masks()
    for f in ("block_gate", "head_gate", "xhead_gate", "ffn_gate"):
        a = masks.get(f)
        if a is not None:
            a = np.ascontiguousarray(a, dtype=np.uint8)
            keep.append(a)
            setattr(m, f, a.ctypes.data)
    out = ctypes.c_void_p()
    _check(lib().dfs_plan_create(ctypes.byref(c), arr, _ptr(w_t), _ptr(b_t), ctypes.byref(m), _ptr(ctx),
                                 _stream(stream), ctypes.byref(out)))
    return Plan(out.value)


def dfs_block_forward(plan, step: int, x, t_emb, out, stream=None):
    """Layer 0 of the plan at MoM step `step`: out = block(x, t_emb) (bf16 device buffers [N, dim], [dim])."""
    _check(lib().dfs_block_forward(_h(plan), step, _ptr(x), _ptr(t_emb), _ptr(out), _stream(stream)))


def dfs_block_forward_layer(plan, step: int, layer: int, x, t_emb, out, stream=None):
    """As dfs_block_forward for layer `layer` of the plan."""
    _check(lib().dfs_block_forward_layer(_h(plan), step, layer, _ptr(x), _ptr(t_emb), _ptr(out),
                                         _stream(stream)))


def dfs_block_forward_host(plan, step: int, layer: int, x_host, t_emb_host, out_host, stream=None):
    """As dfs_block_forward_layer on HOST buffers (pinned for full copy speed); synchronises `stream`."""
    _check(lib().dfs_block_forward_host(_h(plan), step, layer, _ptr(x_host), _ptr(t_emb_host),
                                        _ptr(out_host), _stream(stream)))


def dfs_block_forward_host_async(plan, step: int, layer: int, x_host, t_emb_host, out_host, stream=None):
    """Enqueue-only host-buffer forward; out_host is valid after dfs_plan_sync(plan, stream)."""
    _check(lib().dfs_block_forward_host_async(_h(plan), step, layer, _ptr(x_host), _ptr(t_emb_host),
                                              _ptr(out_host), _stream(stream)))


def dfs_block_forward_noalloc(plan, step: int, layer: int, x, t_emb, out, stream=None):
    """As dfs_block_forward_layer without any device allocation: the workspace lives in
    the library's static 16 MiB device array (see include/dfs.h for its rules)."""
    _check(lib().dfs_block_forward_noalloc(_h(plan), step, layer, _ptr(x), _ptr(t_emb), _ptr(out),
                                           _stream(stream)))


def dfs_denoise(plan, latents, n_steps: int, t_embs, stream=None):
    """Few-step loop on device latents [N, dim] in place: every layer of each step, then x += out / T."""
    _check(lib().dfs_denoise(_h(plan), _ptr(latents), n_steps, _ptr(t_embs), _stream(stream)))


def dfs_model_attach(plan, weights: Dict[str, Any], in_channels: int = 16, freq_dim: int = 256, stream=None):
    """weights: device buffers keyed like dfs_model_weights (bf16)."""
    w = dfs_model_weights()
    w.in_channels, w.freq_dim = in_channels, freq_dim
    for f in MODEL_FIELDS:
        setattr(w, f, _ptr(weights.get(f)))
    _check(lib().dfs_model_attach(_h(plan), ctypes.byref(w), _stream(stream)))


def dfs_model_forward(plan, step: int, latent, t: float, v_out, stream=None):
    """One pass of the attached Wan-shaped model at step `step` and timestep t: latent -> velocity v_out."""
    _check(lib().dfs_model_forward(_h(plan), step, _ptr(latent), float(t), _ptr(v_out), _stream(stream)))


def dfs_model_denoise(plan, latent, n_steps: int, timesteps: Sequence[float], stream=None):
    """Few-step latent denoise with the attached model; `timesteps` holds one host float per step."""
    ts = np.ascontiguousarray(timesteps, dtype=np.float32)
    _check(lib().dfs_model_denoise(_h(plan), _ptr(latent), n_steps, ts.ctypes.data, _stream(stream)))


def dfs_plan_indices(plan, step: int, layer: int, kind) -> np.ndarray:
    """Index list of (step, layer); `kind` is an int or a name of INDEX_KINDS."""
    kind = INDEX_KINDS[kind] if isinstance(kind, str) else kind
    n = ctypes.c_int()
    _check(lib().dfs_plan_indices(_h(plan), step, layer, kind, None, ctypes.byref(n)))
    out = np.zeros(n.value, dtype=np.int32)
    _check(lib().dfs_plan_indices(_h(plan), step, layer, kind,
                                  out.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)), ctypes.byref(n)))
    return out


def dfs_plan_panel(plan, step: int, layer: int, which):
    """(device address, rows, cols, ld) of a compacted panel; `which` is an int or a name."""
    w = PANELS[which] if isinstance(which, str) else which
    p, r, c, ld = ctypes.c_void_p(), ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int64()
    _check(lib().dfs_plan_panel(_h(plan), step, layer, w, ctypes.byref(p), ctypes.byref(r), ctypes.byref(c),
                                ctypes.byref(ld)))
    return p.value or 0, r.value, c.value, ld.value


def dfs_plan_union_panel(plan, layer: int, which):
    """(device address, rows, cols, ld) of a union panel (DFS_ENGINE_UNION plans)."""
    w = UNION_PANELS[which] if isinstance(which, str) else which
    p, r, c, ld = ctypes.c_void_p(), ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int64()
    _check(lib().dfs_plan_union_panel(_h(plan), layer, w, ctypes.byref(p), ctypes.byref(r), ctypes.byref(c),
                                      ctypes.byref(ld)))
    return p.value or 0, r.value, c.value, ld.value


def dfs_plan_memory(plan):
    """(weight bytes, device bytes) held by the plan."""
    wb, db = ctypes.c_int64(), ctypes.c_int64()
    _check(lib().dfs_plan_memory(_h(plan), ctypes.byref(wb), ctypes.byref(db)))
    return wb.value, db.value


def dfs_plan_flops(plan, step: int, layer: int = 0) -> float:
    """Algorithmic FLOPs of (step, layer) (closed form, 2 per multiply-add)."""
    f = ctypes.c_double()
    _check(lib().dfs_plan_flops(_h(plan), step, layer, ctypes.byref(f)))
    return f.value


def dfs_plan_workspace(plan, which):
    """Device address, shape and dtype of a workspace buffer of the last forward (test hook)."""
    w = WORKSPACE[which] if isinstance(which, str) else which
    p, r, c, ld, dt = ctypes.c_void_p(), ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int()
    _check(lib().dfs_plan_workspace(_h(plan), w, ctypes.byref(p), ctypes.byref(r), ctypes.byref(c),
                                    ctypes.byref(ld), ctypes.byref(dt)))
    return p.value or 0, r.value, c.value, ld.value, dt.value


def dfs_plan_sync(plan, stream=None):
    """Waits for `stream` (and the asynchronous host path's copies); raises on a kernel's bounded-wait timeout."""
    _check(lib().dfs_plan_sync(_h(plan), _stream(stream)))


def dfs_selftest_wait_timeout(plan, stream=None):
    """Launches a kernel whose bounded wait runs out on purpose (the timeout path's test hook)."""
    _check(lib().dfs_selftest_wait_timeout(_h(plan), _stream(stream)))


def dfs_plan_profile(plan, enable: bool):
    """Turns per-kernel CUDA-event timing of the plan's launches on or off."""
    _check(lib().dfs_plan_profile(_h(plan), 1 if enable else 0))


def dfs_plan_profile_read(plan, kind):
    """(total event-timed ms, launches) of one kernel kind (index or name of KERNEL_KINDS)."""
    k = KERNEL_KINDS.index(kind) if isinstance(kind, str) else kind
    ms, n = ctypes.c_double(), ctypes.c_int64()
    _check(lib().dfs_plan_profile_read(_h(plan), k, ctypes.byref(ms), ctypes.byref(n)))
    return ms.value, n.value


def dfs_gates_from_soft_masks(kind: int, m: np.ndarray, unit_size: int = 1) -> np.ndarray:
    """kind 0 block, 1 head, 2 FFN chunk; m [rows, units * unit_size] float32."""
    m = np.ascontiguousarray(np.atleast_2d(m), dtype=np.float32)
    rows, width = m.shape
    units = width // unit_size
    g = np.zeros((rows, units), dtype=np.uint8)
    _check(lib().dfs_gates_from_soft_masks(kind, rows, units, unit_size, m.ctypes.data, g.ctypes.data))
    return g


def dfs_plan_destroy(plan):
    """Frees the plan and everything it owns."""
    if isinstance(plan, Plan):
        plan.close()
    elif plan:
        lib().dfs_plan_destroy(int(plan))
