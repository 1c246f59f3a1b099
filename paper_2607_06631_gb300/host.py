"""Device-memory plumbing around the C ABI (torch is used for allocation and copies).

Turns numpy bf16 bit arrays into device tensors, assembles the per-layer weight
pointers for dfs_plan_create, and reads device buffers the library exposes (panels,
workspace) back to numpy.  No block arithmetic happens here.
"""
from __future__ import annotations

from typing import Dict, List, Optional

import numpy as np
import torch

from . import dfs


def to_device(bits: np.ndarray, device="cuda") -> torch.Tensor:
    """uint16 bf16 bits -> torch.bfloat16 tensor on `device`."""
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16))
    return t.to(device).view(torch.bfloat16)


def to_bits(t: torch.Tensor) -> np.ndarray:
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


class _CudaView:
    def __init__(self, ptr: int, shape, typestr: str, itemsize: int, ld: Optional[int] = None):
        strides = None
        if ld is not None and len(shape) == 2:
            strides = (ld * itemsize, itemsize)
        self.__cuda_array_interface__ = {"shape": tuple(int(s) for s in shape), "typestr": typestr,
                                         "data": (int(ptr), False), "version": 2, "strides": strides}


def view_device(ptr: int, rows: int, cols: int, ld: int, dtype: int) -> torch.Tensor:
    """Zero-copy torch view of a library-owned [rows, cols] buffer (dtype 0 bf16, 1 fp32)."""
    if rows * cols == 0 or not ptr:
        return torch.zeros((rows, cols), dtype=torch.bfloat16 if dtype == 0 else torch.float32)
    if dtype == 0:
        t = torch.as_tensor(_CudaView(ptr, (rows, cols), "<i2", 2, ld), device="cuda")
        return t.view(torch.bfloat16)
    return torch.as_tensor(_CudaView(ptr, (rows, cols), "<f4", 4, ld), device="cuda")


def read_panel(plan, step: int, layer: int, which) -> np.ndarray:
    """Compacted panel as uint16 bf16 bits [rows, cols] (host copy)."""
    p, r, c, ld = dfs.dfs_plan_panel(plan, step, layer, which)
    if r * c == 0:
        return np.zeros((r, c), np.uint16)
    return to_bits(view_device(p, r, c, ld, 0).clone())


def read_union_panel(plan, layer: int, which) -> np.ndarray:
    """Union panel (DFS_ENGINE_UNION) as uint16 bf16 bits [rows, cols] (host copy)."""
    p, r, c, ld = dfs.dfs_plan_union_panel(plan, layer, which)
    if r * c == 0:
        return np.zeros((r, c), np.uint16)
    return to_bits(view_device(p, r, c, ld, 0).clone())


def read_workspace(plan, which) -> np.ndarray:
    """Workspace buffer of the last forward: float64 array [rows, cols]."""
    p, r, c, ld, dt = dfs.dfs_plan_workspace(plan, which)
    t = view_device(p, r, c, ld, dt).clone()
    return t.float().cpu().numpy().astype(np.float64)


class DeviceProblem:
    """Device copies of one synthetic problem and the plan built from them."""

    def __init__(self, cfg, shared: Dict[str, np.ndarray], layers: List[Dict[str, np.ndarray]],
                 masks: Dict[str, np.ndarray], acts: Dict[str, np.ndarray], device="cuda"):
        self.cfg = cfg
        self.masks = masks
        self.w_t = to_device(shared["w_t"], device)
        self.b_t = to_device(shared["b_t"], device)
        self.layers = [{k: to_device(v, device) for k, v in lw.items()} for lw in layers]
        self.x = to_device(acts["x"], device)
        self.t_emb = to_device(acts["t_emb"], device)
        self.ctx = to_device(acts["ctx"], device) if "ctx" in acts else None
        self.plan = None

    def create_plan(self, stream=None, masks=None):
        self.plan = dfs.dfs_plan_create(self.cfg, self.layers, self.w_t, self.b_t,
                                        masks if masks is not None else self.masks, self.ctx, stream)
        return self.plan

    def free_weights(self):
        """Drops the full weights once the plan holds its compacted copies."""
        self.layers = None
        self.w_t = self.b_t = None


def random_device_stack(cfg, seed: int = 20260706):
    """Random-init weights of a multi-layer stack drawn directly on the device (torch's
    generator; N(0, 0.02) weights and biases, 1 + 0.1 N(0, 1) norm scales, the shapes of
    synth.layer_shapes): tens of GB would take minutes through the host generator.
    Returns (layers [per-layer dicts of bf16 tensors], w_t, b_t)."""
    import synth
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)

    def draw(shape, std, mean=0.0):
        t = torch.empty(shape, device="cuda", dtype=torch.bfloat16)
        t.normal_(mean, std, generator=g)
        return t
    layers = []
    for _ in range(cfg.n_layers):
        lw = {}
        for k, shp in synth.layer_shapes(cfg).items():
            scale = k in ("gq", "gk", "cgq", "cgk", "cln_w")
            lw[k] = draw(shp, 0.1 if scale else 0.02, 1.0 if scale else 0.0)
        layers.append(lw)
    d = cfg.dim
    return layers, draw((6 * d, d), 0.02), draw((6 * d,), 0.02)
