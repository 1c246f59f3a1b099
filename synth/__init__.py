"""Seeded synthetic inputs for the step-specific pruned DiT block.

This module only draws random numbers and lays them out: configurations (shapes and
per-step keep counts), bf16 weights, activations, timestep embeddings, text context and
the per-step gate masks.  It holds none of the block's arithmetic, so the CPU oracle
and the CUDA library can both be fed from it without sharing any computation.

Every tensor is produced as raw bf16 bits (``numpy.uint16``) so that both sides see
bit-identical values; ``bits_to_f64`` / ``bits_to_f32`` widen them for CPU use.

Distributions (the synthetic stand-in for trained Wan-class weights, which are not
available): linear weights, biases and the per-layer modulation table ~ N(0, 0.02);
norm scales gamma = 1 + 0.1 N(0, 1); block input x, timestep embedding and text context
~ N(0, 1).  Gate masks keep a seeded random subset of heads / FFN chunks per
(step, layer) with the per-step counts of the configuration.
"""
from __future__ import annotations

import concurrent.futures as _cf
import dataclasses
import os
import zlib
from typing import Dict, List, Optional, Sequence

import numpy as np

BASE_SEED = 20260706

# ---------------------------------------------------------------------------------------
# bf16 helpers (bit manipulation only)
# ---------------------------------------------------------------------------------------


def f32_to_bf16_bits(a) -> np.ndarray:
    """Round finite float32 values to bf16 (round to nearest, ties to even); returns
    uint16 bits.  (No finite float32 overflows the 32-bit sum below.)"""
    a = np.ascontiguousarray(np.asarray(a, dtype=np.float32))
    u = a.view(np.uint32)
    u = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return u.astype(np.uint16)


def bits_to_f32(bits) -> np.ndarray:
    b = np.ascontiguousarray(np.asarray(bits, dtype=np.uint16))
    return (b.astype(np.uint32) << 16).view(np.float32)


def bits_to_f64(bits) -> np.ndarray:
    return bits_to_f32(bits).astype(np.float64)


# ---------------------------------------------------------------------------------------
# configurations
# ---------------------------------------------------------------------------------------


@dataclasses.dataclass
class Config:
    name: str
    dim: int
    n_heads: int
    head_dim: int
    ffn_dim: int
    grid: tuple            # (frames, height, width) of the latent token grid
    heads_kept: List[List[int]]   # [n_steps][n_layers] retained head counts
    chunks_kept: List[List[int]]  # [n_steps][n_layers] retained FFN chunk counts
    ffn_chunk: int = 8
    n_layers: int = 1
    n_steps: int = 4
    ctx_len: int = 512
    has_cross: int = 0
    xheads_kept: Optional[List[List[int]]] = None
    ln_eps: float = 1e-6
    rope_theta: float = 10000.0
    qk_norm_mode: int = 0
    block_gate: Optional[List[List[int]]] = None  # [n_steps][n_layers]; None -> all ones
    engine: int = 0        # how the library holds the weights: 0 per-step copies, 1 union
    latent_channels: int = 16   # Wan-shaped model around the blocks: latent video channels
    freq_dim: int = 256         # and timestep-sinusoid width

    @property
    def n_tokens(self) -> int:
        return int(self.grid[0] * self.grid[1] * self.grid[2])

    @property
    def n_chunks(self) -> int:
        return self.ffn_dim // self.ffn_chunk


def keep_count(ratio: float, n: int) -> int:
    """Retained unit count for a keep ratio: round half up of ratio * n."""
    return int(np.floor(ratio * n + 0.5))


def _per_step(counts: Sequence[int], n_layers: int) -> List[List[int]]:
    return [[int(c)] * n_layers for c in counts]


def tiny(n_layers: int = 1, has_cross: int = 0, grid=(2, 16, 16), qk_norm_mode: int = 0) -> Config:
    """Tiny pruned block: d=256, 4 heads x 64, FFN 1024, 2x16x16 tokens."""
    chunks = [c // 8 for c in (1024, 768, 640, 512)]
    return Config(name="tiny", dim=256, n_heads=4, head_dim=64, ffn_dim=1024, grid=tuple(grid),
                  heads_kept=_per_step([4, 3, 3, 2], n_layers),
                  chunks_kept=_per_step(chunks, n_layers), n_layers=n_layers,
                  has_cross=has_cross,
                  xheads_kept=_per_step([4, 3, 3, 2], n_layers) if has_cross else None,
                  ctx_len=512 if has_cross else 0, qk_norm_mode=qk_norm_mode)


def _ratio_config(name, dim, heads, dh, ffn, grid, ratios, n_layers=1, has_cross=0,
                  ctx_len=0) -> Config:
    hk = [keep_count(r, heads) for r in ratios]
    ck = [keep_count(r, ffn // 8) for r in ratios]
    return Config(name=name, dim=dim, n_heads=heads, head_dim=dh, ffn_dim=ffn, grid=tuple(grid),
                  heads_kept=_per_step(hk, n_layers), chunks_kept=_per_step(ck, n_layers),
                  n_layers=n_layers, has_cross=has_cross, ctx_len=ctx_len,
                  xheads_kept=_per_step(hk, n_layers) if has_cross else None)


def wan13b() -> Config:
    """Wan-1.3B-shaped block: d=1536, 12x128 heads, FFN 8960, 21x30x52 tokens."""
    return _ratio_config("wan13b", 1536, 12, 128, 8960, (21, 30, 52), (1.0, 0.85, 0.75, 0.65))


def wan14b() -> Config:
    """Wan-14B-shaped block: d=5120, 40x128 heads, FFN 13824, 21x30x52 tokens."""
    return _ratio_config("wan14b", 5120, 40, 128, 13824, (21, 30, 52), (1.0, 0.8, 0.7, 0.55))


def wan14b_stack(n_layers: int = 40) -> Config:
    """14B-shaped stack of blocks with text cross-attention over 512 context tokens."""
    return _ratio_config("wan14b_x%d" % n_layers, 5120, 40, 128, 13824, (21, 30, 52),
                         (1.0, 0.8, 0.7, 0.55), n_layers=n_layers, has_cross=1, ctx_len=512)


def sweep720(ratio: float) -> Config:
    """720p-shaped block (14B shapes, 21x45x80 tokens) with one uniform keep ratio."""
    return _ratio_config("sweep720_r%.1f" % ratio, 5120, 40, 128, 13824, (21, 45, 80),
                         (ratio,) * 4)


SWEEP_RATIOS = (1.0, 0.9, 0.8, 0.7, 0.6, 0.5)


def sweep720_all() -> Config:
    """720p-shaped block whose six 'steps' are the uniform keep ratios 1.0 .. 0.5, so
    one plan holds every point of the sweep (step i keeps SWEEP_RATIOS[i])."""
    cfg = _ratio_config("sweep720", 5120, 40, 128, 13824, (21, 45, 80), SWEEP_RATIOS)
    cfg.n_steps = len(SWEEP_RATIOS)
    return cfg


def wan14b_cross() -> Config:
    """One Wan-14B-shaped block with text cross-attention over 512 context tokens."""
    return _ratio_config("wan14b_cross", 5120, 40, 128, 13824, (21, 30, 52),
                         (1.0, 0.8, 0.7, 0.55), has_cross=1, ctx_len=512)


# Per-step keep profiles shaped like the learned pruning policy the paper analyses (Sec. 6,
# "U-shaped computational allocation" and "semantic freezing in deep layers"; App. D): the two
# end steps keep more than the two middle ones, deeper layers lose more self / cross-attention
# heads than shallow ones (most at t2 and t3, where the deepest layer is shut down), and the FFN
# keeps more than attention.  At depth u = l / (L - 1) of step s, a unit kind keeps
#     clip(k0 - slope * u, 0, 1)
# of its heads (self and cross alike) / FFN chunks, per step
#     (attention k0, attention slope, FFN k0, FFN slope).
# The constants were chosen so that the 30-layer Wan-1.3B-shaped stack with cross-attention at
# 32760 tokens keeps 88.6 / 78.7 / 77.1 / 89.1 % of its dense FLOPs per step (the paper's learned
# policy: 88.4 / 78.5 / 77.1 / 89.1 %; mean 83.3 % against the final checkpoint's ~83 %).
POLICY_PROFILE = ((1.095, 0.40, 0.97, 0.12),
                  (2.307, 2.30, 0.90, 0.20),
                  (2.282, 2.30, 0.90, 0.20),
                  (1.096, 0.40, 0.97, 0.12))


def policy_counts(n_heads: int, n_chunks: int, n_layers: int, profile=POLICY_PROFILE):
    """[n_steps][n_layers] retained head and FFN chunk counts of the policy-shaped profile."""
    heads, chunks = [], []
    for a0, ba, f0, bf in profile:
        hs, cs = [], []
        for l in range(n_layers):
            u = l / (n_layers - 1) if n_layers > 1 else 0.0
            a = min(1.0, max(0.0, a0 - ba * u))
            f = min(1.0, max(0.0, f0 - bf * u))
            hs.append(keep_count(a, n_heads))
            cs.append(keep_count(f, n_chunks))
        heads.append(hs)
        chunks.append(cs)
    return heads, chunks


def wan13b_policy(n_layers: int = 30, grid=(21, 30, 52)) -> Config:
    """Wan-1.3B-shaped stack (30 blocks, d=1536, 12x128 heads, FFN 8960, text cross-attention
    over 512 context tokens) whose per-(step, layer) masks follow POLICY_PROFILE."""
    hk, ck = policy_counts(12, 8960 // 8, n_layers)
    return Config(name="wan13b_policy", dim=1536, n_heads=12, head_dim=128, ffn_dim=8960, grid=tuple(grid),
                  heads_kept=hk, chunks_kept=ck, n_layers=n_layers, has_cross=1, ctx_len=512,
                  xheads_kept=[list(h) for h in hk])


def policy_small(n_layers: int = 12) -> Config:
    """Tiny-shaped stack (d=256, 4x64 heads, FFN 1024, 2x8x8 tokens, cross-attention over 64
    context tokens) with policy-shaped masks, small enough for the oracle's full denoise."""
    hk, ck = policy_counts(4, 1024 // 8, n_layers)
    return Config(name="policy_small", dim=256, n_heads=4, head_dim=64, ffn_dim=1024, grid=(2, 8, 8),
                  heads_kept=hk, chunks_kept=ck, n_layers=n_layers, has_cross=1, ctx_len=64,
                  xheads_kept=[list(h) for h in hk])


def small_stack(n_layers: int = 4) -> Config:
    """Shrunken stack (d=256, 2x8x8 tokens, cross-attention) for end-to-end denoise checks."""
    cfg = tiny(n_layers=n_layers, has_cross=1, grid=(2, 8, 8))
    cfg.name = "small_stack"
    return cfg


def tiny_model(n_layers: int = 4) -> Config:
    """Tiny-shaped model (d=256, 4x64 heads, FFN 1024, cross-attention over 64 context
    tokens) on a 16 x 2 x 16 x 16 latent video (2 x 8 x 8 = 128 tokens)."""
    cfg = tiny(n_layers=n_layers, has_cross=1, grid=(2, 8, 8))
    cfg.name = "tiny_model"
    cfg.ctx_len = 64
    return cfg


def wan13b_model() -> Config:
    """The 30-layer Wan-1.3B-shaped policy stack inside the model (latent 16 x 21 x 60 x 104)."""
    cfg = wan13b_policy()
    cfg.name = "wan13b_model"
    return cfg


def model_timesteps(n_steps: int = 4) -> List[float]:
    """Host timesteps fed to the model's sinusoid at each step: 1000 (1 - s/T)."""
    return [1000.0 * (1.0 - s / n_steps) for s in range(n_steps)]


# ---------------------------------------------------------------------------------------
# seeded draws
# ---------------------------------------------------------------------------------------


def seed_for(*parts) -> int:
    key = "/".join(str(p) for p in parts).encode()
    return (BASE_SEED * 1000003 + zlib.crc32(key)) & 0xFFFFFFFFFFFF


def _rng(*parts) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(seed_for(*parts)))


_CHUNK = 1 << 22
_POOL = _cf.ThreadPoolExecutor(max_workers=max(1, min(32, os.cpu_count() or 1)))


def normal_bits(shape, std=1.0, mean=0.0, *seed_parts) -> np.ndarray:
    """bf16 bits of mean + std * N(0, 1) draws.  The tensor is filled in chunks of 2^22
    values, chunk i from its own PCG64 stream seeded with (seed, i), in parallel threads."""
    n = int(np.prod(shape)) if len(shape) else 1
    out = np.empty(n, dtype=np.uint16)
    base = seed_for(*seed_parts)

    def fill(i):
        lo, hi = i * _CHUNK, min(n, (i + 1) * _CHUNK)
        rng = np.random.Generator(np.random.PCG64([base, i]))
        a = rng.standard_normal(size=hi - lo, dtype=np.float32)
        if std != 1.0:
            a *= np.float32(std)
        if mean != 0.0:
            a += np.float32(mean)
        out[lo:hi] = f32_to_bf16_bits(a)

    list(_POOL.map(fill, range((n + _CHUNK - 1) // _CHUNK)))
    return out.reshape(shape)


LAYER_KEYS = ("wq", "bq", "wk", "bk", "wv", "bv", "wo", "bo", "gq", "gk",
              "w_up", "b_up", "w_down", "b_down", "e_mod")
CROSS_KEYS = ("cwq", "cbq", "cwk", "cbk", "cwv", "cbv", "cwo", "cbo", "cgq", "cgk",
              "cln_w", "cln_b")


def layer_shapes(cfg: Config) -> Dict[str, tuple]:
    d, F = cfg.dim, cfg.ffn_dim
    s = {"wq": (d, d), "bq": (d,), "wk": (d, d), "bk": (d,), "wv": (d, d), "bv": (d,),
         "wo": (d, d), "bo": (d,), "gq": (d,), "gk": (d,),
         "w_up": (F, d), "b_up": (F,), "w_down": (d, F), "b_down": (d,), "e_mod": (6, d)}
    if cfg.has_cross:
        s.update({"cwq": (d, d), "cbq": (d,), "cwk": (d, d), "cbk": (d,), "cwv": (d, d),
                  "cbv": (d,), "cwo": (d, d), "cbo": (d,), "cgq": (d,), "cgk": (d,),
                  "cln_w": (d,), "cln_b": (d,)})
    return s


def _is_scale(key: str) -> bool:
    return key in ("gq", "gk", "cgq", "cgk", "cln_w")


def make_layer(cfg: Config, layer: int, seed_tag: str = "") -> Dict[str, np.ndarray]:
    out = {}
    for k, shp in layer_shapes(cfg).items():
        tag = (cfg.name + seed_tag, "layer", layer, k)
        if _is_scale(k):
            out[k] = normal_bits(shp, 0.1, 1.0, *tag)
        else:
            out[k] = normal_bits(shp, 0.02, 0.0, *tag)
    return out


def make_shared(cfg: Config, seed_tag: str = "") -> Dict[str, np.ndarray]:
    d = cfg.dim
    return {"w_t": normal_bits((6 * d, d), 0.02, 0.0, cfg.name + seed_tag, "w_t"),
            "b_t": normal_bits((6 * d,), 0.02, 0.0, cfg.name + seed_tag, "b_t")}


def subset_gate(n: int, k: int, *seed_parts) -> np.ndarray:
    """Gate vector of length n keeping a seeded random subset of k units (Fisher-Yates)."""
    g = np.zeros(n, dtype=np.uint8)
    if k > 0:
        perm = _rng(*seed_parts).permutation(n)
        g[np.sort(perm[:k])] = 1
    return g


def make_masks(cfg: Config, seed_tag: str = "") -> Dict[str, np.ndarray]:
    T, L, H, NC = cfg.n_steps, cfg.n_layers, cfg.n_heads, cfg.n_chunks
    head = np.zeros((T, L, H), np.uint8)
    ffn = np.zeros((T, L, NC), np.uint8)
    xhead = np.zeros((T, L, H), np.uint8) if cfg.has_cross else None
    for s in range(T):
        for l in range(L):
            head[s, l] = subset_gate(H, cfg.heads_kept[s][l], cfg.name + seed_tag, "head", s, l)
            ffn[s, l] = subset_gate(NC, cfg.chunks_kept[s][l], cfg.name + seed_tag, "ffn", s, l)
            if cfg.has_cross:
                xhead[s, l] = subset_gate(H, cfg.xheads_kept[s][l], cfg.name + seed_tag,
                                          "xhead", s, l)
    if cfg.block_gate is None:
        block = np.ones((T, L), np.uint8)
    else:
        block = np.asarray(cfg.block_gate, dtype=np.uint8).reshape(T, L)
    return {"block_gate": block, "head_gate": head, "xhead_gate": xhead, "ffn_gate": ffn}


def make_activations(cfg: Config, seed_tag: str = "") -> Dict[str, np.ndarray]:
    d, N = cfg.dim, cfg.n_tokens
    out = {"x": normal_bits((N, d), 1.0, 0.0, cfg.name + seed_tag, "x"),
           "t_emb": normal_bits((cfg.n_steps, d), 1.0, 0.0, cfg.name + seed_tag, "t_emb")}
    if cfg.has_cross:
        out["ctx"] = normal_bits((cfg.ctx_len, d), 1.0, 0.0, cfg.name + seed_tag, "ctx")
    return out


MODEL_KEYS = ("patch_w", "patch_b", "t_w1", "t_b1", "t_w2", "t_b2", "head_mod", "head_w", "head_b")


def model_shapes(cfg: Config) -> Dict[str, tuple]:
    d, p = cfg.dim, 4 * cfg.latent_channels
    return {"patch_w": (d, p), "patch_b": (d,), "t_w1": (d, cfg.freq_dim), "t_b1": (d,),
            "t_w2": (d, d), "t_b2": (d,), "head_mod": (2, d), "head_w": (p, d), "head_b": (p,)}


def make_model_weights(cfg: Config, seed_tag: str = "") -> Dict[str, np.ndarray]:
    """Weights of the model around the blocks, all ~ N(0, 0.02) as bf16 bits."""
    return {k: normal_bits(shp, 0.02, 0.0, cfg.name + seed_tag, "model", k) for k, shp in model_shapes(cfg).items()}


def make_latent(cfg: Config, seed_tag: str = "") -> np.ndarray:
    """Latent video [C, F, H, W] ~ N(0, 1) as bf16 bits (H, W = twice the token grid)."""
    F, gh, gw = cfg.grid
    return normal_bits((cfg.latent_channels, F, 2 * gh, 2 * gw), 1.0, 0.0, cfg.name + seed_tag, "latent")


def make_problem(cfg: Config, seed_tag: str = ""):
    """All inputs of one configuration: (shared, layers, masks, activations), as bf16 bits."""
    shared = make_shared(cfg, seed_tag)
    layers = [make_layer(cfg, l, seed_tag) for l in range(cfg.n_layers)]
    masks = make_masks(cfg, seed_tag)
    acts = make_activations(cfg, seed_tag)
    return shared, layers, masks, acts


def widen(tree):
    """bf16 bits -> float64 for every uint16 array in a dict / list tree."""
    if isinstance(tree, dict):
        return {k: widen(v) for k, v in tree.items()}
    if isinstance(tree, list):
        return [widen(v) for v in tree]
    if isinstance(tree, np.ndarray) and tree.dtype == np.uint16:
        return bits_to_f64(tree)
    return tree
