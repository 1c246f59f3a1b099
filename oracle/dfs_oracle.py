"""CPU oracle for the step-specific pruned video-DiT block ("Dynamic-in-Few-Step").

TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and bench.py's
cpu_baseline / --impl reference leg may import this module.  The CUDA library never
calls it, and it shares no code with the library: it is the plain definition of what
the library computes, written in float64 numpy on bf16-valued inputs.

What the paper fixes (cited per function):
  * Eq. 2 (Sec. 3.2): a gated component's output is multiplied by its binary gate.
  * Sec. 4.1: soft mask -> hard gate rules for blocks, heads (mean of the head's
    D_head mask entries > 0) and FFN chunks of C channels.
  * App. A: chunk size C = 8.
  * Sec. 3.2 (export) and Sec. 4.3 (union super-model + per-step index tables): the
    pruned per-step model is a dense model over the retained units only, so the
    compacted computation is the same function as the masked dense block.
  * Sec. 3.1: T = 4 distilled steps.

What the paper leaves open (numbered readings; parity is unpinned against the
authors' own engine for all of them):
  R1  adaLN parameters: mod = W_t t_emb + b_t + E_l, one linear shared across layers
      plus a per-layer table E_l of shape [6, d].
  R2  order of the six vectors: shift_a, scale_a, gate_a, shift_f, scale_f, gate_f,
      broadcast over tokens.
  R3  LayerNorm: no affine, eps = 1e-6, population variance.
  R4  QK RMSNorm span: mode 0 = over the retained q (resp. k) channels of the row,
      mode 1 = over each head's dh channels; eps = 1e-6; then gamma.
  R5  3D RoPE: dh/2 interleaved pairs (2j, 2j+1) split into frame / height / width
      bands of p_t = dh/2 - 2*floor(dh/6), p_h = p_w = floor(dh/6) pairs; pair j of a
      band of p pairs turns by pos * theta^(-j/p); token n = (f*G_h + y)*G_w + w.
  R6  cross-attention: affine LayerNorm of x1, Q from it, K/V from the context, QK
      RMSNorm as R4, no RoPE, no adaLN gate, its own head gates.
  R7  FFN activation: GELU, tanh approximation.
  R8  a block whose block gate is 0 is the identity.
  R9  4-step sampler: x <- x + (1/T) * v with v the output of the last block.
  R16 patch embedding of the Wan-shaped model around the blocks: latent video
      [C, F, H, W], patches of 1 x 2 x 2; token n = (f*G_h + y)*G_w + x (the RoPE order),
      feature k = c*4 + dy*2 + dx; x = patches W_p^T + b_p.
  R17 timestep embedding: e = [cos(t w_i), sin(t w_i)], w_i = 10000^(-i/(D/2)),
      i < D/2 (D = 256); t_emb = W_2 SiLU(W_1 e + b_1) + b_2.
  R18 output head: LN(x) (no affine) * (1 + scale_h) + shift_h with
      (shift_h, scale_h) = E_h + t_emb (a learned [2, d] table plus t_emb itself), then
      v = y W_h^T + b_h, unpatched back to [C, F, H, W].
  R19 latent sampler: the model predicts a velocity; z <- z + (1/T) v at each of the T
      steps, step s fed with the host timestep t_s (1000 (1 - s/T): noise at s = 0, since
      Sec. 3.1 puts tau = 0 at pure noise and tau = 1 at clean data).
"""
from __future__ import annotations

import math
from typing import Dict, List, Optional

import numpy as np

__all__ = [
    "gates_from_soft_masks", "ffn_channel_gate", "compact_indices", "compact_panels",
    "union_tables", "union_panels",
    "linear", "modulation", "layer_norm", "adaln", "rms_norm", "rope_pairs", "rope_angles",
    "apply_rope", "attention", "gelu_tanh", "block_forward_masked",
    "block_forward_compacted", "block_flops", "denoise", "MacCounter",
    "cross_input_norm", "output_head",
    "patchify", "unpatchify", "timestep_embedding", "time_mlp", "model_forward", "model_denoise",
]


# ---------------------------------------------------------------------------------------
# gates (Sec. 3.2 gate shapes [T, N]; Sec. 4.1 soft -> hard rules; App. A chunk size)
# ---------------------------------------------------------------------------------------

def gates_from_soft_masks(kind: str, m, unit_size: int = 1) -> np.ndarray:
    """Hard gates from continuous masks, Sec. 4.1.

    kind "block": g = I(m > 0) per block.
    kind "head":  m holds D_head entries per head along the last axis; the head is kept
                  iff the mean of its entries is positive.
    kind "ffn":   one scalar per chunk of C channels; the chunk is kept iff m > 0.
    The comparison is made on float64 values.
    """
    m = np.asarray(m, dtype=np.float64)
    if kind in ("block", "ffn"):
        return (m > 0).astype(np.uint8)
    if kind == "head":
        per_head = m.reshape(*m.shape[:-1], m.shape[-1] // unit_size, unit_size)
        return (per_head.mean(axis=-1) > 0).astype(np.uint8)
    raise ValueError(kind)


def ffn_channel_gate(chunk_gate, chunk: int) -> np.ndarray:
    """Per-channel FFN gate: each chunk gate repeated over its C channels (Sec. 4.1)."""
    return np.repeat(np.asarray(chunk_gate, dtype=np.uint8), chunk, axis=-1)


def compact_indices(cfg, masks, step: int, layer: int) -> Dict[str, np.ndarray]:
    """Per-step index table I_t of Sec. 4.3 for one layer.

    heads / chunks / xheads: ascending retained unit ids.
    qk_rows: channel ids of the retained heads (h*dh + j), the rows of Wq/Wk/Wv and the
             columns of Wo that the step uses.
    ffn_ch:  FFN hidden channel ids of the retained chunks (c*C + j).
    """
    dh, C = cfg.head_dim, cfg.ffn_chunk
    heads = np.flatnonzero(masks["head_gate"][step, layer]).astype(np.int32)
    chunks = np.flatnonzero(masks["ffn_gate"][step, layer]).astype(np.int32)
    out = {
        "heads": heads,
        "chunks": chunks,
        "qk_rows": (heads[:, None] * dh + np.arange(dh)[None, :]).reshape(-1).astype(np.int32),
        "ffn_ch": (chunks[:, None] * C + np.arange(C)[None, :]).reshape(-1).astype(np.int32),
    }
    if cfg.has_cross:
        xg = masks.get("xhead_gate")
        xheads = (np.arange(cfg.n_heads, dtype=np.int32) if xg is None
                  else np.flatnonzero(xg[step, layer]).astype(np.int32))
        out["xheads"] = xheads
        out["x_rows"] = (xheads[:, None] * dh + np.arange(dh)[None, :]).reshape(-1).astype(np.int32)
    return out


def compact_panels(layer_w: Dict[str, np.ndarray], idx: Dict[str, np.ndarray]) -> Dict[str, np.ndarray]:
    """Dense per-step weights gathered from the full layer (the export of Sec. 3.2).

    Works on any dtype (bf16 bit patterns included): it only selects rows / columns.
    Linear weights are [out, in]; Wo and W_down are gathered by column.
    """
    r, ch = idx["qk_rows"], idx["ffn_ch"]
    P = {
        "wqkv": np.concatenate([layer_w["wq"][r], layer_w["wk"][r], layer_w["wv"][r]], axis=0),
        "bqkv": np.concatenate([layer_w["bq"][r], layer_w["bk"][r], layer_w["bv"][r]]),
        "gq": layer_w["gq"][r],
        "gk": layer_w["gk"][r],
        "wo": layer_w["wo"][:, r],
        "w_up": layer_w["w_up"][ch],
        "b_up": layer_w["b_up"][ch],
        "w_down": layer_w["w_down"][:, ch],
    }
    if "x_rows" in idx:
        xr = idx["x_rows"]
        P.update({
            "cwq": layer_w["cwq"][xr], "cbq": layer_w["cbq"][xr],
            "cwkv": np.concatenate([layer_w["cwk"][xr], layer_w["cwv"][xr]], axis=0),
            "cbkv": np.concatenate([layer_w["cbk"][xr], layer_w["cbv"][xr]]),
            "cgq": layer_w["cgq"][xr], "cgk": layer_w["cgk"][xr],
            "cwo": layer_w["cwo"][:, xr],
        })
    return P


def union_tables(cfg, masks, layer: int) -> Dict[str, object]:
    """The union super-model of one layer and its per-step index tables (Sec. 4.3,
    Fig. 1(c)): theta_union holds every unit that some step retains, and I_t addresses
    step t's retained units inside it.

    heads / chunks / xheads: ascending unit ids retained at one step or more (block gates
    do not enter: a unit belongs to the union as soon as any step's gate keeps it).
    pos_heads / pos_chunks / pos_xheads: per step, for each retained unit of that step
    (ascending), its index in the union list.
    """
    H = cfg.n_heads
    hg = np.asarray(masks["head_gate"])[:, layer].astype(bool)
    fg = np.asarray(masks["ffn_gate"])[:, layer].astype(bool)
    T = hg.shape[0]
    out = {"heads": [], "chunks": [], "xheads": [], "pos_heads": [], "pos_chunks": [], "pos_xheads": []}
    # a unit is in the union iff some step keeps it
    out["heads"] = np.array([h for h in range(H) if any(hg[s, h] for s in range(T))], dtype=np.int32)
    out["chunks"] = np.array([k for k in range(fg.shape[1]) if any(fg[s, k] for s in range(T))], dtype=np.int32)
    if cfg.has_cross:
        xg = masks.get("xhead_gate")
        xgl = np.ones((T, H), bool) if xg is None else np.asarray(xg)[:, layer].astype(bool)
        out["xheads"] = np.array([h for h in range(H) if any(xgl[s, h] for s in range(T))], dtype=np.int32)
    for s in range(T):
        idx = compact_indices(cfg, masks, s, layer)
        where = {u: i for i, u in enumerate(out["heads"])}
        out["pos_heads"].append(np.array([where[h] for h in idx["heads"]], dtype=np.int32))
        where = {u: i for i, u in enumerate(out["chunks"])}
        out["pos_chunks"].append(np.array([where[k] for k in idx["chunks"]], dtype=np.int32))
        if cfg.has_cross:
            where = {u: i for i, u in enumerate(out["xheads"])}
            out["pos_xheads"].append(np.array([where[h] for h in idx["xheads"]], dtype=np.int32))
    return out


def union_panels(cfg, layer_w: Dict[str, np.ndarray], union: Dict[str, object]) -> Dict[str, np.ndarray]:
    """Weights of the union super-model (Sec. 4.3), gathered from the full layer: the q, k
    and v rows of the union heads stacked, the matching columns of Wo, the union FFN
    channels' rows of W_up and columns of W_down, and with cross-attention the union cross
    heads' rows of cWq and columns of cWo.  Selection only (any dtype)."""
    dh, C = cfg.head_dim, cfg.ffn_chunk
    hu = np.asarray(union["heads"], dtype=np.int64)
    r = (hu[:, None] * dh + np.arange(dh)[None, :]).reshape(-1)
    cu = np.asarray(union["chunks"], dtype=np.int64)
    ch = (cu[:, None] * C + np.arange(C)[None, :]).reshape(-1)
    P = {
        "wqkv": np.concatenate([layer_w["wq"][r], layer_w["wk"][r], layer_w["wv"][r]], axis=0),
        "wo": layer_w["wo"][:, r],
        "w_up": layer_w["w_up"][ch],
        "w_down": layer_w["w_down"][:, ch],
    }
    if cfg.has_cross:
        xu = np.asarray(union["xheads"], dtype=np.int64)
        xr = (xu[:, None] * dh + np.arange(dh)[None, :]).reshape(-1)
        P["cwq"] = layer_w["cwq"][xr]
        P["cwo"] = layer_w["cwo"][:, xr]
    return P


# ---------------------------------------------------------------------------------------
# elementary operations (float64)
# ---------------------------------------------------------------------------------------

class MacCounter:
    """Counts the floating-point operations of the contractions actually executed
    (2 per multiply-add), to check the closed form of ``block_flops``."""

    def __init__(self):
        self.flops = 0

    def add(self, m: int, n: int, k: int):
        self.flops += 2 * int(m) * int(n) * int(k)


def _matmul(a, b, counter: Optional[MacCounter]):
    if counter is not None:
        counter.add(a.shape[0], b.shape[1], a.shape[1])
    return a @ b


def linear(x, w, b=None, counter: Optional[MacCounter] = None):
    """y = x W^T + b with W stored [out, in]."""
    y = _matmul(x, w.T, counter)
    if b is not None:
        y = y + b
    return y


def modulation(w_t, b_t, e_l, t_emb) -> np.ndarray:
    """Six adaLN vectors (R1, R2): rows shift_a, scale_a, gate_a, shift_f, scale_f, gate_f."""
    d = e_l.shape[-1]
    return (w_t @ t_emb + b_t).reshape(6, d) + e_l


def layer_norm(x, eps: float, weight=None, bias=None) -> np.ndarray:
    """LayerNorm over the last axis with population variance (R3)."""
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    y = (x - mu) / np.sqrt(var + eps)
    if weight is not None:
        y = y * weight
    if bias is not None:
        y = y + bias
    return y


def adaln(x, shift, scale, eps: float) -> np.ndarray:
    """adaLN modulation of a LayerNorm without affine: LN(x) * (1 + scale) + shift."""
    return layer_norm(x, eps) * (1.0 + scale) + shift


def rms_norm(x, gamma, keep, eps: float, mode: int, head_dim: int) -> np.ndarray:
    """QK RMSNorm (R4) on rows of x [n, channels].

    keep: 0/1 per channel; pruned channels are excluded from the statistic and zeroed.
    mode 0: one statistic over all retained channels of the row.
    mode 1: one statistic per head (groups of head_dim channels).
    """
    keep = np.asarray(keep, dtype=np.float64)
    xz = x * keep
    if mode == 0:
        cnt = keep.sum()
        ms = (xz ** 2).sum(axis=-1, keepdims=True) / cnt
        y = xz / np.sqrt(ms + eps)
    else:
        n, c = x.shape
        xh = xz.reshape(n, c // head_dim, head_dim)
        ms = (xh ** 2).mean(axis=-1, keepdims=True)
        y = (xh / np.sqrt(ms + eps)).reshape(n, c)
    return y * gamma * keep


def rope_pairs(head_dim: int):
    """Band sizes (p_t, p_h, p_w) in rotation pairs (R5)."""
    half = head_dim // 2
    p_hw = head_dim // 6
    return half - 2 * p_hw, p_hw, p_hw


def rope_angles(grid, head_dim: int, theta: float) -> np.ndarray:
    """Rotation angle of every (token, pair): [N, head_dim/2] (R5)."""
    G_t, G_h, G_w = grid
    p_t, p_h, p_w = rope_pairs(head_dim)
    f, y, w = np.meshgrid(np.arange(G_t), np.arange(G_h), np.arange(G_w), indexing="ij")
    pos = [f.reshape(-1).astype(np.float64), y.reshape(-1).astype(np.float64),
           w.reshape(-1).astype(np.float64)]
    cols = []
    for p_a, pos_a in zip((p_t, p_h, p_w), pos):
        freq = theta ** (-np.arange(p_a, dtype=np.float64) / p_a)
        cols.append(pos_a[:, None] * freq[None, :])
    return np.concatenate(cols, axis=1)


def apply_rope(x, ang) -> np.ndarray:
    """Rotate interleaved pairs (2j, 2j+1) of x [n, heads, dh] by ang [n, dh/2]."""
    c = np.cos(ang)[:, None, :]
    s = np.sin(ang)[:, None, :]
    x0 = x[..., 0::2]
    x1 = x[..., 1::2]
    out = np.empty_like(x)
    out[..., 0::2] = x0 * c - x1 * s
    out[..., 1::2] = x0 * s + x1 * c
    return out


def attention(q, k, v, counter: Optional[MacCounter] = None) -> np.ndarray:
    """Non-causal softmax attention per head: q [n, h, dh], k/v [m, h, dh] -> [n, h, dh]."""
    n, h, dh = q.shape
    out = np.empty((n, h, v.shape[-1]))
    scale = 1.0 / math.sqrt(dh)
    for j in range(h):
        s = _matmul(q[:, j, :], k[:, j, :].T, counter) * scale
        s = s - s.max(axis=1, keepdims=True)
        p = np.exp(s)
        p = p / p.sum(axis=1, keepdims=True)
        out[:, j, :] = _matmul(p, v[:, j, :], counter)
    return out


def gelu_tanh(x) -> np.ndarray:
    """GELU with the tanh approximation (R7)."""
    return 0.5 * x * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (x + 0.044715 * x ** 3)))


# ---------------------------------------------------------------------------------------
# the block
# ---------------------------------------------------------------------------------------

def _rows(x, rows):
    return x if rows is None else x[rows]


def _token_ids(n_tokens, rows):
    return np.arange(n_tokens) if rows is None else np.asarray(rows)


def block_forward_masked(cfg, shared, lw, masks, step: int, layer: int, x, t_emb, ctx=None,
                         rows=None, want: bool = False):
    """Masked dense block at one denoising step: every unit is computed and the
    gated outputs are multiplied by their gates (Eq. 2).  Inputs are float64 arrays.

    rows: optional token subset whose outputs are produced (keys / values still cover
    every token).  want=True also returns a dict of intermediates.
    """
    d, H, dh, C = cfg.dim, cfg.n_heads, cfg.head_dim, cfg.ffn_chunk
    eps = cfg.ln_eps
    N = x.shape[0]
    if int(masks["block_gate"][step, layer]) == 0:          # R8
        out = _rows(x, rows).copy()
        return (out, {}) if want else out
    sh_a, sc_a, g_a, sh_f, sc_f, g_f = modulation(shared["w_t"], shared["b_t"], lw["e_mod"], t_emb)
    hg = masks["head_gate"][step, layer].astype(np.float64)
    keep = np.repeat(hg, dh)
    tok = _token_ids(N, rows)
    inter = {}

    xm = adaln(x, sh_a, sc_a, eps)
    xr = _rows(x, rows)
    x1 = xr.copy()
    if hg.sum() > 0:
        q = linear(_rows(xm, rows), lw["wq"], lw["bq"])
        k = linear(xm, lw["wk"], lw["bk"])
        v = linear(xm, lw["wv"], lw["bv"])
        q = rms_norm(q, lw["gq"], keep, eps, cfg.qk_norm_mode, dh)
        k = rms_norm(k, lw["gk"], keep, eps, cfg.qk_norm_mode, dh)
        ang = rope_angles(cfg.grid, dh, cfg.rope_theta)
        q = apply_rope(q.reshape(-1, H, dh), ang[tok])
        k = apply_rope(k.reshape(N, H, dh), ang)
        o = attention(q, k, v.reshape(N, H, dh))
        o = o * hg[None, :, None]                               # Eq. 2, head gates
        o = o.reshape(-1, d)
        inter.update(q=q, k=k, v=v.reshape(N, H, dh), o=o)
    else:
        o = np.zeros((xr.shape[0], d))
    x1 = x1 + g_a * linear(o, lw["wo"], lw["bo"])

    if cfg.has_cross:
        inter["x1a"] = x1
        x1 = x1 + _cross_masked(cfg, lw, masks, step, layer, x1, ctx, inter)

    xm2 = adaln(x1, sh_f, sc_f, eps)
    u = gelu_tanh(linear(xm2, lw["w_up"], lw["b_up"]))
    u = u * ffn_channel_gate(masks["ffn_gate"][step, layer], C)  # Eq. 2, chunk gates
    out = x1 + g_f * linear(u, lw["w_down"], lw["b_down"])
    if want:
        inter.update(xm=_rows(xm, rows), x1=x1, xm2=xm2, u=u, out=out)
        return out, inter
    return out


def cross_input_norm(x1, cln_w, cln_b, eps: float) -> np.ndarray:
    """Input of the cross-attention (R6): an affine LayerNorm of the residual x1,
    LN(x1) * cln_w + cln_b, with the LayerNorm of R3."""
    return layer_norm(x1, eps, cln_w, cln_b)


def _cross_masked(cfg, lw, masks, step, layer, x1, ctx, inter=None):
    d, H, dh, eps = cfg.dim, cfg.n_heads, cfg.head_dim, cfg.ln_eps
    xg = masks.get("xhead_gate")
    hg = np.ones(H) if xg is None else xg[step, layer].astype(np.float64)
    if hg.sum() == 0:
        return np.zeros_like(x1) + lw["cbo"]
    keep = np.repeat(hg, dh)
    xc = cross_input_norm(x1, lw["cln_w"], lw["cln_b"], eps)
    if inter is not None:
        inter["xc"] = xc
    q = rms_norm(linear(xc, lw["cwq"], lw["cbq"]), lw["cgq"], keep, eps, cfg.qk_norm_mode, dh)
    k = rms_norm(linear(ctx, lw["cwk"], lw["cbk"]), lw["cgk"], keep, eps, cfg.qk_norm_mode, dh)
    v = linear(ctx, lw["cwv"], lw["cbv"])
    L = ctx.shape[0]
    o = attention(q.reshape(-1, H, dh), k.reshape(L, H, dh), v.reshape(L, H, dh))
    o = (o * hg[None, :, None]).reshape(-1, d)
    return linear(o, lw["cwo"], lw["cbo"])


def block_forward_compacted(cfg, shared, lw, masks, step: int, layer: int, x, t_emb, ctx=None,
                            rows=None, want: bool = False, counter: Optional[MacCounter] = None):
    """The exported per-step dense block (Sec. 3.2, Sec. 4.3): weights are gathered by
    the index table and every contraction runs over the retained units only."""
    dh, eps = cfg.head_dim, cfg.ln_eps
    N = x.shape[0]
    if int(masks["block_gate"][step, layer]) == 0:
        out = _rows(x, rows).copy()
        return (out, {}) if want else out
    idx = compact_indices(cfg, masks, step, layer)
    P = compact_panels(lw, idx)
    h_s = len(idx["heads"])
    sh_a, sc_a, g_a, sh_f, sc_f, g_f = modulation(shared["w_t"], shared["b_t"], lw["e_mod"], t_emb)
    tok = _token_ids(N, rows)
    inter = {}

    xm = adaln(x, sh_a, sc_a, eps)
    xr = _rows(x, rows)
    if h_s > 0:
        w = P["wqkv"]
        hd = h_s * dh
        ones = np.ones(hd)
        q = linear(_rows(xm, rows), w[:hd], P["bqkv"][:hd], counter)
        kv = linear(xm, w[hd:], P["bqkv"][hd:], counter)
        k, v = kv[:, :hd], kv[:, hd:]
        q = rms_norm(q, P["gq"], ones, eps, cfg.qk_norm_mode, dh)
        k = rms_norm(k, P["gk"], ones, eps, cfg.qk_norm_mode, dh)
        ang = rope_angles(cfg.grid, dh, cfg.rope_theta)
        q = apply_rope(q.reshape(-1, h_s, dh), ang[tok])
        k = apply_rope(k.reshape(N, h_s, dh), ang)
        o = attention(q, k, v.reshape(N, h_s, dh), counter).reshape(-1, hd)
        inter.update(q=q, k=k, v=v.reshape(N, h_s, dh), o=o)
        x1 = xr + g_a * linear(o, P["wo"], lw["bo"], counter)
    else:
        x1 = xr + g_a * lw["bo"]

    if cfg.has_cross:
        inter["x1a"] = x1
        x1 = x1 + _cross_compacted(cfg, lw, P, idx, x1, ctx, counter, inter)
        inter["x1c"] = x1

    xm2 = adaln(x1, sh_f, sc_f, eps)
    if len(idx["chunks"]) > 0:
        u = gelu_tanh(linear(xm2, P["w_up"], P["b_up"], counter))
        out = x1 + g_f * linear(u, P["w_down"], lw["b_down"], counter)
    else:
        u = np.zeros((x1.shape[0], 0))
        out = x1 + g_f * lw["b_down"]
    if want:
        inter.update(xm=_rows(xm, rows), x1=x1, xm2=xm2, u=u, out=out)
        return out, inter
    return out


def _cross_compacted(cfg, lw, P, idx, x1, ctx, counter, inter=None):
    dh, eps = cfg.head_dim, cfg.ln_eps
    hc = len(idx["xheads"])
    if hc == 0:
        return np.zeros_like(x1) + lw["cbo"]
    hd = hc * dh
    ones = np.ones(hd)
    xc = cross_input_norm(x1, lw["cln_w"], lw["cln_b"], eps)
    if inter is not None:
        inter["xc"] = xc
    q = rms_norm(linear(xc, P["cwq"], P["cbq"], counter), P["cgq"], ones, eps, cfg.qk_norm_mode, dh)
    kv = linear(ctx, P["cwkv"], P["cbkv"], counter)
    k = rms_norm(kv[:, :hd], P["cgk"], ones, eps, cfg.qk_norm_mode, dh)
    v = kv[:, hd:]
    L = ctx.shape[0]
    o = attention(q.reshape(-1, hc, dh), k.reshape(L, hc, dh), v.reshape(L, hc, dh), counter)
    return linear(o.reshape(-1, hd), P["cwo"], lw["cbo"], counter)


# ---------------------------------------------------------------------------------------
# FLOPs and the denoising loop
# ---------------------------------------------------------------------------------------

def block_flops(n_tokens: int, dim: int, head_dim: int, h_s: int, f_s: int,
                hc_s: int = 0, ctx_len: int = 0) -> float:
    """Algorithmic FLOPs of one pruned block at one step (2 per multiply-add).

    QKV (6) + output (2) projections: 8 N d dh h_s; attention QK^T + PV: 4 N^2 dh h_s;
    FFN up + down: 4 N d f_s; cross-attention Q + O projections 4 N d dh hc, context
    K + V projections 4 L d dh hc, attention 4 N L dh hc.
    """
    N, d = float(n_tokens), float(dim)
    f = 8 * N * d * head_dim * h_s + 4 * N * N * head_dim * h_s + 4 * N * d * f_s
    if hc_s:
        f += 4 * N * d * head_dim * hc_s + 4 * ctx_len * d * head_dim * hc_s \
            + 4 * N * ctx_len * head_dim * hc_s
    return f


def denoise(cfg, shared, layers: List[Dict[str, np.ndarray]], masks, latents, t_embs, ctx=None,
            n_steps: Optional[int] = None):
    """Few-step loop (R9): at step s every layer runs with its step-s structure, then
    x <- x + (1/T) * v with v the output of the last layer."""
    T = cfg.n_steps if n_steps is None else n_steps
    x = latents.copy()
    for s in range(T):
        h = x
        for l in range(cfg.n_layers):
            h = block_forward_masked(cfg, shared, layers[l], masks, s, l, h, t_embs[s], ctx)
        x = x + (1.0 / cfg.n_steps) * h
    return x


# ---------------------------------------------------------------------------------------
# the Wan-shaped model around the blocks (R16-R19)
# ---------------------------------------------------------------------------------------

PATCH = (1, 2, 2)


def patchify(latent) -> np.ndarray:
    """[C, F, H, W] -> [F * H/2 * W/2, 4 C] (R16): the 2 x 2 patch at (f, y, x) becomes token
    (f * H/2 + y) * W/2 + x with feature c*4 + dy*2 + dx = latent[c, f, 2y + dy, 2x + dx]."""
    C, F, H, W = latent.shape
    gh, gw = H // 2, W // 2
    out = np.empty((F * gh * gw, 4 * C), dtype=latent.dtype)
    for c in range(C):
        for dy in range(2):
            for dx in range(2):
                out[:, c * 4 + dy * 2 + dx] = latent[c, :, dy::2, dx::2].reshape(-1)
    return out


def unpatchify(tokens, shape) -> np.ndarray:
    """Inverse of ``patchify`` for a latent of the given [C, F, H, W] shape."""
    C, F, H, W = shape
    out = np.empty(shape, dtype=tokens.dtype)
    for c in range(C):
        for dy in range(2):
            for dx in range(2):
                out[c, :, dy::2, dx::2] = tokens[:, c * 4 + dy * 2 + dx].reshape(F, H // 2, W // 2)
    return out


def timestep_embedding(t: float, dim: int) -> np.ndarray:
    """[cos(t w), sin(t w)] with w_i = 10000^(-i / (dim/2)) (R17)."""
    half = dim // 2
    w = 10000.0 ** (-np.arange(half, dtype=np.float64) / half)
    return np.concatenate([np.cos(t * w), np.sin(t * w)])


def time_mlp(mw, t: float) -> np.ndarray:
    """t_emb = W_2 SiLU(W_1 e + b_1) + b_2 (R17)."""
    e = timestep_embedding(t, mw["t_w1"].shape[1])
    h = mw["t_w1"] @ e + mw["t_b1"]
    h = h / (1.0 + np.exp(-h))
    return mw["t_w2"] @ h + mw["t_b2"]


def output_head(x, head_mod, t_emb, head_w, head_b, eps: float) -> np.ndarray:
    """Output head of the model (R18) on token rows x [n, d]: shift_h = head_mod[0] + t_emb,
    scale_h = head_mod[1] + t_emb, y = LN(x) (1 + scale_h) + shift_h, returns y W_h^T + b_h
    ([n, 4 C], still in token layout)."""
    shift = head_mod[0] + t_emb
    scale = head_mod[1] + t_emb
    return linear(adaln(x, shift, scale, eps), head_w, head_b)


def model_forward(cfg, shared, layers, mw, masks, step: int, latent, t: float, ctx=None, want: bool = False):
    """One pass of the Wan-shaped model at denoising step `step` (R16-R18): patch embedding,
    every block with its step-`step` structure (masked-dense form), output head; returns the
    velocity in latent layout [C, F, H, W]."""
    t_emb = time_mlp(mw, t)
    x = linear(patchify(latent), mw["patch_w"], mw["patch_b"])
    for l in range(cfg.n_layers):
        x = block_forward_masked(cfg, shared, layers[l], masks, step, l, x, t_emb, ctx)
    v = unpatchify(output_head(x, mw["head_mod"], t_emb, mw["head_w"], mw["head_b"], cfg.ln_eps),
                   latent.shape)
    return (v, {"t_emb": t_emb, "x_last": x}) if want else v


def model_denoise(cfg, shared, layers, mw, masks, latent, timesteps, ctx=None):
    """T steps of z <- z + (1/T) v(z, t_s) with step s's structure (R19)."""
    z = latent.copy()
    for s, t in enumerate(timesteps):
        z = z + (1.0 / cfg.n_steps) * model_forward(cfg, shared, layers, mw, masks, s, z, t, ctx)
    return z
