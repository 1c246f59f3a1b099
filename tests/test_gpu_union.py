"""GPU parity of the union engine (DFS_ENGINE_UNION, Sec. 4.3 / Fig. 1(c)): one union
super-model per layer plus the per-step index tables I_t, with every projection gathering
its step's rows / columns from the union inside its TMA producer.

Checks, through the C ABI: the union id lists and the I_t positions against the oracle's
union_tables (bit-exact), the union weight panels against the oracle's union_panels
(bit-exact), the block output against the oracle (tolerance) and against the compacted
engine on the same inputs (bit-identical: the same operands reach the tensor cores in the
same order), the denoising loop, and the weight memory against its closed form."""
import copy

import numpy as np
import pytest

import oracle as O
import synth
from gpu_helpers import check_block, run_block
from test_gpu_block import _custom

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2607_06631_gb300 import build
    build.build()


def _union(cfg):
    c = copy.deepcopy(cfg)
    c.engine = 1
    return c


def _hand_masks():
    cfg = synth.tiny(has_cross=1)
    m = synth.make_masks(cfg)
    m["head_gate"][:, 0, :] = np.array([[1, 0, 0, 1], [0, 0, 1, 1], [0, 0, 0, 1], [1, 0, 0, 0]])
    m["xhead_gate"][:, 0, :] = np.array([[0, 0, 0, 1], [0, 0, 0, 1], [0, 1, 0, 0], [0, 1, 0, 1]])
    m["ffn_gate"][:] = 0
    m["ffn_gate"][0, 0, [0, 7]] = 1
    m["ffn_gate"][1, 0, [3]] = 1
    m["ffn_gate"][3, 0, [3, 7, 9]] = 1
    return cfg, m


@pytest.mark.parametrize("hand", [False, True])
def test_union_tables_and_panels_bit_exact(hand):
    from paper_2607_06631_gb300 import dfs, host
    if hand:
        cfg, m = _hand_masks()
    else:
        cfg = synth.tiny(has_cross=1)
        m = None
    cfg = _union(cfg)
    r0, _ = run_block(cfg, masks=m, steps=[], want_intermediates=False)
    plan, m, lw = r0["plan"], r0["masks"], r0["layers"][0]
    u = O.union_tables(cfg, m, 0)
    for kind, key in ((3, "heads"), (4, "chunks"), (5, "xheads")):
        np.testing.assert_array_equal(dfs.dfs_plan_indices(plan, 0, 0, kind), u[key], err_msg=key)
    for s in range(cfg.n_steps):
        for kind, key in ((6, "pos_heads"), (7, "pos_chunks"), (8, "pos_xheads")):
            np.testing.assert_array_equal(dfs.dfs_plan_indices(plan, s, 0, kind), u[key][s], err_msg=(s, key))
        P = O.compact_panels(lw, O.compact_indices(cfg, m, s, 0))
        for name in ("bqkv", "gq", "gk", "b_up", "cbq", "cgq", "cgk"):
            np.testing.assert_array_equal(host.read_panel(plan, s, 0, name)[0], P[name], err_msg=name)
        for name in ("wqkv", "wo", "w_up", "w_down", "cwq", "cwkv", "cwo"):
            assert dfs.dfs_plan_panel(plan, s, 0, name)[0] == 0, name   # no per-step copy
    U = O.union_panels(cfg, lw, u)
    for name in ("wqkv", "wo", "w_up", "w_down", "cwq", "cwo"):
        np.testing.assert_array_equal(host.read_union_panel(plan, 0, name), U[name], err_msg=name)


def _both_engines(cfg, masks=None, steps=None):
    r0c, rc = run_block(cfg, masks=masks, steps=steps)
    r0u, ru = run_block(_union(cfg), masks=masks, steps=steps)
    for a, b in zip(rc, ru):
        np.testing.assert_array_equal(b["out"], a["out"], err_msg="step %d" % a["step"])
    return r0u, ru


@pytest.mark.parametrize("mode", [0, 1])
def test_union_tiny_every_step(mode):
    cfg = synth.tiny(qk_norm_mode=mode)
    r0, res = _both_engines(cfg)
    check_block(_union(cfg), r0, res)


@pytest.mark.parametrize("kw", [dict(grid=(1, 5, 7)), dict(grid=(3, 10, 13)),
                                dict(heads=(1, 2, 1, 4), chunks=(9, 1, 33, 128)),
                                dict(dim=512, n_heads=4, head_dim=128, ffn=1024, heads=(4, 3, 2, 1),
                                     chunks=(128, 100, 50, 16), grid=(2, 8, 20)),
                                dict(dim=1024, n_heads=8, head_dim=128, ffn=2048, heads=(3, 8, 5, 1),
                                     chunks=(17, 256, 131, 40), grid=(2, 6, 30))])
def test_union_ragged_shapes(kw):
    """Ragged token counts, f_s = 72 / 8 (K tails inside a K block of 64), single heads,
    head_dim 128 (one head per 128-row B half) and several N / K tiles."""
    cfg = _custom(**kw)
    r0, res = _both_engines(cfg)
    check_block(_union(cfg), r0, res)


def test_union_cross_attention_and_hand_masks():
    cfg, m = _hand_masks()
    r0, res = _both_engines(cfg, masks=m)
    check_block(_union(cfg), r0, res)


def test_union_empty_masks_and_block_gate():
    cfg = synth.tiny()
    m = synth.make_masks(cfg)
    m["head_gate"][1, 0, :] = 0
    m["ffn_gate"][2, 0, :] = 0
    m["head_gate"][3, 0, :] = 0
    m["ffn_gate"][3, 0, :] = 0
    m["block_gate"][0, 0] = 0
    r0, res = _both_engines(cfg, masks=m)
    check_block(_union(cfg), r0, res, check_intermediates=False)


def test_union_denoise_small_stack_matches_compacted():
    import torch
    from paper_2607_06631_gb300 import dfs, host
    cfg = synth.small_stack(4)
    shared, layers, m, acts = synth.make_problem(cfg)
    m["block_gate"][2, 1] = 0
    outs = []
    for eng in (0, 1):
        c = copy.deepcopy(cfg)
        c.engine = eng
        prob = host.DeviceProblem(c, shared, layers, m, acts)
        plan = prob.create_plan()
        lat = prob.x.clone()
        dfs.dfs_denoise(plan, lat, cfg.n_steps, prob.t_emb)
        dfs.dfs_plan_sync(plan)
        outs.append(host.to_bits(lat))
    np.testing.assert_array_equal(outs[1], outs[0])


def test_union_weight_memory_closed_form():
    """The union engine holds each union unit's weights once; the compacted engine holds
    every step's retained weights (plus, in both, the small per-step vectors)."""
    from paper_2607_06631_gb300 import dfs
    cfg = synth.tiny(has_cross=1)
    cfg.heads_kept = [[2], [3], [1], [2]]
    cfg.chunks_kept = [[40], [90], [7], [64]]
    m = synth.make_masks(cfg, "mem")
    r0c, _ = run_block(cfg, masks=m, steps=[], want_intermediates=False)
    r0u, _ = run_block(_union(cfg), masks=m, steps=[], want_intermediates=False)
    wc, _ = dfs.dfs_plan_memory(r0c["plan"])
    wu, _ = dfs.dfs_plan_memory(r0u["plan"])
    d, dh, C = cfg.dim, cfg.head_dim, cfg.ffn_chunk
    u = O.union_tables(cfg, m, 0)
    vec = 0
    comp = 0
    for s in range(cfg.n_steps):
        idx = O.compact_indices(cfg, m, s, 0)
        hd, xd, fs = len(idx["heads"]) * dh, len(idx["xheads"]) * dh, len(idx["ffn_ch"])
        vec += 2 * (3 * hd + 2 * hd + fs + xd + 2 * xd + 2 * xd)         # bqkv gq gk b_up cbq cbkv cgq cgk
        # wqkv wo w_up w_down cwq cwkv cwo; W_down's rows padded to a multiple of 64 elements
        comp += 2 * (4 * hd * d + fs * d + d * ((fs + 63) // 64 * 64) + 2 * xd * d + 2 * xd * d)
    nu, nf, nx = len(u["heads"]) * dh, len(u["chunks"]) * C, len(u["xheads"]) * dh
    assert wc == comp + vec
    assert wu == 2 * (4 * nu * d + 2 * nf * d + 2 * nx * d) + vec
    assert wu < wc


def test_union_allocation_free_forward_matches_regular_forward():
    """The allocation-free forward on a union-engine plan (its FFN gathers go to the plan's
    scratch, allocated with the plan) gives the regular forward's output."""
    import torch
    from paper_2607_06631_gb300 import dfs, host
    cfg = _union(synth.tiny(has_cross=1))
    r0, _ = run_block(cfg, steps=[], want_intermediates=False)
    plan, prob = r0["plan"], r0["prob"]
    ref, got = torch.empty_like(prob.x), torch.empty_like(prob.x)
    for step in (3, 0):
        dfs.dfs_block_forward_layer(plan, step, 0, prob.x, prob.t_emb[step], ref)
        dfs.dfs_block_forward_noalloc(plan, step, 0, prob.x, prob.t_emb[step], got)
        dfs.dfs_plan_sync(plan)
        np.testing.assert_array_equal(host.to_bits(got), host.to_bits(ref))
