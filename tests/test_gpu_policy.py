"""GPU parity on the policy-shaped mask workload (masks shaped like the learned policy the
paper analyses in Sec. 6: U-shaped per-step retention, deep layers' attention pruned hardest
in the middle steps, the deepest layer's attention shut down, the FFN pruned less).

The whole few-step denoise of a 12-layer tiny-shaped stack against the oracle's denoise
(both engines, bit-identical to each other), and single blocks of the 30-layer
Wan-1.3B-shaped policy at full size (32760 tokens) on sampled query rows, including a
layer whose self- and cross-attention keep no head."""
import copy

import numpy as np
import pytest

import oracle as O
import synth
from gpu_helpers import TOL, branch_err, rel_err

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2607_06631_gb300 import build
    build.build()


def test_policy_small_stack_denoise_both_engines():
    from paper_2607_06631_gb300 import dfs, host
    cfg = synth.policy_small()
    shared, layers, m, acts = synth.make_problem(cfg)
    assert m["head_gate"][1, -1].sum() == 0 and m["xhead_gate"][2, -1].sum() == 0
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
    W, LW, X = synth.widen(shared), synth.widen(layers), synth.widen(acts)
    ref = O.denoise(cfg, W, LW, m, X["x"], X["t_emb"], X["ctx"])
    got = synth.bits_to_f64(outs[0])
    assert rel_err(got, ref) <= TOL
    assert branch_err(got, ref, X["x"]) <= TOL


def _subset(cfg, layers):
    """The same shapes with the policy masks of a subset of the layers."""
    c = copy.deepcopy(cfg)
    c.n_layers = len(layers)
    c.heads_kept = [[h[l] for l in layers] for h in cfg.heads_kept]
    c.chunks_kept = [[k[l] for l in layers] for k in cfg.chunks_kept]
    c.xheads_kept = [[h[l] for l in layers] for h in cfg.xheads_kept]
    c.name = cfg.name + "_layers" + "-".join(map(str, layers))
    return c


@pytest.mark.slow
def test_wan13b_policy_blocks_full_size():
    """Layers 0, 20 and 29 of the 30-layer policy: step 0 of the shallow layer (every head),
    steps 1 and 2 of the deep ones (few heads; layer 29 keeps none)."""
    import torch
    from paper_2607_06631_gb300 import dfs, host
    from test_gpu_large import sample_rows
    full = synth.wan13b_policy()
    pick = (0, 20, 29)
    cfg = _subset(full, pick)
    cases = ((0, 0), (1, 1), (2, 1), (1, 2), (2, 2))   # (step, index into pick)
    assert cfg.heads_kept[1][2] == 0 and cfg.heads_kept[2][2] == 0
    shared, layers, masks, acts = synth.make_problem(cfg)
    prob = host.DeviceProblem(cfg, shared, layers, masks, acts)
    prob.create_plan()
    prob.free_weights()
    out = torch.empty_like(prob.x)
    rows = sample_rows(cfg.n_tokens, 32, 64)
    gpu = {}
    for s, li in cases:
        dfs.dfs_block_forward_layer(prob.plan, s, li, prob.x, prob.t_emb[s], out)
        dfs.dfs_plan_sync(prob.plan)
        gpu[(s, li)] = out[torch.from_numpy(rows).cuda()].clone()
    del prob
    torch.cuda.empty_cache()
    W, LW, X = synth.widen(shared), synth.widen(layers), synth.widen(acts)
    for (s, li), g in gpu.items():
        ref = O.block_forward_compacted(cfg, W, LW[li], masks, s, li, X["x"], X["t_emb"][s], X["ctx"], rows=rows)
        got = synth.bits_to_f64(host.to_bits(g))
        e, b = rel_err(got, ref), branch_err(got, ref, X["x"][rows])
        assert e <= TOL and b <= TOL, (s, pick[li], e, b)
