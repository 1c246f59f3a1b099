"""GPU parity of the Wan-shaped model around the blocks (patch embedding, timestep MLP,
output head, latent-space sampling) against the oracle's model_forward / model_denoise.

Tiny-shaped 4-layer model with cross-attention on a 16 x 2 x 16 x 16 latent: every step's
velocity, the 4-step denoise (both engines, bit-identical), argument checks; and a
one-layer Wan-1.3B-shaped model at full size (latent 16 x 21 x 60 x 104, 32760 tokens) on
sampled tokens."""
import copy

import numpy as np
import pytest

import oracle as O
import synth
from gpu_helpers import TOL, rel_err

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2607_06631_gb300 import build
    build.build()


def _setup(cfg, engine=0, masks=None):
    from paper_2607_06631_gb300 import dfs, host
    c = copy.deepcopy(cfg)
    c.engine = engine
    shared, layers, m, acts = synth.make_problem(c)
    if masks is not None:
        m = masks
    mw = synth.make_model_weights(c)
    lat = synth.make_latent(c)
    prob = host.DeviceProblem(c, shared, layers, m, acts)
    prob.create_plan()
    dmw = {k: host.to_device(v) for k, v in mw.items()}
    dfs.dfs_model_attach(prob.plan, dmw, c.latent_channels, c.freq_dim)
    return prob, (shared, layers, m, acts, mw, lat)


def _f64(problem):
    shared, layers, m, acts, mw, lat = problem
    return synth.widen(shared), synth.widen(layers), m, synth.widen(acts), synth.widen(mw), synth.bits_to_f64(lat)


def test_tiny_model_velocity_every_step():
    import torch
    from paper_2607_06631_gb300 import dfs, host
    cfg = synth.tiny_model()
    prob, pb = _setup(cfg)
    W, LW, m, X, MW, lat = _f64(pb)
    z = host.to_device(pb[5])
    v = torch.empty_like(z)
    ts = synth.model_timesteps(cfg.n_steps)
    for s in range(cfg.n_steps):
        dfs.dfs_model_forward(prob.plan, s, z, ts[s], v)
        dfs.dfs_plan_sync(prob.plan)
        got = synth.bits_to_f64(host.to_bits(v))
        ref = O.model_forward(cfg, W, LW, MW, m, s, lat, ts[s], X["ctx"])
        assert rel_err(got, ref) <= TOL, (s, rel_err(got, ref))


def test_tiny_model_denoise_both_engines():
    from paper_2607_06631_gb300 import dfs, host
    cfg = synth.tiny_model()
    ts = synth.model_timesteps(cfg.n_steps)
    outs = []
    for eng in (0, 1):
        prob, pb = _setup(cfg, eng)
        z = host.to_device(pb[5])
        dfs.dfs_model_denoise(prob.plan, z, cfg.n_steps, ts)
        dfs.dfs_plan_sync(prob.plan)
        outs.append(host.to_bits(z))
    np.testing.assert_array_equal(outs[1], outs[0])
    W, LW, m, X, MW, lat = _f64(pb)
    ref = O.model_denoise(cfg, W, LW, MW, m, lat, ts, X["ctx"])
    got = synth.bits_to_f64(outs[0])
    assert rel_err(got, ref) <= TOL
    # the accumulated update alone, after one bf16 ulp of |z| for storing the latent each step
    from gpu_helpers import branch_err
    assert branch_err(got, ref, lat) <= 2 * TOL


def test_model_arguments_are_checked():
    import torch
    from paper_2607_06631_gb300 import dfs, host
    cfg = synth.tiny_model(n_layers=1)
    shared, layers, m, acts = synth.make_problem(cfg)
    prob = host.DeviceProblem(cfg, shared, layers, m, acts)
    prob.create_plan()
    z = host.to_device(synth.make_latent(cfg))
    v = torch.empty_like(z)
    with pytest.raises(dfs.DfsError) as e:
        dfs.dfs_model_forward(prob.plan, 0, z, 1000.0, v)          # nothing attached
    assert e.value.status == dfs.DFS_EINVAL
    dmw = {k: host.to_device(a) for k, a in synth.make_model_weights(cfg).items()}
    with pytest.raises(dfs.DfsError) as e:
        dfs.dfs_model_attach(prob.plan, dmw, 15, 256)               # odd channel count
    assert e.value.status == dfs.DFS_EINVAL
    dfs.dfs_model_attach(prob.plan, dmw, 16, 256)
    for args in ((0, z, z), (4, z, v)):
        with pytest.raises(dfs.DfsError) as e:
            dfs.dfs_model_forward(prob.plan, args[0], args[1], 1000.0, args[2])
        assert e.value.status == dfs.DFS_EINVAL


@pytest.mark.slow
def test_wan13b_shaped_one_layer_model_full_size():
    """Latent 16 x 21 x 60 x 104: patch embedding, one 1.3B-shaped block with cross-attention
    (policy masks of layer 20: few heads at steps 1 and 2), head; sampled tokens."""
    import torch
    from paper_2607_06631_gb300 import dfs, host
    from test_gpu_large import sample_rows
    full = synth.wan13b_model()
    cfg = copy.deepcopy(full)
    cfg.n_layers = 1
    cfg.heads_kept = [[h[20]] for h in full.heads_kept]
    cfg.chunks_kept = [[k[20]] for k in full.chunks_kept]
    cfg.xheads_kept = [[h[20]] for h in full.xheads_kept]
    cfg.name = "wan13b_model_layer20"
    prob, pb = _setup(cfg)
    W, LW, m, X, MW, lat = _f64(pb)
    z = host.to_device(pb[5])
    v = torch.empty_like(z)
    ts = synth.model_timesteps(cfg.n_steps)
    rows = sample_rows(cfg.n_tokens, 32, 64)
    for s in (0, 2):
        dfs.dfs_model_forward(prob.plan, s, z, ts[s], v)
        dfs.dfs_plan_sync(prob.plan)
        got = O.patchify(synth.bits_to_f64(host.to_bits(v)))[rows]
        t_emb = O.time_mlp(MW, ts[s])
        x = O.linear(O.patchify(lat), MW["patch_w"], MW["patch_b"])
        xo = O.block_forward_masked(cfg, W, LW[0], m, s, 0, x, t_emb, X["ctx"], rows=rows)
        ref = O.output_head(xo, MW["head_mod"], t_emb, MW["head_w"], MW["head_b"], cfg.ln_eps)
        assert rel_err(got, ref) <= TOL, (s, rel_err(got, ref))
