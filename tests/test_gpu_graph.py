"""CUDA graph capture of the forward entry points (through the C ABI).

The block forward, the few-step denoise and the model denoise enqueue only kernel launches
and device-to-device copies on the caller's stream, with no allocation and no
synchronisation, so one call can be captured into a CUDA graph and replayed: every replay
must give the eager call's result bit for bit (including a replay after the inputs were
overwritten in place, since a graph reuses the pointers of its capture)."""
import copy

import numpy as np
import pytest

import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2607_06631_gb300 import build
    build.build()


def _capture(fn):
    import torch
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        fn(torch.cuda.current_stream())
    return g


@pytest.mark.parametrize("engine", [0, 1])
def test_graph_replay_of_denoise_equals_eager(engine):
    import torch
    from paper_2607_06631_gb300 import dfs, host
    cfg = copy.deepcopy(synth.small_stack(4))
    cfg.engine = engine
    shared, layers, m, acts = synth.make_problem(cfg)
    m["block_gate"][2, 1] = 0                     # a gated-off block: a device-to-device copy node
    prob = host.DeviceProblem(cfg, shared, layers, m, acts)
    plan = prob.create_plan()
    lat = prob.x.clone()
    dfs.dfs_denoise(plan, lat, cfg.n_steps, prob.t_emb)
    dfs.dfs_plan_sync(plan)
    want = host.to_bits(lat)

    z = torch.empty_like(prob.x)

    def step(stream):
        z.copy_(prob.x)
        dfs.dfs_denoise(plan, z, cfg.n_steps, prob.t_emb, stream)

    g = _capture(step)
    for _ in range(2):
        z.zero_()
        g.replay()
        torch.cuda.synchronize()
        dfs.dfs_plan_sync(plan)
        np.testing.assert_array_equal(host.to_bits(z), want)


def test_graph_replay_of_block_forwards_follows_new_inputs():
    """Four block forwards (one per step) in one graph; replaying after writing a new x into
    the captured input buffer gives the eager result for that new x."""
    import torch
    from paper_2607_06631_gb300 import dfs, host
    cfg = synth.tiny()
    shared, layers, m, acts = synth.make_problem(cfg)
    prob = host.DeviceProblem(cfg, shared, layers, m, acts)
    plan = prob.create_plan()
    x = prob.x.clone()
    outs = [torch.empty_like(x) for _ in range(cfg.n_steps)]

    def eager(xin):
        res = []
        for s in range(cfg.n_steps):
            o = torch.empty_like(xin)
            dfs.dfs_block_forward(plan, s, xin, prob.t_emb[s], o)
            res.append(o)
        dfs.dfs_plan_sync(plan)
        return [host.to_bits(o) for o in res]

    def fwd(stream):
        for s in range(cfg.n_steps):
            dfs.dfs_block_forward(plan, s, x, prob.t_emb[s], outs[s], stream)

    want0 = eager(x)
    g = _capture(fwd)
    g.replay()
    torch.cuda.synchronize()
    for s in range(cfg.n_steps):
        np.testing.assert_array_equal(host.to_bits(outs[s]), want0[s])
    x.mul_(-0.5)
    want1 = eager(x)
    g.replay()
    torch.cuda.synchronize()
    dfs.dfs_plan_sync(plan)
    for s in range(cfg.n_steps):
        np.testing.assert_array_equal(host.to_bits(outs[s]), want1[s])
    assert any((want0[s] != want1[s]).any() for s in range(cfg.n_steps))


def test_graph_replay_of_model_denoise_equals_eager():
    import torch
    from paper_2607_06631_gb300 import dfs, host
    cfg = synth.tiny_model()
    shared, layers, m, acts = synth.make_problem(cfg)
    prob = host.DeviceProblem(cfg, shared, layers, m, acts)
    prob.create_plan()
    mw = synth.make_model_weights(cfg)
    dmw = {k: host.to_device(v) for k, v in mw.items()}
    dfs.dfs_model_attach(prob.plan, dmw, cfg.latent_channels, cfg.freq_dim)
    lat0 = host.to_device(synth.make_latent(cfg))
    ts = synth.model_timesteps(cfg.n_steps)
    z = lat0.clone()
    dfs.dfs_model_denoise(prob.plan, z, cfg.n_steps, ts)
    dfs.dfs_plan_sync(prob.plan)
    want = host.to_bits(z)

    def step(stream):
        z.copy_(lat0)
        dfs.dfs_model_denoise(prob.plan, z, cfg.n_steps, ts, stream)

    g = _capture(step)
    for _ in range(2):
        z.zero_()
        g.replay()
        torch.cuda.synchronize()
        dfs.dfs_plan_sync(prob.plan)
        np.testing.assert_array_equal(host.to_bits(z), want)
