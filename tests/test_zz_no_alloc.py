"""The allocation-free forward (dfs_block_forward_noalloc) against the regular one.

It serves callers that may not allocate device memory while the model runs (a host that
owns all device memory through its own pool, a latency-critical loop that cannot take
cudaMalloc's implicit synchronisation).  Its workspace is a static 16 MiB device array,
so it must give the same block output as dfs_block_forward_layer on the same plan, call
after call, and refuse problems whose workspace does not fit.  This file is named to be
collected last."""
import numpy as np
import pytest

import synth
from gpu_helpers import TOL, rel_err

pytestmark = pytest.mark.gpu


def _plan(cfg):
    from paper_2607_06631_gb300 import build, host
    build.build()
    shared, layers, masks, acts = synth.make_problem(cfg)
    prob = host.DeviceProblem(cfg, shared, layers, masks, acts)
    prob.create_plan()
    return prob


def test_noalloc_forward_matches_regular_forward_on_consecutive_calls():
    import torch
    from paper_2607_06631_gb300 import dfs, host
    cfg = synth.tiny()
    prob = _plan(cfg)
    ref = torch.empty_like(prob.x)
    got = torch.empty_like(prob.x)
    for step in (1, 3, 1):  # consecutive calls share (and overwrite) the static scratch
        dfs.dfs_block_forward_layer(prob.plan, step, 0, prob.x, prob.t_emb[step], ref)
        got.fill_(0)
        dfs.dfs_block_forward_noalloc(prob.plan, step, 0, prob.x, prob.t_emb[step], got)
        dfs.dfs_plan_sync(prob.plan)
        a = synth.bits_to_f64(host.to_bits(got))
        b = synth.bits_to_f64(host.to_bits(ref))
        assert rel_err(a, b) <= TOL, (step, rel_err(a, b))


def test_noalloc_forward_with_cross_attention():
    import torch
    from paper_2607_06631_gb300 import dfs, host
    cfg = synth.tiny(has_cross=1)
    prob = _plan(cfg)
    ref = torch.empty_like(prob.x)
    got = torch.empty_like(prob.x)
    for step in (0, 2):
        dfs.dfs_block_forward_layer(prob.plan, step, 0, prob.x, prob.t_emb[step], ref)
        dfs.dfs_block_forward_noalloc(prob.plan, step, 0, prob.x, prob.t_emb[step], got)
        dfs.dfs_plan_sync(prob.plan)
        assert rel_err(synth.bits_to_f64(host.to_bits(got)), synth.bits_to_f64(host.to_bits(ref))) <= TOL


def test_noalloc_forward_rejects_workspace_beyond_the_static_array():
    import torch
    from paper_2607_06631_gb300 import dfs
    cfg = synth.tiny(grid=(4, 32, 32))  # 4096 tokens: about 23 MB of workspace
    cfg.name = "tiny_4096"
    prob = _plan(cfg)
    out = torch.empty_like(prob.x)
    with pytest.raises(dfs.DfsError) as e:
        dfs.dfs_block_forward_noalloc(prob.plan, 0, 0, prob.x, prob.t_emb[0], out)
    assert e.value.status == dfs.DFS_EUNSUPPORTED
    assert "scratch" in str(e.value)
