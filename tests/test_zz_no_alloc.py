"""The allocation-free forward (dfs_block_forward_noalloc) against the regular one.

It serves callers that may not allocate device memory while the model runs (a host that
owns all device memory through its own pool, a latency-critical loop that cannot take
cudaMalloc's implicit synchronisation).  Its workspace is a static 16 MiB device array
shared by every call, so each call must give exactly the output of dfs_block_forward_layer
on the same plan (the same kernels run in the same order on the same operands) whatever an
earlier call of another shape left in the array, and must refuse problems whose workspace
does not fit.  This file is named to be collected last."""
import numpy as np
import pytest

import oracle as O
import synth
from gpu_helpers import TOL, branch_err, rel_err

pytestmark = pytest.mark.gpu


def _plan(cfg):
    from paper_2607_06631_gb300 import build, host
    build.build()
    shared, layers, masks, acts = synth.make_problem(cfg)
    prob = host.DeviceProblem(cfg, shared, layers, masks, acts)
    prob.create_plan()
    return prob, (shared, layers, masks, acts)


def _compare(prob, steps):
    """Regular forward, then the allocation-free one on a zero-filled output, per step:
    bit-identical.  Returns the last allocation-free output as float64."""
    import torch
    from paper_2607_06631_gb300 import dfs, host
    ref = torch.empty_like(prob.x)
    got = torch.empty_like(prob.x)
    for step in steps:
        dfs.dfs_block_forward_layer(prob.plan, step, 0, prob.x, prob.t_emb[step], ref)
        got.fill_(0)
        dfs.dfs_block_forward_noalloc(prob.plan, step, 0, prob.x, prob.t_emb[step], got)
        dfs.dfs_plan_sync(prob.plan)
        np.testing.assert_array_equal(host.to_bits(got), host.to_bits(ref), err_msg="step %d" % step)
    return synth.bits_to_f64(host.to_bits(got))


def _oracle_check(cfg, problem, step, got):
    shared, layers, masks, acts = problem
    W, LW, X = synth.widen(shared), synth.widen(layers), synth.widen(acts)
    ref = O.block_forward_compacted(cfg, W, LW[0], masks, step, 0, X["x"], X["t_emb"][step], X.get("ctx"))
    assert rel_err(got, ref) <= TOL, rel_err(got, ref)
    assert branch_err(got, ref, X["x"]) <= TOL, branch_err(got, ref, X["x"])


def test_noalloc_forward_matches_regular_forward_on_consecutive_calls():
    cfg = synth.tiny()
    prob, problem = _plan(cfg)
    # consecutive calls share (and overwrite) the static array; steps differ in h_s and f_s,
    # so each call finds the array carved differently by the one before
    got = _compare(prob, (1, 3, 0, 2, 1))
    _oracle_check(cfg, problem, 1, got)


def test_noalloc_forward_with_cross_attention():
    cfg = synth.tiny(has_cross=1)
    prob, problem = _plan(cfg)
    got = _compare(prob, (0, 2, 3, 1))
    _oracle_check(cfg, problem, 1, got)


def test_noalloc_forward_ragged_tokens_after_a_larger_problem():
    """510 tokens (not a multiple of the 64 / 128 / 256 tiles) right after 512-token calls
    of another plan: the array then holds that plan's values past the 510th row and in
    the V^T padding columns, which no kernel may read."""
    big, _ = _plan(synth.tiny())
    _compare(big, (0, 3))
    cfg = synth.tiny(grid=(2, 15, 17))
    cfg.name = "tiny_ragged_510"
    prob, problem = _plan(cfg)
    got = _compare(prob, (2, 0))
    _oracle_check(cfg, problem, 0, got)


def test_noalloc_forward_on_a_union_engine_plan():
    """Union engine with cross-attention: the FFN panels are gathered into the plan's own
    scratch, the tensor maps of the union gathers are built per call."""
    import copy
    cfg = copy.deepcopy(synth.tiny(has_cross=1))
    cfg.engine = 1
    prob, problem = _plan(cfg)
    got = _compare(prob, (3, 0, 2))
    _oracle_check(cfg, problem, 2, got)


def test_noalloc_forward_rejects_workspace_beyond_the_static_array():
    import torch
    from paper_2607_06631_gb300 import dfs
    cfg = synth.tiny(grid=(4, 32, 32))  # 4096 tokens: about 23 MB of workspace
    cfg.name = "tiny_4096"
    prob, _ = _plan(cfg)
    out = torch.empty_like(prob.x)
    with pytest.raises(dfs.DfsError) as e:
        dfs.dfs_block_forward_noalloc(prob.plan, 0, 0, prob.x, prob.t_emb[0], out)
    assert e.value.status == dfs.DFS_EUNSUPPORTED
    assert "scratch" in str(e.value)
    # the workspace formula of the header, every term rounded up to 256 bytes
    r = lambda b: (b + 255) // 256 * 256
    N, d, dh = cfg.n_tokens, cfg.dim, cfg.head_dim
    h, f = cfg.heads_kept[0][0] * dh, 8 * cfg.chunks_kept[0][0]
    need = (r(24 * d) + r(2 * N * d) + r(4 * N * h) + r(2 * h * ((N + 63) // 64 * 64)) + r(2 * N * h)
            + r(4 * N * d) + r(2 * N * ((f + 63) // 64 * 64)))
    assert ("needs %d bytes" % need) in str(e.value), (need, str(e.value))
