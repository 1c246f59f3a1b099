"""GPU parity of the CUDA path (through the C ABI) against the float64 oracle."""
import copy

import numpy as np
import pytest

import oracle as O
import synth
from gpu_helpers import TOL, branch_err, check_block, rel_err, run_block

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2607_06631_gb300 import build
    build.build()


@pytest.mark.parametrize("mode", [0, 1])
def test_tiny_every_step(mode):
    cfg = synth.tiny(qk_norm_mode=mode)
    r0, res = run_block(cfg)
    check_block(cfg, r0, res)


def test_tiny_index_lists_panels_and_flops_bit_exact():
    from paper_2607_06631_gb300 import dfs, host
    cfg = synth.tiny()
    r0, _ = run_block(cfg, steps=[], want_intermediates=False)
    plan, m, lw = r0["plan"], r0["masks"], r0["layers"][0]
    for s in range(cfg.n_steps):
        idx = O.compact_indices(cfg, m, s, 0)
        np.testing.assert_array_equal(dfs.dfs_plan_indices(plan, s, 0, 0), idx["heads"])
        np.testing.assert_array_equal(dfs.dfs_plan_indices(plan, s, 0, 1), idx["chunks"])
        P = O.compact_panels(lw, idx)
        for name in ("wqkv", "wo", "w_up", "w_down"):
            np.testing.assert_array_equal(host.read_panel(plan, s, 0, name), P[name], err_msg=name)
        for name in ("bqkv", "gq", "gk", "b_up"):
            np.testing.assert_array_equal(host.read_panel(plan, s, 0, name)[0], P[name], err_msg=name)
        f = O.block_flops(cfg.n_tokens, cfg.dim, cfg.head_dim, len(idx["heads"]), len(idx["ffn_ch"]))
        assert dfs.dfs_plan_flops(plan, s, 0) == f


def _custom(grid=(2, 16, 16), heads=(4, 3, 1, 2), chunks=(128, 9, 80, 64), dim=256, n_heads=4, ffn=1024,
            head_dim=64):
    cfg = synth.tiny(grid=grid)
    cfg.dim, cfg.n_heads, cfg.head_dim, cfg.ffn_dim = dim, n_heads, head_dim, ffn
    cfg.heads_kept = [[h] for h in heads]
    cfg.chunks_kept = [[c] for c in chunks]
    cfg.name = "custom_%s_%s_%s_%d" % ("x".join(map(str, grid)), "-".join(map(str, heads)),
                                       "-".join(map(str, chunks)), head_dim)
    return cfg


@pytest.mark.parametrize("grid", [(1, 5, 7), (3, 10, 13), (1, 1, 8)])
def test_ragged_token_counts(grid):
    """N not a multiple of the 128-row tiles: 35, 390 and 8 tokens."""
    cfg = _custom(grid=grid)
    r0, res = run_block(cfg)
    check_block(cfg, r0, res)


def test_ragged_ffn_and_single_head():
    """f_s = 72 (K tail of 8 inside a 64-wide K block), one retained head."""
    cfg = _custom(heads=(1, 2, 1, 4), chunks=(9, 1, 33, 128))
    r0, res = run_block(cfg)
    check_block(cfg, r0, res)


def test_head_dim_128_tiny():
    cfg = _custom(dim=512, n_heads=4, head_dim=128, ffn=1024, heads=(4, 3, 2, 1), chunks=(128, 100, 50, 16),
                  grid=(2, 8, 20))
    r0, res = run_block(cfg)
    check_block(cfg, r0, res)


@pytest.mark.parametrize("head_dim,gamma", [(64, 4.0), (128, 4.0), (64, 8.0)])
def test_peaky_scores_rescale_the_running_max(head_dim, gamma):
    """q / k norm scales multiplied by gamma make the scores gamma^2 times larger, so that in
    many rows a later key block's P, taken with the offset the row had so far, sums to more
    than 2^16: the kernel then redoes that block with the exact row maximum and rescales the
    row's O accumulator and sum (with the default scales that never happens at these sizes;
    the test counts such blocks by the kernel's rule on the GPU's own q and k).  The attention output is compared with the plain softmax of the GPU's
    own bf16 q, k and V (the attention kernel alone; upstream bf16 rounding of q and k moves
    such peaky scores by more than the block tolerance), and, at gamma 4, the block output
    with the oracle at a tolerance that allows for that rounding (630 tokens: a ragged
    last key block)."""
    if head_dim == 64:
        cfg = _custom(grid=(2, 15, 21))
    else:
        cfg = _custom(dim=512, n_heads=4, head_dim=128, ffn=1024, heads=(4, 3, 2, 1), chunks=(128, 100, 50, 16),
                      grid=(2, 15, 21))

    def scale_gammas(layers):
        for lw in layers:
            for k in ("gq", "gk"):
                lw[k] = synth.f32_to_bf16_bits(synth.bits_to_f32(lw[k]) * gamma)

    r0, res = run_block(cfg, steps=[0, 2], patch=scale_gammas)
    dh = cfg.head_dim
    sl2 = np.log2(np.e) / np.sqrt(dh)
    redos = 0
    for r in res:
        N = r["ws_qk"].shape[0]
        hd = r["ws_qk"].shape[1] // 2
        q = r["ws_qk"][:, :hd].reshape(N, -1, dh)
        k = r["ws_qk"][:, hd:].reshape(N, -1, dh)
        v = r["ws_vt"].T.reshape(N, -1, dh)
        want = O.attention(q, k, v).reshape(N, hd)
        assert rel_err(r["ws_attn"], want) <= 1e-2, ("attn vs softmax of the GPU's q, k, v", r["step"],
                                                      rel_err(r["ws_attn"], want))
        for h in range(q.shape[1]):
            S = (q[:, h] @ k[:, h].T) * sl2
            m_run = S[:, :128].max(1)
            for j in range(1, (N + 127) // 128):
                blk = S[:, 128 * j:128 * (j + 1)]
                redo = ~(np.exp2(blk - m_run[:, None]).sum(1) <= 65536.0)
                redos += int(redo.sum())
                m_run = np.where(redo, np.maximum(m_run, blk.max(1)), m_run)
        if gamma <= 4:
            assert branch_err(r["out"], r["ref"], r0["x"]) <= 0.1, ("out - x", r["step"])
    assert redos > 100, redos


def test_wide_rows_above_5120_channels():
    """dim 6144 (48 heads x 128): the LayerNorm's 256-thread row layout, 1536-channel q / k rows."""
    cfg = _custom(dim=6144, n_heads=48, head_dim=128, ffn=2048, heads=(48, 12, 30, 1), chunks=(256, 40, 128, 9),
                  grid=(2, 4, 5))
    r0, res = run_block(cfg)
    check_block(cfg, r0, res)


@pytest.mark.parametrize("case", ["dh128", "ragged", "cross"])
def test_per_head_qk_norm(case):
    """qk_norm_mode 1 (QK RMSNorm per head) with head_dim 128, ragged token counts and
    cross-attention: q, k after RMSNorm + RoPE and the block output against the oracle."""
    if case == "dh128":
        cfg = _custom(dim=512, n_heads=4, head_dim=128, ffn=1024, heads=(4, 3, 2, 1), chunks=(128, 100, 50, 16),
                      grid=(2, 8, 20))
    elif case == "ragged":
        cfg = _custom(grid=(3, 10, 13))
    else:
        cfg = synth.tiny(has_cross=1)
    cfg.qk_norm_mode = 1
    cfg.name += "_mode1"
    r0, res = run_block(cfg)
    check_block(cfg, r0, res)


def test_empty_masks_and_block_gate():
    cfg = synth.tiny()
    m = synth.make_masks(cfg)
    m["head_gate"][1, 0, :] = 0       # step 1: no heads -> x1 = x + gate_a * bo
    m["ffn_gate"][2, 0, :] = 0        # step 2: no FFN chunks -> out = x1 + gate_f * b_down
    m["head_gate"][3, 0, :] = 0
    m["ffn_gate"][3, 0, :] = 0        # step 3: both empty
    m["block_gate"][0, 0] = 0         # step 0: block off -> identity
    r0, res = run_block(cfg, masks=m, want_intermediates=False)
    check_block(cfg, r0, res, check_intermediates=False)
    np.testing.assert_array_equal(res[0]["out"], r0["x"])


def test_cross_attention_block():
    cfg = synth.tiny(has_cross=1)
    r0, res = run_block(cfg)
    check_block(cfg, r0, res)


def test_host_buffers_match_device_buffers():
    import torch
    from paper_2607_06631_gb300 import dfs, host
    cfg = synth.tiny()
    r0, _ = run_block(cfg, steps=[], want_intermediates=False)
    plan, prob = r0["plan"], r0["prob"]
    out = torch.empty_like(prob.x)
    dfs.dfs_block_forward(plan, 2, prob.x, prob.t_emb[2], out)
    dfs.dfs_plan_sync(plan)
    x_h = prob.x.cpu().pin_memory()
    t_h = prob.t_emb[2].cpu().pin_memory()
    o_h = torch.empty_like(x_h).pin_memory()
    dfs.dfs_block_forward_host(plan, 2, 0, x_h, t_h, o_h)
    np.testing.assert_array_equal(host.to_bits(o_h), host.to_bits(out))


def test_async_host_ring_matches_device_buffers():
    """Five asynchronous host-buffer forwards (both staging slots reused, a synchronous call
    in between) give each call's own device-path result."""
    import torch
    from paper_2607_06631_gb300 import dfs, host
    cfg = synth.tiny()
    r0, _ = run_block(cfg, steps=[], want_intermediates=False)
    plan, prob = r0["plan"], r0["prob"]
    g = torch.Generator().manual_seed(7)
    xs = [(prob.x.float().cpu() + 0.1 * k * torch.randn(prob.x.shape, generator=g)).to(prob.x.dtype)
          for k in range(6)]
    steps = [0, 3, 1, 2, 0, 3]
    want = []
    for k, s in enumerate(steps):
        out = torch.empty_like(prob.x)
        dfs.dfs_block_forward(plan, s, xs[k].cuda(), prob.t_emb[s], out)
        want.append(out)
    dfs.dfs_plan_sync(plan)
    x_h = [x.pin_memory() for x in xs]
    t_h = [prob.t_emb[s].cpu().pin_memory() for s in steps]
    o_h = [torch.empty_like(x_h[0]).pin_memory() for _ in steps]
    for k in range(3):
        dfs.dfs_block_forward_host_async(plan, steps[k], 0, x_h[k], t_h[k], o_h[k])
    dfs.dfs_block_forward_host(plan, steps[3], 0, x_h[3], t_h[3], o_h[3])
    for k in range(4, 6):
        dfs.dfs_block_forward_host_async(plan, steps[k], 0, x_h[k], t_h[k], o_h[k])
    dfs.dfs_plan_sync(plan)
    for k in range(len(steps)):
        np.testing.assert_array_equal(host.to_bits(o_h[k]), host.to_bits(want[k]), err_msg=f"call {k}")


def test_denoise_small_stack():
    import torch
    from paper_2607_06631_gb300 import dfs, host
    cfg = synth.small_stack(4)
    shared, layers, m, acts = synth.make_problem(cfg)
    m["block_gate"][2, 1] = 0
    prob = host.DeviceProblem(cfg, shared, layers, m, acts)
    plan = prob.create_plan()
    lat = prob.x.clone()
    dfs.dfs_denoise(plan, lat, cfg.n_steps, prob.t_emb)
    dfs.dfs_plan_sync(plan)
    W, LW, X = synth.widen(shared), synth.widen(layers), synth.widen(acts)
    ref = O.denoise(cfg, W, LW, m, X["x"], X["t_emb"], X["ctx"])
    got = synth.bits_to_f64(host.to_bits(lat))
    assert rel_err(got, ref) <= TOL
    assert branch_err(got, ref, X["x"]) <= TOL


def test_invalid_arguments_are_rejected():
    import torch
    from paper_2607_06631_gb300 import dfs
    cfg = synth.tiny()
    r0, _ = run_block(cfg, steps=[], want_intermediates=False)
    plan, prob = r0["plan"], r0["prob"]
    out = torch.empty_like(prob.x)
    for args in ((4, 0), (-1, 0), (0, 1)):
        with pytest.raises(dfs.DfsError) as e:
            dfs.dfs_block_forward_layer(plan, args[0], args[1], prob.x, prob.t_emb[0], out)
        assert e.value.status == dfs.DFS_EINVAL
    with pytest.raises(dfs.DfsError) as e:
        dfs.dfs_block_forward(plan, 0, prob.x, prob.t_emb[0], prob.x)
    assert e.value.status == dfs.DFS_EINVAL


def test_misaligned_device_pointers_are_rejected_before_any_launch():
    """x / out / t_emb / latents 8 bytes off a 16-byte boundary: DFS_EINVAL, nothing
    launched, and the plan keeps working."""
    import torch
    from paper_2607_06631_gb300 import dfs, host
    cfg = synth.tiny()
    shared, layers, m, acts = synth.make_problem(cfg)
    prob = host.DeviceProblem(cfg, shared, layers, m, acts)
    plan = prob.create_plan()
    buf = torch.zeros(prob.x.numel() + 64, dtype=prob.x.dtype, device=prob.x.device)
    out = torch.empty_like(prob.x)
    x8, out8 = buf.data_ptr() + 8, out.data_ptr() + 8
    for args in ((x8, prob.t_emb[0], out), (prob.x, prob.t_emb[0], out8),
                 (prob.x, prob.t_emb[0].data_ptr() + 8, out)):
        with pytest.raises(dfs.DfsError) as e:
            dfs.dfs_block_forward(plan, 0, *args)
        assert e.value.status == dfs.DFS_EINVAL and "16-byte aligned" in str(e.value)
    with pytest.raises(dfs.DfsError) as e:
        dfs.dfs_denoise(plan, x8, cfg.n_steps, prob.t_emb)
    assert e.value.status == dfs.DFS_EINVAL
    dfs.dfs_plan_sync(plan)
    dfs.dfs_block_forward(plan, 0, prob.x, prob.t_emb[0], out)
    dfs.dfs_plan_sync(plan)


def test_injected_allocation_failure(monkeypatch):
    from paper_2607_06631_gb300 import dfs, host
    cfg = synth.tiny()
    shared, layers, m, acts = synth.make_problem(cfg)
    prob = host.DeviceProblem(cfg, shared, layers, m, acts)
    for n in (1, 7, 40):
        monkeypatch.setenv("DFS_FAULT_ALLOC", str(n))
        with pytest.raises(dfs.DfsError) as e:
            prob.create_plan()
        assert e.value.status == dfs.DFS_ENOMEM
    monkeypatch.delenv("DFS_FAULT_ALLOC")
    prob.create_plan()


def test_injected_launch_failure_is_reported_and_the_plan_recovers(monkeypatch):
    """DFS_FAULT_LAUNCH=n skips the plan's n-th launch and reports it: the forward that hits
    it returns DFS_ECUDA and leaves `out` untouched; the next forward is correct."""
    import torch
    from paper_2607_06631_gb300 import dfs, host
    cfg = synth.tiny()
    shared, layers, m, acts = synth.make_problem(cfg)
    prob = host.DeviceProblem(cfg, shared, layers, m, acts)
    ref_plan = prob.create_plan()
    ref = torch.empty_like(prob.x)
    dfs.dfs_block_forward(ref_plan, 2, prob.x, prob.t_emb[2], ref)
    dfs.dfs_plan_sync(ref_plan)
    monkeypatch.setenv("DFS_FAULT_LAUNCH", "5")
    plan = prob.create_plan()
    monkeypatch.delenv("DFS_FAULT_LAUNCH")
    out = torch.zeros_like(prob.x)
    with pytest.raises(dfs.DfsError) as e:
        dfs.dfs_block_forward(plan, 2, prob.x, prob.t_emb[2], out)
    assert e.value.status == dfs.DFS_ECUDA and "injected" in str(e.value)
    dfs.dfs_plan_sync(plan)
    assert not host.to_bits(out).any()
    dfs.dfs_block_forward(plan, 2, prob.x, prob.t_emb[2], out)
    dfs.dfs_plan_sync(plan)
    np.testing.assert_array_equal(host.to_bits(out), host.to_bits(ref))


def test_injected_launch_failure_in_the_asynchronous_host_path(monkeypatch):
    """A launch failure inside dfs_block_forward_host_async is reported (DFS_ECUDA) and the
    staging slot it used serves the following calls correctly."""
    import torch
    from paper_2607_06631_gb300 import dfs, host
    cfg = synth.tiny()
    shared, layers, m, acts = synth.make_problem(cfg)
    prob = host.DeviceProblem(cfg, shared, layers, m, acts)
    ref_plan = prob.create_plan()
    ref = torch.empty_like(prob.x)
    dfs.dfs_block_forward(ref_plan, 1, prob.x, prob.t_emb[1], ref)
    dfs.dfs_plan_sync(ref_plan)
    monkeypatch.setenv("DFS_FAULT_LAUNCH", "4")
    plan = prob.create_plan()
    monkeypatch.delenv("DFS_FAULT_LAUNCH")
    x_h = prob.x.cpu().pin_memory()
    t_h = prob.t_emb[1].cpu().pin_memory()
    outs = [torch.zeros_like(x_h).pin_memory() for _ in range(3)]
    with pytest.raises(dfs.DfsError) as e:
        dfs.dfs_block_forward_host_async(plan, 1, 0, x_h, t_h, outs[0])
    assert e.value.status == dfs.DFS_ECUDA and "injected" in str(e.value)
    for o in outs[1:]:
        dfs.dfs_block_forward_host_async(plan, 1, 0, x_h, t_h, o)
    dfs.dfs_plan_sync(plan)
    for o in outs[1:]:
        np.testing.assert_array_equal(host.to_bits(o), host.to_bits(ref))


def test_bounded_wait_reports_timeout_and_context_survives():
    """A wait that nothing completes gives up after about a second, the host reads
    DFS_ETIMEOUT, and the next forward on the same context is correct."""
    import time
    import torch
    from paper_2607_06631_gb300 import dfs
    cfg = synth.tiny()
    r0, res = run_block(cfg, steps=[1], want_intermediates=False)
    plan, prob = r0["plan"], r0["prob"]
    t0 = time.time()
    dfs.dfs_selftest_wait_timeout(plan)
    with pytest.raises(dfs.DfsError) as e:
        dfs.dfs_plan_sync(plan)
    assert e.value.status == dfs.DFS_ETIMEOUT
    assert time.time() - t0 < 30
    dfs.dfs_plan_sync(plan)           # the error word was cleared
    out = torch.empty_like(prob.x)
    dfs.dfs_block_forward(plan, 1, prob.x, prob.t_emb[1], out)
    dfs.dfs_plan_sync(plan)
    from paper_2607_06631_gb300 import host
    got = synth.bits_to_f64(host.to_bits(out))
    assert rel_err(got, res[0]["ref"]) <= TOL
