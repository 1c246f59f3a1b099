"""The N>1 bench path on CPU ranks (gloo, world size 2): every rank runs an independent
replica, so the only collective is the timing reduction (max over ranks), and the
whole-job value counts every rank's work against the slowest rank's time."""
import multiprocessing as mp
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    w, r, lr = bench.dist_setup()
    local_ms = 100.0 + 50.0 * rank
    ms_max = bench.dist_max(local_ms, w)
    bench.barrier(w)
    q.put((r, w, lr, ms_max, bench.job_value(2e12, 10, w, ms_max)))
    dist.destroy_process_group()


def test_two_rank_timing_reduction_and_job_value():
    pytest.importorskip("torch.distributed")
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [o[0] for o in out] == [0, 1]
    for r, w, lr, ms_max, val in out:
        assert w == 2 and lr == r
        assert ms_max == 150.0                       # the slower rank sets the time
        assert abs(val - 2e12 * 10 * 2 / 0.150 / 1e12) < 1e-9


# ---------------------------------------------------------------------------------------
# Sequence-parallel partition of one block (CPU ranks against the oracle)
# ---------------------------------------------------------------------------------------
#
# The engine ships replicas only (one independent video per GPU).  Within one block the
# natural sharding is over tokens: every step of the block is row-local except attention,
# whose keys and values span the whole sequence.  These tests run that partition on gloo
# ranks with the oracle's own primitives: each rank owns a contiguous token range, computes
# its rows' q, k, v (RoPE at the global token positions), all-gathers k and v of the
# retained heads (2 N h_s dh elements: the one exchange of the block), attends its queries
# over the gathered keys and finishes its rows alone; the gathered rows must equal the
# monolithic oracle block.

def _sp_rank(rank, world, port, q, cfg_kind, step):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import numpy as np
    import torch
    import torch.distributed as dist
    import oracle as O
    from oracle import dfs_oracle as OD
    import synth
    dist.init_process_group("gloo", rank=rank, world_size=world)
    cfg = synth.tiny(has_cross=1) if cfg_kind == "cross" else synth.tiny(grid=(1, 15, 26))
    shared, layers, m, acts = synth.make_problem(cfg)
    W, LW, X = synth.widen(shared), synth.widen(layers), synth.widen(acts)
    lw, x, t_emb = LW[0], X["x"], X["t_emb"][step]
    N, dh, eps = x.shape[0], cfg.head_dim, cfg.ln_eps
    parts = np.array_split(np.arange(N), world)
    rows = parts[rank]
    idx = O.compact_indices(cfg, m, step, 0)
    P = O.compact_panels(lw, idx)
    h_s = len(idx["heads"])
    hd = h_s * dh
    sh_a, sc_a, g_a, sh_f, sc_f, g_f = O.modulation(W["w_t"], W["b_t"], lw["e_mod"], t_emb)

    xm = O.adaln(x[rows], sh_a, sc_a, eps)                                   # row-local
    qkv = O.linear(xm, P["wqkv"], P["bqkv"])
    ones = np.ones(hd)
    qr = O.rms_norm(qkv[:, :hd], P["gq"], ones, eps, cfg.qk_norm_mode, dh)
    kr = O.rms_norm(qkv[:, hd:2 * hd], P["gk"], ones, eps, cfg.qk_norm_mode, dh)
    vr = qkv[:, 2 * hd:]
    ang = O.rope_angles(cfg.grid, dh, cfg.rope_theta)[rows]                  # global positions
    qr = O.apply_rope(qr.reshape(-1, h_s, dh), ang)
    kr = O.apply_rope(kr.reshape(-1, h_s, dh), ang)

    # the exchange: all-gather k and v of the retained heads (padded to the longest part)
    L = max(len(p) for p in parts)
    mine = np.zeros((2, L, h_s, dh))
    mine[0, :len(rows)] = kr
    mine[1, :len(rows)] = vr.reshape(-1, h_s, dh)
    got = [torch.zeros(2, L, h_s, dh, dtype=torch.float64) for _ in range(world)]
    dist.all_gather(got, torch.from_numpy(mine))
    K = np.concatenate([g.numpy()[0, :len(p)] for g, p in zip(got, parts)])
    V = np.concatenate([g.numpy()[1, :len(p)] for g, p in zip(got, parts)])
    exchanged = sum(2 * len(p) * h_s * dh for p in parts)

    o = O.attention(qr, K, V).reshape(-1, hd)
    x1 = x[rows] + g_a * O.linear(o, P["wo"], lw["bo"])                      # row-local from here
    if cfg.has_cross:
        x1 = x1 + OD._cross_compacted(cfg, lw, P, idx, x1, X["ctx"], None)
    xm2 = O.adaln(x1, sh_f, sc_f, eps)
    u = O.gelu_tanh(O.linear(xm2, P["w_up"], P["b_up"]))
    out = x1 + g_f * O.linear(u, P["w_down"], lw["b_down"])

    outs = [torch.zeros(L, x.shape[1], dtype=torch.float64) for _ in range(world)]
    pad = np.zeros((L, x.shape[1]))
    pad[:len(rows)] = out
    dist.all_gather(outs, torch.from_numpy(pad))
    if rank == 0:
        full = np.concatenate([g.numpy()[:len(p)] for g, p in zip(outs, parts)])
        ref = O.block_forward_compacted(cfg, W, lw, m, step, 0, x, t_emb, X.get("ctx"))
        err = float(np.abs(full - ref).max() / np.abs(ref).max())
        q.put((err, exchanged, 2 * N * h_s * dh))
    dist.destroy_process_group()


@pytest.mark.parametrize("world,cfg_kind,step", [(2, "self", 0), (3, "self", 3), (2, "cross", 1)])
def test_sequence_parallel_block_partition_equals_the_block(world, cfg_kind, step):
    pytest.importorskip("torch.distributed")
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_sp_rank, args=(r, world, port, q, cfg_kind, step)) for r in range(world)]
    for p in procs:
        p.start()
    import queue
    import time
    deadline = time.monotonic() + 300
    while True:                                   # fail fast if a rank dies before reporting
        try:
            err, exchanged, closed_form = q.get(timeout=2)
            break
        except queue.Empty:
            assert any(p.is_alive() for p in procs) and time.monotonic() < deadline, \
                "a rank exited without a result: %s" % [p.exitcode for p in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert err < 1e-12, err
    assert exchanged == closed_form
