#!/usr/bin/env python
"""Benchmark of the step-specific pruned video-DiT block on GB300.

One bench step = one pass of the whole hot path over one synthetic latent: the four
distilled denoising steps of one Wan-14B-shaped block (d=5120, 40 heads x 128, FFN
13824, 21x30x52 = 32760 tokens), each with its own retained heads / FFN chunks (keep
1.0 / 0.8 / 0.7 / 0.55, i.e. 40/32/28/22 heads and 13824/11056/9680/7600 channels),
run through the C ABI (dfs_block_forward).  Weights and inputs are seeded synthetic
bf16 values (synth/), resident in HBM before timing; every input is larger than L2.

Reported: TFLOP/s of algorithmic (pruned) FLOPs, its fraction of the measured bf16
peak, the roofline of the dominant kernel (CUDA-event timed inside the timed region),
the per-step pruned/dense speedup against the ideal FLOP ratio, an end-to-end number
through the host-buffer entry point, and the CPU oracle's throughput on a bounded
sample.  `--impl reference` times that CPU oracle alone (the reference arm).
"""
from __future__ import annotations

import argparse
import copy
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import synth  # noqa: E402

METRIC = "pruned-block TFLOP/s and % bf16 tensor peak; pruned/dense speedup vs ideal"
KINDS = ("modulation", "adaln", "gemm_qkv", "qk_norm_rope", "attention", "gemm_o", "gemm_up", "gemm_down",
         "cross", "other", "gather", "model")
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def get_config(name: str, grid=None):
    cfg = _named_config(name)
    if grid:
        cfg.grid = tuple(int(v) for v in grid.split(","))
        cfg.name = cfg.name + "_grid" + "x".join(map(str, cfg.grid))
    return cfg


def _named_config(name: str):
    if name == "wan14b":
        return synth.wan14b()
    if name == "wan14b_cross":
        return synth.wan14b_cross()
    if name == "sweep720":
        return synth.sweep720_all()
    if name.startswith("wan14b_x"):
        return synth.wan14b_stack(int(name[len("wan14b_x"):]))
    if name == "wan13b":
        return synth.wan13b()
    if name == "tiny":
        return synth.tiny()
    if name == "wan13b_policy":
        return synth.wan13b_policy()
    if name == "wan13b_model":
        return synth.wan13b_model()
    if name == "tiny_model":
        return synth.tiny_model()
    if name.startswith("sweep720:"):
        return synth.sweep720(float(name.split(":")[1]))
    raise SystemExit("unknown config " + name)


def _is_model(cfg) -> bool:
    return cfg.name.endswith("_model")


def _policy_shaped(cfg) -> bool:
    return any(len(set(h)) > 1 for h in cfg.heads_kept) or any(len(set(c)) > 1 for c in cfg.chunks_kept)


def workload_desc(cfg) -> str:
    if _policy_shaped(cfg):
        hk = "/".join("%d-%d" % (min(cfg.heads_kept[s]), max(cfg.heads_kept[s])) for s in range(cfg.n_steps))
        fk = "/".join("%d-%d" % (8 * min(cfg.chunks_kept[s]), 8 * max(cfg.chunks_kept[s]))
                      for s in range(cfg.n_steps))
        hk += " per layer (policy-shaped: U-shaped per-step retention, deep layers pruned most)"
    else:
        hk = "/".join(str(cfg.heads_kept[s][0]) for s in range(cfg.n_steps))
        fk = "/".join(str(8 * cfg.chunks_kept[s][0]) for s in range(cfg.n_steps))
    what = ("%d-layer %d-step denoise (dfs_denoise)" % (cfg.n_layers, cfg.n_steps) if cfg.n_layers > 1
            else "%d MoM steps per bench step" % cfg.n_steps)
    if _is_model(cfg):
        what = ("Wan-shaped model (patch embedding of a %dx%dx%dx%d latent, timestep MLP, head) around %d layers, "
                "%d-step latent denoise (dfs_model_denoise, timesteps %s)"
                % (cfg.latent_channels, cfg.grid[0], 2 * cfg.grid[1], 2 * cfg.grid[2], cfg.n_layers, cfg.n_steps,
                   "/".join("%g" % t for t in synth.model_timesteps(cfg.n_steps))))
    cross = (", text cross-attention over %d context tokens (cross heads kept as self heads)" % cfg.ctx_len
             if cfg.has_cross else "")
    return ("%s-shaped pruned DiT block, %s: d=%d, %dx%d heads, FFN %d, %s=%d tokens, kept heads %s, "
            "kept FFN channels %s%s"
            % (cfg.name, what, cfg.dim, cfg.n_heads, cfg.head_dim, cfg.ffn_dim,
               "x".join(map(str, cfg.grid)), cfg.n_tokens, hk, fk, cross))


def panel_mb(cfg):
    """Smallest and largest per-step compacted weight bytes of one layer (MB)."""
    d, dh = cfg.dim, cfg.head_dim
    mb = [(4 * cfg.heads_kept[s][l] * dh * d + 2 * 8 * cfg.chunks_kept[s][l] * d) * 2 / 1e6
          for s in range(cfg.n_steps) for l in range(cfg.n_layers)]
    return min(mb), max(mb)


def kernel_units(cfg):
    """Algorithmic work of each kernel kind summed over the MoM steps of one bench step:
    ('tensor', FLOPs) or ('hbm', bytes)."""
    N, d, dh = cfg.n_tokens, cfg.dim, cfg.head_dim
    u = {k: 0.0 for k in KINDS}
    for s in range(cfg.n_steps):
        for l in range(cfg.n_layers):
            hd = cfg.heads_kept[s][l] * dh
            fs = 8 * cfg.chunks_kept[s][l]
            u["gemm_qkv"] += 2.0 * N * d * 3 * hd
            u["attention"] += 4.0 * N * N * hd
            u["gemm_o"] += 2.0 * N * hd * d
            u["gemm_up"] += 2.0 * N * d * fs
            u["gemm_down"] += 2.0 * N * fs * d
            u["adaln"] += N * d * (2 + 2) + N * d * (4 + 2)      # x bf16 -> xm, x1 fp32 -> xm2
            u["qk_norm_rope"] += 2.0 * N * 2 * hd * 2              # q, k read + written
            u["modulation"] += 6.0 * d * d * 2                     # W_t read once
            if cfg.engine == 1:                                    # union engine: FFN panels gathered
                u["gather"] += 2.0 * (2 * fs * d * 2)              # W_up_s, W_down_s read + written
            if cfg.has_cross:
                hc = cfg.xheads_kept[s][l] * dh
                u["cross"] += 4.0 * N * d * hc + 4.0 * N * cfg.ctx_len * hc
    if cfg.n_layers > 1:  # the stack's modulation GEMV runs once per step, not per layer
        u["modulation"] = cfg.n_steps * 6.0 * d * d * 2
    if _is_model(cfg):    # model around the blocks, per step: token rows (4C wide) written by patchify and
        # read by the embedding, the embedding's output, the head's LayerNorm in / out and GEMM input, the
        # head's token rows and the latent read + written by the update (bf16)
        C4 = 4 * cfg.latent_channels
        u["model"] = cfg.n_steps * 2.0 * N * (2 * C4 + 4 * d + C4 + 2 * C4)
    bound = {k: ("tensor" if k.startswith("gemm") or k in ("attention", "cross") else "hbm") for k in KINDS}
    return u, bound


# ------------------------------------------------------------------------------ clocks

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        self.proc = None
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(gpu_index), "--query-gpu=" + self.FIELDS,
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.file, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        self.file.flush()
        self.file.seek(0)
        rows = [l.strip().split(",") for l in self.file.read().splitlines() if l.strip()]
        self.file.close()
        os.unlink(self.file.name)
        sm, mx, reasons = [], 0.0, set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for r in rows:
            try:
                sm.append(float(r[1]))
                mx = max(mx, float(r[2]))
                for n, v in zip(names, r[5:9]):
                    if v.strip().lower().startswith("active"):
                        reasons.add(n)
            except (ValueError, IndexError):
                continue
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx or None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------------------------------ distributed

def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def dist_max(x: float, world: int) -> float:
    """Maximum of x over the ranks (timing only; the block itself exchanges nothing)."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_value(flops_per_step: float, steps: int, world: int, ms_max: float) -> float:
    """Whole-job TFLOP/s: every rank runs its own replica, so the units of all ranks are
    divided by the slowest rank's time."""
    return flops_per_step * steps * world / (ms_max / 1e3) / 1e12


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


# ------------------------------------------------------------------------------ CPU oracle

def cpu_cores() -> int:
    try:
        from threadpoolctl import threadpool_info
        n = [i.get("num_threads", 0) for i in threadpool_info() if i.get("user_api") == "blas"]
        if n:
            return int(max(n))
    except Exception:
        pass
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def oracle_sample(cfg, problem_f64, step: int, rows: int, seed: int = 0):
    """Runs the float64 oracle (compacted block) for `rows` query rows of one MoM step;
    keys / values cover every token.  Returns (seconds, counted FLOPs)."""
    import oracle as O
    W, LW, M, X = problem_f64
    r = np.sort(np.random.default_rng(seed).choice(cfg.n_tokens, size=rows, replace=False))
    c = O.MacCounter()
    t0 = time.perf_counter()
    O.block_forward_compacted(cfg, W, LW[0], M, step, 0, X["x"], X["t_emb"][step], X.get("ctx"), rows=r,
                              counter=c)
    return time.perf_counter() - t0, c.flops


def load_problem_f64(cfg):
    shared, layers, masks, acts = synth.make_problem(cfg)
    return synth.widen(shared), synth.widen(layers), masks, synth.widen(acts)


CPU_SLICE = 512    # query rows of the oracle's timed slice (cpu_baseline and the reference arm)


def one_layer(cfg):
    """Layer 0 of a stack as a one-layer configuration (its own seeded weights and masks)."""
    if cfg.n_layers == 1:
        return cfg
    c = copy.deepcopy(cfg)
    c.name = cfg.name + "_layer0"
    c.n_layers = 1
    c.heads_kept = [[h[0]] for h in cfg.heads_kept]
    c.chunks_kept = [[k[0]] for k in cfg.chunks_kept]
    if cfg.xheads_kept is not None:
        c.xheads_kept = [[h[0]] for h in cfg.xheads_kept]
    if cfg.block_gate is not None:
        c.block_gate = [[g[0]] for g in cfg.block_gate]
    return c


def stack_flops(cfg) -> float:
    """Closed-form FLOPs of every (step, layer) block of a configuration (gated-off blocks: 0)."""
    import oracle as O
    tot = 0.0
    for s in range(cfg.n_steps):
        for l in range(cfg.n_layers):
            if cfg.block_gate is not None and not cfg.block_gate[s][l]:
                continue
            hc = cfg.xheads_kept[s][l] if cfg.has_cross else 0
            tot += O.block_flops(cfg.n_tokens, cfg.dim, cfg.head_dim, cfg.heads_kept[s][l], 8 * cfg.chunks_kept[s][l],
                                 hc, cfg.ctx_len)
    return tot


def cpu_baseline(cfg):
    """The float64 oracle on the host cores, timed on a bounded sample of the workload.

    One block (layer 0, the last MoM step): T_KV = the oracle on a single query row, i.e. the
    adaLN, K and V projections, K norm and RoPE over all N tokens plus one row; T_call = the
    same with a 512-row slice; T_rows = T_call - T_KV; the block is extrapolated as
    T = T_KV + (N / 512) T_rows.  Up to 512 tokens the whole block is timed instead.  A stack
    (L layers x T steps) is extrapolated at that block's FLOP rate over its closed-form FLOPs
    (the Wan-14B-shaped stack: the config-3-shaped block x 40 layers x 4 steps x keep)."""
    import oracle as O
    one = one_layer(cfg)
    prob = load_problem_f64(one)
    step = one.n_steps - 1
    N = one.n_tokens
    h_s, f_s = one.heads_kept[step][0], 8 * one.chunks_kept[step][0]
    hc = one.xheads_kept[step][0] if one.has_cross else 0
    flops = O.block_flops(N, one.dim, one.head_dim, h_s, f_s, hc, one.ctx_len)
    out = {"unit": "TFLOP/s", "cores": cpu_cores(), "kind": "oracle"}
    if N <= CPU_SLICE:
        t_call, _ = oracle_sample(one, prob, step, N)
        t_block = t_call
        out["sample"] = ("float64 oracle, MoM step %d of the whole %d-token block, timed in full (%.2f s)"
                         % (step, N, t_call))
    else:
        t_kv, _ = oracle_sample(one, prob, step, 1, seed=7)
        t_call, _ = oracle_sample(one, prob, step, CPU_SLICE)
        t_rows = max(t_call - t_kv, 1e-9)
        t_block = t_kv + (N / CPU_SLICE) * t_rows
        out.update({"T_KV_s": round(t_kv, 3), "T_rows_s": round(t_rows, 3), "slice_rows": CPU_SLICE,
                    "formula": "T = T_KV + (N / %d) T_rows = %.3f + (%d / %d) x %.3f" % (CPU_SLICE, t_kv, N,
                                                                                    CPU_SLICE, t_rows)})
        out["sample"] = ("float64 oracle, MoM step %d: T_KV = one query row with keys / values over all %d "
                         "tokens (%.2f s); a %d-row slice through the whole block (%.2f s in the same call "
                         "as its K / V) gives T_rows = %.2f s" % (step, N, t_kv, CPU_SLICE, t_call, t_rows))
    rate = flops / t_block
    out["block_seconds_extrapolated"] = round(t_block, 2)
    out["block_flops"] = flops
    if cfg.n_layers == 1:
        out["value"] = rate / 1e12
        out["extrapolation"] = "one full block of MoM step %d (%.3e algorithmic FLOPs)" % (step, flops)
    else:
        tot = stack_flops(cfg)
        out["value"] = rate / 1e12
        out["stack_seconds_extrapolated"] = round(tot / rate, 1)
        out["extrapolation"] = ("the %d-layer %d-step workload (%.3e closed-form FLOPs, every layer at its own "
                                "keep) at the FLOP rate of layer 0's block at MoM step %d" %
                                (cfg.n_layers, cfg.n_steps, tot, step))
    return out


def oracle_block_seconds(cfg, prob, step: int, t_kv_cache: dict):
    """The oracle's time for one whole block of a MoM step, measured on a bounded sample: the
    whole block up to 512 tokens, else T_KV (one query row with keys / values over all N
    tokens; measured once per MoM step) plus (N / 512) T_rows from a 512-row slice.
    Returns (seconds, wall seconds spent)."""
    N = cfg.n_tokens
    if N <= CPU_SLICE:
        t, _ = oracle_sample(cfg, prob, step, N)
        return t, t
    wall = 0.0
    if step not in t_kv_cache:
        t_kv_cache[step], _ = oracle_sample(cfg, prob, step, 1, seed=7)
        wall += t_kv_cache[step]
    t_kv = t_kv_cache[step]
    t_call, _ = oracle_sample(cfg, prob, step, CPU_SLICE, seed=step)
    return t_kv + (N / CPU_SLICE) * max(t_call - t_kv, 1e-9), wall + t_call


def run_reference(args):
    world, rank, _ = dist_setup()
    if rank != 0:
        return 0
    import oracle as O
    cfg = one_layer(get_config(args.config, args.grid))
    prob = load_problem_f64(cfg)

    def step_flops(s):
        hc = cfg.xheads_kept[s][0] if cfg.has_cross else 0
        return O.block_flops(cfg.n_tokens, cfg.dim, cfg.head_dim, cfg.heads_kept[s][0], 8 * cfg.chunks_kept[s][0], hc,
                             cfg.ctx_len)

    for i in range(args.warmup):  # a single query row each (the K / V pass dominates)
        oracle_sample(cfg, prob, i % cfg.n_steps, 1, seed=1000 + i)
    tot_t = tot_f = tot_wall = 0.0
    t_kv = {}
    for i in range(args.steps):
        s = i % cfg.n_steps
        t, wall = oracle_block_seconds(cfg, prob, s, t_kv)
        tot_t += t
        tot_wall += wall
        tot_f += step_flops(s)
    val = tot_f / tot_t / 1e12
    sample = ("each step: the float64 oracle on one MoM step (cycling 0..%d) of one block, its whole-block time "
              "taken as T_KV + (N / %d) T_rows (T_KV: one query row with keys / values over all %d tokens; T_rows: "
              "a %d-row slice through the block); value = closed-form block FLOPs / that time"
              % (cfg.n_steps - 1, CPU_SLICE, cfg.n_tokens, CPU_SLICE)) if cfg.n_tokens > CPU_SLICE else \
             ("each step: the float64 oracle on one whole MoM step (cycling 0..%d) of the %d-token block"
              % (cfg.n_steps - 1, cfg.n_tokens))
    line = {"impl": "reference", "metric": METRIC, "value": val, "unit": "TFLOP/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot_wall / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": workload_desc(get_config(args.config, args.grid))},
            "cpu_baseline": {"kind": "oracle", "cores": cpu_cores(), "value": val, "unit": "TFLOP/s",
                             "sample": sample, "block_seconds_extrapolated_mean": round(tot_t / args.steps, 2)},
            "e2e": {"value": val, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------------------------------ our arm

def device_stack(cfg, seed: int = 20260706):
    """Random-init stack weights drawn on the device (host.random_device_stack); masks,
    inputs and text context come from synth."""
    from paper_2607_06631_gb300 import host
    layers, w_t, b_t = host.random_device_stack(cfg, seed)
    acts = synth.make_activations(cfg)
    x = host.to_device(acts["x"])
    temb = host.to_device(acts["t_emb"])
    ctx = host.to_device(acts["ctx"]) if "ctx" in acts else None
    return layers, w_t, b_t, synth.make_masks(cfg), x, temb, ctx

def run_ours(args):
    import torch
    world, rank, local = dist_setup()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    else:
        torch.cuda.set_device(0)
    from paper_2607_06631_gb300 import build, dfs, host
    build.build()
    peaks, peak_src = load_peaks()
    cfg = get_config(args.config, args.grid)
    cfg.engine = dfs.ENGINES[args.engine]
    cfg.qk_norm_mode = args.qk_norm_mode
    T, L = cfg.n_steps, cfg.n_layers
    stream = torch.cuda.current_stream()
    # the dense reference of the speedups: step 0 when it keeps every unit, else a separate
    # one-step plan over the same weights that keeps every unit
    dense_step0 = all(h == cfg.n_heads for h in cfg.heads_kept[0]) and \
        all(c == cfg.n_chunks for c in cfg.chunks_kept[0]) and \
        (not cfg.has_cross or all(h == cfg.n_heads for h in cfg.xheads_kept[0]))
    dense_plan = None

    def make_dense(layers_dev, w_t_dev, b_t_dev, ctx_dev):
        dc = copy.deepcopy(cfg)
        dc.n_steps = 1
        ones = {"block_gate": np.ones((1, L), np.uint8), "head_gate": np.ones((1, L, cfg.n_heads), np.uint8),
                "xhead_gate": np.ones((1, L, cfg.n_heads), np.uint8) if cfg.has_cross else None,
                "ffn_gate": np.ones((1, L, cfg.n_chunks), np.uint8)}
        return dfs.dfs_plan_create(dc, layers_dev, w_t_dev, b_t_dev, ones, ctx_dev, stream)

    if L == 1:
        shared, layers, masks, acts = synth.make_problem(cfg)
        prob = host.DeviceProblem(cfg, shared, layers, masks, acts)
        del shared, layers
        plan = prob.create_plan(stream)
        if not dense_step0:
            dense_plan = make_dense(prob.layers, prob.w_t, prob.b_t, prob.ctx)
        prob.free_weights()
        x, temb = prob.x, prob.t_emb
    else:
        dl, w_t, b_t, masks, x, temb, ctx = device_stack(cfg)
        plan = dfs.dfs_plan_create(cfg, dl, w_t, b_t, masks, ctx, stream)
        if not dense_step0:
            dense_plan = make_dense(dl, w_t, b_t, ctx)
        del dl, w_t, b_t
        torch.cuda.empty_cache()
        prob = None
    out = torch.empty_like(x)
    lat = x.clone()
    model = _is_model(cfg)
    if model:  # the model around the blocks: weights drawn on the device, latent from synth
        g = torch.Generator(device="cuda")
        g.manual_seed(7)
        mw = {}
        for k, shp in synth.model_shapes(cfg).items():
            mw[k] = torch.empty(shp, device="cuda", dtype=torch.bfloat16)
            mw[k].normal_(0.0, 0.02, generator=g)
        for pl in (plan, dense_plan):
            if pl is not None:
                dfs.dfs_model_attach(pl, mw, cfg.latent_channels, cfg.freq_dim, stream)
        del mw
        latent0 = host.to_device(synth.make_latent(cfg))
        lat = latent0.clone()
        vbuf = torch.empty_like(latent0)
        tsteps = synth.model_timesteps(T)
    weight_bytes, device_bytes = dfs.dfs_plan_memory(plan)
    # model: patch embedding and head GEMMs of every step count too (2 N (4C) d FLOPs each)
    extra = 4.0 * cfg.n_tokens * 4 * cfg.latent_channels * cfg.dim if model else 0.0
    flops = [sum(dfs.dfs_plan_flops(plan, s, l) for l in range(L)) + extra for s in range(T)]
    flops_step = sum(flops)

    def one_step(st=stream):
        if model:
            lat.copy_(latent0)
            dfs.dfs_model_denoise(plan, lat, T, tsteps, st)
        elif L == 1:
            for s in range(T):
                dfs.dfs_block_forward(plan, s, x, temb[s], out, st)
        else:
            lat.copy_(x)
            dfs.dfs_denoise(plan, lat, T, temb, st)

    for _ in range(args.warmup):
        one_step()
    dfs.dfs_plan_sync(plan, stream)
    graph = None
    if args.graph:
        # one bench step recorded once as a CUDA graph; the timed region replays it
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            one_step(torch.cuda.current_stream())
        for _ in range(args.warmup):
            graph.replay()
        dfs.dfs_plan_sync(plan, stream)
    barrier(world)
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    if graph is None:
        dfs.dfs_plan_profile(plan, True)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        if graph is None:
            one_step()
        else:
            graph.replay()
    e1.record(stream)
    torch.cuda.synchronize()
    if graph is None:
        dfs.dfs_plan_profile(plan, False)
    ck = clocks.stop()
    if graph is not None:
        # per-kernel timings from the same steps run eagerly right after (event records
        # cannot sit inside the replayed graph); the graph holds the same launches
        dfs.dfs_plan_sync(plan, stream)
        dfs.dfs_plan_profile(plan, True)
        for _ in range(args.steps):
            one_step()
        torch.cuda.synchronize()
        dfs.dfs_plan_profile(plan, False)
    barrier(world)
    ms = e0.elapsed_time(e1)
    ms_max = dist_max(ms, world)
    value = job_value(flops_step, args.steps, world, ms_max)
    dfs.dfs_plan_sync(plan, stream)

    # per-kernel event timings inside the timed region
    units, bound = kernel_units(cfg)
    kernels, launches = {}, 0
    for k in KINDS:
        kms, n = dfs.dfs_plan_profile_read(plan, k)
        launches += n
        if n == 0:
            continue
        work = units[k] * args.steps
        if bound[k] == "tensor":
            ach = work / (kms / 1e3) / 1e12
            peak = peaks["bf16_tflops_sustained"]
            unit = "TFLOP/s"
        else:
            ach = work / (kms / 1e3) / 1e9
            peak = peaks["hbm_gbs"]
            unit = "GB/s"
        kernels[k] = {"launches": n, "ms_total": round(kms, 4), "ms_per_launch": round(kms / n, 5),
                      "share": None, "achieved": round(ach, 2), "unit": unit, "peak": peak,
                      "frac": round(ach / peak, 4), "bound": bound[k]}
    tot_k = sum(v["ms_total"] for v in kernels.values())
    for v in kernels.values():
        v["share"] = round(v["ms_total"] / tot_k, 4)
    dom = max(kernels, key=lambda k: kernels[k]["ms_total"])
    dk = kernels[dom]
    traffic = None
    tfile = os.path.join(ROOT, "profiles", "traffic.json")
    if os.path.exists(tfile) and args.grid is None:
        tr = json.load(open(tfile)).get(args.config, {}).get(dom)
        if tr:
            import hashlib
            src = os.path.join(ROOT, tr["source"])
            sha = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16] if os.path.exists(src) else None
            if sha == tr["source_sha"]:  # counters taken on this very kernel source
                traffic = tr["bytes_per_launch"]
    roofline = {"kernel": dom, "bound": dk["bound"], "achieved": dk["achieved"], "peak": dk["peak"],
                "unit": dk["unit"], "frac": dk["frac"], "traffic": traffic,
                "peak_source": "%s (%s)" % (peak_src, "bf16_tflops_sustained" if dk["bound"] == "tensor"
                                            else "hbm_gbs")}

    # per-MoM-step latency: pruned vs dense (step 0 keeps every head and channel)
    # per-MoM-step latency (every layer of the step, as the denoising loop runs it) against the
    # dense reference
    bufs = (out, torch.empty_like(x)) if L > 1 else (out,)

    def run_step(pl, s):
        if model:
            dfs.dfs_model_forward(pl, s, latent0, tsteps[s], vbuf, stream)
            return
        cur = x
        for l in range(L):
            dst = bufs[l % len(bufs)]
            dfs.dfs_block_forward_layer(pl, s, l, cur, temb[s], dst, stream)
            cur = dst

    def time_step(pl, s):
        reps = max(3, min(10, args.steps)) if L == 1 else 2
        for _ in range(2 if L == 1 else 1):
            run_step(pl, s)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(reps):
            run_step(pl, s)
        b.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(b) / reps

    step_ms = [time_step(plan, s) for s in range(T)]
    if dense_plan is None:
        ref_ms, ref_flops, ref_desc = step_ms[0], flops[0], "step 0 (keeps every unit)"
    else:
        ref_ms = time_step(dense_plan, 0)
        ref_flops = sum(dfs.dfs_plan_flops(dense_plan, 0, l) for l in range(L)) + extra
        ref_desc = "separate plan keeping every unit (%.2f ms)" % ref_ms
        dense_plan.close()
    ideal = [ref_flops / f for f in flops]
    mean_ideal = ref_flops / (sum(flops) / T)
    speed = [ref_ms / t for t in step_ms]
    mean_meas = ref_ms / (sum(step_ms) / T)

    # end to end through the host-buffer entry point (pinned host memory)
    e2e = None
    if not args.no_e2e and L == 1:
        xh = x.cpu().pin_memory()
        th = temb.cpu().pin_memory()
        oh = [torch.empty_like(xh).pin_memory() for _ in range(2)]
        ke = max(1, min(args.steps, 20))  # the device-timed step count (its copies' pipeline fill and drain amortise alike)
        dfs.dfs_block_forward_host(plan, 0, 0, xh, th[0], oh[0], stream)
        dfs.dfs_block_forward_host_async(plan, 0, 0, xh, th[0], oh[0], stream)
        dfs.dfs_block_forward_host_async(plan, 1 % T, 0, xh, th[1 % T], oh[1], stream)
        dfs.dfs_plan_sync(plan, stream)
        torch.cuda.synchronize()

        def host_loop(fn):
            barrier(world)
            t0 = time.perf_counter()
            k = 0
            for _ in range(ke):
                for s in range(T):
                    fn(plan, s, 0, xh, th[s], oh[k % 2], stream)
                    k += 1
            dfs.dfs_plan_sync(plan, stream)
            return dist_max(time.perf_counter() - t0, world)

        # every step copies its input from pinned host memory and its result back; the
        # asynchronous entry point overlaps those copies with the neighbouring steps' forwards
        dt = host_loop(dfs.dfs_block_forward_host_async)
        dt_sync = host_loop(dfs.dfs_block_forward_host)
        nbytes = x.numel() * 2
        e2e = {"value": flops_step * ke * world / dt / 1e12, "unit": "TFLOP/s",
               "h2d_bytes_per_step": T * (nbytes + cfg.dim * 2), "d2h_bytes_per_step": T * nbytes,
               "steps": ke, "api": "dfs_block_forward_host_async",
               "value_synchronous": flops_step * ke * world / dt_sync / 1e12}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        del prob
        cpu = cpu_baseline(cfg)

    if rank == 0:
        line = {
            "metric": METRIC, "value": round(value, 2), "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(ms_max / args.steps, 4), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": workload_desc(cfg),
                       "engine": args.engine, "qk_norm_mode": args.qk_norm_mode,
                       "plan_weight_gb": round(weight_bytes / 1e9, 3),
                       "plan_device_gb": round(device_bytes / 1e9, 3),
                       "l2": ("inputs larger than L2 (x %.0f MB, per-step weights read %.0f-%.0f MB); no flush "
                              "between steps" % (cfg.n_tokens * cfg.dim * 2 / 1e6, panel_mb(cfg)[0],
                                                 panel_mb(cfg)[1]))
                             if cfg.n_tokens * cfg.dim * 2 > 129e6 else
                             ("inputs fit in L2 (x %.2f MB): L2-warm small-case timing, not a full-size "
                              "measurement" % (cfg.n_tokens * cfg.dim * 2 / 1e6)),
                       "launch": "CUDA graph replay of one bench step" if args.graph else "eager",
                       "parallelism": "replicas (one independent block per GPU)" if world > 1 else "1 GPU"},
            "frac_of_peak": round(value / world / peaks["bf16_tflops_sustained"], 4),
            "peak_tflops": peaks["bf16_tflops_sustained"], "peak_source": peak_src + " bf16_tflops_sustained",
            "step_ms": [round(t, 4) for t in step_ms], "step_tflops": [round(f / t / 1e9, 1) for f, t in
                                                                       zip(flops, step_ms)],
            "step_flop_keep": [round(f / ref_flops, 4) for f in flops], "speedup_reference": ref_desc,
            "speedup": [round(v, 4) for v in speed] if speed else None,
            "speedup_ideal": [round(v, 4) for v in ideal],
            "speedup_vs_ideal": [round(a / b, 4) for a, b in zip(speed, ideal)] if speed else None,
            "mean_speedup": round(mean_meas, 4) if mean_meas else None,
            "mean_speedup_ideal": round(mean_ideal, 4),
            "mean_speedup_vs_ideal": round(mean_meas / mean_ideal, 4) if mean_meas else None,
            "roofline": roofline, "kernels": kernels, "cpu_baseline": cpu, "e2e": e2e,
            "gpu_launches": launches, "clocks": ck,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--config", default="wan14b",
                    help="wan14b (default), wan13b, wan14b_cross, sweep720 (keep 1.0..0.5 as six steps), "
                         "sweep720:<ratio>, wan14b_x<L> (L-layer 4-step denoise with cross-attention), "
                         "wan13b_policy (30-layer 4-step denoise, policy-shaped masks), wan13b_model (the same "
                         "layers inside the Wan-shaped model on a latent video), tiny")
    ap.add_argument("--grid", default=None, help="override the latent grid T,H,W (smaller profiling cases)")
    ap.add_argument("--qk-norm-mode", type=int, choices=(0, 1), default=0,
                    help="QK RMSNorm over the retained channels of a row (0, default) or per head (1)")
    ap.add_argument("--engine", choices=("compacted", "union"), default="compacted",
                    help="weights per (step, layer) compacted once (default), or one union super-model per "
                         "layer gathered by the projections' TMA producers (Sec. 4.3)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--graph", action="store_true",
                    help="time replays of one bench step captured as a CUDA graph (per-kernel table from an "
                         "eager pass of the same steps)")
    args = ap.parse_args()
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
