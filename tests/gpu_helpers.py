"""Shared helpers of the GPU parity tests: run the CUDA path through the C ABI and the
oracle on the same seeded inputs, and compare."""
import numpy as np

import oracle as O
import synth

TOL = 2e-2  # max|err| / max|ref| on bf16 outputs with fp32 accumulation


def rel_err(got, ref) -> float:
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    den = np.abs(ref).max()
    if den == 0:
        return float(np.abs(got).max())
    return float(np.abs(got - ref).max() / den)


def bf16_ulp(v):
    """Spacing of bf16 numbers at |v| (8 significant bits)."""
    a = np.maximum(np.abs(np.asarray(v, dtype=np.float64)), 2.0 ** -126)
    return 2.0 ** (np.floor(np.log2(a)) - 7)


def branch_err(out, ref, x) -> float:
    """Error of the residual branch out - x, relative to its largest reference value,
    after allowing one bf16 ulp of |out| for storing the block output in bf16."""
    extra = np.maximum(np.abs(out - ref) - bf16_ulp(ref), 0.0)
    den = np.abs(ref - x).max()
    return float(extra.max() / den) if den > 0 else float(extra.max())


def run_block(cfg, seed_tag="", masks=None, steps=None, layer=0, want_intermediates=True, rows=None,
              patch=None):
    """Runs every requested step of `layer` on the GPU and the oracle (compacted mode).
    `patch(layers)`, if given, edits the seeded bf16 layer weights in place first.

    Returns a list of dicts with the GPU output, the oracle output and intermediates."""
    import torch
    from paper_2607_06631_gb300 import dfs, host

    shared, layers, m, acts = synth.make_problem(cfg, seed_tag)
    if patch is not None:
        patch(layers)
    if masks is not None:
        m = masks
    prob = host.DeviceProblem(cfg, shared, layers, m, acts)
    plan = prob.create_plan()
    W, LW, X = synth.widen(shared), synth.widen(layers), synth.widen(acts)
    out = torch.empty_like(prob.x)
    res = []
    for s in (range(cfg.n_steps) if steps is None else steps):
        dfs.dfs_block_forward_layer(plan, s, layer, prob.x, prob.t_emb[s], out)
        dfs.dfs_plan_sync(plan)
        got = host.to_bits(out)
        r = {"step": s, "out": synth.bits_to_f64(got)}
        if want_intermediates and m["block_gate"][s, layer]:
            for k in ("qk", "vt", "attn", "x1", "h", "xm", "mod"):
                r["ws_" + k] = host.read_workspace(plan, k)
        ref, it = O.block_forward_compacted(cfg, W, LW[layer], m, s, layer, X["x"], X["t_emb"][s],
                                            X.get("ctx"), rows=rows, want=True)
        r["ref"] = ref
        r["it"] = it
        r["mod_ref"] = O.modulation(W["w_t"], W["b_t"], LW[layer]["e_mod"], X["t_emb"][s])
        res.append(r)
    r0 = {"plan": plan, "prob": prob, "masks": m, "layers": layers, "x": X["x"]}
    return r0, res


def check_block(cfg, r0, res, check_intermediates=True, tol=TOL):
    x = r0["x"]
    m = r0["masks"]
    dh = cfg.head_dim
    for r in res:
        s = r["step"]
        e_out = rel_err(r["out"], r["ref"])
        e_branch = branch_err(r["out"], r["ref"], x)
        assert e_out <= tol, ("out", s, e_out)
        assert e_branch <= tol, ("out - x", s, e_branch)
        if not check_intermediates or not m["block_gate"][s, 0]:
            continue
        it = r["it"]
        assert rel_err(r["ws_mod"], r["mod_ref"]) <= 1e-5, ("mod", s)
        assert rel_err(r["ws_x1"], it["x1"]) <= tol, ("x1", s, rel_err(r["ws_x1"], it["x1"]))
        # the attention branch alone: x1 is stored in fp32
        assert rel_err(r["ws_x1"] - x, it["x1"] - x) <= tol, ("x1 - x", s, rel_err(r["ws_x1"] - x, it["x1"] - x))
        assert rel_err(r["ws_xm"], it["xm2"]) <= tol, ("xm2", s, rel_err(r["ws_xm"], it["xm2"]))
        if it["u"].shape[1]:
            assert rel_err(r["ws_h"], it["u"]) <= tol, ("h", s, rel_err(r["ws_h"], it["u"]))
        if "q" in it and not cfg.has_cross:
            N = x.shape[0]
            hd = it["q"].shape[1] * dh
            q, k = r["ws_qk"][:, :hd], r["ws_qk"][:, hd:]
            assert rel_err(q, it["q"].reshape(N, hd)) <= tol, ("q", s, rel_err(q, it["q"].reshape(N, hd)))
            assert rel_err(k, it["k"].reshape(N, hd)) <= tol, ("k", s)
            assert rel_err(r["ws_vt"].T, it["v"].reshape(N, hd)) <= tol, ("v", s)
            assert rel_err(r["ws_attn"], it["o"]) <= tol, ("attn", s, rel_err(r["ws_attn"], it["o"]))
