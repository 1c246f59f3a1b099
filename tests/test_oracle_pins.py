"""Pins of the CPU oracle against facts that do not come from the oracle itself:
values the paper prints, closed forms, invariants, textbook / library special cases
and brute force on tiny inputs.  CPU only."""
import json
import math
import os

import numpy as np
import pytest

import oracle as O
import synth

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_numbers.json")))


def rng(seed=0):
    return np.random.default_rng(seed)


# --------------------------------------------------------------------------- gates (Sec. 4.1)

def test_block_and_ffn_gate_rule():
    m = np.array([[0.3, -0.1, 0.0, 1e-30], [-2.0, 5.0, -0.0, 0.5]])
    assert O.gates_from_soft_masks("block", m).tolist() == [[1, 0, 0, 1], [0, 1, 0, 1]]
    assert O.gates_from_soft_masks("ffn", m).tolist() == [[1, 0, 0, 1], [0, 1, 0, 1]]


def test_head_gate_rule_mean_of_head_entries():
    # 3 heads of D_head = 4: mean positive / exactly zero / negative despite a large entry
    m = np.array([0.1, 0.2, -0.05, 0.0,
                  1.0, -1.0, 2.0, -2.0,
                  5.0, -3.0, -3.0, -0.5])
    assert O.gates_from_soft_masks("head", m, unit_size=4).tolist() == [1, 0, 0]


def test_ffn_chunk_gate_expands_to_c_channels():
    C = GOLD["ffn_chunk"]["value"]
    g = O.ffn_channel_gate([1, 0, 1], C)
    assert g.shape == (3 * C,)
    assert g.tolist() == [1] * C + [0] * C + [1] * C


def test_index_lists_follow_gates():
    cfg = synth.tiny()
    masks = synth.make_masks(cfg)
    for s in range(4):
        idx = O.compact_indices(cfg, masks, s, 0)
        assert len(idx["heads"]) == cfg.heads_kept[s][0]
        assert len(idx["chunks"]) == cfg.chunks_kept[s][0]
        assert np.all(np.diff(idx["heads"]) > 0) and np.all(np.diff(idx["chunks"]) > 0)
        # channels are whole heads / whole chunks of the retained units
        assert set(idx["qk_rows"] // cfg.head_dim) == set(idx["heads"].tolist())
        assert set(idx["ffn_ch"] // cfg.ffn_chunk) == set(idx["chunks"].tolist())
        assert len(idx["ffn_ch"]) == 8 * len(idx["chunks"])


def test_compact_panels_are_row_and_column_selections():
    cfg = synth.tiny()
    lw = synth.make_layer(cfg, 0)
    masks = synth.make_masks(cfg)
    idx = O.compact_indices(cfg, masks, 2, 0)
    P = O.compact_panels(lw, idx)
    hd = len(idx["heads"]) * cfg.head_dim
    for i, h in enumerate(idx["heads"]):
        for j in (0, cfg.head_dim - 1):
            r = h * cfg.head_dim + j
            np.testing.assert_array_equal(P["wqkv"][i * cfg.head_dim + j], lw["wq"][r])
            np.testing.assert_array_equal(P["wqkv"][hd + i * cfg.head_dim + j], lw["wk"][r])
            np.testing.assert_array_equal(P["wqkv"][2 * hd + i * cfg.head_dim + j], lw["wv"][r])
            np.testing.assert_array_equal(P["wo"][:, i * cfg.head_dim + j], lw["wo"][:, r])
    c0 = idx["chunks"][1]
    np.testing.assert_array_equal(P["w_up"][8:16], lw["w_up"][c0 * 8:(c0 + 1) * 8])
    np.testing.assert_array_equal(P["w_down"][:, 8:16], lw["w_down"][:, c0 * 8:(c0 + 1) * 8])


# --------------------------------------------------------------------------- union super-model (Sec. 4.3)

def _hand_masks():
    """Tiny config, one layer, hand-made gates: head 1 and chunk 5 are kept at no step."""
    cfg = synth.tiny(has_cross=1)
    m = synth.make_masks(cfg)
    m["head_gate"][:, 0, :] = np.array([[1, 0, 0, 1], [0, 0, 1, 1], [0, 0, 0, 1], [1, 0, 0, 0]])
    m["xhead_gate"][:, 0, :] = np.array([[0, 0, 0, 1], [0, 0, 0, 1], [0, 1, 0, 0], [0, 1, 0, 1]])
    m["ffn_gate"][:] = 0
    m["ffn_gate"][0, 0, [0, 7]] = 1
    m["ffn_gate"][1, 0, [3]] = 1
    m["ffn_gate"][3, 0, [3, 7, 9]] = 1
    return cfg, m


def test_union_tables_on_hand_made_gates():
    cfg, m = _hand_masks()
    u = O.union_tables(cfg, m, 0)
    assert u["heads"].tolist() == [0, 2, 3]
    assert [p.tolist() for p in u["pos_heads"]] == [[0, 2], [1, 2], [2], [0]]
    assert u["chunks"].tolist() == [0, 3, 7, 9]
    assert [p.tolist() for p in u["pos_chunks"]] == [[0, 2], [1], [], [1, 2, 3]]
    assert u["xheads"].tolist() == [1, 3]
    assert [p.tolist() for p in u["pos_xheads"]] == [[1], [1], [0], [0, 1]]


def test_union_with_a_keep_all_step_is_every_unit():
    cfg = synth.tiny()          # step 0 keeps all 4 heads and all 128 chunks
    u = O.union_tables(cfg, synth.make_masks(cfg), 0)
    assert u["heads"].tolist() == list(range(cfg.n_heads))
    assert u["chunks"].tolist() == list(range(cfg.n_chunks))
    assert u["pos_heads"][0].tolist() == list(range(cfg.n_heads))


@pytest.mark.parametrize("hand", [False, True])
def test_union_panels_indexed_by_positions_are_the_step_panels(hand):
    """theta_union gathered through I_t gives exactly the exported per-step weights."""
    if hand:
        cfg, m = _hand_masks()
    else:
        cfg = synth.tiny(has_cross=1)
        cfg.heads_kept = [[2], [3], [1], [2]]
        cfg.chunks_kept = [[40], [90], [7], [64]]
        m = synth.make_masks(cfg, "union")
    lw = synth.make_layer(cfg, 0)
    u = O.union_tables(cfg, m, 0)
    U = O.union_panels(cfg, lw, u)
    dh, C = cfg.head_dim, cfg.ffn_chunk
    nu = len(u["heads"])
    for s in range(cfg.n_steps):
        P = O.compact_panels(lw, O.compact_indices(cfg, m, s, 0))
        ph = np.asarray(u["pos_heads"][s], dtype=np.int64)
        r = (ph[:, None] * dh + np.arange(dh)[None, :]).reshape(-1)
        rows = np.concatenate([r, nu * dh + r, 2 * nu * dh + r])
        np.testing.assert_array_equal(U["wqkv"][rows], P["wqkv"])
        np.testing.assert_array_equal(U["wo"][:, r], P["wo"])
        pc = np.asarray(u["pos_chunks"][s], dtype=np.int64)
        ch = (pc[:, None] * C + np.arange(C)[None, :]).reshape(-1)
        np.testing.assert_array_equal(U["w_up"][ch], P["w_up"])
        np.testing.assert_array_equal(U["w_down"][:, ch], P["w_down"])
        px = np.asarray(u["pos_xheads"][s], dtype=np.int64)
        xr = (px[:, None] * dh + np.arange(dh)[None, :]).reshape(-1)
        np.testing.assert_array_equal(U["cwq"][xr], P["cwq"])
        np.testing.assert_array_equal(U["cwo"][:, xr], P["cwo"])


# --------------------------------------------------------------------------- elementary ops

def test_linear_orientation_out_in():
    w = np.zeros((3, 5))
    w[2, 4] = 1.0
    x = rng().standard_normal((7, 5))
    y = O.linear(x, w, np.array([0.0, 0.0, 0.5]))
    np.testing.assert_allclose(y[:, 2], x[:, 4] + 0.5)
    np.testing.assert_allclose(y[:, :2], 0.0)


def test_modulation_affine_in_t_emb():
    d = 8
    r = rng(1)
    w_t, b_t, e = r.standard_normal((6 * d, d)), r.standard_normal(6 * d), r.standard_normal((6, d))
    np.testing.assert_allclose(O.modulation(w_t, b_t, e, np.zeros(d)), b_t.reshape(6, d) + e)
    t = np.zeros(d)
    t[3] = 1.0
    np.testing.assert_allclose(O.modulation(w_t, b_t, e, t), (w_t[:, 3] + b_t).reshape(6, d) + e)


def test_layer_norm_against_library_and_constant_row():
    torch = pytest.importorskip("torch")
    x = rng(2).standard_normal((9, 33)) * 3 + 1
    ref = torch.nn.functional.layer_norm(torch.from_numpy(x), (33,), eps=1e-6).numpy()
    np.testing.assert_allclose(O.layer_norm(x, 1e-6), ref, rtol=1e-12, atol=1e-12)
    w, b = rng(3).standard_normal(33), rng(4).standard_normal(33)
    ref = torch.nn.functional.layer_norm(torch.from_numpy(x), (33,), torch.from_numpy(w),
                                         torch.from_numpy(b), eps=1e-6).numpy()
    np.testing.assert_allclose(O.layer_norm(x, 1e-6, w, b), ref, rtol=1e-12, atol=1e-12)
    # a constant row normalises to zero, so adaLN returns the shift
    shift, scale = rng(5).standard_normal(33), rng(6).standard_normal(33)
    np.testing.assert_allclose(O.adaln(np.full((2, 33), 4.25), shift, scale, 1e-6),
                               np.tile(shift, (2, 1)), atol=1e-12)
    y = O.layer_norm(x, 0.0)
    np.testing.assert_allclose(y.mean(-1), 0, atol=1e-12)
    np.testing.assert_allclose((y ** 2).mean(-1), 1, atol=1e-12)


def test_rms_norm_closed_forms():
    a = 2.5
    signs = rng(7).choice([-1.0, 1.0], size=(4, 16))
    g = 1 + 0.1 * rng(8).standard_normal(16)
    keep = np.ones(16)
    y = O.rms_norm(a * signs, g, keep, 0.0, 0, 8)
    np.testing.assert_allclose(y, signs * g, rtol=1e-14)
    # pruned channels do not enter the statistic (mode 0) and come out zero
    keep = np.array([1] * 8 + [0] * 8, dtype=np.float64)
    x = a * signs
    x2 = x.copy()
    x2[:, 8:] = 1e3 * rng(9).standard_normal((4, 8))
    y1, y2 = O.rms_norm(x, g, keep, 0.0, 0, 8), O.rms_norm(x2, g, keep, 0.0, 0, 8)
    np.testing.assert_array_equal(y1, y2)
    np.testing.assert_allclose(y1[:, :8], signs[:, :8] * g[:8], rtol=1e-14)
    np.testing.assert_array_equal(y1[:, 8:], 0.0)
    # mode 1: each head has its own statistic, so scaling one head changes nothing
    x = rng(10).standard_normal((3, 16))
    xs = x.copy()
    xs[:, 8:] *= 17.0
    np.testing.assert_allclose(O.rms_norm(x, g, np.ones(16), 0.0, 1, 8),
                               O.rms_norm(xs, g, np.ones(16), 0.0, 1, 8), rtol=1e-13)
    # ... while in mode 0 it does
    assert not np.allclose(O.rms_norm(x, g, np.ones(16), 0.0, 0, 8)[:, :8],
                           O.rms_norm(xs, g, np.ones(16), 0.0, 0, 8)[:, :8])


@pytest.mark.parametrize("dh,bands", [(128, (22, 21, 21)), (64, (12, 10, 10))])
def test_rope_band_sizes(dh, bands):
    assert O.rope_pairs(dh) == bands
    assert sum(bands) == dh // 2


def test_rope_angles_explicit_values():
    grid, dh, th = (3, 4, 5), 64, 10000.0
    p_t, p_h, p_w = O.rope_pairs(dh)
    ang = O.rope_angles(grid, dh, th)
    tok = lambda f, y, w: (f * grid[1] + y) * grid[2] + w
    assert np.all(ang[tok(0, 0, 0)] == 0)
    # the first pair of each band turns by the position itself
    assert ang[tok(2, 0, 0), 0] == 2.0
    assert ang[tok(0, 3, 0), p_t] == 3.0
    assert ang[tok(0, 0, 4), p_t + p_h] == 4.0
    # pair j of the frame band turns by f * theta^(-j / p_t)
    np.testing.assert_allclose(ang[tok(1, 0, 0), 5], th ** (-5 / p_t), rtol=1e-15)
    np.testing.assert_allclose(ang[tok(0, 2, 0), p_t + 3], 2 * th ** (-3 / p_h), rtol=1e-15)
    # a token that differs only in w shares the frame and height angles
    a, b = ang[tok(1, 2, 0)], ang[tok(1, 2, 3)]
    np.testing.assert_array_equal(a[:p_t + p_h], b[:p_t + p_h])
    assert np.all(a[p_t + p_h + 1:] != b[p_t + p_h + 1:])


def test_rope_equals_complex_multiplication_and_is_relative():
    grid, dh = (2, 3, 4), 64
    ang = O.rope_angles(grid, dh, 10000.0)
    N = ang.shape[0]
    x = rng(11).standard_normal((N, 2, dh))
    y = O.apply_rope(x, ang)
    z = (x[..., 0::2] + 1j * x[..., 1::2]) * np.exp(1j * ang)[:, None, :]
    np.testing.assert_allclose(y[..., 0::2], z.real, atol=1e-13)
    np.testing.assert_allclose(y[..., 1::2], z.imag, atol=1e-13)
    np.testing.assert_allclose(np.linalg.norm(y, axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-13)
    # <R(p) q, R(p') k> = <q, R(p' - p) k> along one axis (width, here)
    q, k = rng(12).standard_normal((1, 1, dh)), rng(13).standard_normal((1, 1, dh))
    tok = lambda f, y_, w: (f * grid[1] + y_) * grid[2] + w
    lhs = np.sum(O.apply_rope(q, ang[[tok(1, 1, 1)]]) * O.apply_rope(k, ang[[tok(1, 1, 3)]]))
    rhs = np.sum(q * O.apply_rope(k, ang[[tok(0, 0, 2)]]))
    np.testing.assert_allclose(lhs, rhs, rtol=1e-12)


def _attention_brute(q, k, v):
    n, h, dh = q.shape
    m = k.shape[0]
    out = np.zeros((n, h, v.shape[2]))
    for j in range(h):
        for i in range(n):
            logits = [sum(q[i, j, c] * k[t, j, c] for c in range(dh)) / math.sqrt(dh)
                      for t in range(m)]
            mx = max(logits)
            w = [math.exp(l - mx) for l in logits]
            z = sum(w)
            for c in range(v.shape[2]):
                out[i, j, c] = sum(w[t] * v[t, j, c] for t in range(m)) / z
    return out


def test_attention_brute_force():
    r = rng(14)
    q, k, v = r.standard_normal((5, 2, 4)) * 2, r.standard_normal((7, 2, 4)), r.standard_normal((7, 2, 4))
    np.testing.assert_allclose(O.attention(q, k, v), _attention_brute(q, k, v), rtol=1e-12, atol=1e-14)


def test_attention_special_cases():
    r = rng(15)
    dh = 4
    # identical keys -> uniform weights -> mean of V
    q = r.standard_normal((3, 1, dh))
    k = np.tile(r.standard_normal((1, 1, dh)), (6, 1, 1))
    v = r.standard_normal((6, 1, dh))
    np.testing.assert_allclose(O.attention(q, k, v)[:, 0], np.tile(v[:, 0].mean(0), (3, 1)), rtol=1e-13)
    # logit gap of ln 2 after the 1/sqrt(dh) scale -> weights 2/3 and 1/3
    q = np.zeros((1, 1, dh)); q[0, 0, 0] = 2 * math.log(2.0)
    k = np.zeros((2, 1, dh)); k[0, 0, 0] = 1.0
    v = np.zeros((2, 1, dh)); v[0, 0, 0] = 3.0; v[1, 0, 0] = 0.0
    np.testing.assert_allclose(O.attention(q, k, v)[0, 0, 0], 2.0, rtol=1e-14)
    # one dominant logit selects its value row
    q = np.zeros((1, 1, dh)); q[0, 0, 1] = 2000.0
    k = r.standard_normal((5, 1, dh)) * 0.01; k[3, 0, 1] = 1.0
    v = r.standard_normal((5, 1, dh))
    np.testing.assert_allclose(O.attention(q, k, v)[0, 0], v[3, 0], rtol=1e-12)


def test_gelu_tanh_textbook():
    x = np.linspace(-6, 6, 241)
    g = O.gelu_tanh(x)
    assert O.gelu_tanh(np.array([0.0]))[0] == 0.0
    np.testing.assert_allclose(g - O.gelu_tanh(-x), x, atol=1e-14)
    exact = np.array([v * 0.5 * (1 + math.erf(v / math.sqrt(2))) for v in x])
    assert np.max(np.abs(g - exact)) < 1e-3
    assert np.max(np.abs(g - exact)) > 1e-5        # it is the tanh form, not the erf form


# --------------------------------------------------------------------------- the block

def _problem(has_cross=0, mode=0, grid=(2, 4, 4), ctx_len=16, seed_tag=""):
    cfg = synth.tiny(has_cross=has_cross, grid=grid, qk_norm_mode=mode)
    cfg.ctx_len = ctx_len if has_cross else 0
    sh, L, M, A = synth.make_problem(cfg, seed_tag)
    return cfg, synth.widen(sh), synth.widen(L), M, synth.widen(A)


@pytest.mark.parametrize("has_cross,mode", [(0, 0), (0, 1), (1, 0)])
def test_masked_dense_equals_compacted(has_cross, mode):
    """Eq. 2 + export (Sec. 3.2) + index tables (Sec. 4.3): same function."""
    cfg, W, LW, M, X = _problem(has_cross, mode)
    for s in range(4):
        a, ia = O.block_forward_masked(cfg, W, LW[0], M, s, 0, X["x"], X["t_emb"][s],
                                       X.get("ctx"), want=True)
        b, ib = O.block_forward_compacted(cfg, W, LW[0], M, s, 0, X["x"], X["t_emb"][s],
                                          X.get("ctx"), want=True)
        np.testing.assert_allclose(a, b, rtol=0, atol=1e-12 * np.abs(a).max())
        np.testing.assert_allclose(ia["x1"], ib["x1"], rtol=0, atol=1e-12 * np.abs(ia["x1"]).max())
        # the pruned branch is not the identity
        assert np.abs(a - X["x"]).max() > 1e-2


def test_row_slice_equals_full():
    cfg, W, LW, M, X = _problem(1, 0)
    rows = np.array([0, 5, 17, 31])
    full = O.block_forward_compacted(cfg, W, LW[0], M, 1, 0, X["x"], X["t_emb"][1], X["ctx"])
    part = O.block_forward_compacted(cfg, W, LW[0], M, 1, 0, X["x"], X["t_emb"][1], X["ctx"], rows=rows)
    np.testing.assert_allclose(part, full[rows], rtol=1e-13, atol=1e-13)
    part = O.block_forward_masked(cfg, W, LW[0], M, 1, 0, X["x"], X["t_emb"][1], X["ctx"], rows=rows)
    np.testing.assert_allclose(part, full[rows], rtol=1e-11, atol=1e-11)


def test_keep_all_is_the_unpruned_block():
    cfg, W, LW, M, X = _problem()
    M1 = dict(M)
    M1["head_gate"] = np.ones_like(M["head_gate"])
    M1["ffn_gate"] = np.ones_like(M["ffn_gate"])
    a, ia = O.block_forward_compacted(cfg, W, LW[0], M1, 3, 0, X["x"], X["t_emb"][3], want=True)
    # mode-0 QK norm over all retained channels is then the full-row RMSNorm
    q_raw = O.linear(ia["xm"], LW[0]["wq"], LW[0]["bq"])
    full = q_raw / np.sqrt((q_raw ** 2).mean(-1, keepdims=True) + cfg.ln_eps) * LW[0]["gq"]
    ang = O.rope_angles(cfg.grid, cfg.head_dim, cfg.rope_theta)
    np.testing.assert_allclose(ia["q"], O.apply_rope(full.reshape(-1, 4, 64), ang), rtol=1e-12, atol=1e-12)
    b = O.block_forward_masked(cfg, W, LW[0], M1, 3, 0, X["x"], X["t_emb"][3])
    np.testing.assert_allclose(a, b, atol=1e-12)


def test_empty_masks_reduce_to_bias_branches():
    cfg, W, LW, M, X = _problem()
    M0 = dict(M)
    M0["head_gate"] = np.zeros_like(M["head_gate"])
    M0["ffn_gate"] = np.zeros_like(M["ffn_gate"])
    mod = O.modulation(W["w_t"], W["b_t"], LW[0]["e_mod"], X["t_emb"][0])
    for fn in (O.block_forward_masked, O.block_forward_compacted):
        out, it = fn(cfg, W, LW[0], M0, 0, 0, X["x"], X["t_emb"][0], want=True)
        x1 = X["x"] + mod[2] * LW[0]["bo"]
        np.testing.assert_allclose(it["x1"], x1, atol=1e-14)
        np.testing.assert_allclose(out, x1 + mod[5] * LW[0]["b_down"], atol=1e-14)


def test_block_gate_zero_is_identity():
    cfg, W, LW, M, X = _problem()
    Mb = dict(M)
    Mb["block_gate"] = np.zeros_like(M["block_gate"])
    for fn in (O.block_forward_masked, O.block_forward_compacted):
        np.testing.assert_array_equal(fn(cfg, W, LW[0], Mb, 1, 0, X["x"], X["t_emb"][1]), X["x"])


def test_modulation_vectors_land_where_read():
    """Zeroing gate_a removes the attention branch; 1+scale_f = 0 makes xm2 = shift_f."""
    cfg, W, LW, M, X = _problem()
    t = X["t_emb"][2]
    base = (W["w_t"] @ t + W["b_t"]).reshape(6, cfg.dim)
    lw = dict(LW[0])
    e = lw["e_mod"].copy()
    e[2] = -base[2]
    e[4] = -1.0 - base[4]
    lw["e_mod"] = e
    out, it = O.block_forward_compacted(cfg, W, lw, M, 2, 0, X["x"], t, want=True)
    np.testing.assert_array_equal(it["x1"], X["x"])
    np.testing.assert_allclose(it["xm2"], np.tile(base[3] + e[3], (cfg.n_tokens, 1)), atol=1e-12)


def _cross_branch(fn, cfg, W, lw, M, s, X):
    """The cross-attention branch of one block (R6): x1 after the cross-attention minus x1
    before it, with the cross-attention's input and its LayerNorm output."""
    _, it = fn(cfg, W, lw, M, s, 0, X["x"], X["t_emb"][s], X["ctx"], want=True)
    return it["x1"] - it["x1a"], it["x1a"], it["xc"]


@pytest.mark.parametrize("form", ["masked", "compacted"])
def test_cross_layer_norm_weight_zero_gives_one_query_row(form):
    """R6 with cln_w = 0: LN(x1) cln_w + cln_b = cln_b for every token, so every query row is
    the same, the branch is one row repeated, and that row is the softmax of a single query
    over the context keys (brute force) projected by Wo_c."""
    fn = O.block_forward_masked if form == "masked" else O.block_forward_compacted
    cfg, W, LW, M, X = _problem(has_cross=1)
    lw = dict(LW[0])
    lw["cln_w"] = np.zeros_like(lw["cln_w"])
    s = 1
    br, x1a, xc = _cross_branch(fn, cfg, W, lw, M, s, X)
    np.testing.assert_array_equal(xc, np.tile(lw["cln_b"], (x1a.shape[0], 1)))
    np.testing.assert_allclose(br, np.tile(br[0], (br.shape[0], 1)), rtol=0, atol=1e-12 * np.abs(br).max())
    # the one row by hand: retained cross heads, full-row RMSNorm over their channels (R4 mode 0)
    H, dh, eps = cfg.n_heads, cfg.head_dim, cfg.ln_eps
    heads = np.flatnonzero(M["xhead_gate"][s, 0])
    r = (heads[:, None] * dh + np.arange(dh)[None, :]).reshape(-1)

    def rms(a, g):
        return a / np.sqrt((a ** 2).mean(-1, keepdims=True) + eps) * g

    q = rms(lw["cwq"][r] @ lw["cln_b"] + lw["cbq"][r], lw["cgq"][r])
    k = rms(X["ctx"] @ lw["cwk"][r].T + lw["cbk"][r], lw["cgk"][r])
    v = X["ctx"] @ lw["cwv"][r].T + lw["cbv"][r]
    L, h = X["ctx"].shape[0], len(heads)
    o = _attention_brute(q.reshape(1, h, dh), k.reshape(L, h, dh), v.reshape(L, h, dh)).reshape(-1)
    want = lw["cwo"][:, r] @ o + lw["cbo"]
    np.testing.assert_allclose(br[0], want, rtol=1e-10, atol=1e-12)


@pytest.mark.parametrize("form", ["masked", "compacted"])
def test_cross_layer_norm_is_the_library_affine_layer_norm(form):
    """R6: the cross-attention reads torch's affine LayerNorm of x1 (weight cln_w, bias cln_b);
    with cln_w = 1 and cln_b = 0 that is the plain LayerNorm."""
    torch = pytest.importorskip("torch")
    fn = O.block_forward_masked if form == "masked" else O.block_forward_compacted
    cfg, W, LW, M, X = _problem(has_cross=1)
    d = cfg.dim
    for w, b in ((LW[0]["cln_w"], LW[0]["cln_b"]), (np.ones(d), np.zeros(d))):
        lw = dict(LW[0], cln_w=w, cln_b=b)
        _, x1a, xc = _cross_branch(fn, cfg, W, lw, M, 2, X)
        ref = torch.nn.functional.layer_norm(torch.from_numpy(x1a), (d,), torch.from_numpy(w),
                                             torch.from_numpy(b), eps=cfg.ln_eps).numpy()
        np.testing.assert_allclose(xc, ref, rtol=1e-12, atol=1e-12)


# --------------------------------------------------------------------------- FLOPs

@pytest.mark.parametrize("has_cross", [0, 1])
def test_flop_closed_form_matches_executed_contractions(has_cross):
    cfg, W, LW, M, X = _problem(has_cross)
    for s in range(4):
        c = O.MacCounter()
        O.block_forward_compacted(cfg, W, LW[0], M, s, 0, X["x"], X["t_emb"][s], X.get("ctx"), counter=c)
        idx = O.compact_indices(cfg, M, s, 0)
        f = O.block_flops(cfg.n_tokens, cfg.dim, cfg.head_dim, len(idx["heads"]), len(idx["ffn_ch"]),
                          len(idx["xheads"]) if has_cross else 0, cfg.ctx_len)
        assert c.flops == f


def test_flop_keep_reproduces_paper_cut():
    """The 14B-shaped keep schedule removes the paper's 24% of per-step FLOPs."""
    cfg = synth.wan14b()
    f = [O.block_flops(cfg.n_tokens, cfg.dim, cfg.head_dim, cfg.heads_kept[s][0],
                       8 * cfg.chunks_kept[s][0]) for s in range(4)]
    mean_keep = np.mean(f) / f[0]
    assert abs((1 - mean_keep) - GOLD["wan14b_per_step_flop_cut"]["value"]) < 0.01
    assert mean_keep <= GOLD["stop_criterion_mean_flops"]["value"] + 0.02
    # the paper's U-shaped 1.3B retention averages to its ~83% final checkpoint
    assert abs(np.mean(GOLD["wan13b_step_retention"]["value"]) - GOLD["wan13b_final_flop_ratio"]["value"]) < 0.01
    # closed-form dense 14B block: 38.1 TFLOP, attention the largest share
    assert abs(f[0] - 3.8125e13) / 3.8125e13 < 1e-3


def test_policy_shaped_masks_reproduce_the_paper_retention():
    """The policy-shaped workload keeps the per-step FLOP fractions the paper reports for its
    learned Wan-1.3B policy (Sec. 6) and has its described shape."""
    cfg = synth.wan13b_policy()
    N, d, dh = cfg.n_tokens, cfg.dim, cfg.head_dim
    dense = O.block_flops(N, d, dh, cfg.n_heads, cfg.ffn_dim, cfg.n_heads, cfg.ctx_len)
    ret = []
    for s in range(4):
        f = [O.block_flops(N, d, dh, cfg.heads_kept[s][l], 8 * cfg.chunks_kept[s][l], cfg.xheads_kept[s][l],
                           cfg.ctx_len) for l in range(cfg.n_layers)]
        ret.append(sum(f) / (cfg.n_layers * dense))
    paper = GOLD["wan13b_step_retention"]["value"]
    assert max(abs(a - b) for a, b in zip(ret, paper)) < 0.005, ret
    assert abs(np.mean(ret) - GOLD["wan13b_final_flop_ratio"]["value"]) < 0.01
    assert ret[0] > ret[1] and ret[3] > ret[2] and min(ret[0], ret[3]) > max(ret[1], ret[2])  # U shape
    for s in range(4):
        h, c = cfg.heads_kept[s], cfg.chunks_kept[s]
        assert all(a >= b for a, b in zip(h, h[1:])) and all(a >= b for a, b in zip(c, c[1:]))  # depth
        # attention keeps a smaller fraction than the FFN in the deepest layer
        assert h[-1] / cfg.n_heads < c[-1] / cfg.n_chunks
    assert cfg.heads_kept[1][-1] == 0 and cfg.heads_kept[2][-1] == 0       # deepest layer shut down
    assert cfg.heads_kept[0][-1] > 0 and cfg.heads_kept[3][-1] > 0


def test_denoise_with_all_blocks_off_is_geometric():
    cfg, W, LW, M, X = _problem()
    Mb = dict(M)
    Mb["block_gate"] = np.zeros_like(M["block_gate"])
    out = O.denoise(cfg, W, LW, Mb, X["x"], X["t_emb"])
    np.testing.assert_allclose(out, X["x"] * (1 + 1 / GOLD["n_steps"]["value"]) ** 4, rtol=1e-14)


# --------------------------------------------------------------------------- model around the blocks (R16-R19)

def test_patchify_places_each_latent_element_by_hand():
    C, F, H, W = 2, 2, 4, 6
    lat = np.zeros((C, F, H, W))
    for c in range(C):
        for f in range(F):
            for y in range(H):
                for x in range(W):
                    lat[c, f, y, x] = 1000 * c + 100 * f + 10 * y + x
    tok = O.patchify(lat)
    assert tok.shape == (F * 2 * 3, 4 * C)
    # the patch at frame 1, patch row 1, patch column 1 (token grid 2 x 3): latent rows 2, 3 and
    # columns 2, 3; token (1 * 2 + 1) * 3 + 1 = 10; features c*4 + dy*2 + dx
    n = (1 * 2 + 1) * 3 + 1
    assert tok[n].tolist() == [100 + 20 + 2, 100 + 20 + 3, 100 + 30 + 2, 100 + 30 + 3,
                               1100 + 20 + 2, 1100 + 20 + 3, 1100 + 30 + 2, 1100 + 30 + 3]
    np.testing.assert_array_equal(O.unpatchify(tok, lat.shape), lat)


def test_timestep_embedding_textbook_values():
    np.testing.assert_array_equal(O.timestep_embedding(0.0, 8), [1, 1, 1, 1, 0, 0, 0, 0])
    e = O.timestep_embedding(1.0, 4)      # w = [1, 10000^-0.5]
    np.testing.assert_allclose(e, [math.cos(1), math.cos(0.01), math.sin(1), math.sin(0.01)], rtol=1e-15)
    e = O.timestep_embedding(750.0, 256)
    np.testing.assert_allclose(e[:128] ** 2 + e[128:] ** 2, 1.0, rtol=1e-12)


def test_time_mlp_silu():
    d, D = 4, 8
    mw = {"t_w1": np.zeros((d, D)), "t_b1": np.array([0.0, 1.0, -1.0, 3.0]), "t_w2": np.eye(d),
          "t_b2": np.array([0.5, 0, 0, 0])}
    sig = lambda v: 1 / (1 + math.exp(-v))
    np.testing.assert_allclose(O.time_mlp(mw, 123.0), [0.5, sig(1.0), -sig(-1.0), 3 * sig(3.0)], rtol=1e-15)


def _model_problem(seed_tag=""):
    cfg = synth.tiny_model(n_layers=2)
    cfg.grid = (2, 4, 4)
    sh, L, M, A = synth.make_problem(cfg, seed_tag)
    mw = synth.widen(synth.make_model_weights(cfg, seed_tag))
    lat = synth.bits_to_f64(synth.make_latent(cfg, seed_tag))
    return cfg, synth.widen(sh), synth.widen(L), M, synth.widen(A), mw, lat


def test_model_head_reads_only_its_bias_when_its_weights_vanish():
    cfg, W, LW, M, X, mw, lat = _model_problem()
    mw = dict(mw)
    mw["head_w"] = np.zeros_like(mw["head_w"])
    v = O.model_forward(cfg, W, LW, mw, M, 1, lat, 750.0, X["ctx"])
    want = O.unpatchify(np.tile(mw["head_b"], (cfg.n_tokens, 1)), lat.shape)
    np.testing.assert_allclose(v, want, rtol=0, atol=0)


def test_model_head_scale_minus_one_returns_the_shift():
    """R18: with head_mod[1] = -1 - t_emb the head's 1 + scale_h vanishes, so every token's
    head input is shift_h = head_mod[0] + t_emb and the velocity is that one row projected."""
    cfg, W, LW, M, X, mw, lat = _model_problem()
    t = 500.0
    t_emb = O.time_mlp(mw, t)
    mw = dict(mw)
    hm = mw["head_mod"].copy()
    hm[1] = -1.0 - t_emb
    mw["head_mod"] = hm
    v = O.model_forward(cfg, W, LW, mw, M, 2, lat, t, X["ctx"])
    row = mw["head_w"] @ (hm[0] + t_emb) + mw["head_b"]
    want = O.unpatchify(np.tile(row, (cfg.n_tokens, 1)), lat.shape)
    np.testing.assert_allclose(v, want, rtol=1e-12, atol=1e-12)


def test_model_head_without_modulation_is_the_library_layer_norm():
    """R18: with shift_h = scale_h = 0 (head_mod = -t_emb in both rows) the head is torch's
    plain LayerNorm of the last block's output followed by the head projection."""
    torch = pytest.importorskip("torch")
    cfg, W, LW, M, X, mw, lat = _model_problem()
    t = 250.0
    t_emb = O.time_mlp(mw, t)
    mw = dict(mw)
    mw["head_mod"] = np.stack([-t_emb, -t_emb])
    v, it = O.model_forward(cfg, W, LW, mw, M, 3, lat, t, X["ctx"], want=True)
    y = torch.nn.functional.layer_norm(torch.from_numpy(it["x_last"]), (cfg.dim,), eps=cfg.ln_eps).numpy()
    want = O.unpatchify(y @ mw["head_w"].T + mw["head_b"], lat.shape)
    np.testing.assert_allclose(v, want, rtol=1e-10, atol=1e-12)


def test_model_blocks_off_leave_the_embedded_patches():
    """With every block gated off the head sees the patch embedding itself."""
    cfg, W, LW, M, X, mw, lat = _model_problem()
    Mb = dict(M)
    Mb["block_gate"] = np.zeros_like(M["block_gate"])
    v, it = O.model_forward(cfg, W, LW, mw, Mb, 0, lat, 1000.0, X["ctx"], want=True)
    np.testing.assert_array_equal(it["x_last"], O.patchify(lat) @ mw["patch_w"].T + mw["patch_b"])
    np.testing.assert_allclose(it["t_emb"], O.time_mlp(mw, 1000.0))


def test_model_denoise_sums_the_step_velocities():
    cfg, W, LW, M, X, mw, lat = _model_problem()
    ts = synth.model_timesteps(4)
    assert ts == [1000.0, 750.0, 500.0, 250.0]
    z = lat.copy()
    vs = []
    for s in range(4):
        v = O.model_forward(cfg, W, LW, mw, M, s, z, ts[s], X["ctx"])
        vs.append(v)
        z = z + v / 4
    np.testing.assert_allclose(O.model_denoise(cfg, W, LW, mw, M, lat, ts, X["ctx"]), lat + sum(vs) / 4,
                               rtol=1e-12, atol=1e-12)


# --------------------------------------------------------------------------- input generator

def test_bf16_rounding_matches_torch():
    torch = pytest.importorskip("torch")
    a = np.concatenate([rng(16).standard_normal(5000).astype(np.float32),
                        np.array([1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -1.0 - 2 ** -8, 0.0], np.float32)])
    ref = torch.from_numpy(a).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(synth.f32_to_bf16_bits(a), ref)


def test_config_keep_counts():
    c2, c3 = synth.wan13b(), synth.wan14b()
    assert [c2.heads_kept[s][0] for s in range(4)] == [12, 10, 9, 8]
    assert [8 * c2.chunks_kept[s][0] for s in range(4)] == [8960, 7616, 6720, 5824]
    assert [c3.heads_kept[s][0] for s in range(4)] == [40, 32, 28, 22]
    assert [8 * c3.chunks_kept[s][0] for s in range(4)] == [13824, 11056, 9680, 7600]
    assert c3.n_tokens == 32760 and synth.sweep720(0.5).n_tokens == 75600
