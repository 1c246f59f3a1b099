"""bench.py's per-kernel algorithmic units (the roofline numerators) against the oracle's FLOP
closed form: the tensor kinds of one bench step must add up to the oracle's block FLOPs of
every (step, layer), and the HBM byte counts must be the stated per-kernel formulas."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import oracle as O  # noqa: E402
import synth  # noqa: E402


@pytest.mark.parametrize("name", ["tiny", "wan13b", "wan14b", "wan14b_cross", "sweep720", "wan13b_policy"])
def test_tensor_units_equal_the_oracle_block_flops(name):
    import bench
    cfg = bench.get_config(name)
    units, bound = bench.kernel_units(cfg)
    tensor = sum(v for k, v in units.items() if bound[k] == "tensor")
    want = 0.0
    for s in range(cfg.n_steps):
        for l in range(cfg.n_layers):
            hc = cfg.xheads_kept[s][l] if cfg.has_cross else 0
            want += O.block_flops(cfg.n_tokens, cfg.dim, cfg.head_dim, cfg.heads_kept[s][l], 8 * cfg.chunks_kept[s][l],
                                  hc, cfg.ctx_len)
    # the cross-attention context K / V projections are computed once per plan, not per step
    if cfg.has_cross:
        want -= sum(4.0 * cfg.ctx_len * cfg.dim * cfg.head_dim * cfg.xheads_kept[s][l]
                    for s in range(cfg.n_steps) for l in range(cfg.n_layers))
    assert tensor == pytest.approx(want, rel=1e-12)


def test_wan14b_step_flops_are_the_closed_form_values():
    """Per-step FLOPs of the 14B-shaped block at its keep schedule (40/32/28/22 heads,
    13824/11056/9680/7600 FFN channels): 8 N d dh h + 4 N^2 dh h + 4 N d f."""
    cfg = synth.wan14b()
    got = [O.block_flops(cfg.n_tokens, cfg.dim, cfg.head_dim, cfg.heads_kept[s][0], 8 * cfg.chunks_kept[s][0])
           for s in range(4)]
    N, d, dh = 32760, 5120, 128
    for g, (h, f) in zip(got, [(40, 13824), (32, 11056), (28, 9680), (22, 7600)]):
        assert g == 8 * N * d * dh * h + 4 * N * N * dh * h + 4 * N * d * f
    assert [round(g / 1e13, 4) for g in got] == [3.8125, 3.0498, 2.6689, 2.0966]


def test_hbm_units_are_the_stated_byte_counts():
    import bench
    cfg = synth.wan14b()
    units, bound = bench.kernel_units(cfg)
    N, d = cfg.n_tokens, cfg.dim
    assert bound["adaln"] == "hbm" and units["adaln"] == cfg.n_steps * (N * d * 4 + N * d * 6)
    hsum = sum(cfg.heads_kept[s][0] for s in range(cfg.n_steps)) * cfg.head_dim
    assert units["qk_norm_rope"] == 2.0 * N * 2 * hsum * 2
    assert units["modulation"] == cfg.n_steps * 6.0 * d * d * 2


def test_reference_arm_prints_one_contract_line_on_the_tiny_block():
    """`bench.py --impl reference` (the oracle timed on the host cores) prints one JSON line with
    the contract's keys; on the tiny configuration each step is the whole block."""
    import json
    import subprocess
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--config", "tiny",
                        "--steps", "1", "--warmup", "0"], capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["unit"] == "TFLOP/s" and d["value"] > 0 and d["higher_is_better"]
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["value"] == d["value"]
    assert "whole MoM step" in d["cpu_baseline"]["sample"] and "512-token block" in d["cpu_baseline"]["sample"]


def test_cpu_baseline_slice_extrapolation_on_a_small_block():
    """cpu_baseline times K / V over all N once (one query row) and a 512-row slice, and
    extrapolates the block as T_KV + (N / 512) T_rows; a stack at that block's FLOP rate."""
    import copy
    import bench
    cfg = synth.tiny(grid=(2, 16, 32))  # 1024 tokens: two slices' worth
    cfg.name = "tiny_1024"
    c = bench.cpu_baseline(cfg)
    N = cfg.n_tokens
    assert c["kind"] == "oracle" and c["value"] > 0 and c["slice_rows"] == 512
    t = c["T_KV_s"] + (N / 512) * c["T_rows_s"]
    assert abs(c["block_seconds_extrapolated"] - t) <= 0.02 + 1e-3 * t
    assert "T = T_KV + (N / 512) T_rows" in c["formula"]
    stack = copy.deepcopy(synth.tiny(n_layers=3))
    s = bench.cpu_baseline(stack)
    assert s["stack_seconds_extrapolated"] > 0
    rate = s["block_flops"] / s["block_seconds_extrapolated"]
    assert abs(s["stack_seconds_extrapolated"] - bench.stack_flops(stack) / rate) <= 0.1 + 1e-3 * s["stack_seconds_extrapolated"]
