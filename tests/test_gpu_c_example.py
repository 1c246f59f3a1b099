"""The C ABI from plain C: paper_2607_06631_gb300/examples/block_forward.c (CUDA runtime +
libdfs.so, no Python in the process) gives the same block output, bit for bit, as the
Python binding on the same inputs."""
import os
import subprocess

import numpy as np
import pytest

import synth

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
LAYER0 = ("wq", "bq", "wk", "bk", "wv", "bv", "wo", "bo", "gq", "gk", "w_up", "b_up", "w_down", "b_down", "e_mod")


def test_plain_c_program_matches_the_python_binding(tmp_path):
    import torch
    from paper_2607_06631_gb300 import build, dfs, host
    lib = build.build()
    cfg = synth.tiny()
    shared, layers, m, acts = synth.make_problem(cfg)
    d = str(tmp_path)
    with open(os.path.join(d, "config.txt"), "w") as f:
        f.write("%d %d %d %d %d %d %d %d %d\n" % (cfg.dim, cfg.n_heads, cfg.head_dim, cfg.ffn_dim, cfg.n_layers,
                                                cfg.n_steps, *cfg.grid))
    for name, arr in list(shared.items()) + [(k, layers[0][k]) for k in LAYER0] + [("x", acts["x"]),
                                                                                  ("t_emb", acts["t_emb"])]:
        np.ascontiguousarray(arr, dtype=np.uint16).tofile(os.path.join(d, name + ".bin"))
    for g in ("block_gate", "head_gate", "ffn_gate"):
        np.ascontiguousarray(m[g], dtype=np.uint8).tofile(os.path.join(d, g + ".bin"))
    exe = os.path.join(d, "block_forward")
    libdir = os.path.dirname(lib)
    subprocess.run([build._nvcc(), "-O2", "-I", os.path.join(ROOT, "include"),
                    os.path.join(ROOT, "paper_2607_06631_gb300", "examples", "block_forward.c"),
                    "-L", libdir, "-ldfs", "-lcudart", "-Xlinker", "-rpath=" + libdir, "-o", exe],
                   check=True, capture_output=True, text=True)
    step = 2
    r = subprocess.run([exe, d, str(step)], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stdout + r.stderr
    got = np.fromfile(os.path.join(d, "out.bin"), dtype=np.uint16)

    prob = host.DeviceProblem(cfg, shared, layers, m, acts)
    plan = prob.create_plan()
    out = torch.empty_like(prob.x)
    dfs.dfs_block_forward(plan, step, prob.x, prob.t_emb[step], out)
    dfs.dfs_plan_sync(plan)
    np.testing.assert_array_equal(got.reshape(-1), host.to_bits(out).reshape(-1))
