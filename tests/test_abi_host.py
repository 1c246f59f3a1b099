"""CPU-side checks of the C ABI: the library builds, loads without a GPU and exports
every entry point the header declares; host-only logic (argument validation before any
CUDA call, the soft-mask -> gate rules of Sec. 4.1) matches the oracle."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle as O
import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def dfs():
    from paper_2607_06631_gb300 import build, dfs as D
    build.build()
    return D


def header_symbols():
    src = open(os.path.join(ROOT, "include", "dfs.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(dfs_[a-z_]+)\s*\(", src)))


def test_library_exports_every_declared_symbol(dfs):
    syms = header_symbols()
    assert len(syms) >= 13
    lib = ctypes.CDLL(dfs.lib()._name)
    for s in syms:
        assert hasattr(lib, s), s
    assert set(syms) == set(dfs.EXPORTED)


def _valid_args(dfs, cfg):
    layers = [{k: 16 for k in dfs.LAYER_FIELDS}]  # non-null dummy pointers; never dereferenced
    masks = synth.make_masks(cfg)
    return layers, masks


@pytest.mark.parametrize("field,value", [("head_dim", 96), ("dim", 300), ("ffn_chunk", 16), ("ffn_dim", 1020),
                                         ("n_steps", 0), ("n_steps", 9), ("qk_norm_mode", 2),
                                         ("has_cross", 2), ("n_layers", 0)])
def test_plan_create_rejects_bad_config_without_touching_cuda(dfs, field, value):
    cfg = synth.tiny()
    layers, masks = _valid_args(dfs, cfg)
    c = dfs.make_config(cfg)
    setattr(c, field, value)
    with pytest.raises(dfs.DfsError) as e:
        dfs.dfs_plan_create(c, layers, 16, 16, masks, None, 0)
    assert e.value.status in (dfs.DFS_EINVAL, dfs.DFS_EUNSUPPORTED)
    assert dfs.dfs_last_error()


def test_plan_create_rejects_bad_masks_and_pointers(dfs):
    cfg = synth.tiny()
    layers, masks = _valid_args(dfs, cfg)
    bad = dict(masks)
    bad["head_gate"] = masks["head_gate"].copy()
    bad["head_gate"][1, 0, 2] = 2
    with pytest.raises(dfs.DfsError) as e:
        dfs.dfs_plan_create(cfg, layers, 16, 16, bad, None, 0)
    assert e.value.status == dfs.DFS_EINVAL and "0 or 1" in dfs.dfs_last_error()
    nul = [dict(layers[0])]
    nul[0]["w_up"] = None
    with pytest.raises(dfs.DfsError) as e:
        dfs.dfs_plan_create(cfg, nul, 16, 16, masks, None, 0)
    assert e.value.status == dfs.DFS_EINVAL
    with pytest.raises(dfs.DfsError) as e:
        dfs.dfs_plan_create(cfg, layers, None, 16, masks, None, 0)
    assert e.value.status == dfs.DFS_EINVAL
    xc = synth.tiny(has_cross=1)
    with pytest.raises(dfs.DfsError) as e:  # cross-attention without a context
        dfs.dfs_plan_create(xc, [{k: 16 for k in dfs.LAYER_FIELDS}], 16, 16, synth.make_masks(xc), None, 0)
    assert e.value.status == dfs.DFS_EINVAL


def test_plan_create_rejects_misaligned_device_pointers(dfs):
    """Device buffers are read with 16-byte vectors and TMA: an address that is not
    16-byte aligned is refused before any CUDA call."""
    cfg = synth.tiny()
    layers, masks = _valid_args(dfs, cfg)
    bad = [dict(layers[0])]
    bad[0]["w_down"] = 24
    with pytest.raises(dfs.DfsError) as e:
        dfs.dfs_plan_create(cfg, bad, 16, 16, masks, None, 0)
    assert e.value.status == dfs.DFS_EINVAL and "16-byte aligned" in dfs.dfs_last_error()
    with pytest.raises(dfs.DfsError) as e:
        dfs.dfs_plan_create(cfg, layers, 40, 16, masks, None, 0)
    assert e.value.status == dfs.DFS_EINVAL and "16-byte aligned" in dfs.dfs_last_error()


def test_forward_rejects_null_plan(dfs):
    with pytest.raises(dfs.DfsError) as e:
        dfs.dfs_block_forward(0, 0, 16, 16, 32, 0)
    assert e.value.status == dfs.DFS_EINVAL


@pytest.mark.parametrize("call", ["layer", "host", "host_async", "noalloc", "denoise", "model_forward",
                                  "model_denoise", "sync", "memory", "flops"])
def test_every_entry_point_rejects_a_null_plan_before_any_cuda_call(dfs, call):
    import numpy as np
    h = np.zeros(64, dtype=np.uint16)
    calls = {
        "layer": lambda: dfs.dfs_block_forward_layer(0, 0, 0, 16, 16, 32, 0),
        "host": lambda: dfs.dfs_block_forward_host(0, 0, 0, h, h[:16], h[32:], 0),
        "host_async": lambda: dfs.dfs_block_forward_host_async(0, 0, 0, h, h[:16], h[32:], 0),
        "noalloc": lambda: dfs.dfs_block_forward_noalloc(0, 0, 0, 16, 16, 32, 0),
        "denoise": lambda: dfs.dfs_denoise(0, 16, 4, 32, 0),
        "model_forward": lambda: dfs.dfs_model_forward(0, 0, 16, 1.0, 32, 0),
        "model_denoise": lambda: dfs.dfs_model_denoise(0, 16, 4, [1000.0, 750.0, 500.0, 250.0], 0),
        "sync": lambda: dfs.dfs_plan_sync(0, 0),
        "memory": lambda: dfs.dfs_plan_memory(0),
        "flops": lambda: dfs.dfs_plan_flops(0, 0, 0),
    }
    with pytest.raises(dfs.DfsError) as e:
        calls[call]()
    assert e.value.status == dfs.DFS_EINVAL


@pytest.mark.parametrize("kind,unit", [(0, 1), (1, 64), (1, 128), (2, 1)])
def test_soft_mask_gate_rules_match_oracle(dfs, kind, unit):
    rng = np.random.default_rng(kind * 100 + unit)
    m = rng.standard_normal((4, 12 * unit)).astype(np.float32) + 0.05
    m[0, :unit] = 0.0                 # mean exactly zero -> pruned
    if unit > 1:
        m[1, :unit] = -1.0
        m[1, 0] = float(unit)         # mean +1/unit... positive
    g = dfs.dfs_gates_from_soft_masks(kind, m, unit)
    ref = O.gates_from_soft_masks({0: "block", 1: "head", 2: "ffn"}[kind], m, unit)
    np.testing.assert_array_equal(g, ref)
    assert g[0, 0] == 0


def test_header_and_c_example_are_plain_c(tmp_path):
    """include/dfs.h is a C header (no C++ or torch types): it and the plain-C example compile
    as strict C99 with warnings as errors, and the header also as C++17."""
    import shutil
    import subprocess
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no gcc")
    inc = os.path.join(ROOT, "include")
    src = tmp_path / "h.c"
    src.write_text('#include "dfs.h"\nint main(void) { dfs_plan* p = 0; (void)p; return 0; }\n')
    for cmd in ([gcc, "-std=c99", "-Wall", "-Wextra", "-Werror", "-pedantic", "-fsyntax-only", "-I", inc, str(src)],
                ["g++", "-std=c++17", "-Wall", "-Werror", "-fsyntax-only", "-I", inc, "-x", "c++", str(src)]):
        r = subprocess.run(cmd, capture_output=True, text=True)
        assert r.returncode == 0, r.stderr
    cuda_inc = next((d for d in ("/usr/local/cuda/include",) if os.path.exists(os.path.join(d, "cuda_runtime_api.h"))),
                    None)
    if cuda_inc:
        ex = os.path.join(ROOT, "paper_2607_06631_gb300", "examples", "block_forward.c")
        r = subprocess.run([gcc, "-std=c99", "-Wall", "-Wextra", "-Werror", "-fsyntax-only", "-I", inc, "-I", cuda_inc, ex],
                           capture_output=True, text=True)
        assert r.returncode == 0, r.stderr
