"""Planted mistakes: each plausible error in the oracle (a dropped term, a wrong sign, a
swapped or transposed operand, a wrong constant, a band in the wrong order) must make at
least one of the pins in test_oracle_pins.py fail.  The mistakes are planted in the oracle
on the CPU, one at a time, by replacing one of its functions for the duration of a test."""
import functools
import inspect
import math

import numpy as np
import pytest

import oracle
from oracle import dfs_oracle as D
import test_oracle_pins as pins


def _ln_unbiased(orig):
    def f(x, eps, weight=None, bias=None):
        mu = x.mean(axis=-1, keepdims=True)
        var = ((x - mu) ** 2).sum(axis=-1, keepdims=True) / (x.shape[-1] - 1)
        y = (x - mu) / np.sqrt(var + eps)
        if weight is not None:
            y = y * weight
        return y + bias if bias is not None else y
    return f


def _adaln_no_one(orig):
    return lambda x, shift, scale, eps: D.layer_norm(x, eps) * scale + shift


def _rms_no_gamma(orig):
    return lambda x, gamma, keep, eps, mode, head_dim: orig(x, np.ones_like(gamma), keep, eps, mode, head_dim)


def _rope_sign(orig):
    return lambda x, ang: orig(x, -ang)


def _rope_band_order(orig):
    def f(grid, head_dim, theta):
        ang = orig(grid, head_dim, theta)
        p_t, p_h, p_w = D.rope_pairs(head_dim)
        return np.concatenate([ang[:, p_t + p_h:], ang[:, p_t:p_t + p_h], ang[:, :p_t]], axis=1)
    return f


def _attn_no_scale(orig):
    return lambda q, k, v, counter=None: orig(q * math.sqrt(q.shape[-1]), k, v, counter)


def _attn_wrong_axis(orig):
    def f(q, k, v, counter=None):
        n, h, dh = q.shape
        out = np.empty((n, h, v.shape[-1]))
        for j in range(h):
            s = q[:, j, :] @ k[:, j, :].T / math.sqrt(dh)
            p = np.exp(s - s.max(axis=0, keepdims=True))
            p = p / p.sum(axis=0, keepdims=True)
            out[:, j, :] = p @ v[:, j, :]
        return out
    return f


def _gelu_erf(orig):
    erf = np.vectorize(math.erf)
    return lambda x: 0.5 * x * (1.0 + erf(np.asarray(x) / math.sqrt(2.0)))


def _linear_transposed(orig):
    return lambda x, w, b=None, counter=None: orig(x, np.ascontiguousarray(w.T), b, counter)


def _modulation_swapped(orig):
    def f(w_t, b_t, e_l, t_emb):
        m = orig(w_t, b_t, e_l, t_emb)
        return m[[1, 0, 2, 4, 3, 5]]
    return f


def _time_cos_sin_swapped(orig):
    def f(t, dim):
        e = orig(t, dim)
        return np.concatenate([e[dim // 2:], e[:dim // 2]])
    return f


def _gelu_coefficient(orig):
    return lambda x: 0.5 * x * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (x + 0.0447 * x ** 2)))


def _cross_ln_weight_bias_swapped(orig):
    return lambda x1, cln_w, cln_b, eps: orig(x1, cln_b, cln_w, eps)


def _head_shift_scale_swapped(orig):
    return lambda x, head_mod, t_emb, head_w, head_b, eps: orig(x, head_mod[::-1], t_emb, head_w, head_b, eps)


MUTATIONS = {
    "LayerNorm with the unbiased variance": ("layer_norm", _ln_unbiased),
    "adaLN scale without the 1 +": ("adaln", _adaln_no_one),
    "QK RMSNorm without gamma": ("rms_norm", _rms_no_gamma),
    "RoPE rotating the wrong way": ("apply_rope", _rope_sign),
    "RoPE bands in w, h, t order": ("rope_angles", _rope_band_order),
    "attention without 1/sqrt(dh)": ("attention", _attn_no_scale),
    "softmax over the keys' axis": ("attention", _attn_wrong_axis),
    "GELU erf form instead of tanh": ("gelu_tanh", _gelu_erf),
    "GELU cubic term squared": ("gelu_tanh", _gelu_coefficient),
    "linear with W not transposed": ("linear", _linear_transposed),
    "shift and scale swapped": ("modulation", _modulation_swapped),
    "timestep sinusoid halves swapped": ("timestep_embedding", _time_cos_sin_swapped),
    "cross-attention LayerNorm weight and bias swapped": ("cross_input_norm", _cross_ln_weight_bias_swapped),
    "output head shift and scale swapped": ("output_head", _head_shift_scale_swapped),
}


def _pin_calls():
    """Every pin of test_oracle_pins.py as a no-argument call (parametrized ones expanded)."""
    calls = []
    for name, fn in inspect.getmembers(pins, inspect.isfunction):
        if not name.startswith("test_"):
            continue
        marks = [m for m in getattr(fn, "pytestmark", []) if m.name == "parametrize"]
        if not marks:
            calls.append((name, fn))
            continue
        argnames, values = marks[0].args
        argnames = [a.strip() for a in argnames.split(",")] if isinstance(argnames, str) else list(argnames)
        for v in values:
            v = v if isinstance(v, (tuple, list)) and len(argnames) > 1 else (v,)
            calls.append(("%s%s" % (name, v), functools.partial(fn, **dict(zip(argnames, v)))))
    return calls


def test_every_pin_passes_on_the_oracle_as_written():
    for name, call in _pin_calls():
        call()


@pytest.mark.parametrize("mistake", list(MUTATIONS))
def test_planted_mistake_fails_a_pin(mistake, monkeypatch):
    attr, make = MUTATIONS[mistake]
    bad = make(getattr(D, attr))
    monkeypatch.setattr(D, attr, bad)
    monkeypatch.setattr(oracle, attr, bad)
    for name, call in _pin_calls():
        try:
            call()
        except (AssertionError, ValueError):
            return          # caught by pin `name`: a failed check, or operands whose shapes no longer fit
    pytest.fail("no pin caught: %s" % mistake)
