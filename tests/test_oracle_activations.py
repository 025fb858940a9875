"""Pins for the oracle's other bottleneck activations (Section 4.4, Table 5):
tanh, LeakyReLU and GELU, one layer (sigma(h) = f(h)) or two layers around the
mixing matrix (sigma(h) = f(f(h) M)).  No GPU needed.

Each check is fixed by the mathematics, not by the oracle's own formulas:
  * textbook values: tanh(1) = 0.7615941559557649 and the standard normal
    distribution function Phi(1) = 0.8413447460685429 (so GELU(1) = Phi(1));
    the two-layer cases choose M so that the second layer sees exactly 1 again;
  * symmetries: tanh is odd; GELU(u) - GELU(-u) = u (erf is odd);
  * LeakyReLU is the identity for positive inputs and 0.01 x for negative ones,
    which reduces the branch to the linear collapse x W_down (M) W_up;
  * small-input limits: tanh(e u) / e -> u and GELU(e u) / e -> u / 2, which fix
    the orientation of M and the factor 1/2 in each GELU layer;
  * central finite differences for every gradient, in every mode.
A planted mistake in the activation code (a dropped factor, a wrong sign,
a wrong slope) fails one of these; see test_activation_pins_catch_planted_mistakes.
"""
import math
import os

import numpy as np
import pytest

import oracle
from tests.test_oracle_pins import PARAM_OF_GRAD, rand_params, rel

TANH_1 = 0.7615941559557649
PHI_1 = 0.8413447460685429
ACT_MODES = ["tanh1", "tanh2", "leaky1", "leaky2", "gelu1", "gelu2"]


def fwd(p, mode):
    return oracle.fwd(p["x"], p["W"], p.get("bias"), p["W_down"], p["omega1"], p["phi1"],
                      p["M"], p["omega2"], p["phi2"], p["W_up"], mode=oracle.MODES[mode])


def bwd(p, mode):
    return oracle.bwd(p["x"], p["W"], p["W_down"], p["omega1"], p["phi1"], p["M"],
                      p["omega2"], p["phi2"], p["W_up"], p["dy"], mode=oracle.MODES[mode])


def scalar_case(h, m):
    """T = d_in = d_out = r = 1, W = 0, bias = 0, W_up = 1: y = sigma(h)."""
    one = np.ones((1, 1))
    return dict(x=one, W=np.zeros((1, 1)), bias=np.zeros(1), W_down=np.full((1, 1), h),
                omega1=np.ones(1), phi1=np.zeros(1), M=np.full((1, 1), m), omega2=np.ones(1),
                phi2=np.zeros(1), W_up=one, dy=one)


@pytest.mark.parametrize("mode,h,m,want", [
    ("tanh1", 1.0, 0.0, TANH_1),
    ("tanh2", 1.0, 1.0 / TANH_1, TANH_1),
    ("gelu1", 1.0, 0.0, PHI_1),
    ("gelu2", 1.0, 1.0 / PHI_1, PHI_1),
    ("leaky1", -2.0, 0.0, -0.02),
    ("leaky1", 3.0, 0.0, 3.0),
    ("leaky2", -2.0, 50.0, -0.01),
    ("leaky2", -2.0, -50.0, 1.0),
])
def test_textbook_values(mode, h, m, want):
    assert abs(fwd(scalar_case(h, m), mode)[0, 0] - want) < 1e-15


def test_tanh_single_layer_is_odd():
    rng = np.random.default_rng(11)
    p = rand_params(rng, 20, 12, 9, 8)
    base = p["x"] @ p["W"] + p["bias"]
    neg = dict(p, W_down=-p["W_down"])
    assert np.max(np.abs(fwd(p, "tanh1") + fwd(neg, "tanh1") - 2 * base)) < 1e-13


def test_gelu_odd_part_is_the_identity():
    # GELU(u) - GELU(-u) = u: the branch difference is x W_down W_up exactly
    rng = np.random.default_rng(12)
    p = rand_params(rng, 20, 12, 9, 8)
    neg = dict(p, W_down=-p["W_down"])
    diff = fwd(p, "gelu1") - fwd(neg, "gelu1")
    assert rel(diff, p["x"] @ p["W_down"] @ p["W_up"]) < 1e-13


@pytest.mark.parametrize("sign,scale", [(1.0, 1.0), (-1.0, 0.01)])
def test_leaky_single_layer_on_one_side(sign, scale):
    rng = np.random.default_rng(13)
    p = rand_params(rng, 15, 10, 7, 6)
    p["x"] = np.abs(p["x"])
    p["W_down"] = sign * np.abs(p["W_down"])  # every h on one side of 0
    want = p["x"] @ p["W"] + p["bias"] + scale * (p["x"] @ p["W_down"] @ p["W_up"])
    assert rel(fwd(p, "leaky1"), want) < 1e-13


def test_leaky_two_layers_positive_is_linear():
    rng = np.random.default_rng(14)
    p = rand_params(rng, 15, 10, 7, 6)
    p["x"], p["W_down"], p["M"] = np.abs(p["x"]), np.abs(p["W_down"]), np.abs(p["M"])
    want = p["x"] @ p["W"] + p["bias"] + p["x"] @ p["W_down"] @ p["M"] @ p["W_up"]
    assert rel(fwd(p, "leaky2"), want) < 1e-13


@pytest.mark.parametrize("mode,factor", [("tanh1", 1.0), ("tanh2", 1.0), ("gelu1", 0.5),
                                         ("gelu2", 0.25)])
def test_small_input_limit(mode, factor):
    # branch / eps -> factor * x W_down [M] W_up with an O(eps) (GELU) or
    # O(eps^2) (tanh) remainder: the error must shrink as eps does
    rng = np.random.default_rng(15)
    p = rand_params(rng, 10, 8, 6, 5)
    lin = p["x"] @ p["W_down"] @ (p["M"] if mode.endswith("2") else np.eye(5)) @ p["W_up"]
    errs = []
    for eps in (1e-3, 1e-4):
        q = dict(p, W_down=eps * p["W_down"])
        branch = fwd(q, mode) - (p["x"] @ p["W"] + p["bias"])
        errs.append(rel(branch / eps, factor * lin))
    assert errs[1] < 0.2 * errs[0] + 1e-9 and errs[1] < 1e-3, errs


def _loss(p, mode):
    return float(np.sum(fwd(p, mode) * p["dy"]))


@pytest.mark.parametrize("mode", ACT_MODES)
def test_finite_difference_gradients(mode):
    rng = np.random.default_rng(16)
    p = rand_params(rng, 3, 5, 4, 3, branch_std=1.0)
    g = bwd(p, mode)
    step = 1e-6
    for gname, pname in PARAM_OF_GRAD.items():
        base = p[pname]
        fd = np.zeros_like(base)
        for idx in np.ndindex(base.shape):
            plus, minus = base.copy(), base.copy()
            plus[idx] += step
            minus[idx] -= step
            fd[idx] = (_loss(dict(p, **{pname: plus}), mode)
                       - _loss(dict(p, **{pname: minus}), mode)) / (2 * step)
        scale = max(np.max(np.abs(fd)), 1e-3)
        assert np.max(np.abs(g[gname] - fd)) / scale < 1e-7, (gname, mode)


def test_activation_pins_catch_planted_mistakes(tmp_path):
    """Plant mistakes in a copy of the activation code; each must fail a pin."""
    import ctypes
    import subprocess
    src = open(os.path.join(os.path.dirname(oracle.__file__), "noble_oracle.c")).read()
    mistakes = {
        "GELU without 1/2": ("return 0.5 * u * (1.0 + erf(u / sqrt(2.0)));",
                             "return u * (1.0 + erf(u / sqrt(2.0)));"),
        "GELU erf scaling": ("return 0.5 * u * (1.0 + erf(u / sqrt(2.0)));",
                             "return 0.5 * u * (1.0 + erf(u));"),
        "GELU derivative density": ("u * exp(-0.5 * u * u) / sqrt(2.0 * acos(-1.0))",
                                    "u * exp(-u * u) / sqrt(2.0 * acos(-1.0))"),
        "leaky slope": ("return u > 0.0 ? u : 0.01 * u;", "return u > 0.0 ? u : 0.1 * u;"),
        "leaky derivative": ("return u > 0.0 ? 1.0 : 0.01;", "return u > 0.0 ? 1.0 : 0.0;"),
        "tanh derivative sign": ("return 1.0 - t * t;", "return 1.0 + t * t;"),
        "two-layer da uses M": ("                    for (j = 0; j < r; ++j) s += db[j] * M[i * r + j];\n"
                                "                    da[i] = s;\n                }\n"
                                "                for (i = 0; i < r; ++i) {\n"
                                "                    du1[i] = act_df(act, h[i]) * da[i];",
                                "                    for (j = 0; j < r; ++j) s += db[j] * M[j * r + i];\n"
                                "                    da[i] = s;\n                }\n"
                                "                for (i = 0; i < r; ++i) {\n"
                                "                    du1[i] = act_df(act, h[i]) * da[i];"),
    }
    checks = [lambda: test_textbook_values(m, h, mm, w) for (m, h, mm, w) in [
        ("tanh1", 1.0, 0.0, TANH_1), ("gelu1", 1.0, 0.0, PHI_1), ("leaky1", -2.0, 0.0, -0.02)]]
    checks += [test_gelu_odd_part_is_the_identity,
               lambda: test_leaky_single_layer_on_one_side(-1.0, 0.01)]
    checks += [lambda m=m: test_finite_difference_gradients(m) for m in ACT_MODES]
    saved = oracle._lib
    oracle._lib = None
    oracle._load()
    real = oracle._lib
    try:
        for name, (old, new) in mistakes.items():
            assert src.count(old) == 1, name
            path = tmp_path / f"m{abs(hash(name))}.c"
            path.write_text(src.replace(old, new))
            so = str(path) + ".so"
            subprocess.run(["gcc", "-O1", "-shared", "-fPIC", "-std=c99", "-o", so, str(path), "-lm"],
                           check=True)
            lib = ctypes.CDLL(so)
            for fn in ("oracle_fwd", "oracle_bwd"):
                getattr(lib, fn).argtypes = getattr(real, fn).argtypes
            oracle._lib = lib
            caught = False
            for chk in checks:
                try:
                    chk()
                except AssertionError:
                    caught = True
                    break
            assert caught, f"planted mistake not caught: {name}"
            oracle._lib = real
    finally:
        oracle._lib = saved
