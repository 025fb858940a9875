"""Pins for the oracle's three-layer cosine bottleneck (Section 4.4, Table 5):
    a = cos(omega1 h + phi1), b = a M, a2 = cos(omega2 b + phi2), b2 = a2 M2,
    c = cos(omega3 b2 + phi3).
No GPU needed.  Independent of the oracle's own formulas:
  * the linear limit (phases -pi/2, small omega1) reduces the branch to
    x W_down M M2 W_up, which fixes the orientation of M2 and that the third
    layer reads b2;
  * M2 = 0 makes c = cos(phi3) for every token exactly and zeroes every
    gradient upstream of M2;
  * 2 pi periodicity in phi3;
  * central finite differences for all 13 gradients;
  * planted mistakes in the three-layer code each fail one of these.
"""
import math
import os

import numpy as np
import pytest

import oracle
from tests.test_oracle_pins import rand_params, rel


def params3(rng, T, d_in, d_out, r, branch_std=0.5):
    p = rand_params(rng, T, d_in, d_out, r, branch_std)
    p["M2"] = rng.standard_normal((r, r)) / math.sqrt(r)
    p["omega3"] = rng.uniform(0.5, 2.0, r)
    p["phi3"] = rng.uniform(-math.pi, math.pi, r)
    return p


def fwd(p):
    return oracle.fwd3(p["x"], p["W"], p["bias"], p)


def bwd(p):
    return oracle.bwd3(p["x"], p["W"], p, p["dy"])


def test_linear_limit_fixes_orientation():
    rng = np.random.default_rng(21)
    p = params3(rng, 12, 9, 7, 5)
    for k in ("phi1", "phi2", "phi3"):
        p[k] = np.full(5, -math.pi / 2)
    p["omega2"] = np.ones(5)
    p["omega3"] = np.ones(5)
    lin = p["x"] @ p["W_down"] @ p["M"] @ p["M2"] @ p["W_up"]
    base = p["x"] @ p["W"] + p["bias"]
    errs = []
    for eps in (1e-2, 1e-3):
        q = dict(p, omega1=np.full(5, eps))
        errs.append(rel((fwd(q) - base) / eps, lin))
    assert errs[1] < errs[0] / 50 and errs[1] < 1e-5, errs
    # the transposed reading of M2 is far off
    q = dict(p, omega1=np.full(5, 1e-3))
    assert rel((fwd(q) - base) / 1e-3, p["x"] @ p["W_down"] @ p["M"] @ p["M2"].T @ p["W_up"]) > 1e-2


def test_zero_second_matrix():
    rng = np.random.default_rng(22)
    p = params3(rng, 10, 8, 6, 4)
    p["M2"] = np.zeros((4, 4))
    y = fwd(p)
    want = p["x"] @ p["W"] + p["bias"] + np.cos(p["phi3"]) @ p["W_up"]
    assert rel(y, want) < 1e-13
    g = bwd(p)
    for k in ("dW_down", "dM", "domega1", "dphi1", "domega2", "dphi2", "domega3"):
        assert np.all(g[k] == 0.0), k
    dc = p["dy"] @ p["W_up"].T
    du3 = -np.sin(p["phi3"]) * dc
    assert rel(g["dphi3"], du3.sum(0)) < 1e-13
    assert np.max(np.abs(g["dM2"])) > 1e-3


def test_phase_periodicity():
    rng = np.random.default_rng(23)
    p = params3(rng, 10, 8, 6, 4)
    y0, g0 = fwd(p), bwd(p)
    q = dict(p, phi3=p["phi3"] + 2 * math.pi * 3)
    assert rel(fwd(q), y0) < 1e-12
    g1 = bwd(q)
    for k in oracle.GRAD_NAMES3:
        assert np.max(np.abs(g1[k] - g0[k])) <= 1e-10 * max(1.0, np.max(np.abs(g0[k]))), k


PARAM_OF_GRAD3 = {"dx": "x", "dW": "W", "dbias": "bias", "dW_down": "W_down", "dM": "M",
                  "domega1": "omega1", "dphi1": "phi1", "domega2": "omega2", "dphi2": "phi2",
                  "dM2": "M2", "domega3": "omega3", "dphi3": "phi3", "dW_up": "W_up"}


def test_finite_difference_gradients():
    rng = np.random.default_rng(24)
    p = params3(rng, 3, 5, 4, 3, branch_std=1.0)
    g = bwd(p)

    def loss(q):
        return float(np.sum(fwd(q) * q["dy"]))

    step = 1e-6
    for gname, pname in PARAM_OF_GRAD3.items():
        base = p[pname]
        fd = np.zeros_like(base)
        for idx in np.ndindex(base.shape):
            plus, minus = base.copy(), base.copy()
            plus[idx] += step
            minus[idx] -= step
            fd[idx] = (loss(dict(p, **{pname: plus})) - loss(dict(p, **{pname: minus}))) / (2 * step)
        scale = max(np.max(np.abs(fd)), 1e-3)
        assert np.max(np.abs(g[gname] - fd)) / scale < 1e-7, gname


def test_cos3_pins_catch_planted_mistakes(tmp_path):
    import ctypes
    import subprocess
    src = open(os.path.join(os.path.dirname(oracle.__file__), "noble_oracle.c")).read()
    mistakes = {
        "M2 transposed": ("s += a2[i] * M2[i * r + j];", "s += a2[i] * M2[j * r + i];"),
        "third layer reads b": ("c[j] = cos(om3[j] * b2[j] + ph3[j]);", "c[j] = cos(om3[j] * b[j] + ph3[j]);"),
        "da2 uses M2": ("s += db2[j] * M2[i * r + j];", "s += db2[j] * M2[j * r + i];"),
        "du3 sign": ("du3[j] = -sin(om3[j] * b2[j] + ph3[j]) * dc[j];",
                     "du3[j] = sin(om3[j] * b2[j] + ph3[j]) * dc[j];"),
        "domega3 with b": ("s[4] += DU3[t * r + k] * B2[t * r + k];", "s[4] += DU3[t * r + k] * B[t * r + k];"),
        "dM2 with a": ("dM2[i * r + j] += A2[t * r + i] * DB2[t * r + j];",
                       "dM2[i * r + j] += A[t * r + i] * DB2[t * r + j];"),
    }
    checks = [test_linear_limit_fixes_orientation, test_zero_second_matrix, test_finite_difference_gradients]
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
            for fn in ("oracle_fwd3", "oracle_bwd3"):
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
