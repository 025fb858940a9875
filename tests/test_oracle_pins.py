"""Pins for the fp64 oracle, independent of the oracle itself (no GPU needed).

Each check is a property that the paper or the mathematics fixes:
  * W_up = 0 reduces the layer to x W + bias exactly (Section 3.3: the branch
    contributes nothing at zero W_up) and zeroes every branch gradient;
  * the identity sigma collapses to x (W + W_down W_up) (Sections 1 and 3.1);
  * the linear limit of CosNet reduces to ((omega1 h) M omega2) W_up, fixing the
    orientation of M and where each frequency and phase enters (Eq. 2);
  * a hand-derived two-token case on textbook cosine values (Eq. 1, Eq. 2);
  * 2 pi periodicity of the phases and token-permutation equivariance;
  * central finite differences for every gradient (all three sigma modes).
A planted mistake in the oracle (sign, transposed M, dropped term) fails one
of these; ``test_pins_catch_planted_mistakes`` checks that on copies.
"""
import json
import math
import os

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def rand_params(rng, T, d_in, d_out, r, branch_std=0.5):
    """Paper-orientation fp64 tensors with O(1) branch so every term matters."""
    return dict(
        x=rng.standard_normal((T, d_in)),
        W=rng.standard_normal((d_in, d_out)) / math.sqrt(d_in),
        bias=rng.standard_normal(d_out) * 0.1,
        W_down=rng.standard_normal((d_in, r)) / math.sqrt(d_in),
        omega1=rng.uniform(0.5, 2.0, r),
        phi1=rng.uniform(-math.pi, math.pi, r),
        M=rng.standard_normal((r, r)) / math.sqrt(r),
        omega2=rng.uniform(0.5, 2.0, r),
        phi2=rng.uniform(-math.pi, math.pi, r),
        W_up=rng.standard_normal((r, d_out)) * branch_std,
        dy=rng.standard_normal((T, d_out)),
    )


def fwd(p, mode=oracle.COSNET, **kw):
    return oracle.fwd(p["x"], p["W"], p.get("bias"), p["W_down"], p["omega1"], p["phi1"],
                      p["M"], p["omega2"], p["phi2"], p["W_up"], mode=mode, **kw)


def bwd(p, mode=oracle.COSNET, **kw):
    return oracle.bwd(p["x"], p["W"], p["W_down"], p["omega1"], p["phi1"], p["M"],
                      p["omega2"], p["phi2"], p["W_up"], p["dy"], mode=mode, **kw)


def rel(a, b):
    a, b = np.asarray(a), np.asarray(b)
    return float(np.max(np.abs(a - b)) / max(np.max(np.abs(b)), 1e-300))


# --------------------------------------------------------------------- S1
def test_zero_up_reduces_to_plain_layer():
    rng = np.random.default_rng(1)
    p = rand_params(rng, 37, 24, 19, 8)
    p["W_up"] = np.zeros_like(p["W_up"])
    y = fwd(p)
    plain = oracle.fwd(p["x"], p["W"], p["bias"], None, None, None, None, None, None, None)
    assert np.array_equal(y, plain)  # same loop order, +0.0 branch: bit-exact
    assert rel(y, p["x"] @ p["W"] + p["bias"]) < 1e-13
    g = bwd(p, want_intermediates=True)
    for k in ("dW_down", "dM", "domega1", "dphi1", "domega2", "dphi2"):
        assert np.all(g[k] == 0.0), k
    assert np.all(g["dh"] == 0.0)
    assert rel(g["dx"], p["dy"] @ p["W"].T) < 1e-13
    assert rel(g["dW"], p["x"].T @ p["dy"]) < 1e-13
    assert rel(g["dbias"], p["dy"].sum(0)) < 1e-13
    assert np.max(np.abs(g["dW_up"])) > 0.1  # c^T dy does not vanish
    assert rel(g["dW_up"], g["c"].T @ p["dy"]) < 1e-13


# --------------------------------------------------------------------- S2
def test_identity_sigma_collapses_to_merged_weight():
    rng = np.random.default_rng(2)
    p = rand_params(rng, 29, 16, 12, 5)
    Wm = p["W"] + p["W_down"] @ p["W_up"]
    assert rel(fwd(p, oracle.IDENTITY), p["x"] @ Wm + p["bias"]) < 1e-12
    g = bwd(p, oracle.IDENTITY)
    assert rel(g["dx"], p["dy"] @ Wm.T) < 1e-12
    assert rel(g["dW_down"], p["x"].T @ (p["dy"] @ p["W_up"].T)) < 1e-12
    assert rel(g["dW_up"], (p["x"] @ p["W_down"]).T @ p["dy"]) < 1e-12
    assert rel(g["dW"], p["x"].T @ p["dy"]) < 1e-12
    for k in ("dM", "domega1", "dphi1", "domega2", "dphi2"):
        assert np.all(g[k] == 0.0), k


# --------------------------------------------------------------------- S4
def _linear_limit_error(p, eps, transpose_M=False):
    q = dict(p)
    r = p["M"].shape[0]
    q["phi1"] = np.full(r, -math.pi / 2)
    q["phi2"] = np.full(r, -math.pi / 2)
    q["omega1"] = eps * p["w1"]
    q["omega2"] = eps * p["w2"]
    y = fwd(q)
    q0 = dict(q, W_up=np.zeros_like(q["W_up"]))
    branch = (y - fwd(q0)) / eps**2
    M = p["M"].T if transpose_M else p["M"]
    pred = (((p["x"] @ p["W_down"]) * p["w1"]) @ M * p["w2"]) @ p["W_up"]
    return rel(branch, pred)


def test_linear_limit_fixes_composition_and_orientation():
    """phi = -pi/2 turns cos into sin; with omega = eps*w, sin(z) = z + O(z^3)
    so the branch divided by eps^2 tends to ((w1 * h) M * w2) W_up."""
    rng = np.random.default_rng(4)
    p = rand_params(rng, 33, 20, 14, 6)
    p["w1"] = rng.uniform(0.5, 2.0, 6)
    p["w2"] = rng.uniform(0.5, 2.0, 6)
    e2, e3 = _linear_limit_error(p, 1e-2), _linear_limit_error(p, 1e-3)
    assert e3 < 1e-4
    assert 30 < e2 / e3 < 300  # second-order convergence
    # The transposed mixing matrix is not a valid reading of this oracle.
    assert _linear_limit_error(p, 1e-3, transpose_M=True) > 1e-2


# ------------------------------------------------------- closed form golden
def _golden():
    with open(os.path.join(GOLDEN, "cosnet_closed_form.json")) as f:
        g = json.load(f)
    env = {"__builtins__": {}, "pi": math.pi, "sqrt": math.sqrt}
    ev = lambda v: (np.array([ev(e) for e in v]) if isinstance(v, list)
                    else float(eval(v, env)))
    return {k: ev(v) for k, v in g["inputs"].items()}, {k: ev(v) for k, v in g["expected"].items()}


def test_closed_form_two_tokens():
    p, e = _golden()
    y, h, b, c = fwd(p, want_intermediates=True)
    for name, got in (("h", h), ("b", b), ("c", c), ("y", y)):
        assert np.max(np.abs(got - e[name])) < 1e-12, name
    g = bwd(p)
    for k in oracle.GRAD_NAMES:
        assert np.max(np.abs(g[k] - e[k])) < 1e-12, k


# --------------------------------------------------------------------- S5
def test_phase_periodicity():
    rng = np.random.default_rng(5)
    p = rand_params(rng, 21, 10, 9, 4)
    y0, g0 = fwd(p), bwd(p)
    for k in (1, 2, 4):
        q = dict(p, phi1=p["phi1"] + 2 * math.pi * k, phi2=p["phi2"] - 2 * math.pi * k)
        assert rel(fwd(q), y0) < 1e-12 * k
        g = bwd(q)
        for name in oracle.GRAD_NAMES:
            assert rel(g[name], g0[name]) < 1e-11 * k, name


# --------------------------------------------------------------------- S6
def test_token_permutation():
    rng = np.random.default_rng(6)
    p = rand_params(rng, 40, 12, 10, 4)
    perm = rng.permutation(40)
    q = dict(p, x=p["x"][perm], dy=p["dy"][perm])
    assert np.array_equal(fwd(q), fwd(p)[perm])  # rows are independent
    g, gq = bwd(p), bwd(q)
    assert np.array_equal(gq["dx"], g["dx"][perm])
    for name in oracle.GRAD_NAMES[1:]:
        assert rel(gq[name], g[name]) < 1e-12, name


# --------------------------------------------------------------------- S3
def _loss(p, mode):
    return float(np.sum(fwd(p, mode) * p["dy"]))


PARAM_OF_GRAD = {"dx": "x", "dW": "W", "dbias": "bias", "dW_down": "W_down", "dM": "M",
                 "domega1": "omega1", "dphi1": "phi1", "domega2": "omega2",
                 "dphi2": "phi2", "dW_up": "W_up"}


@pytest.mark.parametrize("mode", [oracle.COSNET, oracle.IDENTITY, oracle.COS1])
def test_finite_difference_gradients(mode):
    rng = np.random.default_rng(3)
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


def test_outer_elems_is_the_gradient_element():
    rng = np.random.default_rng(7)
    P, Q = rng.standard_normal((50, 7)), rng.standard_normal((50, 9))
    rows, cols = rng.integers(0, 7, 20), rng.integers(0, 9, 20)
    assert rel(oracle.outer_elems(P, Q, rows, cols), (P.T @ Q)[rows, cols]) < 1e-13


# ------------------------------------------------------ discriminative power
def test_pins_catch_planted_mistakes(tmp_path):
    """Plant mistakes in a copy of the oracle source; each must fail a pin."""
    import ctypes
    import subprocess
    src = open(os.path.join(os.path.dirname(oracle.__file__), "noble_oracle.c")).read()
    mistakes = {
        "transposed M": ("s += a[i] * M[i * r + j];\n        b[j] = s;\n    }\n    for (j = 0; j < r; ++j) c[j]",
                         "s += a[i] * M[j * r + i];\n        b[j] = s;\n    }\n    for (j = 0; j < r; ++j) c[j]"),
        "phase sign": ("cos(om2[j] * b[j] + ph2[j])", "cos(om2[j] * b[j] - ph2[j])"),
        "dropped sin sign": ("du1[i] = -sin(u1[i]) * da[i];", "du1[i] = sin(u1[i]) * da[i];"),
        "da uses M not M^T": ("s += db[j] * M[i * r + j];\n                    da[i] = s;\n                }\n"
                              "                for (i = 0; i < r; ++i) {\n                    du1[i] = -sin",
                              "s += db[j] * M[j * r + i];\n                    da[i] = s;\n                }\n"
                              "                for (i = 0; i < r; ++i) {\n                    du1[i] = -sin"),
        "dropped dh term": ("dx[t * d_in + i] = s + sb;\n            }\n        }\n",
                            "dx[t * d_in + i] = s;\n            }\n        }\n"),
    }
    p, e = _golden()
    for name, (old, new) in mistakes.items():
        assert src.count(old) == 1, name
        path = tmp_path / f"m{abs(hash(name))}.c"
        path.write_text(src.replace(old, new))
        so = str(path) + ".so"
        subprocess.run(["gcc", "-O1", "-shared", "-fPIC", "-o", so, str(path), "-lm"], check=True)
        lib = ctypes.CDLL(so)
        saved = oracle._lib
        try:
            oracle._lib = None
            oracle._load()  # set argtypes on the real library first
            real = oracle._lib
            for fn in ("oracle_fwd", "oracle_bwd"):
                getattr(lib, fn).argtypes = getattr(real, fn).argtypes
            oracle._lib = lib
            y = fwd(p)
            g = bwd(p)
            bad = np.max(np.abs(y - e["y"])) > 1e-6 or any(
                np.max(np.abs(g[k] - e[k])) > 1e-6 for k in oracle.GRAD_NAMES)
            assert bad, f"planted mistake not caught: {name}"
        finally:
            oracle._lib = saved
