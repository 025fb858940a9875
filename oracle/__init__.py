"""fp64 CPU oracle for the NOBLE linear layer with the CosNet branch.

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the CPU
baseline leg of ``bench.py`` may use this package; the library under
``paper_2603_06492_gb300`` never imports it and never falls back to it.

The arithmetic lives in ``noble_oracle.c`` (plain C, fp64, ascending-order
sums); this module only compiles it with gcc and marshals numpy arrays.

Orientation is the paper's (Eq. 1, Section 3.1, row vectors):
``W[d_in][d_out]``, ``W_down[d_in][r]``, ``W_up[r][d_out]``, ``M[r][r]`` with
``b = a M``.  Callers holding nn.Linear-style ``[out][in]`` weights transpose
them before calling.

Parity status: pinned by ``tests/test_oracle_pins.py`` (no GPU needed).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

COSNET, IDENTITY, COS1 = 0, 1, 2
# the other activations of the ablation (Section 4.4, Table 5): one layer
# sigma(h) = f(h), or two layers sigma(h) = f(f(h) M), without frequency/phase
TANH1, TANH2, LEAKY1, LEAKY2, GELU1, GELU2 = 3, 4, 5, 6, 7, 8
MODES = {"cosnet": COSNET, "identity": IDENTITY, "cos1": COS1, "tanh1": TANH1, "tanh2": TANH2,
         "leaky1": LEAKY1, "leaky2": LEAKY2, "gelu1": GELU1, "gelu2": GELU2}

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "noble_oracle.c")
_LIB = os.path.join(_HERE, "libnoble_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (fp64, no FMA contraction, OpenMP)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fopenmp", "-shared",
               "-fPIC", "-std=c99", "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB)
            p = ctypes.c_void_p
            i64 = ctypes.c_int64
            lib.oracle_fwd.argtypes = [ctypes.c_int, i64, i64, i64, i64] + [p] * 14
            lib.oracle_fwd.restype = None
            lib.oracle_bwd.argtypes = [ctypes.c_int, i64, i64, i64, i64] + [p] * 24
            lib.oracle_bwd.restype = None
            lib.oracle_fwd3.argtypes = [i64, i64, i64, i64] + [p] * 18
            lib.oracle_fwd3.restype = None
            lib.oracle_bwd3.argtypes = [i64, i64, i64, i64] + [p] * 26
            lib.oracle_bwd3.restype = None
            lib.oracle_outer_elems.argtypes = [i64, p, i64, p, i64, i64, p, p, p]
            lib.oracle_outer_elems.restype = None
            _lib = lib
    return _lib


def _c(a):
    """fp64 C-contiguous copy (or view) of ``a``; None stays None."""
    if a is None:
        return None
    return np.ascontiguousarray(a, dtype=np.float64)


def _ptr(a):
    return None if a is None else a.ctypes.data


def fwd(x, W, bias, W_down, omega1, phi1, M, omega2, phi2, W_up, mode=COSNET,
        want_intermediates=False):
    """Forward pass, Eq. 1 with sigma = CosNet (Eq. 2).

    Shapes (paper orientation): x [T,d_in], W [d_in,d_out], bias [d_out] or
    None, W_down [d_in,r], omega/phi [r], M [r,r], W_up [r,d_out].  Returns y
    [T,d_out], or (y, h, b, c) with ``want_intermediates``.
    """
    lib = _load()
    x, W, bias = _c(x), _c(W), _c(bias)
    T, d_in = x.shape
    d_out = W.shape[1]
    r = 0 if W_down is None else np.asarray(W_down).shape[1]
    W_down, W_up = _c(W_down), _c(W_up)
    om1, ph1, M, om2, ph2 = _c(omega1), _c(phi1), _c(M), _c(omega2), _c(phi2)
    y = np.empty((T, d_out))
    h = np.empty((T, r)) if want_intermediates else None
    b = np.empty((T, r)) if want_intermediates else None
    c = np.empty((T, r)) if want_intermediates else None
    lib.oracle_fwd(mode, T, d_in, d_out, r, _ptr(x), _ptr(W), _ptr(bias), _ptr(W_down),
                   _ptr(om1), _ptr(ph1), _ptr(M), _ptr(om2), _ptr(ph2), _ptr(W_up),
                   _ptr(y), _ptr(h), _ptr(b), _ptr(c))
    return (y, h, b, c) if want_intermediates else y


GRAD_NAMES = ("dx", "dW", "dbias", "dW_down", "dM", "domega1", "dphi1", "domega2",
              "dphi2", "dW_up")


def bwd(x, W, W_down, omega1, phi1, M, omega2, phi2, W_up, dy, mode=COSNET,
        skip=(), want_intermediates=False):
    """Backward pass of ``L = sum(y * dy)``; returns a dict of gradients.

    Gradient names: dx, dW, dbias, dW_down, dM, domega1, dphi1, domega2, dphi2,
    dW_up, each in the orientation of its parameter above.  Names listed in
    ``skip`` are not computed (for large shapes).  With
    ``want_intermediates`` the dict also holds the per-token c, a, db and dh.
    """
    lib = _load()
    x, W, dy = _c(x), _c(W), _c(dy)
    T, d_in = x.shape
    d_out = W.shape[1]
    r = 0 if W_down is None else np.asarray(W_down).shape[1]
    W_down, W_up = _c(W_down), _c(W_up)
    om1, ph1, M, om2, ph2 = _c(omega1), _c(phi1), _c(M), _c(omega2), _c(phi2)
    shapes = {"dx": (T, d_in), "dW": (d_in, d_out), "dbias": (d_out,),
              "dW_down": (d_in, r), "dM": (r, r), "domega1": (r,), "dphi1": (r,),
              "domega2": (r,), "dphi2": (r,), "dW_up": (r, d_out)}
    out = {k: (None if k in skip else np.empty(s)) for k, s in shapes.items()}
    inter = {k: (np.empty((T, r)) if want_intermediates else None)
             for k in ("c", "a", "db", "dh")}
    lib.oracle_bwd(mode, T, d_in, d_out, r, _ptr(x), _ptr(W), _ptr(W_down), _ptr(om1),
                   _ptr(ph1), _ptr(M), _ptr(om2), _ptr(ph2), _ptr(W_up), _ptr(dy),
                   *[_ptr(out[k]) for k in GRAD_NAMES],
                   _ptr(inter["c"]), _ptr(inter["a"]), _ptr(inter["db"]), _ptr(inter["dh"]))
    res = {k: v for k, v in out.items() if v is not None}
    if want_intermediates:
        res.update(inter)
    return res


# the three-layer cosine (Section 4.4, Table 5), with M2 [r,r], omega3, phi3 [r]
PARAMS3 = ("W_down", "omega1", "phi1", "M", "omega2", "phi2", "M2", "omega3", "phi3", "W_up")
GRAD_NAMES3 = ("dx", "dW", "dbias", "dW_down", "dM", "domega1", "dphi1", "domega2", "dphi2",
               "dM2", "domega3", "dphi3", "dW_up")


def fwd3(x, W, bias, p, want_intermediates=False):
    """Forward with the three-layer cosine; ``p`` maps the names of PARAMS3
    (paper orientation) to arrays.  Returns y, or (y, h, b, b2, c)."""
    lib = _load()
    x, W, bias = _c(x), _c(W), _c(bias)
    T, d_in = x.shape
    d_out = W.shape[1]
    r = np.asarray(p["W_down"]).shape[1]
    q = [_c(p[k]) for k in PARAMS3]
    y = np.empty((T, d_out))
    inter = [np.empty((T, r)) if want_intermediates else None for _ in range(4)]
    lib.oracle_fwd3(T, d_in, d_out, r, _ptr(x), _ptr(W), _ptr(bias), *[_ptr(a) for a in q], _ptr(y),
                    *[_ptr(a) for a in inter])
    return (y, *inter) if want_intermediates else y


def bwd3(x, W, p, dy):
    """Backward of ``L = sum(y * dy)`` with the three-layer cosine; returns a
    dict over GRAD_NAMES3, each in the orientation of its parameter."""
    lib = _load()
    x, W, dy = _c(x), _c(W), _c(dy)
    T, d_in = x.shape
    d_out = W.shape[1]
    r = np.asarray(p["W_down"]).shape[1]
    q = [_c(p[k]) for k in PARAMS3]
    shapes = {"dx": (T, d_in), "dW": (d_in, d_out), "dbias": (d_out,), "dW_down": (d_in, r),
              "dM": (r, r), "domega1": (r,), "dphi1": (r,), "domega2": (r,), "dphi2": (r,),
              "dM2": (r, r), "domega3": (r,), "dphi3": (r,), "dW_up": (r, d_out)}
    out = {k: np.empty(shapes[k]) for k in GRAD_NAMES3}
    lib.oracle_bwd3(T, d_in, d_out, r, _ptr(x), _ptr(W), *[_ptr(a) for a in q], _ptr(dy),
                    *[_ptr(out[k]) for k in GRAD_NAMES3])
    return out


def outer_elems(P, Q, rows, cols):
    """``out[p] = sum_t P[t, rows[p]] * Q[t, cols[p]]`` in ascending t."""
    lib = _load()
    P, Q = _c(P), _c(Q)
    rows = np.ascontiguousarray(rows, dtype=np.int64)
    cols = np.ascontiguousarray(cols, dtype=np.int64)
    assert P.shape[0] == Q.shape[0] and rows.shape == cols.shape
    out = np.empty(rows.shape[0])
    lib.oracle_outer_elems(P.shape[0], _ptr(P), P.shape[1], _ptr(Q), Q.shape[1],
                           rows.shape[0], _ptr(rows), _ptr(cols), _ptr(out))
    return out
