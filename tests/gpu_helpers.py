"""Helpers shared by the GPU parity tests: run the CUDA path through the C ABI
and the oracle on the same seeded inputs, and compare.

Tolerance metric (per output tensor): max|got - ref| / max|ref|; where
max|ref| is 0 the absolute error is compared instead.
"""
from __future__ import annotations

import numpy as np

import oracle
from paper_2603_06492_gb300 import binding
from paper_2603_06492_gb300.inputs import Layer, to_paper_orientation

TOL = {"fp32": 1e-5, "bf16": 1e-2}
ABS_TOL_ZERO = {"fp32": 1e-6, "bf16": 1e-3}
OUT_NAMES = ("y", "dx", "dW", "dbias", "dW_down", "dM", "domega1", "dphi1", "domega2", "dphi2",
             "dW_up")


def rel_err(got, ref) -> float:
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    if ref.size == 0:
        return 0.0
    scale = np.max(np.abs(ref))
    err = np.max(np.abs(got - ref))
    return float(err / scale) if scale > 0 else float(err)


def run_gpu(layer: Layer, inp: dict, with_dbias=True, repeat=1, flags=0):
    """fwd + bwd through the C ABI; returns numpy fp64 outputs (library layout)."""
    import torch
    dev = binding.params_to_device(inp, layer.dtype)
    buf = binding.NobleLinearBuffers(layer.T, layer.d_in, layer.d_out, layer.r, layer.dtype, flags=flags)
    for _ in range(repeat):
        binding.forward(buf, dev["x"], dev)
        binding.backward(buf, dev["x"], dev["dy"], dev, with_dbias=with_dbias)
    torch.cuda.synchronize()
    binding.noble_get_device_status(None)
    out = {"y": buf.y, "dx": buf.dx}
    out.update(buf.grads)
    if not with_dbias:
        out.pop("dbias")
    return {k: v.float().cpu().numpy().astype(np.float64) for k, v in out.items()}


def run_oracle(layer: Layer, inp: dict) -> dict:
    """Full fp64 oracle in the library layout."""
    p = to_paper_orientation(inp)
    r = layer.r
    br = (lambda k: p[k]) if r > 0 else (lambda k: None)
    y = oracle.fwd(p["x"], p["W"], p["bias"], br("W_down"), br("omega1"), br("phi1"), br("M"),
                   br("omega2"), br("phi2"), br("W_up"))
    g = oracle.bwd(p["x"], p["W"], br("W_down"), br("omega1"), br("phi1"), br("M"),
                   br("omega2"), br("phi2"), br("W_up"), p["dy"])
    out = {"y": y, "dx": g["dx"], "dW": g["dW"].T, "dbias": g["dbias"]}
    if r > 0:
        out.update(dW_down=g["dW_down"].T, dM=g["dM"], domega1=g["domega1"], dphi1=g["dphi1"],
                   domega2=g["domega2"], dphi2=g["dphi2"], dW_up=g["dW_up"].T)
    return out


def compare(got: dict, ref: dict, dtype: str, names=None) -> dict:
    errs = {}
    for k in names or ref.keys():
        if k not in got:
            continue
        scale = np.max(np.abs(ref[k])) if np.size(ref[k]) else 0.0
        e = rel_err(got[k], ref[k])
        tol = TOL[dtype] if scale > 0 else ABS_TOL_ZERO[dtype]
        errs[k] = (e, tol)
    return errs


def assert_close(got: dict, ref: dict, dtype: str, names=None, ctx=""):
    errs = compare(got, ref, dtype, names)
    bad = {k: v for k, v in errs.items() if not v[0] <= v[1]}
    assert not bad, f"{ctx} out of tolerance: {bad}; all: {errs}"
    return errs
