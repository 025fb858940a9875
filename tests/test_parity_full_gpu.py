"""Parity at the measured layer shapes (configs 1-4), in the same launch
configuration bench.py times, on outputs the oracle can compute one by one:

  * y and dx on one sampled token of every 128-token tile (up to 256 tiles)
    and the last token (tokens are independent, so the oracle runs on just
    those rows);
  * one element of dW in every 256 x 256 tile, 1024 more at random, and all
    of dbias (each is one sum over tokens);
  * every branch gradient (dW_down, dW_up, dM, domega, dphi) in full, from one
    full-batch oracle pass of the r-wide branch.
"""
import numpy as np
import pytest

import oracle
from paper_2603_06492_gb300.inputs import (CONFIGS, PAPER_WORKLOAD_SEED, PAPER_WORKLOADS, layer_seed,
                                           make_layer_inputs, to_paper_orientation)
from tests.gpu_helpers import TOL, rel_err, run_gpu

pytestmark = pytest.mark.gpu

CASES = [(1, 0), (1, 1), (2, 0), (2, 1), (3, 0), (3, 1), (3, 2),
         (4, 0), (4, 7), (4, 14), (4, 11)]  # config 4: r16 qkv, r64 ffn_up, r256 ffn_down, r128 ffn_down


@pytest.fixture(scope="module", autouse=True)
def lib():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2603_06492_gb300.build import build
    build()


@pytest.mark.parametrize("cfg,li", CASES, ids=lambda v: str(v))
def test_full_size_sampled(cfg, li):
    layer = CONFIGS[cfg][li]
    check_full_size(layer, layer_seed(cfg, li), 100 + cfg * 31 + li, f"config {cfg}")


@pytest.mark.parametrize("li", [0, 1, 2], ids=["ffn_up", "ffn_down", "qkv"])
def test_full_size_strong_branch(li):
    # the 1.5B-scale layers with W_up ~ N(0, 1/r): the branch is as large as
    # the main path, so an error in the second K segment ([x | c] at
    # K = d_in + r, [dy | dh] at K = d_out + r) cannot hide under the main
    # path's magnitude; the branch delta y - (x W^T + bias) is checked too
    layer = CONFIGS[3][li]
    check_full_size(layer, layer_seed(3, li) + 500, 900 + li, "config 3 strong branch", init="strong_branch",
                    branch_delta=True)


@pytest.mark.parametrize("li", [0, 2], ids=["gate_2048x5504", "down_5504x2048"])
def test_paper_geglu_shapes_sampled(li):
    # the paper's Large-model GeGLU FFN projections: a hidden width (5504) that
    # leaves a half-filled last 256-wide tile
    w = "geglu-large"
    layer = PAPER_WORKLOADS[w][li]
    check_full_size(layer, layer_seed(PAPER_WORKLOAD_SEED[w], li), 700 + li, w)


def check_full_size(layer, seed, rng_seed, ctx, init="config", branch_delta=False):
    inp = make_layer_inputs(layer, seed, init=init)
    got = run_gpu(layer, inp)
    p = to_paper_orientation(inp)
    rng = np.random.default_rng(rng_seed)
    tol = TOL[layer.dtype]

    # one token from each 128-token tile (at most 256 tiles), and the last token
    # (the ragged tail tile): every row tile of every kernel is checked
    nblk = -(-layer.T // 128)
    blks = np.sort(rng.choice(nblk, min(nblk, 256), replace=False))
    rows = np.minimum(blks * 128 + rng.integers(0, 128, blks.size), layer.T - 1)
    rows = np.unique(np.append(rows, layer.T - 1))
    sub = {k: (v[rows] if k in ("x", "dy") else v) for k, v in p.items()}
    y_ref = oracle.fwd(sub["x"], sub["W"], sub["bias"], sub["W_down"], sub["omega1"], sub["phi1"],
                       sub["M"], sub["omega2"], sub["phi2"], sub["W_up"])
    g_sub = oracle.bwd(sub["x"], sub["W"], sub["W_down"], sub["omega1"], sub["phi1"], sub["M"],
                       sub["omega2"], sub["phi2"], sub["W_up"], sub["dy"],
                       skip=("dW", "dbias", "dW_down", "dM", "domega1", "dphi1", "domega2",
                             "dphi2", "dW_up"))
    errs = {"y": rel_err(got["y"][rows], y_ref), "dx": rel_err(got["dx"][rows], g_sub["dx"])}
    if branch_delta:
        # x W^T + bias from the oracle (W_up = 0 leaves exactly that)
        plain = oracle.fwd(sub["x"], sub["W"], sub["bias"], sub["W_down"], sub["omega1"], sub["phi1"],
                           sub["M"], sub["omega2"], sub["phi2"], np.zeros_like(sub["W_up"]))
        errs["branch"] = rel_err(got["y"][rows] - plain, y_ref - plain)

    # dW: one element in each 256 x 256 output tile of the weight-gradient
    # launch, 1024 more at random, and the far corner
    tm, tn = -(-layer.d_out // 256), -(-layer.d_in // 256)
    gm, gn = np.meshgrid(np.arange(tm), np.arange(tn), indexing="ij")
    o_idx = np.minimum(gm.ravel() * 256 + rng.integers(0, 256, gm.size), layer.d_out - 1)
    i_idx = np.minimum(gn.ravel() * 256 + rng.integers(0, 256, gn.size), layer.d_in - 1)
    o_idx = np.concatenate([o_idx, rng.integers(0, layer.d_out, 1024), [layer.d_out - 1]])
    i_idx = np.concatenate([i_idx, rng.integers(0, layer.d_in, 1024), [layer.d_in - 1]])
    dW_ref = oracle.outer_elems(p["dy"], p["x"], o_idx, i_idx)
    errs["dW"] = rel_err(got["dW"][o_idx, i_idx], dW_ref)
    ones = np.ones((layer.T, 1))
    dbias_ref = oracle.outer_elems(p["dy"], ones, np.arange(layer.d_out), np.zeros(layer.d_out, np.int64))
    errs["dbias"] = rel_err(got["dbias"], dbias_ref)

    g = oracle.bwd(p["x"], p["W"], p["W_down"], p["omega1"], p["phi1"], p["M"], p["omega2"],
                   p["phi2"], p["W_up"], p["dy"], skip=("dx", "dW", "dbias"))
    errs["dW_down"] = rel_err(got["dW_down"], g["dW_down"].T)
    errs["dW_up"] = rel_err(got["dW_up"], g["dW_up"].T)
    for k in ("dM", "domega1", "dphi1", "domega2", "dphi2"):
        errs[k] = rel_err(got[k], g[k])
    bad = {k: e for k, e in errs.items() if not e <= tol}
    assert not bad, f"{ctx} {layer.name}: {bad} (all {errs})"
