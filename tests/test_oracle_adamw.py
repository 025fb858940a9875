"""Pins for the fp64 optimizer reference (oracle/adamw.py): a library
implementation of the same rule (torch.optim.AdamW on the CPU, fp64), the
first step in closed form, and exact cases of the paper's learning-rate
multipliers (Section 3.3, Appendix A)."""
import math

import numpy as np
import pytest

from oracle import adamw


def test_matches_library_adamw_over_several_steps():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(3)
    shapes = [(7, 5), (13,), (4, 4)]
    mults = [1.0, 5.0, 3.0]
    decays = [True, False, True]
    lr, wd = 3e-3, 0.01
    ps = [rng.standard_normal(s) for s in shapes]
    tp = [torch.tensor(p, dtype=torch.float64, requires_grad=True) for p in ps]
    groups = [{"params": [t], "lr": lr * k, "weight_decay": wd if d else 0.0}
              for t, k, d in zip(tp, mults, decays)]
    opt = torch.optim.AdamW(groups, betas=(0.9, 0.98), eps=1e-8)
    ms = [np.zeros(s) for s in shapes]
    vs = [np.zeros(s) for s in shapes]
    for step in range(1, 6):
        gs = [rng.standard_normal(s) for s in shapes]
        for t, g in zip(tp, gs):
            t.grad = torch.tensor(g, dtype=torch.float64)
        opt.step()
        for i in range(len(ps)):
            ps[i], ms[i], vs[i] = adamw.adamw_step(ps[i], gs[i], ms[i], vs[i], step, lr * mults[i],
                                                   weight_decay=wd, decay=decays[i])
        for p, t in zip(ps, tp):
            np.testing.assert_allclose(p, t.detach().numpy(), rtol=1e-13, atol=1e-15)


def test_first_step_closed_form():
    # m = v = 0 at step 1: the bias-corrected moments are g and g^2, so the
    # step is a * g / (|g| + eps) after the decay factor (1 - a wd)
    rng = np.random.default_rng(5)
    p0, g = rng.standard_normal(50), rng.standard_normal(50)
    a, wd, eps = 1e-2, 0.1, 1e-8
    p1, m1, v1 = adamw.adamw_step(p0, g, np.zeros(50), np.zeros(50), 1, a, weight_decay=wd, eps=eps)
    np.testing.assert_allclose(p1, p0 * (1 - a * wd) - a * g / (np.abs(g) + eps), rtol=1e-12)
    np.testing.assert_allclose(m1, 0.1 * g, rtol=1e-15)
    np.testing.assert_allclose(v1, 0.02 * g * g, rtol=1e-14)


def test_zero_gradient_only_decays():
    p0 = np.linspace(-1, 1, 9)
    p, m, v = p0, np.zeros(9), np.zeros(9)
    for step in range(1, 4):
        p, m, v = adamw.adamw_step(p, np.zeros(9), m, v, step, 0.5, weight_decay=0.2)
    np.testing.assert_allclose(p, p0 * 0.9 ** 3, rtol=1e-15)


def test_learning_rate_multipliers_exact_cases():
    # min(d_in, d_out) / r = 32: W_up gets 32^(2*0.3) = 2^3 = 8 exactly
    k = adamw.lr_multipliers(2048, 4096, 64)
    assert k["W_up"] == pytest.approx(8.0, rel=1e-15)
    assert k["M"] == pytest.approx(2.0 ** 2.25, rel=1e-15)  # 32^0.45 = 2^(5 * 0.45)
    assert (k["W"], k["bias"], k["W_down"], k["omega"], k["phi"]) == (1.0, 1.0, 1.0, 3.0, 5.0)
    # the smaller of the two widths sets the ratio; r equal to it gives 1
    k = adamw.lr_multipliers(8192, 128, 128)
    assert k["W_up"] == 1.0 and k["M"] == 1.0
    assert math.isclose(adamw.lr_multipliers(1024, 4096, 64)["W_up"], 16 ** 0.6)
