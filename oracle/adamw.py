"""fp64 reference of the optimizer step with NOBLE's per-group learning rates.

Test infrastructure only (used by tests/, never by the library).

AdamW with decoupled weight decay, the optimizer of the paper's training
runs (Section 4.1: beta1 = 0.9, beta2 = 0.98, weight decay 0.01), applied
per parameter tensor with the learning rate of its group (Section 3.3,
"Learning Rate Scaling", and the hyperparameter defaults of Appendix A):

    W, bias, W_down : lr
    W_up            : lr * (min(d_in, d_out) / r) ** (2 gamma),  gamma = 0.3
    M               : lr * (min(d_in, d_out) / r) ** gamma_M,    gamma_M = 0.45
    omega1, omega2  : lr * 3
    phi1, phi2      : lr * 5

One step t >= 1 for a tensor p with gradient g, moments m, v and group
learning rate a (elementwise):

    p <- p - a * wd * p                (decoupled decay, if the tensor decays)
    m <- beta1 m + (1 - beta1) g
    v <- beta2 v + (1 - beta2) g^2
    p <- p - (a / (1 - beta1^t)) * m / (sqrt(v) / sqrt(1 - beta2^t) + eps)
"""
from __future__ import annotations

import math

import numpy as np


def lr_multipliers(d_in: int, d_out: int, r: int, gamma: float = 0.3, gamma_m: float = 0.45,
                   omega_mult: float = 3.0, phi_mult: float = 5.0) -> dict:
    """Per-group multipliers of the base learning rate (Section 3.3, Appendix A)."""
    ratio = min(d_in, d_out) / r
    return {"W": 1.0, "bias": 1.0, "W_down": 1.0, "W_up": ratio ** (2.0 * gamma), "M": ratio ** gamma_m,
            "omega": omega_mult, "phi": phi_mult}


def adamw_step(p, g, m, v, step: int, lr: float, beta1: float = 0.9, beta2: float = 0.98,
               eps: float = 1e-8, weight_decay: float = 0.01, decay: bool = True):
    """One AdamW step in fp64 on copies; returns (p, m, v)."""
    p = np.array(p, dtype=np.float64)
    g = np.asarray(g, dtype=np.float64)
    m = np.array(m, dtype=np.float64)
    v = np.array(v, dtype=np.float64)
    if decay:
        p = p - lr * weight_decay * p
    m = beta1 * m + (1.0 - beta1) * g
    v = beta2 * v + (1.0 - beta2) * g * g
    bc1 = 1.0 - beta1 ** step
    bc2 = 1.0 - beta2 ** step
    p = p - (lr / bc1) * m / (np.sqrt(v) / math.sqrt(bc2) + eps)
    return p, m, v
