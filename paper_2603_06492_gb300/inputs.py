"""Seeded synthetic inputs for the NOBLE linear layer.

This module draws random tensors and nothing else: it holds none of the
layer's arithmetic, imports neither the CUDA library nor the oracle, and is
the only code that both sides share.

Layer shapes mirror the paper's models (Section 4.1.1: the 250M decoder,
d=1024, sequence 1024; the 1.5B decoder, d=2048; Section 4.2.1 ViT, here at
ViT-Base width 768 with 197 tokens per image).  No dataset is used: every
tensor is drawn from a seeded numpy PCG64 generator in a fixed order

    x, W, bias, W_down, omega1, phi1, M, omega2, phi2, W_up, dy

in fp64 and then rounded to the operand type (bf16 by round-to-nearest-even
through fp32, or fp32).  omega, phi, M and bias are always fp32.

Tensors are returned in the library's layout (nn.Linear "out x in"):
    x [T, d_in], W [d_out, d_in], bias [d_out], W_down [r, d_in],
    omega1, phi1, omega2, phi2 [r], M [r, r] (b = a M), W_up [d_out, r],
    dy [T, d_out].
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np


@dataclass(frozen=True)
class Layer:
    name: str
    T: int
    d_in: int
    d_out: int
    r: int
    dtype: str  # "bf16" or "fp32": operand type of x, W, W_down, W_up, dy, y, dx

    def flops(self) -> float:
        """Algorithmic fwd+bwd FLOPs: 6 T (d_in d_out + r (d_in + d_out) + r^2).

        Three products (forward, data gradient, weight gradient) of each of the
        four contractions x W, x W_down, a M and c W_up, 2 FLOPs per
        multiply-add.  Cosines, bias and the elementwise chain are not counted.
        """
        return 6.0 * self.T * (self.d_in * self.d_out + self.r * (self.d_in + self.d_out)
                               + self.r * self.r)

    def plain(self) -> "Layer":
        return Layer(self.name + "_plain", self.T, self.d_in, self.d_out, 0, self.dtype)


# The five measured configurations; layer i of config k draws from seed layer_seed(k, i).
CONFIGS = {
    0: [Layer("tiny", 256, 128, 128, 16, "fp32")],
    1: [Layer("qkv", 8192, 1024, 3072, 64, "bf16"),
        Layer("attn_out", 8192, 1024, 1024, 64, "bf16")],
    2: [Layer("ffn_up", 8192, 1024, 4096, 64, "bf16"),
        Layer("ffn_down", 8192, 4096, 1024, 64, "bf16")],
    3: [Layer("ffn_up", 16384, 2048, 8192, 128, "bf16"),
        Layer("ffn_down", 16384, 8192, 2048, 128, "bf16"),
        Layer("qkv", 16384, 2048, 6144, 128, "bf16")],
    4: [Layer(f"{n}_r{r}", 50432, di, do, r, "bf16")
        for r in (16, 32, 64, 128, 256)
        for (n, di, do) in (("qkv", 768, 2304), ("ffn_up", 768, 3072), ("ffn_down", 3072, 768))],
}


def round_bf16(a: np.ndarray) -> np.ndarray:
    """Round to the nearest bfloat16 (ties to even) through fp32; returns fp64."""
    f = np.ascontiguousarray(a, dtype=np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    out = (u.astype(np.uint32) << 16).view(np.float32)
    return out.astype(np.float64)


def round_fp32(a: np.ndarray) -> np.ndarray:
    return np.asarray(a, dtype=np.float32).astype(np.float64)


def bf16_bits(a: np.ndarray) -> np.ndarray:
    """uint16 bit patterns of values that are already bf16-representable."""
    f = np.ascontiguousarray(a, dtype=np.float32)
    return (f.view(np.uint32) >> 16).astype(np.uint16)


def make_layer_inputs(layer: Layer, seed: int, init: str = "config") -> dict:
    """Draw one layer's inputs (fp64 arrays holding dtype-representable values).

    ``init`` selects the distributions:
      "config"        x, dy ~ N(0,1); W, W_down ~ N(0, 1/d_in); M ~ N(0, 1/r);
                      W_up ~ N(0, 0.02^2); omega ~ U(0.5, 2); phi ~ U(-pi, pi);
                      bias ~ N(0, 0.02^2).
      "strong_branch" as "config" but W_up ~ N(0, 1/r), so that the branch is
                      as large as the main path and branch errors are visible.
      "paper"         the paper's initialisation (Section 3.3, Appendix A):
                      W ~ N(0, (0.5/sqrt(d_in))^2), W_up ~ N(0, (0.01/sqrt(r))^2),
                      omega ~ U(0.8, 1.2), phi ~ N(0, 0.1^2), M Xavier-uniform.
    """
    T, d_in, d_out, r = layer.T, layer.d_in, layer.d_out, layer.r
    rng = np.random.Generator(np.random.PCG64(seed))
    q = round_bf16 if layer.dtype == "bf16" else round_fp32
    out = {}
    out["x"] = q(rng.standard_normal((T, d_in)))
    w_std = 0.5 / math.sqrt(d_in) if init == "paper" else 1.0 / math.sqrt(d_in)
    out["W"] = q(rng.standard_normal((d_out, d_in)) * w_std)
    out["bias"] = round_fp32(rng.standard_normal(d_out) * 0.02)
    if r > 0:
        out["W_down"] = q(rng.standard_normal((r, d_in)) / math.sqrt(d_in))
        if init == "paper":
            lim = math.sqrt(6.0 / (2 * r))
            out["omega1"] = round_fp32(rng.uniform(0.8, 1.2, r))
            out["phi1"] = round_fp32(rng.standard_normal(r) * 0.1)
            out["M"] = round_fp32(rng.uniform(-lim, lim, (r, r)))
            out["omega2"] = round_fp32(rng.uniform(0.8, 1.2, r))
            out["phi2"] = round_fp32(rng.standard_normal(r) * 0.1)
            out["W_up"] = q(rng.standard_normal((d_out, r)) * (0.01 / math.sqrt(r)))
        else:
            out["omega1"] = round_fp32(rng.uniform(0.5, 2.0, r))
            out["phi1"] = round_fp32(rng.uniform(-math.pi, math.pi, r))
            out["M"] = round_fp32(rng.standard_normal((r, r)) / math.sqrt(r))
            out["omega2"] = round_fp32(rng.uniform(0.5, 2.0, r))
            out["phi2"] = round_fp32(rng.uniform(-math.pi, math.pi, r))
            up_std = 1.0 / math.sqrt(r) if init == "strong_branch" else 0.02
            out["W_up"] = q(rng.standard_normal((d_out, r)) * up_std)
    out["dy"] = q(rng.standard_normal((T, d_out)))
    return out


def make_cos3_inputs(r: int, seed: int) -> dict:
    """The extra parameters of the three-layer cosine bottleneck: M2 [r, r]
    (b2 = a2 M2) ~ N(0, 1/r), omega3 ~ U(0.5, 2), phi3 ~ U(-pi, pi), drawn in
    that order from their own PCG64 stream, fp32."""
    rng = np.random.default_rng(seed)
    return {"M2": round_fp32(rng.standard_normal((r, r)) / math.sqrt(r)),
            "omega3": round_fp32(rng.uniform(0.5, 2.0, r)),
            "phi3": round_fp32(rng.uniform(-math.pi, math.pi, r))}


def to_paper_orientation(inp: dict) -> dict:
    """The same tensors in the paper's row-vector orientation (Eq. 1):
    W [d_in, d_out], W_down [d_in, r], W_up [r, d_out]; others unchanged."""
    out = dict(inp)
    out["W"] = inp["W"].T
    if "W_down" in inp:
        out["W_down"] = inp["W_down"].T
        out["W_up"] = inp["W_up"].T
    return out


def geglu_hidden(d: int) -> int:
    """GeGLU FFN hidden width of the paper's language models: 8/3 d rounded up
    to a multiple of 64 (Section 4.1)."""
    return -(-8 * d // (3 * 64)) * 64


# The paper's own FFN shapes (GeGLU: gate and up projections d -> hidden,
# down projection hidden -> d, NOBLE on all three), as extra workloads next
# to the numbered configurations: the Base model (d = 1024, T = 8192 tokens
# per GPU, r = 64) and the Large model (d = 2048, T = 16384, r = 128).
PAPER_WORKLOADS = {
    "geglu-base": [Layer("gate", 8192, 1024, geglu_hidden(1024), 64, "bf16"),
                   Layer("up", 8192, 1024, geglu_hidden(1024), 64, "bf16"),
                   Layer("down", 8192, geglu_hidden(1024), 1024, 64, "bf16")],
    "geglu-large": [Layer("gate", 16384, 2048, geglu_hidden(2048), 128, "bf16"),
                    Layer("up", 16384, 2048, geglu_hidden(2048), 128, "bf16"),
                    Layer("down", 16384, geglu_hidden(2048), 2048, 128, "bf16")],
}
PAPER_WORKLOAD_SEED = {"geglu-base": 10, "geglu-large": 11}


def layer_seed(config: int, layer_index: int) -> int:
    """Seed of layer ``layer_index`` of configuration ``config`` (config 0 -> 0)."""
    return config * 1000 + layer_index
