"""Bottleneck variants of the ablation (Section 4.4, Table 5) on the GPU: the
single cosine sigma(h) = cos(omega1 h + phi1) (NOBLE_FLAG_SIGMA_COS1), the
identity sigma(h) = h (NOBLE_FLAG_SIGMA_IDENTITY), and tanh, LeakyReLU and
GELU with one layer (sigma(h) = f(h)) or two around the mixing matrix
(sigma(h) = f(f(h) M)), against the oracle's modes of the same name.
Parameters a variant does not use are passed as NULL; their gradients must
come back as exact zeros.

LeakyReLU's derivative is a decision on the sign of h (and of b): the GPU
takes it in fp32, the oracle in fp64, and where a pre-activation is within
rounding of zero the two may take different branches.  Rows are independent,
so the tokens whose oracle h lies within 2e-5, or b within 2e-4, of zero
(relative to the largest magnitude; the GPU's h and b carry ~1e-6 and ~1e-5
relative error) get a zero dy row: every term that multiplies the ambiguous
derivative is then exactly zero on both sides, and all outputs are compared.
The forward output y is continuous in h and b and is compared on every row."""
import numpy as np
import pytest

import oracle
from paper_2603_06492_gb300 import binding
from paper_2603_06492_gb300.inputs import Layer, make_layer_inputs, to_paper_orientation
from tests.gpu_helpers import assert_close

pytestmark = pytest.mark.gpu

VARIANTS = {k: (binding.SIGMA_FLAGS[k], oracle.MODES[k], binding.SIGMA_UNUSED[k])
            for k in ("cos1", "identity", "tanh1", "tanh2", "leaky1", "leaky2", "gelu1", "gelu2")}
# gradients that must be exact zeros
ZERO = {"cos1": ("dM", "domega2", "dphi2"), "identity": ("dM", "domega1", "dphi1", "domega2", "dphi2")}
for _n in ("tanh", "leaky", "gelu"):
    ZERO[_n + "1"] = ("dM", "domega1", "dphi1", "domega2", "dphi2")
    ZERO[_n + "2"] = ("domega1", "dphi1", "domega2", "dphi2")


@pytest.fixture(scope="module", autouse=True)
def lib():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2603_06492_gb300.build import build
    build()
    binding.load()


def run_variant(layer, inp, flags, unused):
    import torch
    dev = binding.params_to_device(inp, layer.dtype)
    for k in unused:
        dev[k] = None
    buf = binding.NobleLinearBuffers(layer.T, layer.d_in, layer.d_out, layer.r, layer.dtype, flags=flags)
    binding.forward(buf, dev["x"], dev)
    binding.backward(buf, dev["x"], dev["dy"], dev)
    torch.cuda.synchronize()
    binding.noble_get_device_status(None)
    out = {"y": buf.y, "dx": buf.dx}
    out.update(buf.grads)
    return {k: v.float().cpu().numpy().astype(np.float64) for k, v in out.items()}


def oracle_variant(inp, mode):
    p = to_paper_orientation(inp)
    args = [p[k] for k in ("W_down", "omega1", "phi1", "M", "omega2", "phi2", "W_up")]
    y = oracle.fwd(p["x"], p["W"], p["bias"], *args, mode=mode)
    g = oracle.bwd(p["x"], p["W"], *args, p["dy"], mode=mode)
    return {"y": y, "dx": g["dx"], "dW": g["dW"].T, "dbias": g["dbias"], "dW_down": g["dW_down"].T,
            "dW_up": g["dW_up"].T, "dM": g["dM"], "domega1": g["domega1"], "dphi1": g["dphi1"],
            "domega2": g["domega2"], "dphi2": g["dphi2"]}


def variant_inputs(layer, variant, seed, init="strong_branch"):
    """Seeded inputs; for LeakyReLU, dy is zero on the tokens whose
    pre-activations (the oracle's h, and b with two layers) come within
    rounding of 0.  Returns (inputs, number of zeroed rows)."""
    inp = make_layer_inputs(layer, seed, init=init)
    if not variant.startswith("leaky"):
        return inp, 0
    p = to_paper_orientation(inp)
    args = [p[k] for k in ("W_down", "omega1", "phi1", "M", "omega2", "phi2", "W_up")]
    _, h, b, _ = oracle.fwd(p["x"], p["W"], p["bias"], *args, mode=oracle.MODES[variant],
                            want_intermediates=True)
    pre = [(h, 2e-5)] + ([(b, 2e-4)] if variant.endswith("2") else [])
    near = np.zeros(layer.T, dtype=bool)
    for v, tol in pre:
        near |= np.any(np.abs(v) <= tol * np.max(np.abs(v)), axis=1)
    inp = dict(inp)
    inp["dy"] = np.where(near[:, None], 0.0, inp["dy"]).astype(inp["dy"].dtype)
    return inp, int(near.sum())


@pytest.mark.parametrize("variant", sorted(VARIANTS))
@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("shape", [(300, 200, 264, 16), (257, 192, 328, 64), (200, 256, 136, 128),
                                   (130, 264, 256, 256)], ids=lambda s: "x".join(map(str, s)))
def test_variant_matches_oracle(variant, dtype, shape):
    flags, mode, unused = VARIANTS[variant]
    layer = Layer(variant, *shape, dtype)
    inp, zeroed = variant_inputs(layer, variant, 41)
    assert zeroed < layer.T // 4, zeroed  # most rows still carry a gradient
    got = run_variant(layer, inp, flags, unused)
    ref = oracle_variant(inp, mode)
    assert_close(got, ref, dtype, ctx=f"{variant} {dtype} {shape} ({zeroed} dy rows zeroed)")
    for k in ZERO[variant]:
        assert np.all(got[k] == 0), k


@pytest.mark.parametrize("variant", sorted(VARIANTS))
def test_variant_simt_path_agrees(variant):
    """bf16 on the CUDA-core kernels (NOBLE_FLAG_SIMT_ONLY) against the oracle too."""
    flags, mode, unused = VARIANTS[variant]
    layer = Layer(variant, 200, 136, 264, 32, "bf16")
    inp, _ = variant_inputs(layer, variant, 43, init="config")
    got = run_variant(layer, inp, flags | binding.NOBLE_FLAG_SIMT_ONLY, unused)
    assert_close(got, oracle_variant(inp, mode), "bf16", ctx=f"{variant} simt")
