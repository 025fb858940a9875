"""Bottleneck variants of the ablation (Section 4.4, Table 5) on the GPU: the
single cosine sigma(h) = cos(omega1 h + phi1) (NOBLE_FLAG_SIGMA_COS1) and the
identity sigma(h) = h (NOBLE_FLAG_SIGMA_IDENTITY), against the oracle's modes
of the same name (the identity mode is pinned by the collapse to
x (W + W_down W_up)).  Parameters a variant does not use are passed as NULL;
their gradients must come back as exact zeros."""
import numpy as np
import pytest

import oracle
from paper_2603_06492_gb300 import binding
from paper_2603_06492_gb300.inputs import Layer, make_layer_inputs, to_paper_orientation
from tests.gpu_helpers import assert_close

pytestmark = pytest.mark.gpu

VARIANTS = {"cos1": (binding.NOBLE_FLAG_SIGMA_COS1, oracle.COS1, ("M", "omega2", "phi2")),
            "identity": (binding.NOBLE_FLAG_SIGMA_IDENTITY, oracle.IDENTITY,
                         ("omega1", "phi1", "M", "omega2", "phi2"))}


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


@pytest.mark.parametrize("variant", sorted(VARIANTS))
@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("shape", [(300, 200, 264, 16), (257, 192, 328, 64), (200, 256, 136, 128),
                                   (130, 264, 256, 256)], ids=lambda s: "x".join(map(str, s)))
def test_variant_matches_oracle(variant, dtype, shape):
    flags, mode, unused = VARIANTS[variant]
    layer = Layer(variant, *shape, dtype)
    inp = make_layer_inputs(layer, 41, init="strong_branch")
    got = run_variant(layer, inp, flags, unused)
    ref = oracle_variant(inp, mode)
    assert_close(got, ref, dtype, ctx=f"{variant} {dtype} {shape}")
    zero = {"cos1": ("dM", "domega2", "dphi2"),
            "identity": ("dM", "domega1", "dphi1", "domega2", "dphi2")}[variant]
    for k in zero:
        assert np.all(got[k] == 0), k


@pytest.mark.parametrize("variant", sorted(VARIANTS))
def test_variant_simt_path_agrees(variant):
    """bf16 on the CUDA-core kernels (NOBLE_FLAG_SIMT_ONLY) against the oracle too."""
    flags, mode, unused = VARIANTS[variant]
    layer = Layer(variant, 200, 136, 264, 32, "bf16")
    inp = make_layer_inputs(layer, 43)
    got = run_variant(layer, inp, flags | binding.NOBLE_FLAG_SIMT_ONLY, unused)
    assert_close(got, oracle_variant(inp, mode), "bf16", ctx=f"{variant} simt")
