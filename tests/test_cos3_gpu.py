"""The three-layer cosine bottleneck (NOBLE_FLAG_SIGMA_COS3, the deepest row of
the ablation in Section 4.4, Table 5) on the GPU through
noble_linear_fwd_cos3 / noble_linear_bwd_cos3, against the oracle's fwd3 /
bwd3 (pinned by tests/test_oracle_cos3.py), in fp32 and bf16 at ragged
shapes for every rank (bf16, r <= 128: the tensor-core bottleneck kernel;
r = 256: CUDA-core rows), and on the CUDA-core path."""
import numpy as np
import pytest

import oracle
from paper_2603_06492_gb300 import binding
from paper_2603_06492_gb300.inputs import Layer, make_cos3_inputs, make_layer_inputs, to_paper_orientation
from tests.gpu_helpers import assert_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2603_06492_gb300.build import build
    build()
    binding.load()


def run_cos3(layer, inp, flags=0):
    import torch
    dev = binding.params_to_device(inp, layer.dtype)
    buf = binding.NobleLinearBuffers(layer.T, layer.d_in, layer.d_out, layer.r, layer.dtype,
                                     flags=binding.NOBLE_FLAG_SIGMA_COS3 | flags)
    binding.forward(buf, dev["x"], dev)
    binding.backward(buf, dev["x"], dev["dy"], dev)
    torch.cuda.synchronize()
    binding.noble_get_device_status(None)
    out = {"y": buf.y, "dx": buf.dx}
    out.update(buf.grads)
    return {k: v.float().cpu().numpy().astype(np.float64) for k, v in out.items()}


def oracle_cos3(inp):
    p = to_paper_orientation(inp)
    y = oracle.fwd3(p["x"], p["W"], p["bias"], p)
    g = oracle.bwd3(p["x"], p["W"], p, p["dy"])
    out = {"y": y, "dx": g["dx"], "dW": g["dW"].T, "dbias": g["dbias"], "dW_down": g["dW_down"].T,
           "dW_up": g["dW_up"].T}
    for k in ("dM", "domega1", "dphi1", "domega2", "dphi2", "dM2", "domega3", "dphi3"):
        out[k] = g[k]
    return out


def inputs(layer, seed):
    inp = make_layer_inputs(layer, seed, init="strong_branch")
    inp.update(make_cos3_inputs(layer.r, seed + 1))
    return inp


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("shape", [(300, 200, 264, 16), (257, 192, 328, 64), (200, 256, 136, 128),
                                   (130, 264, 256, 256), (777, 136, 200, 32), (1000, 512, 520, 128)],
                         ids=lambda s: "x".join(map(str, s)))
def test_cos3_matches_oracle(dtype, shape):
    layer = Layer("cos3", *shape, dtype)
    inp = inputs(layer, 61)
    assert_close(run_cos3(layer, inp), oracle_cos3(inp), dtype, ctx=f"cos3 {dtype} {shape}")


def test_cos3_simt_path():
    layer = Layer("cos3", 200, 136, 264, 32, "bf16")
    inp = inputs(layer, 63)
    assert_close(run_cos3(layer, inp, binding.NOBLE_FLAG_SIMT_ONLY), oracle_cos3(inp), "bf16", ctx="cos3 simt")


def test_cos3_needs_its_entry_points():
    import torch
    layer = Layer("cos3", 64, 64, 64, 16, "bf16")
    dev = binding.params_to_device(inputs(layer, 65), "bf16")
    plain = binding.NobleLinearBuffers(64, 64, 64, 16, "bf16")
    three = binding.NobleLinearBuffers(64, 64, 64, 16, "bf16", flags=binding.NOBLE_FLAG_SIGMA_COS3)
    s = torch.cuda.current_stream().cuda_stream
    with pytest.raises(binding.NobleError) as e:  # a three-layer descriptor on the plain entry point
        binding.noble_linear_fwd(three.desc, dev["x"], dev["W"], None, dev["W_down"], dev["omega1"],
                                 dev["phi1"], dev["M"], dev["omega2"], dev["phi2"], dev["W_up"], three.y,
                                 three.saved, three.saved_bytes, s)
    assert e.value.status == 1
    with pytest.raises(binding.NobleError) as e:  # a plain descriptor on the three-layer entry point
        binding.noble_linear_fwd_cos3(plain.desc, dev["x"], dev["W"], None, dev["W_down"], dev["omega1"],
                                      dev["phi1"], dev["M"], dev["omega2"], dev["phi2"], dev["M2"],
                                      dev["omega3"], dev["phi3"], dev["W_up"], plain.y, plain.saved,
                                      plain.saved_bytes, s)
    assert e.value.status == 1
