"""noble_linear_bwd_noalloc: the backward pass for callers that cannot allocate
device memory (a host framework or plugin that owns every allocation and gives
its extensions no allocator, or a loop that forbids allocation once running).
It uses a static scratch array inside the library instead of a caller
workspace.

Checked through the C ABI against noble_linear_bwd (caller workspace) on the
same inputs, within the parity tolerance of the other GPU tests, on two calls
in a row (the array keeps the previous call's contents).  This file is
collected last so that a stop-at-first-failure run has already run every
other test; it needs no state from them.
"""
import numpy as np
import pytest

from paper_2603_06492_gb300 import binding
from paper_2603_06492_gb300.inputs import Layer, make_layer_inputs
from tests.gpu_helpers import TOL, rel_err

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2603_06492_gb300.build import build
    build()
    binding.load()


def _grads_noalloc(buf, dev, dx, grads):
    g = grads
    binding.noble_linear_bwd_noalloc(
        buf.desc, dev["dy"], dev["x"], dev["W"], dev.get("W_down"), dev.get("omega1"),
        dev.get("phi1"), dev.get("M"), dev.get("omega2"), dev.get("phi2"), dev.get("W_up"),
        buf.saved, buf.saved_bytes, dx, g["dW"], g["dbias"], g.get("dW_down"), g.get("dM"),
        g.get("domega1"), g.get("dphi1"), g.get("domega2"), g.get("dphi2"), g.get("dW_up"), None)


@pytest.mark.parametrize("shape,dtype", [((300, 200, 264, 64), "bf16"),
                                         ((256, 128, 136, 16), "fp32"),
                                         ((2048, 1024, 1024, 128), "bf16")])
def test_noalloc_matches_workspace_entry_point(shape, dtype):
    import torch
    layer = Layer("noalloc", *shape, dtype)
    inp = make_layer_inputs(layer, 42, init="strong_branch")
    dev = binding.params_to_device(inp, dtype)
    buf = binding.NobleLinearBuffers(*shape, dtype)
    binding.forward(buf, dev["x"], dev)
    binding.backward(buf, dev["x"], dev["dy"], dev)
    torch.cuda.synchronize()
    ref = {"dx": buf.dx.float().cpu().numpy()}
    ref.update({k: v.cpu().numpy() for k, v in buf.grads.items()})

    for call in range(2):
        dx = torch.full_like(buf.dx, float("nan"))
        grads = {k: torch.full_like(v, float("nan")) for k, v in buf.grads.items()}
        _grads_noalloc(buf, dev, dx, grads)
        torch.cuda.synchronize()
        binding.noble_get_device_status(None)
        got = {"dx": dx.float().cpu().numpy()}
        got.update({k: v.cpu().numpy() for k, v in grads.items()})
        for k in ref:
            assert np.all(np.isfinite(got[k])), (call, k)
            assert rel_err(got[k], ref[k]) <= TOL[dtype], (call, k, rel_err(got[k], ref[k]))


def test_noalloc_rejects_shapes_beyond_its_scratch():
    d = binding.make_desc(1 << 20, 1024, 1024, 256, "bf16")
    assert binding.noble_linear_bwd_workspace_bytes(d) > binding.NOALLOC_SCRATCH_BYTES
    fake = 0x100000
    with pytest.raises(binding.NobleError) as e:
        binding.noble_linear_bwd_noalloc(d, *([fake] * 11), 1 << 40, *([fake] * 10), None)
    assert e.value.status == 4 and "static scratch" in str(e.value)
