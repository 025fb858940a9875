"""noble_linear_bwd_noalloc: the backward pass for callers that cannot allocate
device memory (a host framework or plugin that owns every allocation and gives
its extensions no allocator, or a loop that forbids allocation once running).
It uses a static scratch array inside the library instead of a caller
workspace.

Checked through the C ABI against noble_linear_bwd (caller workspace): both
run the same kernels with fixed-order reductions, so the results must be
bit-identical.  The array keeps the previous call's contents, so the checked
calls are separated by a call on other inputs of the same shape (another dy):
a scratch value read before it is written would then carry that call's data
into the next one.  This file is collected last so that a stop-at-first-failure
run has already run every other test; it needs no state from them.
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


def _to_numpy(dx, grads):
    out = {"dx": dx.float().cpu().numpy()}
    out.update({k: v.cpu().numpy() for k, v in grads.items()})
    return out


@pytest.mark.parametrize("shape,dtype", [((300, 200, 264, 64), "bf16"),
                                         ((256, 128, 136, 16), "fp32"),
                                         ((2048, 1024, 1024, 128), "bf16")])
def test_noalloc_matches_workspace_entry_point(shape, dtype):
    import torch
    layer = Layer("noalloc", *shape, dtype)
    inp = make_layer_inputs(layer, 42, init="strong_branch")
    dev = binding.params_to_device(inp, dtype)
    # a second dy of the same shape (another seed)
    dy_other = binding.params_to_device({"dy": make_layer_inputs(layer, 43, init="strong_branch")["dy"]},
                                        dtype)["dy"]
    buf = binding.NobleLinearBuffers(*shape, dtype)
    binding.forward(buf, dev["x"], dev)
    refs = {}
    for name, dy in (("a", dev["dy"]), ("b", dy_other)):
        binding.backward(buf, dev["x"], dy, dev)
        torch.cuda.synchronize()
        refs[name] = _to_numpy(buf.dx, buf.grads)

    # a, then b (other scratch contents), then a again
    for call, name in enumerate(("a", "b", "a")):
        dy = dev["dy"] if name == "a" else dy_other
        dx = torch.full_like(buf.dx, float("nan"))
        grads = {k: torch.full_like(v, float("nan")) for k, v in buf.grads.items()}
        _grads_noalloc(buf, dict(dev, dy=dy), dx, grads)
        torch.cuda.synchronize()
        binding.noble_get_device_status(None)
        got = _to_numpy(dx, grads)
        for k, ref in refs[name].items():
            assert np.all(np.isfinite(got[k])), (call, k)
            assert np.array_equal(got[k], ref), (call, name, k, rel_err(got[k], ref))
        # and within the parity tolerance of the other input's result: the two
        # dy differ, so the test would notice results that ignore dy
        other = refs["b" if name == "a" else "a"]
        assert rel_err(got["dx"], other["dx"]) > TOL[dtype], (call, name)


def test_noalloc_rejects_shapes_beyond_its_scratch():
    d = binding.make_desc(1 << 20, 1024, 1024, 256, "bf16")
    assert binding.noble_linear_bwd_workspace_bytes(d) > binding.NOALLOC_SCRATCH_BYTES
    fake = 0x100000
    with pytest.raises(binding.NobleError) as e:
        binding.noble_linear_bwd_noalloc(d, *([fake] * 11), 1 << 40, *([fake] * 10), None)
    assert e.value.status == 4 and "static scratch" in str(e.value)
