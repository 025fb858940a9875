"""The inference forward (NOBLE_FLAG_INFERENCE): y must be bit-identical to the
training forward's y on the same inputs (the flag only drops the saved h and
b), and the smaller saved buffer must hold the same c."""
import pytest

from paper_2603_06492_gb300 import binding
from paper_2603_06492_gb300.inputs import Layer, make_layer_inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2603_06492_gb300.build import build
    build()
    binding.load()


@pytest.mark.parametrize("T,d_in,d_out,r", [(300, 256, 320, 16), (1000, 512, 384, 64), (257, 1024, 512, 128),
                                           (4096, 2048, 1024, 256)])
def test_inference_forward_matches_training_forward(T, d_in, d_out, r):
    import torch
    layer = Layer("inf", T, d_in, d_out, r, "bf16")
    dev = binding.params_to_device(make_layer_inputs(layer, 7 + r), "bf16")
    train = binding.NobleLinearBuffers(T, d_in, d_out, r, "bf16", with_grads=False)
    infer = binding.NobleLinearBuffers(T, d_in, d_out, r, "bf16", with_grads=False,
                                       flags=binding.NOBLE_FLAG_INFERENCE)
    assert infer.saved_bytes == (T * r * 2 + 255) // 256 * 256 < train.saved_bytes
    infer.y.fill_(float("nan"))
    binding.forward(train, dev["x"], dev)
    binding.forward(infer, dev["x"], dev)
    torch.cuda.synchronize()
    binding.noble_get_device_status(None)
    assert torch.equal(train.y, infer.y)
    # c: the last [T][r] bf16 block of the training buffer, all of the inference one
    off = ((T * r * 4 + 255) // 256 * 256) * 2  # after h and b, each 256-byte aligned
    c_train = train.saved[off:off + T * r * 2]
    assert torch.equal(c_train, infer.saved[:T * r * 2])
