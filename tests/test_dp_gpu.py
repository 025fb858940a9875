"""The data-parallel gradient exchange on the GPU (one rank, NCCL): a layer's
backward writes its gradients into the flat bucket that
noble_linear_grad_bucket lays out, and dp.GradAllReduce reduces that bucket
with an asynchronous NCCL all-reduce ordered after the backward on the
stream.  With one rank the sum is the bucket itself, so the gradients read
from the bucket after the reduction must equal the oracle's (Eq. 1 / Eq. 2
chain rule), and the padding between slots must stay zero."""
import os

import numpy as np
import pytest

from paper_2603_06492_gb300 import binding
from paper_2603_06492_gb300.inputs import Layer, make_layer_inputs
from tests.gpu_helpers import assert_close, run_oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def nccl_group():
    import torch
    import torch.distributed as dist
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2603_06492_gb300.build import build
    build()
    binding.load()
    os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
    os.environ.setdefault("MASTER_PORT", str(29900 + os.getpid() % 1000))
    dist.init_process_group("nccl", rank=0, world_size=1, device_id=torch.device("cuda", 0))
    yield dist
    dist.destroy_process_group()


def test_bucket_allreduce_one_rank(nccl_group):
    import torch
    from paper_2603_06492_gb300.dp import GradAllReduce
    layer = Layer("dp_gpu", 777, 256, 520, 64, "bf16")
    inp = make_layer_inputs(layer, 41, init="strong_branch")
    dev = binding.params_to_device(inp, "bf16")
    buf = binding.NobleLinearBuffers(layer.T, layer.d_in, layer.d_out, layer.r, "bf16")
    buf.bucket.fill_(float("nan"))
    used = torch.zeros_like(buf.bucket, dtype=torch.bool)
    for name, slot in buf.layout.items():
        if name != "total_bytes":
            off, n = slot
            used[off // 4: off // 4 + n] = True
    buf.bucket[~used] = 0.0
    stream = torch.cuda.current_stream()
    binding.forward(buf, dev["x"], dev, stream)
    binding.backward(buf, dev["x"], dev["dy"], dev, stream)
    ar = GradAllReduce()
    ar.launch(buf.bucket)
    ar.wait()
    torch.cuda.synchronize()
    binding.noble_get_device_status(None)
    assert not torch.any(buf.bucket[~used] != 0)
    got = {"y": buf.y, "dx": buf.dx}
    got.update(buf.grads)
    got = {k: v.float().cpu().numpy().astype(np.float64) for k, v in got.items()}
    assert_close(got, run_oracle(layer, inp), "bf16", ctx="bucket after the all-reduce")
