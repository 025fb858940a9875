"""Data-parallel gradient exchange on the host (gloo, world size 2).

Two ranks each take a contiguous share of a layer's tokens, compute the
layer's parameter gradients on their share with the fp64 oracle, place them
in the flat bucket that noble_linear_grad_bucket lays out, and sum the
buckets with the library's all-reduce helper.  Every parameter gradient of
Eq. 1 / Eq. 2 is a sum over tokens, so the reduced bucket must equal the
oracle's gradients of the whole batch: the property the data-parallel
training of Section 4.1.1 rests on.
"""
import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

# name in the oracle -> (bucket slot, transpose into the library layout)
ORACLE_TO_SLOT = {"dW": ("dW", True), "dbias": ("dbias", False), "dW_down": ("dW_down", True),
                  "dW_up": ("dW_up", True), "dM": ("dM", False), "domega1": ("domega1", False),
                  "dphi1": ("dphi1", False), "domega2": ("domega2", False), "dphi2": ("dphi2", False)}


def _layer():
    from paper_2603_06492_gb300.inputs import Layer
    return Layer("dp", 21, 16, 24, 16, "fp32")


def _shard_grads(inp, start, stop):
    """Oracle parameter gradients of tokens [start, stop), library layout."""
    import oracle
    from paper_2603_06492_gb300.inputs import to_paper_orientation
    p = to_paper_orientation(inp)
    g = oracle.bwd(p["x"][start:stop], p["W"], p["W_down"], p["omega1"], p["phi1"], p["M"], p["omega2"],
                   p["phi2"], p["W_up"], p["dy"][start:stop])
    return {ORACLE_TO_SLOT[k][0]: (v.T if ORACLE_TO_SLOT[k][1] else v) for k, v in g.items() if k in ORACLE_TO_SLOT}


def _pack(grads, layout, total_bytes):
    bucket = np.zeros(total_bytes // 4, dtype=np.float32)
    for name, (off, n) in _slots(layout):
        bucket[off // 4: off // 4 + n] = np.asarray(grads[name], dtype=np.float64).reshape(-1)
    return bucket


def _slots(layout):
    return [(k, v) for k, v in layout.items() if k != "total_bytes"]


def _worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import torch
    import torch.distributed as dist
    from paper_2603_06492_gb300 import binding
    from paper_2603_06492_gb300.dp import GradAllReduce, token_shard
    from paper_2603_06492_gb300.inputs import make_layer_inputs
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        layer = _layer()
        inp = make_layer_inputs(layer, 5, init="strong_branch")
        layout = binding.noble_linear_grad_bucket(binding.make_desc(layer.T, layer.d_in, layer.d_out, layer.r, "fp32"))
        start, stop = token_shard(layer.T, rank, world)
        bucket = torch.from_numpy(_pack(_shard_grads(inp, start, stop), layout, layout["total_bytes"]))
        ar = GradAllReduce()
        ar.launch(bucket)
        assert ar.pending == 1
        ar.wait()
        q.put((rank, bucket.numpy().copy()))
    finally:
        dist.destroy_process_group()


@pytest.fixture(scope="module")
def built():
    import oracle
    from paper_2603_06492_gb300.build import build
    build()
    oracle.build()


def test_token_shard_partitions_tokens():
    from paper_2603_06492_gb300.dp import token_shard
    for T in (0, 1, 7, 21, 16384):
        for world in (1, 2, 3, 8):
            spans = [token_shard(T, r, world) for r in range(world)]
            assert spans[0][0] == 0 and spans[-1][1] == T
            assert all(a[1] == b[0] for a, b in zip(spans, spans[1:]))
            sizes = [b - a for a, b in spans]
            assert max(sizes) - min(sizes) <= 1
    with pytest.raises(ValueError):
        token_shard(5, 2, 2)


def test_bucket_layout(built):
    from paper_2603_06492_gb300 import binding
    for r, flags in ((16, 0), (0, 0), (128, binding.NOBLE_FLAG_SIGMA_COS3)):
        d_in, d_out = 2048, 6144
        lay = binding.noble_linear_grad_bucket(binding.make_desc(4096, d_in, d_out, r, "bf16", flags))
        shapes = binding.grad_shapes(d_in, d_out, r)
        slots = [s for s in binding.BUCKET_SLOTS if s in lay]
        expect = ["dW", "dbias"] + (["dW_down", "dW_up", "dM", "domega1", "dphi1", "domega2", "dphi2"] if r else [])
        expect += ["dM2", "domega3", "dphi3"] if flags else []
        assert slots == expect
        end = 0
        for s in slots:
            off, n = lay[s]
            assert off % binding.GRAD_ALIGN == 0 and off >= end
            assert n == int(np.prod(shapes[s]))
            end = off + 4 * n
        assert lay["total_bytes"] % binding.GRAD_ALIGN == 0 and end <= lay["total_bytes"] < end + binding.GRAD_ALIGN
    with pytest.raises(binding.NobleError):
        binding.noble_linear_grad_bucket(binding.make_desc(16, 100, 128, 16, "bf16"))


def test_bucket_views_alias_the_slots(built):
    import torch
    from paper_2603_06492_gb300 import binding
    d_in, d_out, r = 200, 264, 16
    lay = binding.noble_linear_grad_bucket(binding.make_desc(300, d_in, d_out, r, "fp32", binding.NOBLE_FLAG_SIGMA_COS3))
    bucket = torch.zeros(lay["total_bytes"] // 4)
    views = binding.bucket_views(bucket, lay, binding.grad_shapes(d_in, d_out, r))
    assert set(views) == set(binding.BUCKET_SLOTS)
    for i, name in enumerate(binding.BUCKET_SLOTS):
        off, n = lay[name]
        assert tuple(views[name].shape) == binding.grad_shapes(d_in, d_out, r)[name]
        views[name].fill_(i + 1)
        assert torch.all(bucket[off // 4: off // 4 + n] == i + 1)
    assert int((bucket != 0).sum()) == sum(lay[k][1] for k in binding.BUCKET_SLOTS)


def test_allreduce_of_token_shards_equals_full_batch_gradients(built):
    import torch.multiprocessing as mp
    from paper_2603_06492_gb300 import binding
    from paper_2603_06492_gb300.dp import token_shard
    from paper_2603_06492_gb300.inputs import make_layer_inputs

    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = 29700 + os.getpid() % 1000
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    got = dict(q.get(timeout=300) for _ in range(world))
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0

    layer = _layer()
    inp = make_layer_inputs(layer, 5, init="strong_branch")
    layout = binding.noble_linear_grad_bucket(binding.make_desc(layer.T, layer.d_in, layer.d_out, layer.r, "fp32"))
    total = layout["total_bytes"]
    # every rank holds the same reduced bucket: the fp32 sum of the two shards' buckets
    shards = [_pack(_shard_grads(inp, *token_shard(layer.T, r, world)), layout, total) for r in range(world)]
    assert np.array_equal(got[0], got[1])
    assert np.array_equal(got[0], shards[0] + shards[1])
    # and that sum is the gradient of the whole batch
    full = _shard_grads(inp, 0, layer.T)
    for name, (off, n) in _slots(layout):
        ref = np.asarray(full[name], dtype=np.float64).reshape(-1)
        err = np.max(np.abs(got[0][off // 4: off // 4 + n] - ref)) / np.max(np.abs(ref))
        assert err < 1e-6, (name, err)
        # a single shard is not the whole-batch gradient
        assert np.max(np.abs(shards[0][off // 4: off // 4 + n] - ref)) / np.max(np.abs(ref)) > 1e-3, name
    # padding between slots is never written
    used = np.zeros(total // 4, dtype=bool)
    for name, (off, n) in _slots(layout):
        used[off // 4: off // 4 + n] = True
    assert not np.any(got[0][~used])
