"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle on the
same seeded inputs, element by element, at sizes the oracle finishes in
seconds (several tiles and a ragged tail), plus the special cases of the
method and the edge cases of the interface."""
import math

import numpy as np
import pytest

from paper_2603_06492_gb300 import binding
from paper_2603_06492_gb300.inputs import CONFIGS, Layer, layer_seed, make_layer_inputs
from tests.gpu_helpers import assert_close, rel_err, run_gpu, run_oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2603_06492_gb300.build import build
    build()
    binding.load()


def test_config0_fp32_full():
    layer = CONFIGS[0][0]
    inp = make_layer_inputs(layer, layer_seed(0, 0))
    assert_close(run_gpu(layer, inp), run_oracle(layer, inp), "fp32", ctx="config 0")


SMALL = [
    # (T, d_in, d_out, r): multiple tiles in every dimension plus ragged tails
    (300, 200, 264, 16),
    (129, 136, 72, 32),
    (257, 192, 328, 64),
    (200, 256, 136, 128),
    (130, 264, 256, 256),
    (1, 128, 128, 64),
    (33, 128, 136, 128),  # one row in the second 32-row box, the last two boxes past T
    (31, 64, 72, 128),    # fewer tokens than one 32-row store box; a single k-block
    (127, 72, 40, 16),
    (333, 200, 264, 0),
]


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("shape", SMALL, ids=lambda s: "x".join(map(str, s)))
@pytest.mark.parametrize("init", ["config", "strong_branch"])
def test_small_shapes(dtype, shape, init):
    layer = Layer("small", *shape, dtype)
    inp = make_layer_inputs(layer, 1234 + sum(shape), init=init)
    got, ref = run_gpu(layer, inp), run_oracle(layer, inp)
    assert_close(got, ref, dtype, ctx=f"{shape} {dtype} {init}")


# The bottleneck fused into the output GEMMs (NOBLE_FLAG_FUSED_BRANCH, the
# CosNet with r in {64, 128}) and the separate kernels: both against the
# oracle, on shapes with several groups of 8 row pairs, a ragged last group
# and ragged column tiles (the fused tile order and its ready flags).
FUSED = [
    (5000, 256, 520, 128),
    (5000, 192, 264, 64),
    (2049, 512, 1000, 128),
    (300, 136, 264, 64),   # d_in % 64 != 0: fused forward, separate backward
    (600, 128, 128, 128),  # d_in = d_out = r: leader tiles only
    (1000, 320, 192, 64),  # forward: leader + 128-wide tail; backward: leader + 256-wide tiles
    (20000, 192, 448, 64),  # more row pairs than clusters: several waves of leaders
]


@pytest.mark.parametrize("shape", FUSED, ids=lambda s: "x".join(map(str, s)))
@pytest.mark.parametrize("separate", [False, True], ids=["fused", "separate"])
def test_fused_bottleneck(shape, separate):
    layer = Layer("fused", *shape, "bf16")
    inp = make_layer_inputs(layer, 4321 + sum(shape), init="strong_branch")
    flags = 0 if separate else binding.NOBLE_FLAG_FUSED_BRANCH
    got, ref = run_gpu(layer, inp, flags=flags), run_oracle(layer, inp)
    assert_close(got, ref, "bf16", ctx=f"{shape} {'separate' if separate else 'fused'}")


def _bf16_ulp(v):
    # spacing of bf16 numbers at |v| (8 significant bits)
    e = np.floor(np.log2(np.maximum(np.abs(v), np.finfo(np.float32).tiny)))
    return np.exp2(e - 7)


def _is_bf16(v):
    import torch
    return np.array_equal(v, torch.from_numpy(v).to(torch.bfloat16).double().numpy())


def test_fused_matches_separate():
    # same arithmetic up to summation order: far tighter than the oracle bound.
    # Both runs accumulate in fp32 in different orders, so an output stored in
    # bf16 may round the other way: there an element may differ by one bf16
    # step of its own magnitude, and few elements may differ at all.
    layer = Layer("fused", 3000, 256, 520, 128, "bf16")
    inp = make_layer_inputs(layer, 99)
    a = run_gpu(layer, inp, flags=binding.NOBLE_FLAG_FUSED_BRANCH)
    b = run_gpu(layer, inp)
    for k in a:
        if _is_bf16(a[k]) and _is_bf16(b[k]):
            d = np.abs(a[k] - b[k])
            step = _bf16_ulp(np.maximum(np.abs(a[k]), np.abs(b[k])))
            scale = np.max(np.abs(b[k]))
            assert np.all(d <= np.maximum(step, 2e-3 * scale)), (k, float(np.max(d / step)))
            assert np.mean(d > 0) <= 0.02, (k, float(np.mean(d > 0)))
        else:
            assert rel_err(a[k], b[k]) <= 2e-3, (k, rel_err(a[k], b[k]))


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_paper_init(dtype):
    layer = Layer("paper_init", 257, 192, 264, 64, dtype)
    inp = make_layer_inputs(layer, 77, init="paper")
    assert_close(run_gpu(layer, inp), run_oracle(layer, inp), dtype, ctx="paper init")


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_branch_delta(dtype):
    """The branch term alone, y - (x W^T + bias), so branch errors cannot hide
    under the main path's magnitude."""
    layer = Layer("delta", 256, 128, 192, 32, dtype)
    inp = make_layer_inputs(layer, 5)
    plain = {k: v for k, v in inp.items() if k in ("x", "W", "bias", "dy")}
    lp = layer.plain()
    got = run_gpu(layer, inp)["y"] - run_gpu(lp, plain)["y"]
    ref = run_oracle(layer, inp)["y"] - run_oracle(lp, plain)["y"]
    # y itself is rounded to the operand type; compare against that rounding
    scale = np.max(np.abs(run_oracle(layer, inp)["y"]))
    ulp = scale * (2.0**-8 if dtype == "bf16" else 2.0**-23)
    err = np.max(np.abs(got - ref))
    assert err <= 2 * ulp + 1e-2 * np.max(np.abs(ref)), (err, ulp, np.max(np.abs(ref)))


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_zero_up_equals_plain_path(dtype):
    """W_up = 0: y and dx equal the r = 0 path bit for bit; branch gradients
    other than dW_up vanish."""
    layer = Layer("s1", 200, 136, 264, 32, dtype)
    inp = make_layer_inputs(layer, 11)
    inp["W_up"] = np.zeros_like(inp["W_up"])
    got = run_gpu(layer, inp)
    plain = run_gpu(layer.plain(), {k: inp[k] for k in ("x", "W", "bias", "dy")})
    assert np.array_equal(got["y"], plain["y"])
    assert np.array_equal(got["dx"], plain["dx"])
    assert np.array_equal(got["dW"], plain["dW"])
    for k in ("dW_down", "dM", "domega1", "dphi1", "domega2", "dphi2"):
        assert np.all(got[k] == 0), k
    assert_close(got, run_oracle(layer, inp), dtype, ctx="W_up = 0")


def test_linear_limit_fp32():
    """phi = -pi/2, small omega: CosNet is nearly linear; checked against the
    oracle in fp32 (fixes the orientation of M on the device too)."""
    layer = Layer("lin", 192, 128, 136, 16, "fp32")
    inp = make_layer_inputs(layer, 21, init="strong_branch")
    rng = np.random.default_rng(0)
    for k in ("phi1", "phi2"):
        inp[k] = np.full(16, np.float32(-math.pi / 2), dtype=np.float64)
    inp["omega1"] = np.float32(1e-2) * rng.uniform(0.5, 2, 16).astype(np.float32).astype(np.float64)
    inp["omega2"] = rng.uniform(0.5, 2, 16).astype(np.float32).astype(np.float64)
    assert_close(run_gpu(layer, inp), run_oracle(layer, inp), "fp32", ctx="linear limit")


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_phase_periodicity(dtype):
    layer = Layer("per", 256, 128, 128, 16, dtype)
    inp = make_layer_inputs(layer, 9)
    base = run_gpu(layer, inp)
    shifted = dict(inp, phi1=(inp["phi1"] + 2 * math.pi).astype(np.float32).astype(np.float64))
    got = run_gpu(layer, shifted)
    ref = run_oracle(layer, shifted)
    assert_close(got, ref, dtype, ctx="phase + 2 pi")
    for k in base:
        assert rel_err(got[k], base[k]) < (1e-4 if dtype == "fp32" else 2e-2), k


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_deterministic(dtype):
    layer = Layer("det", 300, 200, 264, 64, dtype)
    inp = make_layer_inputs(layer, 3)
    a, b = run_gpu(layer, inp), run_gpu(layer, inp, repeat=2)
    for k in a:
        assert np.array_equal(a[k], b[k]), k


def test_deterministic_fused():
    layer = Layer("det", 2049, 256, 520, 128, "bf16")
    inp = make_layer_inputs(layer, 5)
    f = binding.NOBLE_FLAG_FUSED_BRANCH
    a, b = run_gpu(layer, inp, flags=f), run_gpu(layer, inp, repeat=3, flags=f)
    for k in a:
        assert np.array_equal(a[k], b[k]), k


def test_token_permutation_bf16():
    layer = Layer("perm", 256, 128, 136, 32, "bf16")
    inp = make_layer_inputs(layer, 8)
    perm = np.random.default_rng(1).permutation(256)
    q = dict(inp, x=inp["x"][perm], dy=inp["dy"][perm])
    a, b = run_gpu(layer, inp), run_gpu(layer, q)
    assert np.array_equal(b["y"], a["y"][perm])
    assert np.array_equal(b["dx"], a["dx"][perm])


def test_empty_batch():
    import torch
    layer = Layer("empty", 0, 128, 64, 16, "bf16")
    inp = make_layer_inputs(layer, 0)
    dev = binding.params_to_device(inp, "bf16")
    buf = binding.NobleLinearBuffers(0, 128, 64, 16, "bf16")
    for g in buf.grads.values():
        g.fill_(7.0)
    binding.forward(buf, dev["x"], dev)
    binding.backward(buf, dev["x"], dev["dy"], dev)
    torch.cuda.synchronize()
    for k, g in buf.grads.items():
        assert torch.all(g == 0), k


def test_device_status_reporting():
    binding.noble_get_device_status(None)
    binding.noble_debug_raise_device_status(1)
    with pytest.raises(binding.NobleError) as e:
        binding.noble_get_device_status(None)
    assert e.value.status == 6
    binding.noble_get_device_status(None)  # cleared


def test_device_side_wait_expiry():
    """A kernel's bounded mbarrier wait really expires on the device: the test
    kernel waits 1 ms on a barrier nothing arrives at, records the timeout in
    the status word and exits; the host reads NOBLE_ERR_TIMEOUT, and a normal
    fwd+bwd right after still matches the oracle."""
    import torch
    binding.noble_get_device_status(None)
    result = torch.zeros(4, dtype=torch.int32, device="cuda")
    binding.noble_debug_wait_expiry(1_000_000, result)
    with pytest.raises(binding.NobleError) as e:
        binding.noble_get_device_status(None)
    assert e.value.status == 6 and "bounded wait" in str(e.value)
    assert int(result[0]) == 2  # the wait returned false
    binding.noble_get_device_status(None)  # cleared
    layer = Layer("after_timeout", 300, 256, 264, 64, "bf16")
    inp = make_layer_inputs(layer, 5, init="strong_branch")
    assert_close(run_gpu(layer, inp), run_oracle(layer, inp), "bf16", ctx="after the expired wait")
    with pytest.raises(binding.NobleError) as e:
        binding.noble_debug_wait_expiry(0, result)
    assert e.value.status == 1


def test_launch_counter_advances():
    layer = Layer("cnt", 128, 128, 128, 16, "bf16")
    inp = make_layer_inputs(layer, 2)
    n0 = binding.noble_kernel_launch_count()
    run_gpu(layer, inp)
    assert binding.noble_kernel_launch_count() > n0


@pytest.mark.parametrize("d_out,r", [(768, 256), (2304, 16), (6144, 128), (1024, 64)])
def test_dbias_from_cosnet_kernel(d_out, r):
    """dbias is summed from the dy tiles streamed by the CosNet backward
    kernel; check it against an fp64 column sum on shapes with many k-blocks
    per tile, eight times in a row (the sums race with the ring reuse that
    follows the main loop, or with the refill of a stage by the copy engine,
    if their ordering is wrong)."""
    import torch
    layer = Layer("dbias", 4096, 256, d_out, r, "bf16")
    inp = make_layer_inputs(layer, 31)
    ref = inp["dy"].sum(axis=0)
    dev = binding.params_to_device(inp, "bf16")
    buf = binding.NobleLinearBuffers(4096, 256, d_out, r, "bf16")
    binding.forward(buf, dev["x"], dev)
    for _ in range(8):
        buf.grads["dbias"].fill_(float("nan"))
        binding.backward(buf, dev["x"], dev["dy"], dev)
        torch.cuda.synchronize()
        got = buf.grads["dbias"].cpu().numpy().astype(np.float64)
        assert rel_err(got, ref) < 1e-5, rel_err(got, ref)


@pytest.mark.parametrize("T,d_out", [(4096, 8192), (1000, 264)])
def test_dbias_without_branch(T, d_out):
    """r = 0: dbias (the all-ones operand's column of the weight-gradient
    launch) against an fp64 column sum, and bit-identical over repeated
    calls."""
    import torch
    layer = Layer("dbias0", T, 256, d_out, 0, "bf16")
    inp = make_layer_inputs(layer, 37)
    ref = inp["dy"].sum(axis=0)
    dev = binding.params_to_device(inp, "bf16")
    buf = binding.NobleLinearBuffers(T, 256, d_out, 0, "bf16")
    binding.forward(buf, dev["x"], dev)
    first = None
    for _ in range(2):
        buf.grads["dbias"].fill_(float("nan"))
        binding.backward(buf, dev["x"], dev["dy"], dev)
        torch.cuda.synchronize()
        got = buf.grads["dbias"].cpu().numpy().astype(np.float64)
        assert rel_err(got, ref) < 1e-5, rel_err(got, ref)
        if first is None:
            first = got
        assert np.array_equal(first, got)
