"""C-ABI checks that need no GPU: the library builds, loads, exports every
function include/noble.h declares, and rejects bad arguments on the host
before it touches a device."""
import ctypes

import pytest

from paper_2603_06492_gb300 import binding
from paper_2603_06492_gb300.build import build


@pytest.fixture(scope="module")
def lib():
    build()
    return binding.load()


def test_exports_every_declared_function(lib):
    names = binding.declared_functions()
    assert "noble_linear_fwd" in names and "noble_linear_bwd" in names
    for n in names:
        assert hasattr(lib, n), n


def test_status_strings(lib):
    for code in range(8):
        assert lib.noble_status_string(code)


def test_buffer_size_queries(lib):
    d = binding.make_desc(256, 128, 128, 16, "fp32")
    sb, wb = binding.noble_linear_saved_bytes(d), binding.noble_linear_bwd_workspace_bytes(d)
    assert sb >= 256 * 16 * (4 + 4 + 4)
    assert wb >= 256 * 16 * 4
    assert binding.noble_linear_saved_bytes(binding.make_desc(256, 128, 128, 0, "bf16")) == 0
    assert binding.noble_linear_bwd_workspace_bytes(binding.make_desc(0, 128, 128, 0, "bf16")) > 0
    # invalid descriptors report 0
    assert binding.noble_linear_saved_bytes(binding.make_desc(256, 128, 128, 24, "bf16")) == 0
    assert binding.noble_linear_bwd_workspace_bytes(binding.make_desc(256, 100, 128, 16, "bf16")) == 0


FAKE = 0x100000  # 16-byte aligned and never dereferenced: validation fails first


def _fwd(desc, **over):
    args = dict(x=FAKE, W=FAKE, bias=None, W_down=FAKE, omega1=FAKE, phi1=FAKE, M=FAKE,
                omega2=FAKE, phi2=FAKE, W_up=FAKE, y=FAKE, saved=FAKE,
                saved_bytes=1 << 40, stream=None)
    args.update(over)
    return binding.noble_linear_fwd(desc, **args)


@pytest.mark.parametrize("shape,code", [
    ((256, 128, 128, 24), 3),   # rank not supported
    ((256, 100, 128, 16), 3),   # d_in not a multiple of 8
    ((256, 128, 4, 16), 3),     # d_out below 8
    ((-1, 128, 128, 16), 1),    # negative T
])
def test_bad_shapes_rejected(lib, shape, code):
    with pytest.raises(binding.NobleError) as e:
        _fwd(binding.make_desc(*shape, "bf16"))
    assert e.value.status == code


def test_bad_pointers_rejected(lib):
    d = binding.make_desc(256, 128, 128, 16, "bf16")
    with pytest.raises(binding.NobleError) as e:
        _fwd(d, x=None)
    assert e.value.status == 1 and "x" in str(e.value)
    with pytest.raises(binding.NobleError) as e:
        _fwd(d, W_up=FAKE + 8)
    assert e.value.status == 2
    with pytest.raises(binding.NobleError) as e:
        _fwd(d, M=None)
    assert e.value.status == 1
    with pytest.raises(binding.NobleError) as e:
        _fwd(d, saved_bytes=16)
    assert e.value.status == 4
    bad = binding.make_desc(256, 128, 128, 16, "bf16")
    bad.flags = 0x100  # unknown flag bit
    with pytest.raises(binding.NobleError) as e:
        _fwd(bad)
    assert e.value.status == 3
    with pytest.raises(binding.NobleError) as e:
        binding._check(binding.load().noble_linear_fwd(None, *([None] * 12), 0, None))
    assert e.value.status == 1


def test_branch_pointers_optional_without_rank(lib):
    d = binding.make_desc(256, 128, 128, 0, "bf16")
    # valid arguments reach the device check; on a machine without a GPU that
    # is the first failure, on a GPU machine it is not reached here.
    import torch
    if torch.cuda.is_available():
        pytest.skip("device present")
    with pytest.raises(binding.NobleError) as e:
        _fwd(d, W_down=None, omega1=None, phi1=None, M=None, omega2=None, phi2=None,
             W_up=None, saved=None, saved_bytes=0)
    assert e.value.status == 7


def test_inference_flag(lib):
    # the tensor-core forward saves only c; the CUDA-core paths keep the full layout
    T, r = 256, 16
    full = binding.noble_linear_saved_bytes(binding.make_desc(T, 128, 128, r, "bf16"))
    inf = binding.noble_linear_saved_bytes(
        binding.make_desc(T, 128, 128, r, "bf16", binding.NOBLE_FLAG_INFERENCE))
    assert inf == T * r * 2 and full >= T * r * (4 + 4 + 2)
    simt = binding.make_desc(T, 128, 128, r, "bf16", binding.NOBLE_FLAG_INFERENCE | binding.NOBLE_FLAG_SIMT_ONLY)
    assert binding.noble_linear_saved_bytes(simt) == full
    f32 = binding.make_desc(T, 128, 128, r, "fp32", binding.NOBLE_FLAG_INFERENCE)
    assert binding.noble_linear_saved_bytes(f32) == binding.noble_linear_saved_bytes(
        binding.make_desc(T, 128, 128, r, "fp32"))
    # the backward of an inference descriptor is rejected before anything runs
    d = binding.make_desc(T, 128, 128, r, "bf16", binding.NOBLE_FLAG_INFERENCE)
    kw = dict(dy=FAKE, x=FAKE, W=FAKE, W_down=FAKE, omega1=FAKE, phi1=FAKE, M=FAKE, omega2=FAKE,
              phi2=FAKE, W_up=FAKE, saved=FAKE, saved_bytes=1 << 40, dx=FAKE, dW=FAKE, dbias=None,
              dW_down=FAKE, dM=FAKE, domega1=FAKE, dphi1=FAKE, domega2=FAKE, dphi2=FAKE,
              dW_up=FAKE, stream=None)
    with pytest.raises(binding.NobleError) as e:
        binding.noble_linear_bwd(d, workspace=FAKE, workspace_bytes=1 << 40, **kw)
    assert e.value.status == 1 and "inference" in str(e.value)
    with pytest.raises(binding.NobleError) as e:
        binding.noble_linear_bwd_noalloc(d, **kw)
    assert e.value.status == 1


def test_bwd_workspace_size_checked(lib):
    d = binding.make_desc(64, 128, 128, 16, "bf16")
    sb = binding.noble_linear_saved_bytes(d)
    wb = binding.noble_linear_bwd_workspace_bytes(d)
    kw = dict(dy=FAKE, x=FAKE, W=FAKE, W_down=FAKE, omega1=FAKE, phi1=FAKE, M=FAKE, omega2=FAKE,
              phi2=FAKE, W_up=FAKE, saved=FAKE, saved_bytes=sb, dx=FAKE, dW=FAKE, dbias=None,
              dW_down=FAKE, dM=FAKE, domega1=FAKE, dphi1=FAKE, domega2=FAKE, dphi2=FAKE,
              dW_up=FAKE, workspace=FAKE, workspace_bytes=wb - 1, stream=None)
    with pytest.raises(binding.NobleError) as e:
        binding.noble_linear_bwd(d, **kw)
    assert e.value.status == 4
    kw.update(workspace_bytes=wb, dM=None)
    with pytest.raises(binding.NobleError) as e:
        binding.noble_linear_bwd(d, **kw)
    assert e.value.status == 1 and "dM" in str(e.value)


def test_lr_multipliers_host(lib):
    from oracle import adamw
    for d_in, d_out, r in [(2048, 8192, 128), (1024, 1024, 64), (768, 3072, 16)]:
        got = binding.noble_linear_lr_multipliers(binding.make_desc(256, d_in, d_out, r, "bf16"))
        ref = adamw.lr_multipliers(d_in, d_out, r)
        assert got == pytest.approx([ref["W"], ref["W_up"], ref["M"], ref["omega"], ref["phi"]], rel=1e-6)
    with pytest.raises(binding.NobleError) as e:
        binding.noble_linear_lr_multipliers(binding.make_desc(256, 128, 128, 0, "bf16"))
    assert e.value.status == 1


def test_adamw_arguments_validated(lib):
    t = dict(param=FAKE, grad=FAKE, exp_avg=FAKE, exp_avg_sq=FAKE, n=64)
    with pytest.raises(binding.NobleError) as e:
        binding.noble_adamw_step([t], lr=1e-3, step=0)
    assert e.value.status == 1
    with pytest.raises(binding.NobleError) as e:
        binding.noble_adamw_step([dict(t, grad=None)], lr=1e-3)
    assert e.value.status == 1
    with pytest.raises(binding.NobleError) as e:
        binding.noble_adamw_step([dict(t, exp_avg=FAKE + 4)], lr=1e-3)
    assert e.value.status == 2
    with pytest.raises(binding.NobleError) as e:
        binding.noble_adamw_step([dict(t, param_bf16=FAKE + 2)], lr=1e-3)
    assert e.value.status == 2
    with pytest.raises(binding.NobleError) as e:
        binding.noble_adamw_step([t], lr=1e-3, beta2=1.0)
    assert e.value.status == 1


def test_activation_flags(lib):
    # ACT_* with the identity is rejected; the other combinations validate and
    # reach the device check (no GPU here), with the pointers a variant does
    # not read passed as NULL
    import torch
    bad = binding.make_desc(256, 128, 128, 16, "bf16",
                            binding.NOBLE_FLAG_ACT_GELU | binding.NOBLE_FLAG_SIGMA_IDENTITY)
    with pytest.raises(binding.NobleError) as e:
        _fwd(bad)
    assert e.value.status == 1
    if torch.cuda.is_available():
        pytest.skip("device present")
    for name, flags in binding.SIGMA_FLAGS.items():
        d = binding.make_desc(256, 128, 128, 16, "bf16", flags)
        unused = {k: None for k in binding.SIGMA_UNUSED[name]}
        with pytest.raises(binding.NobleError) as e:
            _fwd(d, **unused)
        assert e.value.status == 7, name
    # a two-layer variant needs M
    with pytest.raises(binding.NobleError) as e:
        _fwd(binding.make_desc(256, 128, 128, 16, "bf16", binding.NOBLE_FLAG_ACT_TANH), M=None)
    assert e.value.status == 1


def test_cos3_flag_validation(lib):
    # the three-layer flag excludes the other bottleneck flags; the plain entry
    # points refuse a three-layer descriptor (before any device check)
    for other in (binding.NOBLE_FLAG_SIGMA_COS1, binding.NOBLE_FLAG_SIGMA_IDENTITY, binding.NOBLE_FLAG_ACT_GELU):
        bad = binding.make_desc(256, 128, 128, 16, "bf16", binding.NOBLE_FLAG_SIGMA_COS3 | other)
        with pytest.raises(binding.NobleError) as e:
            _fwd(bad)
        assert e.value.status == 1
    three = binding.make_desc(256, 128, 128, 16, "bf16", binding.NOBLE_FLAG_SIGMA_COS3)
    with pytest.raises(binding.NobleError) as e:
        _fwd(three)
    assert e.value.status == 1 and "cos3" in str(e.value)
    # h, b, b2 (fp32) and c (bf16), each 256-byte aligned
    T, r = 256, 16
    assert binding.noble_linear_saved_bytes(three) == 3 * T * r * 4 + T * r * 2


@pytest.mark.parametrize("r", [16, 32, 64, 128, 256])
@pytest.mark.parametrize("T", [1, 300, 4096])
def test_saved_layout_sizes(lib, T, r):
    # the documented saved-buffer layouts: h, b (fp32) and c; c alone for an
    # inference forward on the tensor-core path; h, b, b2 and c for the
    # three-layer cosine; plus one ready flag per 128 tokens (whole row pairs)
    # when the fused bottleneck runs (CosNet, r in {64, 128})
    al = lambda n: (n + 255) // 256 * 256
    tr = T * r
    flags_bytes = al(2 * ((T + 255) // 256) * 4) if r in (64, 128) else 0
    B = binding
    size = lambda flags, dt="bf16": B.noble_linear_saved_bytes(B.make_desc(T, 128, 128, r, dt, flags))
    assert size(0) == al(tr * 4) * 2 + al(tr * 2)
    assert size(0, "fp32") == al(tr * 4) * 3
    assert size(B.NOBLE_FLAG_INFERENCE) == al(tr * 2)
    assert size(B.NOBLE_FLAG_INFERENCE | B.NOBLE_FLAG_SIMT_ONLY) == size(0)
    assert size(B.NOBLE_FLAG_SIGMA_COS3) == al(tr * 4) * 3 + al(tr * 2)
    assert size(B.NOBLE_FLAG_FUSED_BRANCH) == size(0) + flags_bytes
    assert size(B.NOBLE_FLAG_FUSED_BRANCH | B.NOBLE_FLAG_INFERENCE) == al(tr * 2) + flags_bytes
    # the fused bottleneck is the CosNet's only: other variants keep the plain layout
    assert size(B.NOBLE_FLAG_FUSED_BRANCH | B.NOBLE_FLAG_ACT_GELU) == size(0)
    for flags in (0, B.NOBLE_FLAG_SIGMA_COS1, B.NOBLE_FLAG_ACT_TANH, B.NOBLE_FLAG_SIGMA_COS3,
                  B.NOBLE_FLAG_FUSED_BRANCH, B.NOBLE_FLAG_SIMT_ONLY):
        assert B.noble_linear_bwd_workspace_bytes(B.make_desc(T, 128, 128, r, "bf16", flags)) > 0
