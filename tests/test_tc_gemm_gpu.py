"""The tensor-core GEMM on its own, through the noble_test_gemm_bf16 hook,
against an fp64 product of the same bf16 values: every operand layout the
layer uses, both K segments, split-K, ragged M/N/K and the N tiles 16..256."""
import numpy as np
import pytest

from paper_2603_06492_gb300 import binding
from paper_2603_06492_gb300.inputs import round_bf16

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2603_06492_gb300.build import build
    build()
    binding.load()


def _dev(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16).cuda()


def run_case(M, N, K0, K1, a_mn, b_mn, bn, c_fp32, bias=False, kb_per_split=0, seed=0):
    import torch
    rng = np.random.default_rng(seed)
    A0 = round_bf16(rng.standard_normal((M, K0)))
    B0 = round_bf16(rng.standard_normal((N, K0)))
    A1 = round_bf16(rng.standard_normal((M, K1))) if K1 else None
    B1 = round_bf16(rng.standard_normal((N, K1))) if K1 else None
    bvec = rng.standard_normal(N).astype(np.float32) if bias else None
    nsplit = 1
    kb_total = -(-K0 // 64) + (-(-K1 // 64) if K1 else 0)
    if kb_per_split:
        nsplit = -(-kb_total // kb_per_split)
    lay_a = (lambda a: a.T) if a_mn else (lambda a: a)
    lay_b = (lambda b: b.T) if b_mn else (lambda b: b)
    dA0, dB0 = _dev(lay_a(A0)), _dev(lay_b(B0))
    dA1 = _dev(lay_a(A1)) if K1 else None
    dB1 = _dev(lay_b(B1)) if K1 else None
    dbias = torch.from_numpy(bvec).cuda() if bias else None
    C = torch.full((nsplit, M, N), float("nan"), dtype=torch.float32 if c_fp32 else torch.bfloat16,
                   device="cuda")
    binding.noble_test_gemm_bf16(M, N, K0, K1, a_mn, b_mn, bn, dA0, dB0, dA1, dB1, dbias, C,
                                 c_fp32, kb_per_split, nsplit, None)
    torch.cuda.synchronize()
    binding.noble_get_device_status(None)
    got = C.float().cpu().numpy().astype(np.float64)
    if kb_per_split:
        # reference per split: k-blocks of 64 over the concatenated K axis
        Acat = np.concatenate([A0, A1], 1) if K1 else A0
        Bcat = np.concatenate([B0, B1], 1) if K1 else B0
        kidx = np.concatenate([np.arange(K0), np.arange(K1) + 64 * -(-K0 // 64)]) if K1 else np.arange(K0)
        refs = []
        for z in range(nsplit):
            sel = (kidx >= z * kb_per_split * 64) & (kidx < (z + 1) * kb_per_split * 64)
            refs.append(Acat[:, sel] @ Bcat[:, sel].T)
        ref = np.stack(refs)
    else:
        ref = A0 @ B0.T + (A1 @ B1.T if K1 else 0) + (bvec if bias else 0)
        ref = ref[None]
    err = np.max(np.abs(got - ref)) / np.max(np.abs(ref))
    tol = 1e-5 if c_fp32 else 8e-3
    assert err < tol, (err, M, N, K0, K1, a_mn, b_mn, bn)


@pytest.mark.parametrize("bn", [16, 32, 64, 128, 256])
def test_kmajor_both(bn):
    run_case(300, bn * 2 + 8 if bn < 256 else 264, 200, 0, 0, 0, bn, 1)


def test_kmajor_two_segments_bias_bf16():
    run_case(300, 264, 200, 16, 0, 0, 256, 0, bias=True)
    run_case(129, 520, 136, 128, 0, 0, 256, 0, bias=True, seed=1)


def test_kmajor_a_mnmajor_b_two_segments():
    run_case(300, 264, 200, 32, 0, 1, 256, 0)
    run_case(256, 512, 1024, 64, 0, 1, 256, 1, seed=2)


@pytest.mark.parametrize("bn", [64, 128, 256])
def test_mnmajor_both(bn):
    run_case(200, 264 if bn == 256 else bn, 333 - 333 % 8, 0, 1, 1, bn, 1)


def test_mnmajor_small_rank_columns():
    # N = r < 64 inside a 64-wide tile (dW_up with r = 16), M = r < 128 (dW_down)
    run_case(264, 16, 512, 0, 1, 1, 64, 1)
    run_case(16, 264, 512, 0, 1, 1, 256, 1)


def test_split_k():
    run_case(128, 128, 1024, 0, 1, 1, 128, 1, kb_per_split=3)


def test_large_square():
    run_case(1024, 1024, 2048, 0, 0, 0, 256, 1, seed=5)


@pytest.mark.parametrize("amn,bmn,cf", [(0, 1, 0), (1, 1, 1), (1, 1, 0)])
def test_mnmajor_tiled_layout(amn, bmn, cf):
    # extents that tile by 64 (MN) and 8 (K): MN-major operands use the 4-D
    # TMA layout with interleaved 64-wide chunks
    run_case(384, 512, 1032, 0, amn, bmn, 256, cf, seed=11)
    run_case(256, 128, 520, 0, amn, bmn, 128, cf, seed=12)


def test_mnmajor_tiled_two_segments():
    run_case(256, 512, 1024, 128, 0, 1, 256, 0, seed=13)
