"""Host-side input recipe: the paper's GeGLU hidden width and workload shapes,
and reproducibility of the seeded generators (no GPU)."""
import numpy as np

from paper_2603_06492_gb300.inputs import (CONFIGS, PAPER_WORKLOADS, geglu_hidden, make_cos3_inputs,
                                           make_layer_inputs)


def test_geglu_hidden_width():
    # 8/3 d rounded up to a multiple of 64 (Section 4.1.1's GeGLU FFN)
    for d in (768, 1024, 2048, 4096):
        h = geglu_hidden(d)
        assert h % 64 == 0 and h >= 8 * d / 3 > h - 64
    assert geglu_hidden(1024) == 2752 and geglu_hidden(2048) == 5504


def test_paper_workloads():
    base, large = PAPER_WORKLOADS["geglu-base"], PAPER_WORKLOADS["geglu-large"]
    assert [(l.d_in, l.d_out) for l in base] == [(1024, 2752), (1024, 2752), (2752, 1024)]
    assert [(l.d_in, l.d_out) for l in large] == [(2048, 5504), (2048, 5504), (5504, 2048)]
    assert {l.T for l in base} == {8192} and {l.T for l in large} == {16384}
    assert {l.r for l in base} == {64} and {l.r for l in large} == {128}


def test_generators_are_seeded():
    layer = CONFIGS[0][0]
    a, b = make_layer_inputs(layer, 5), make_layer_inputs(layer, 5)
    assert a.keys() == b.keys() and all(np.array_equal(a[k], b[k]) for k in a)
    c = make_layer_inputs(layer, 6)
    assert not np.array_equal(a["x"], c["x"])
    p, q = make_cos3_inputs(16, 3), make_cos3_inputs(16, 3)
    assert all(np.array_equal(p[k], q[k]) for k in p)
    assert p["M2"].shape == (16, 16) and p["omega3"].min() >= 0.5 and p["omega3"].max() <= 2.0
