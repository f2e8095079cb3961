"""The seeded synthetic workloads (CPU only): the GPT-2 parameter sets, the
single-matrix case and the stress set have the shapes, element counts,
dtypes, anisotropy, learning rates and step counts they stand for, and the
draws are reproducible and distributed as stated."""
import numpy as np
import pytest

from paper_2608_05088_gb300 import inputs

W = inputs.WORKLOADS


@pytest.mark.parametrize("name,layers,d,elements,variant,lr", [
    # learning rates: the paper's tuned values (Section 5.1 table) for the
    # optimizer each set runs with
    ("gpt2_small", 12, 768, 84_934_656, "malt", 0.0013),
    ("gpt2_medium", 24, 1024, 301_989_888, "malter", 0.009),
    ("gpt2_large", 36, 1280, 707_788_800, "malt", 0.0007),
])
def test_gpt2_parameter_sets(name, layers, d, elements, variant, lr):
    wl = W[name]
    assert len(wl.shapes) == 4 * layers
    per_layer = [(d, 3 * d), (d, d), (d, 4 * d), (4 * d, d)]   # c_attn, attn c_proj, c_fc, mlp c_proj
    assert list(wl.shapes) == per_layer * layers
    assert wl.elements == elements
    assert (wl.weight_dtype, wl.sigma, wl.variant, wl.lr, wl.steps, wl.ns_steps) == \
        ("bf16", 1.5, variant, lr, 10, 5)


def test_single_matrix_and_stress_set():
    wl = W["single_256x512"]
    assert (wl.shapes, wl.weight_dtype, wl.sigma, wl.lr, wl.variant, wl.steps, wl.ns_steps) == \
        (((256, 512),), "f32", 1.0, 0.02, "malt", 3, 5)
    seen = set()
    for rows, cols in ((4096, 4096), (4096, 16384), (16384, 4096)):
        for sigma in (0.0, 1.0, 3.0):
            for k in (5, 8):
                s = inputs.stress_workload(rows, cols, sigma, k)
                assert (s.shapes, s.weight_dtype, s.sigma, s.ns_steps, s.lr, s.steps) == \
                    (((rows, cols),), "bf16", sigma, k, 0.02, 3)
                seen.add(s.wid)
    assert len(seen) == 6          # one seed per (sigma, k), shared by the three shapes


def test_flop_counts_of_gpt2_large():
    wl = W["gpt2_large"]
    # dense 4 p^2 q + 2 p^3 and symmetric 3 p^2 q + p^3 per matrix and iteration
    assert wl.ns_flops_dense() == pytest.approx(21.139e12, rel=1e-4)
    assert wl.ns_flops_min() == pytest.approx(15.099e12, rel=1e-4)
    # 1280 = 5 tiles of 256: diagonal tiles are issued whole
    assert wl.ns_flops_min() < wl.ns_flops_issued() < wl.ns_flops_dense()


def test_draws_are_reproducible_and_independent():
    wl = W["gpt2_small"]
    g0 = inputs.gradient(wl, 3, 0)
    assert g0.dtype == np.float32 and g0.shape == wl.shapes[3]
    assert np.array_equal(g0, inputs.gradient(wl, 3, 0))
    g1 = inputs.gradient(wl, 3, 1)
    assert not np.array_equal(g0, g1)
    # same row / column scales every step: G / z differs between steps only by z
    a, b = inputs.row_col_scales(wl, 3)
    assert np.array_equal(a, inputs.row_col_scales(wl, 3)[0])
    assert not np.array_equal(a, inputs.row_col_scales(wl, 4)[0][: a.size])
    # another matrix of the same shape draws other values
    assert not np.array_equal(inputs.gradient(wl, 7, 0), g0)
    # the first layers of a set draw exactly what the full set draws
    part = inputs.first_layers(wl, 2)
    for i in range(len(part.shapes)):
        assert np.array_equal(inputs.gradient(part, i, 2), inputs.gradient(wl, i, 2))
        assert np.array_equal(inputs.initial_weight(part, i), inputs.initial_weight(wl, i))
    par = inputs.gradients_for_step(part, 1, workers=3)
    for i, g in enumerate(par):
        assert np.array_equal(g, inputs.gradient(part, i, 1))


def test_distributions():
    wl = W["gpt2_medium"]            # sigma 1.5, bf16 weights
    idx = 2                          # 1024 x 4096
    a, b = inputs.row_col_scales(wl, idx)
    for s in (a, b):
        assert s.min() > 0
        assert abs(np.log(s).std() - 1.5) < 0.15
        assert abs(np.log(s).mean()) < 0.15
    g = inputs.gradient(wl, idx, 0)
    z = g / a[:, None] / b[None, :]
    assert abs(z.mean()) < 0.01 and abs(z.std() - 1.0) < 0.01
    w = inputs.initial_weight(wl, idx)
    assert w.dtype == np.float32 and abs(w.std() - 0.02) < 2e-4
    # bf16 weights: every value has a zero low half (exactly representable)
    assert not np.any(w.view(np.uint32) & 0xFFFF)
    w32 = inputs.initial_weight(W["single_256x512"], 0)
    assert np.any(w32.view(np.uint32) & 0xFFFF)   # fp32 weights are not rounded


def test_bf16_representable_is_nearest_even():
    x = np.array([1.0, 1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, 1.0 + 2.0 ** -9, -2.5,
                  1.0 + 2.0 ** -8 + 2.0 ** -20], dtype=np.float32)
    want = np.array([1.0, 1.0, 1.0 + 2.0 ** -6, 1.0, -2.5, 1.0 + 2.0 ** -7], dtype=np.float32)
    # ties go to the even mantissa; above a tie rounds up
    assert np.array_equal(inputs.bf16_representable(x), want)


def test_random_shapes():
    s = inputs.random_shapes(3, 10)
    assert s == inputs.random_shapes(3, 10)
    assert len(s) == 10 and s[-1] == s[0][::-1]
    assert all(r % 8 == 0 and c % 8 == 0 and 8 <= r <= 776 and 8 <= c <= 776 for r, c in s)
    big = inputs.random_shapes(11, 5, max_dim=2056)
    assert all(8 <= r <= 2056 and 8 <= c <= 2056 for r, c in big)


def test_gpt2_whole_parameter_counts_match_the_paper():
    """The 2-D matrices MALT updates plus the tensors AdamW updates add up to
    the model sizes Section 5.1 states: GPT-2 Small 124M, Medium 355M, Large
    774M parameters (NanoGPT's padded vocabulary, tied head)."""
    for name, millions in (("gpt2_small", 124), ("gpt2_medium", 355), ("gpt2_large", 774)):
        total = inputs.WORKLOADS[name].elements + inputs.ADAMW_SETS[name].elements
        assert round(total / 1e6) == millions, (name, total)


def test_adamw_set_recipe():
    aset = inputs.ADAMW_SETS["gpt2_small"]
    names = [t[0] for t in aset.tensors]
    assert names[:2] == ["wte", "wpe"] and len(names) == 2 + 8 * 12 + 2
    assert all(wd == (0.1 if len(shape) == 2 else 0.0) for _, shape, wd in aset.tensors)
    assert aset.lr == 0.0013 and inputs.ADAMW_SETS["gpt2_large"].lr == 0.0009
    w = inputs.adamw_initial(aset, 0)
    assert w.dtype == np.float32 and w.shape == (50304, 768) and abs(w.std() - 0.02) < 1e-3
    assert np.all(inputs.adamw_initial(aset, names.index("h0.ln_1.weight")) == 1.0)
    assert not np.any(inputs.adamw_initial(aset, names.index("h0.mlp.c_fc.bias")))
    g0 = inputs.adamw_gradient(aset, 5, 0)
    assert np.array_equal(g0, inputs.adamw_gradient(aset, 5, 0))
    assert not np.array_equal(g0, inputs.adamw_gradient(aset, 5, 1))
