"""CUDA path vs the fp64 oracle, element by element, on seeded inputs.

Bars: momentum / statistics / ||Mt|| within 1e-5 relative (fp32 arithmetic);
orthogonalised direction O and the grafting norms within 2e-2 relative
Frobenius (bf16 Newton-Schulz operands with fp32 accumulation); final weights
within 5e-3 relative Frobenius and the update within 2e-2; bf16 weights
within |x_gpu - x_oracle| + 1 ulp of the oracle's round-to-nearest-even
result (x the pre-rounding values) and equal to the rounding of the GPU's own
pre-rounding value.
"""
import numpy as np
import pytest

from paper_2608_05088_gb300 import inputs
from tests.gpu_harness import Run, bf16_rounding

pytestmark = pytest.mark.gpu


def test_single_256x512_malt():
    """The 256 x 512 fp32 matrix, 3 MALT steps, checked after every step."""
    wl = inputs.WORKLOADS["single_256x512"]
    run = Run(wl)
    for s in range(wl.steps):
        run.step()
        assert run.status() == 0
        run.assert_close(0, f"step {s}")
    run.close()


RAGGED = ((200, 328), (392, 136), (8, 8), (136, 1000), (520, 520), (64, 2056), (1032, 264),
          (256, 512))


@pytest.mark.parametrize("variant", ["malt", "malter"])
def test_ragged_mixed_shapes(variant):
    """Shapes that leave ragged tiles in every direction, tall matrices (NS on
    the transpose), several shape classes in one grouped launch, fp32 and bf16
    weights side by side."""
    wl = inputs.Workload("ragged", 31, RAGGED, "f32", 1.5, 0.02, variant, 3)
    w_dtypes = ["f32", "bf16"] * (len(RAGGED) // 2)
    run = Run(wl, w_dtypes=w_dtypes)
    for s in range(wl.steps):
        run.step()
        assert run.status() == 0
        for i in range(len(RAGGED)):
            run.assert_close(i, f"{variant} step {s}")
    run.close()


@pytest.mark.parametrize("seed,variant", [(1, "malt"), (2, "malter"), (3, "malt")])
def test_seeded_random_shapes(seed, variant):
    """Ten seeded random shapes (multiples of 8 up to 776: wide, tall and
    square, every tile edge ragged), fp32 and bf16 weights side by side,
    2 steps, every matrix checked against the oracle."""
    shapes = inputs.random_shapes(seed, 10)
    wl = inputs.Workload(f"random{seed}", 40 + seed, shapes, "f32", 1.5, 0.02, variant, 2)
    run = Run(wl, w_dtypes=["f32", "bf16"] * 5)
    for s in range(wl.steps):
        run.step()
        assert run.status() == 0
    for i in range(len(shapes)):
        run.assert_close(i, f"seed {seed} {variant}")
    run.close()


@pytest.mark.parametrize("seed", [11, 12])
def test_seeded_random_large_shapes(seed):
    """Five seeded random shapes up to 2056 (up to 9 x 9 GEMM tiles, ragged),
    bf16 weights, one MALTER step, checked in full against the oracle."""
    shapes = inputs.random_shapes(seed, 5, max_dim=2056)
    wl = inputs.Workload(f"random{seed}", 40 + seed, shapes, "bf16", 1.5, 0.02, "malter", 1)
    run = Run(wl)
    run.step()
    assert run.status() == 0
    for i in range(len(shapes)):
        run.assert_close(i, f"seed {seed}")
    run.close()


def test_bf16_gradients_and_k8():
    """bf16 gradients, 8 Newton-Schulz iterations, strong anisotropy (sigma 3)."""
    wl = inputs.Workload("bf16g", 32, ((512, 768), (768, 256)), "bf16", 3.0, 0.02, "malt", 3,
                         ns_steps=8)
    run = Run(wl, g_dtype="bf16")
    for _ in range(wl.steps):
        run.step()
    assert run.status() == 0
    for i in range(2):
        run.assert_close(i)
    run.close()


def test_zero_gradient_leaves_weights():
    """G = 0 at t = 1: Mt = 0, O = 0, the grafted scale is 0, W is unchanged."""
    wl = inputs.Workload("zero", 33, ((128, 256), (264, 136)), "f32", 1.0, 0.02, "malter", 1)
    run = Run(wl)
    W0 = [run.host(w).copy() for w in run.W]
    run.step(grads=[np.zeros(s, np.float32) for s in wl.shapes])
    assert run.status() == 0
    for i in range(2):
        assert np.array_equal(run.host(run.W[i]), W0[i])
        assert not np.any(run.host(run.opt.direction(i)))
    run.close()


def test_bitwise_deterministic():
    """Two identical runs give bitwise identical W, M, l, r (no atomics)."""
    wl = inputs.Workload("det", 34, RAGGED[:5], "bf16", 1.5, 0.02, "malter", 2)
    outs = []
    for _ in range(2):
        run = Run(wl, check=[])
        for _ in range(wl.steps):
            run.step(oracle=False)
        assert run.status() == 0
        outs.append([run.host(t) for t in run.W + run.M + run.l + run.r])
        run.close()
    for a, b in zip(*outs):
        assert np.array_equal(a, b)


def test_checkpoint_roundtrip():
    """3 steps straight == 1 step, save (M, l, r, nu, t), fresh state, restore,
    2 more steps; bitwise."""
    import torch
    wl = inputs.Workload("ckpt", 35, ((256, 384), (392, 136)), "f32", 1.5, 0.02, "malter", 3)
    a = Run(wl, check=[])
    for _ in range(3):
        a.step(oracle=False)
    b = Run(wl, check=[])
    b.step(oracle=False)
    nu, t = b.opt.scalars()
    assert t == 1
    saved = [[x.clone() for x in (b.W[i], b.M[i], b.l[i], b.r[i])] for i in range(2)]
    b.close()
    c = Run(wl, check=[])
    for i in range(2):
        for dst, src in zip((c.W[i], c.M[i], c.l[i], c.r[i]), saved[i]):
            dst.copy_(src)
    c.opt.set_scalars(nu, t)
    c.steps_done = 1
    for _ in range(2):
        c.step(oracle=False)
    torch.cuda.synchronize()
    for i in range(2):
        for x, y in zip((a.W[i], a.M[i], a.l[i], a.r[i]), (c.W[i], c.M[i], c.l[i], c.r[i])):
            assert torch.equal(x, y)
    nu_a, t_a = a.opt.scalars()
    nu_c, t_c = c.opt.scalars()
    assert t_a == t_c == 3 and np.array_equal(nu_a, nu_c)
    a.close()
    c.close()


def test_gpt2_small_sampled():
    """GPT-2 Small 2-D parameter set (48 matrices, bf16 W), 2 MALT steps in one
    grouped step; one matrix of each shape checked in full against the oracle."""
    wl = inputs.WORKLOADS["gpt2_small"]
    check = [0, 1, 2, 3, 45, 46, 47]
    run = Run(wl, check=check)
    for _ in range(2):
        run.step()
    assert run.status() == 0
    for i in check:
        run.assert_close(i)
    run.close()


def test_gpt2_medium_malter_sampled():
    """GPT-2 Medium (96 matrices), 2 MALTER steps, one matrix per shape checked."""
    wl = inputs.WORKLOADS["gpt2_medium"]
    check = [4, 5, 6, 7]
    run = Run(wl, check=check)
    for _ in range(2):
        run.step()
    assert run.status() == 0
    for i in check:
        run.assert_close(i)
    run.close()


def test_gpt2_large_bench_configuration():
    """The benchmark's own configuration: all 144 GPT-2 Large matrices in one
    grouped step (bf16 W, fp32 state, 5 NS iterations), 2 MALT steps.

    * Ten matrices, every shape of the first, a middle and the last layer
      (the first and last entries of the launch's work lists), are checked in
      full against the oracle.
    * Every matrix's statistics l, r against fp64 row / column sums of its
      gradients.
    * Every matrix's graft and update against the step's own intermediates
      (properties that hold at any size): ||O||_F and ||D||_F = ||L O R||_F
      from the last GEMM epilogue's partial sums against fp64 norms of the
      step's O, L, R (Algorithm 1, graft line), and the stored bf16 W against
      the round-to-nearest-even of W_prev - s L O R with the step's scale s
      (Algorithm 1, update line)."""
    import torch
    wl = inputs.WORKLOADS["gpt2_large"]
    check = [0, 1, 2, 3, 69, 70, 140, 141, 142, 143]
    run = Run(wl, check=check)
    sq_rows = {}
    sq_cols = {}
    mu2 = run.hp_ref.mu2
    for s in range(2):
        grads = inputs.gradients_for_step(wl, s)
        for i, G in enumerate(grads):
            G64 = G.astype(np.float64)
            r_, c_ = np.sum(G64 * G64, axis=1), np.sum(G64 * G64, axis=0)
            sq_rows[i] = mu2 * sq_rows.get(i, 0.0) + (1 - mu2) * r_
            sq_cols[i] = mu2 * sq_cols.get(i, 0.0) + (1 - mu2) * c_
        if s == 1:
            w_prev = [w.cpu() for w in run.W]
        run.step(grads=grads)
    assert run.status() == 0
    for i in check:
        run.assert_close(i)
    scalars = run.opt.debug_scalars()
    for i in range(len(wl.shapes)):
        l_gpu = run.host(run.l[i])
        r_gpu = run.host(run.r[i])
        assert np.max(np.abs(l_gpu - sq_rows[i]) / sq_rows[i]) < 1e-5, i
        assert np.max(np.abs(r_gpu - sq_cols[i]) / sq_cols[i]) < 1e-5, i
        W = run.host(run.W[i])
        assert np.all(np.isfinite(W))
        O = run.host(run.opt.direction(i))
        Lg, Rg = (run.host(t) for t in run.opt.precond(i))
        D = Lg[:, None] * O * Rg[None, :]
        nO, nD = np.linalg.norm(O), np.linalg.norm(D)
        sc = scalars[i]
        assert abs(sc[0] - nO) / nO < 1e-4 and abs(sc[1] - nD) / nD < 1e-4, (i, sc[:2], nO, nD)
        dW = float(sc[6]) * D
        W_pre = run.decay_gpu * w_prev[i].to(torch.float64).numpy() - dW
        e = bf16_rounding(W, W_pre, W_pre, 2.0 ** -21 * (np.abs(W_pre) + np.abs(dW)), dW)
        assert e["own_mismatch"] == 0, (i, e)
    run.close()


@pytest.mark.parametrize("rows,cols,sigma,ns_steps", [(4096, 4096, 3.0, 8), (4096, 16384, 1.0, 5),
                                                      (16384, 4096, 0.0, 5)])
def test_stress_shapes(rows, cols, sigma, ns_steps):
    """Largest single matrices of the stress set (bf16 W, fp32 state), one
    MALT step each, checked in full against the oracle."""
    wl = inputs.stress_workload(rows, cols, sigma, ns_steps)
    run = Run(wl)
    run.step()
    assert run.status() == 0
    run.assert_close(0, f"stress {rows}x{cols} sigma={sigma} k={ns_steps}")
    run.close()


def test_muon_through_the_same_engine():
    """muon_step = the engine with identity preconditioners, against the
    oracle's identity-preconditioner MALT step (plain Muon with the EMA
    momentum, Section 3.1); l and r stay untouched."""
    wl = inputs.Workload("muon", 36, RAGGED[:6], "f32", 1.5, 0.02, "muon", 3)
    run = Run(wl, w_dtypes=["f32", "bf16"] * 3)
    for s in range(wl.steps):
        run.step()
        assert run.status() == 0
        for i in range(len(wl.shapes)):
            run.assert_close(i, f"muon step {s}")
            assert not np.any(run.host(run.l[i])) and not np.any(run.host(run.r[i]))
    run.close()


@pytest.mark.parametrize("variant", ["malt", "malter"])
@pytest.mark.parametrize("hyper", [
    dict(weight_decay=0.1),                       # decoupled weight decay (reading 7)
    dict(mu1=0.0, mu2=0.0),                       # no momentum, statistics of this G only
    dict(eps=1e-3),                               # damping that dominates small rows
    dict(mu1=0.9, mu2=0.999, ns_eps=1e-5),
], ids=["wd0.1", "mu0", "eps1e-3", "mu0.9_0.999"])
def test_hyperparameter_variants(variant, hyper):
    """Non-default hyperparameters reach every kernel the same way they reach
    the oracle (f32 and bf16 weights, 3 steps)."""
    wl = inputs.Workload("hyper", 37, ((256, 512), (392, 136)), "f32", 1.5, 0.05, variant, 3)
    run = Run(wl, w_dtypes=["f32", "bf16"], **hyper)
    for s in range(wl.steps):
        run.step()
        assert run.status() == 0
        for i in range(2):
            run.assert_close(i, f"{hyper} step {s}")
    run.close()


@pytest.mark.parametrize("ns_steps,coeffs", [(1, (3.4445, -4.7750, 2.0315)),
                                             (12, (1.5, -0.5, 0.0))])
def test_newton_schulz_settings(ns_steps, coeffs):
    """One quintic iteration, and twelve iterations of the cubic polynomial
    (1.5, -0.5, 0), through the whole step."""
    wl = inputs.Workload("nsset", 38, ((256, 512), (392, 136)), "f32", 1.0, 0.02, "malt", 2,
                         ns_steps=ns_steps)
    run = Run(wl, ns_coeffs=coeffs)
    for _ in range(wl.steps):
        run.step()
    assert run.status() == 0
    for i in range(2):
        run.assert_close(i)
    run.close()


UNALIGNED = ((1, 1), (7, 13), (13, 7), (100, 3), (3, 1000), (255, 511), (1001, 999), (250, 509),
             (256, 512))


@pytest.mark.parametrize("variant,g_dtype", [("malt", "f32"), ("malter", "bf16"), ("muon", "f32")])
def test_unaligned_shapes(variant, g_dtype):
    """Rows and cols that are not multiples of 8 (a 1 x 1 matrix, odd and
    prime sizes, wide and tall): such a matrix runs on zero-padded copies.
    250 x 509 shares its padded frame (256 x 512) with an aligned matrix.
    fp32 and bf16 weights, 3 steps, every matrix checked against the oracle."""
    wl = inputs.Workload("unaligned", 46, UNALIGNED, "f32", 1.5, 0.02, variant, 3)
    run = Run(wl, w_dtypes=["f32", "bf16", "bf16", "f32", "f32", "bf16", "f32", "bf16", "f32"],
              g_dtype=g_dtype)
    for s_ in range(wl.steps):
        run.step()
        assert run.status() == 0
        for i in range(len(UNALIGNED)):
            run.assert_close(i, f"{variant} step {s_}")
    run.close()


@pytest.mark.parametrize("seed", [21, 22])
def test_seeded_random_odd_shapes(seed):
    """Ten seeded random shapes of any size up to 517 (most not multiples of
    8), fp32 and bf16 weights, 2 MALTER steps, every matrix against the oracle."""
    shapes = inputs.random_shapes(seed, 10, max_dim=517, multiple=1)
    wl = inputs.Workload(f"odd{seed}", 47 + seed, shapes, "f32", 1.5, 0.02, "malter", 2)
    run = Run(wl, w_dtypes=["f32", "bf16"] * 5)
    for _ in range(wl.steps):
        run.step()
        assert run.status() == 0
    for i in range(len(shapes)):
        run.assert_close(i, f"seed {seed}")
    run.close()
