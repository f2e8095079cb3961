"""Pins that tie the fp64 oracle to what the paper and the mathematics fix.

Each check takes the oracle module as an argument so the same checks can run
against the real oracle (test_oracle_pins.py) and against copies with planted
mistakes (test_oracle_mutations.py).  No check re-types the oracle's own
formula: each uses brute force, a closed form, a library routine that the
special case reduces to, or an invariant of the method.
"""
from __future__ import annotations

import json
import math
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _golden():
    with open(os.path.join(GOLDEN, "paper_tables.json")) as f:
        return json.load(f)


def _rel(a, b):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def _int_grad(rng, m, n):
    return rng.integers(-3, 4, size=(m, n)).astype(np.float64)


# --------------------------------------------------------------------------
# Statistics (Algorithm 1, l_t / r_t lines; eq. dp_preconditioner)
# --------------------------------------------------------------------------

def check_row_col_brute_force(ref):
    """Row/column squared norms of an integer matrix against explicit loops
    (exact in fp64)."""
    rng = np.random.default_rng(11)
    m, n = 7, 5
    G = _int_grad(rng, m, n)
    rows = [0.0] * m
    cols = [0.0] * n
    for i in range(m):
        for j in range(n):
            rows[i] += G[i][j] ** 2
            cols[j] += G[i][j] ** 2
    s_row, s_col = ref.row_col_sq_norms(G)
    assert s_row.shape == (m,) and s_col.shape == (n,)
    assert np.array_equal(s_row, np.array(rows)), (s_row, rows)
    assert np.array_equal(s_col, np.array(cols)), (s_col, cols)


def check_ema_unrolled(ref):
    """Three steps of the statistics and momentum EMAs from zero state equal
    the unrolled geometric sums (mu = 1/2 and 1/4 keep fp64 exact)."""
    rng = np.random.default_rng(12)
    m, n = 6, 9
    Gs = [_int_grad(rng, m, n) for _ in range(3)]
    hp = ref.Hyper(lr=0.01, mu1=0.25, mu2=0.5)
    st = ref.State.zeros(m, n)
    W = np.zeros((m, n))
    for G in Gs:
        W, _ = ref.malt_step_ref(W, G, st, hp)
    s = [np.sum(G * G, axis=1) for G in Gs]
    c = [np.sum(G * G, axis=0) for G in Gs]
    l3 = 0.5 * (0.25 * s[0] + 0.5 * s[1] + s[2])
    r3 = 0.5 * (0.25 * c[0] + 0.5 * c[1] + c[2])
    M3 = 0.75 * (0.0625 * Gs[0] + 0.25 * Gs[1] + Gs[2])
    assert np.array_equal(st.l, l3)
    assert np.array_equal(st.r, r3)
    assert np.allclose(st.M, M3, rtol=0, atol=1e-15)
    assert st.t == 3


def check_preconditioner_root(ref):
    """L = (l + eps)^(-1/8): raising it to the -8th power gives l + eps back;
    l = 0 with eps = 1e-8 gives exactly 10; l + eps = 256 gives 1/2."""
    l = np.array([0.0, 256.0 - 1e-8, 3.7, 1e-3, 5e4])
    L = ref.diag_preconditioner(l, 1e-8)
    assert np.allclose(L ** -8, l + 1e-8, rtol=1e-12, atol=0)
    assert abs(L[0] - 10.0) < 1e-12
    assert abs(L[1] - 0.5) < 1e-12


def check_two_sided_entrywise(ref):
    """Diag(L) X Diag(R) against loops and against dense diagonal matmuls."""
    rng = np.random.default_rng(13)
    m, n = 5, 4
    X = rng.standard_normal((m, n))
    Ld = rng.uniform(0.5, 2, m)
    Rd = rng.uniform(0.5, 2, n)
    Y = ref.two_sided(Ld, X, Rd)
    for i in range(m):
        for j in range(n):
            assert abs(Y[i, j] - Ld[i] * X[i, j] * Rd[j]) < 1e-15
    assert np.allclose(Y, np.diag(Ld) @ X @ np.diag(Rd), rtol=1e-14, atol=0)


# --------------------------------------------------------------------------
# Orth (Section 3.1) and Newton-Schulz
# --------------------------------------------------------------------------

def check_ns_singular_value_map(ref):
    """Newton-Schulz acts on singular values only: NS_k(X) = U phi_k(S/nrm) V^T
    with phi_k the scalar quintic iterated k times, nrm = ||X||_F + ns_eps.
    Checked on wide and tall matrices, k = 5 and 8."""
    rng = np.random.default_rng(14)
    for shape in ((12, 20), (20, 12), (16, 16)):
        X = rng.standard_normal(shape)
        U, S, Vt = np.linalg.svd(X, full_matrices=False)
        for k in (5, 8):
            a, b, c = ref.DEFAULT_NS_COEFFS
            x = S / (math.sqrt(float(np.sum(S ** 2))) + ref.DEFAULT_NS_EPS)
            for _ in range(k):
                x = a * x + b * x ** 3 + c * x ** 5
            expect = (U * x[None, :]) @ Vt
            got = ref.newton_schulz(X, steps=k)
            assert got.shape == X.shape
            assert _rel(got, expect) < 1e-10, (shape, k, _rel(got, expect))


def check_ns_band(ref):
    """The singular values of the NS output lie in the band that the scalar
    map takes the normalised input range to."""
    rng = np.random.default_rng(15)
    X = rng.standard_normal((24, 40)) * np.exp(rng.standard_normal(40))[None, :]
    S_in = np.linalg.svd(X, compute_uv=False)
    xs = np.linspace(S_in.min(), S_in.max(), 20001) / np.linalg.norm(X)
    band = ref.ns_scalar_map(xs)
    S_out = np.linalg.svd(ref.newton_schulz(X), compute_uv=False)
    assert S_out.min() >= band.min() - 1e-9 and S_out.max() <= band.max() + 1e-9
    # the default quintic leaves the well-conditioned part near 1, not at 1
    assert 0.5 < np.median(S_out) < 1.3


def check_ns_scalar_map_closed_forms(ref):
    """The scalar map that Newton-Schulz applies to each normalised singular
    value, against facts fixed by the polynomial p(x) = a x + b x^3 + c x^5
    itself: p(0) = 0, p(1) = a + b + c, p is odd, p'(0) = a (so k steps scale
    tiny inputs by a^k); and k steps equal the k-fold composition p(p(...)),
    built as a polynomial by numpy.polynomial for k <= 2 and evaluated by its
    polyval k times for k <= 6 (library routines working from the coefficient
    vector), for the quintic, a second quintic and the cubic (1.5, -0.5, 0),
    whose fixed point is 1."""
    from numpy.polynomial import Polynomial
    from numpy.polynomial.polynomial import polyval
    for coeffs in (ref.DEFAULT_NS_COEFFS, (1.5, -0.5, 0.0), (2.0, -1.5, 0.5)):
        a, b, c = coeffs
        assert ref.ns_scalar_map(0.0, 1, coeffs) == 0.0
        assert abs(ref.ns_scalar_map(1.0, 1, coeffs) - (a + b + c)) < 1e-15
        xs = np.linspace(-1.2, 1.2, 241)
        assert np.allclose(ref.ns_scalar_map(-xs, 3, coeffs), -ref.ns_scalar_map(xs, 3, coeffs),
                           rtol=0, atol=1e-13)
        tiny = 1e-9
        for k in (1, 4):
            assert abs(ref.ns_scalar_map(tiny, k, coeffs) / tiny - a ** k) < 1e-6 * a ** k
        coef = [0.0, a, 0.0, b, 0.0, c]
        xs = np.linspace(0.0, 1.1, 111)
        # one and two steps: the composed polynomial itself (degree 5, 25)
        p = Polynomial(coef)
        assert np.allclose(ref.ns_scalar_map(xs, 1, coeffs), p(xs), rtol=1e-12, atol=1e-13)
        assert np.allclose(ref.ns_scalar_map(xs, 2, coeffs), p(p)(xs), rtol=1e-9, atol=1e-10)
        # more steps: the library's evaluation of p, applied k times
        y = xs.copy()
        for k in range(1, 7):
            y = polyval(y, coef)
            assert np.allclose(ref.ns_scalar_map(xs, k, coeffs), y, rtol=1e-12, atol=1e-13), (coeffs, k)
    assert ref.ns_scalar_map(1.0, 7, (1.5, -0.5, 0.0)) == 1.0


def check_cubic_ns_is_polar(ref):
    """With the cubic coefficients (1.5, -0.5, 0) and many steps Newton-Schulz
    converges to the polar factor U V^T (Section 3.1): compare with an SVD and
    with the defining properties O O^T = I and O^T X symmetric PSD."""
    rng = np.random.default_rng(16)
    U0, _ = np.linalg.qr(rng.standard_normal((16, 16)))
    V0, _ = np.linalg.qr(rng.standard_normal((24, 16)))
    X = U0 @ np.diag(np.linspace(1.0, 4.0, 16)) @ V0.T          # kappa = 4, 16 x 24
    O = ref.newton_schulz(X, steps=40, coeffs=(1.5, -0.5, 0.0), ns_eps=0.0)
    assert np.allclose(O @ O.T, np.eye(16), atol=1e-10)
    P = O.T @ X
    assert np.allclose(P, P.T, atol=1e-10)
    assert np.linalg.eigvalsh(0.5 * (P + P.T)).min() > -1e-10
    assert abs(np.linalg.norm(O) - 4.0) < 1e-10                 # sqrt(min(m, n))
    assert _rel(O, U0 @ V0.T) < 1e-10
    Oe = ref.orth_exact(X)
    assert _rel(Oe, U0 @ V0.T) < 1e-12
    assert _rel(ref.orth_exact(X.T), (U0 @ V0.T).T) < 1e-12


# --------------------------------------------------------------------------
# The whole step (Algorithm 1 / 2)
# --------------------------------------------------------------------------

def _phi(S, k, nrm, coeffs):
    a, b, c = coeffs
    x = S / nrm
    for _ in range(k):
        x = a * x + b * x ** 3 + c * x ** 5
    return x


def check_step_internals(ref):
    """One anisotropic MALT step on a square matrix, every intermediate
    recomputed independently: stats by loops, L/R by the -8th power relation,
    Mt and D entrywise, O by the singular-value map, the graft magnitude and
    the direction of W_t - W_{t-1}."""
    rng = np.random.default_rng(17)
    m = n = 9
    hp = ref.Hyper(lr=0.05)
    W0 = rng.standard_normal((m, n)) * 0.1
    G1 = rng.standard_normal((m, n)) * np.exp(rng.standard_normal(m))[:, None]
    G2 = rng.standard_normal((m, n)) * np.exp(2 * rng.standard_normal(n))[None, :]
    st = ref.State.zeros(m, n)
    W1, _ = ref.malt_step_ref(W0, G1, st, hp)
    W2, info = ref.malt_step_ref(W1, G2, st, hp)
    mu1, mu2, eps = hp.mu1, hp.mu2, hp.eps
    Mb = (1 - mu1) * (mu1 * G1 + G2)
    lb = np.array([(1 - mu2) * (mu2 * sum(G1[i, j] ** 2 for j in range(n))
                                + sum(G2[i, j] ** 2 for j in range(n))) for i in range(m)])
    rb = np.array([(1 - mu2) * (mu2 * sum(G1[i, j] ** 2 for i in range(m))
                                + sum(G2[i, j] ** 2 for i in range(m))) for j in range(n)])
    assert np.allclose(info["L"] ** -8 - eps, lb, rtol=1e-10, atol=0)
    assert np.allclose(info["R"] ** -8 - eps, rb, rtol=1e-10, atol=0)
    Lb, Rb = info["L"], info["R"]
    Mt = np.array([[Lb[i] * Mb[i, j] * Rb[j] for j in range(n)] for i in range(m)])
    assert _rel(info["Mt"], Mt) < 1e-12
    U, S, Vt = np.linalg.svd(Mt)
    O = (U * _phi(S, hp.ns_steps, np.linalg.norm(Mt) + hp.ns_eps, hp.ns_coeffs)[None, :]) @ Vt
    assert _rel(info["O"], O) < 1e-10
    D = np.array([[Lb[i] * O[i, j] * Rb[j] for j in range(n)] for i in range(m)])
    assert _rel(info["D"], D) < 1e-10
    step = W1 - W2
    want = hp.lr * np.linalg.norm(O) * np.linalg.norm(D) / (np.linalg.norm(D) + eps)
    assert abs(np.linalg.norm(step) - want) < 1e-10 * want
    cos = float(np.sum(step * D) / (np.linalg.norm(step) * np.linalg.norm(D)))
    assert cos > 1 - 1e-12


def check_muon_reduction(ref):
    """Gradients with +-1 entries have equal row norms and equal column norms,
    so L and R are multiples of I and the graft cancels them: MALT becomes
    Muon with EMA momentum, W <- W - lr * NS_k(M) (Section 3.4: the diagonal
    scaling only matters through row/column differences).  Compared with a
    Muon written here from the singular-value map."""
    rng = np.random.default_rng(18)
    m, n = 10, 14
    hp = ref.Hyper(lr=0.03)
    W = rng.standard_normal((m, n)) * 0.1
    Wm = W.copy()
    M = np.zeros((m, n))
    st = ref.State.zeros(m, n)
    for _ in range(3):
        G = rng.choice([-1.0, 1.0], size=(m, n))
        W, _ = ref.malt_step_ref(W, G, st, hp)
        M = hp.mu1 * M + (1 - hp.mu1) * G
        U, S, Vt = np.linalg.svd(M, full_matrices=False)
        Wm = Wm - hp.lr * (U * _phi(S, hp.ns_steps, np.linalg.norm(M), hp.ns_coeffs)[None, :]) @ Vt
    assert _rel(W, Wm) < 1e-6, _rel(W, Wm)


def check_transpose_equivariance(ref):
    """step(W^T, G^T) = step(W, G)^T for MALT and MALTER (the row and column
    statistics trade places; Orth commutes with transposition)."""
    rng = np.random.default_rng(19)
    m, n = 8, 13
    for variant in ("malt", "malter"):
        W = rng.standard_normal((m, n)) * 0.1
        Gs = [rng.standard_normal((m, n)) * np.exp(rng.standard_normal(m))[:, None] for _ in range(3)]
        Wa, _, _ = ref.run_steps(W, Gs, ref.Hyper(lr=0.02), variant=variant)
        Wb, _, _ = ref.run_steps(W.T, [G.T for G in Gs], ref.Hyper(lr=0.02), variant=variant)
        assert _rel(Wb.T, Wa) < 1e-12


def check_permutation_equivariance(ref):
    """Permuting rows and columns of W and G permutes the result the same way
    (the preconditioners are diagonal, Orth is equivariant under orthogonal
    maps as Section 3.4 states for the SOAP rotation)."""
    rng = np.random.default_rng(20)
    m, n = 7, 11
    pr, pc = rng.permutation(m), rng.permutation(n)
    W = rng.standard_normal((m, n)) * 0.1
    Gs = [rng.standard_normal((m, n)) * np.exp(rng.standard_normal(n))[None, :] for _ in range(2)]
    Wa, _, _ = ref.run_steps(W, Gs, ref.Hyper(), variant="malter")
    Wb, _, _ = ref.run_steps(W[pr][:, pc], [G[pr][:, pc] for G in Gs], ref.Hyper(), variant="malter")
    assert _rel(Wb, Wa[pr][:, pc]) < 1e-12


def check_gradient_scale_invariance(ref):
    """G -> 4G leaves the MALT and MALTER updates unchanged up to eps terms:
    L and R scale by 4^(-1/4), NS normalises its input and the graft (and
    alpha) are ratios."""
    rng = np.random.default_rng(21)
    m, n = 9, 6
    W = rng.standard_normal((m, n)) * 0.1
    Gs = [rng.standard_normal((m, n)) * np.exp(rng.standard_normal(m))[:, None] for _ in range(3)]
    for variant in ("malt", "malter"):
        Wa, _, _ = ref.run_steps(W, Gs, ref.Hyper(), variant=variant)
        Wb, _, _ = ref.run_steps(W, [4.0 * G for G in Gs], ref.Hyper(), variant=variant)
        assert _rel(Wb - W, Wa - W) < 1e-6


def check_malter_first_alpha(ref):
    """From zero state, alpha_1 = 1 up to eps terms: M_1 = (1-mu1) G_1 and
    nu_1 = (1-mu2) ||L G_1 R||^2, so both bias corrections cancel exactly."""
    rng = np.random.default_rng(22)
    G = rng.standard_normal((6, 10)) * np.exp(rng.standard_normal(10))[None, :]
    st = ref.State.zeros(6, 10)
    _, info = ref.malt_step_ref(np.zeros((6, 10)), G, st, ref.Hyper(), variant="malter")
    assert abs(info["alpha"] - 1.0) < 1e-6, info["alpha"]


def check_malter_pm1_closed_form(ref):
    """+-1 gradients make every MALTER quantity a scalar recurrence:
    l_t = n (1 - mu2^t), r_t = m (1 - mu2^t), ||L G R||^2 = L^2 R^2 m n,
    ||Mt|| = L R ||M||.  alpha_t from these scalars must equal the oracle's,
    and the step must be lr * alpha_t * NS_k(M) (the graft cancels L R)."""
    rng = np.random.default_rng(23)
    m, n = 5, 8
    hp = ref.Hyper(lr=0.01)
    st = ref.State.zeros(m, n)
    W = np.zeros((m, n))
    M = np.zeros((m, n))
    nu = 0.0
    for t in range(1, 5):
        G = rng.choice([-1.0, 1.0], size=(m, n))
        W_prev = W
        W, info = ref.malt_step_ref(W, G, st, hp, variant="malter")
        M = hp.mu1 * M + (1 - hp.mu1) * G
        Lt = (n * (1 - hp.mu2 ** t) + hp.eps) ** -0.125
        Rt = (m * (1 - hp.mu2 ** t) + hp.eps) ** -0.125
        nu = hp.mu2 * nu + (1 - hp.mu2) * Lt * Lt * Rt * Rt * m * n
        alpha = (math.sqrt(1 - hp.mu2 ** t) / (1 - hp.mu1 ** t + hp.eps)
                 * Lt * Rt * np.linalg.norm(M) / (math.sqrt(nu) + hp.eps))
        assert abs(info["nu"] - nu) < 1e-12 * nu
        assert abs(info["alpha"] - alpha) < 1e-10 * alpha, (t, info["alpha"], alpha)
        # L, R are scalars, so the grafted MALTER step is lr * alpha * NS_k(M)
        U, S, Vt = np.linalg.svd(M, full_matrices=False)
        O = (U * _phi(S, hp.ns_steps, np.linalg.norm(M), hp.ns_coeffs)[None, :]) @ Vt
        assert _rel(W_prev - W, hp.lr * alpha * O) < 1e-6


def check_zero_gradient(ref):
    """G = 0 at t = 1: Mt = 0, O = 0, the graft scale is 0, W is unchanged."""
    W = np.random.default_rng(24).standard_normal((4, 6))
    for variant in ("malt", "malter"):
        st = ref.State.zeros(4, 6)
        Wn, info = ref.malt_step_ref(W, np.zeros((4, 6)), st, ref.Hyper(), variant=variant)
        assert np.array_equal(Wn, W)
        assert not np.any(info["O"])


def check_decoupled_weight_decay(ref):
    """Weight decay in the decoupled form (reading: W <- (1 - lr wd) W before
    the update; the algorithms leave it out).  With G = 0 every step the
    direction is 0, so t steps shrink W geometrically: W_t = (1 - lr wd)^t W_0.
    With a gradient, the decay changes neither the statistics, the direction
    nor the graft scale, only W, and it acts on the weights the step starts
    from, not on the updated ones."""
    rng = np.random.default_rng(26)
    W0 = rng.standard_normal((8, 12))
    hp = ref.Hyper(lr=0.05, weight_decay=0.3)
    for variant in ("malt", "malter"):
        st = ref.State.zeros(8, 12)
        W = W0
        for _ in range(5):
            W, _ = ref.malt_step_ref(W, np.zeros((8, 12)), st, hp, variant=variant)
        assert _rel(W, (1.0 - 0.05 * 0.3) ** 5 * W0) < 1e-14
    G = rng.standard_normal((8, 12))
    a, b = ref.State.zeros(8, 12), ref.State.zeros(8, 12)
    Wa, ia = ref.malt_step_ref(W0, G, a, hp, variant="malter")
    Wb, ib = ref.malt_step_ref(W0, G, b, ref.Hyper(lr=0.05), variant="malter")
    for key in ("O", "D", "L", "R"):
        assert np.array_equal(ia[key], ib[key])
    assert ia["scale"] == ib["scale"] and a.nu == b.nu
    # Wb = W0 - delta; the decayed step removes the same delta from the shrunk W0
    assert _rel(Wa, (1.0 - 0.05 * 0.3) * W0 - (W0 - Wb)) < 1e-13


def check_bf16_rounding(ref):
    """Round-to-nearest-even to bf16 against torch's fp32 -> bf16 conversion
    (a library routine), on random values and on exact ties."""
    import torch
    rng = np.random.default_rng(25)
    x = (rng.standard_normal(20000) * np.exp(4 * rng.standard_normal(20000))).astype(np.float32)
    # exact ties: bf16 value plus half an ulp, for even and odd last bits
    base = (np.arange(1, 2001, dtype=np.uint32) << 16) | np.uint32(0x3F000000)
    ties = (base | np.uint32(0x8000)).view(np.float32)
    x = np.concatenate([x, ties, -ties, np.float32([0.0, 1e-40, -3e-39])])
    want = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    got = ref.round_to_bf16(x.astype(np.float64))
    assert np.array_equal(got, want)


def check_state_memory_matches_paper(ref):
    """Section 5.5: MALT's state exceeds Muon's by 1.50 MB on GPT-2 Medium
    (1554.88 vs 1553.38); MALTER adds one scalar per matrix and prints the
    same figure.  Recompute from the oracle's own state layout in fp32."""
    g = _golden()
    mem = g["state_memory_gpt2_medium_MB"]
    shapes = [tuple(s) for s in g["gpt2_medium_matrices"]["shapes"]] * g["gpt2_medium_matrices"]["layers"]
    extra_malt = sum(ref.state_floats(m, n, "malt") - m * n for m, n in shapes) * 4 / 2 ** 20
    extra_malter = sum(ref.state_floats(m, n, "malter") - m * n for m, n in shapes) * 4 / 2 ** 20
    assert abs(extra_malt - (mem["malt"] - mem["muon"])) < 0.005
    assert abs(extra_malter - (mem["malter"] - mem["muon"])) < 0.005


def check_defaults_match_paper(ref):
    """The oracle's default mu1, mu2, eps are the appendix table's."""
    hpg = _golden()["hyperparameters"]
    hp = ref.Hyper()
    assert (hp.mu1, hp.mu2, hp.eps) == (hpg["mu1"], hpg["mu2"], hpg["eps"])


ALL_CHECKS = [
    check_row_col_brute_force,
    check_ema_unrolled,
    check_preconditioner_root,
    check_two_sided_entrywise,
    check_ns_singular_value_map,
    check_ns_scalar_map_closed_forms,
    check_ns_band,
    check_cubic_ns_is_polar,
    check_step_internals,
    check_muon_reduction,
    check_transpose_equivariance,
    check_permutation_equivariance,
    check_gradient_scale_invariance,
    check_malter_first_alpha,
    check_malter_pm1_closed_form,
    check_zero_gradient,
    check_decoupled_weight_decay,
    check_bf16_rounding,
    check_state_memory_matches_paper,
    check_defaults_match_paper,
]
