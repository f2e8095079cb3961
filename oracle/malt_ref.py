"""Reference (oracle) implementation of the MALT / MALTER per-matrix update.

TEST INFRASTRUCTURE ONLY.  This module is a plain, slow, fp64 NumPy restatement
of the paper's update and exists to check the CUDA library against.  Only the
test suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py``
may import it; the library itself never does, and it imports nothing from the
library.

What it computes (paper: "MALT: Lightweight Curvature-Aware Muon via Diagonal
Preconditioning"):

* Algorithm 1 (MALT update) for one m x n matrix, step by step:
  momentum EMA, row/column squared-norm EMAs (eq. dp_preconditioner), the
  diagonal preconditioners L = Diag((l+eps)^(-1/8)), R = Diag((r+eps)^(-1/8)),
  the preconditioned momentum Mt = L M R, O = Orth(Mt), the back-map
  D = L O R and the norm-grafted update W <- W - lr * ||O||_F/(||D||_F+eps) * D.
* Algorithm 2 (MALTER) adds the scalar nu <- mu2 nu + (1-mu2) ||L G R||_F^2 and
  the adaptive factor alpha_t of Section 3.5 (the displayed equation with no
  learning rate in it), and updates W <- W - lr * alpha * ||O||/(||D||+eps) * D.
* Orth (Section 3.1, eq. muon-update) is either the exact polar factor U V^T
  from an SVD, or the quintic Newton-Schulz iteration the paper names but does
  not spell out (readings below).

Readings of points the paper leaves open:

1. Newton-Schulz: X <- X / (||X||_F + ns_eps); k times A = X X^T,
   B = b A + c A A, X <- a X + B X; done on the transpose when m > n.
   Default (a, b, c) = (3.4445, -4.7750, 2.0315), k = 5, ns_eps = 1e-7.
2. alpha_t carries no learning rate; the learning rate appears once, in the
   W update (Algorithm 2 would otherwise apply it twice).
3. One epsilon everywhere (preconditioner damping, graft denominator,
   bias-correction and sqrt(nu) guards); default 1e-8 (appendix table).
4. t is 1-based; bias corrections use the incremented t.
5. Optional decoupled weight decay W <- (1 - lr*wd) W before the update
   (the appendix table lists 0.1, the algorithms do not); default 0.
6. bf16 weights are rounded once per step, round-to-nearest-even.

Every function below cites the passage it follows.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

# Appendix C hyperparameter table: (mu1, mu2) = (0.95, 0.99), eps = 1e-8.
DEFAULT_MU1 = 0.95
DEFAULT_MU2 = 0.99
DEFAULT_EPS = 1e-8
# Reading 1: the quintic Newton-Schulz coefficients commonly used with Muon.
DEFAULT_NS_COEFFS = (3.4445, -4.7750, 2.0315)
DEFAULT_NS_STEPS = 5
DEFAULT_NS_EPS = 1e-7
# Eq. dp_preconditioner: the inverse eighth root taken from Shampoo.
PRECOND_EXPONENT = -1.0 / 8.0


@dataclasses.dataclass
class Hyper:
    """Hyperparameters of Algorithms 1 and 2 (their Require lines) plus the
    Newton-Schulz settings the paper leaves unspecified."""
    lr: float = 0.02
    mu1: float = DEFAULT_MU1
    mu2: float = DEFAULT_MU2
    eps: float = DEFAULT_EPS
    weight_decay: float = 0.0
    ns_steps: int = DEFAULT_NS_STEPS
    ns_coeffs: tuple = DEFAULT_NS_COEFFS
    ns_eps: float = DEFAULT_NS_EPS


@dataclasses.dataclass
class State:
    """Per-matrix optimizer state (Algorithm 1 INITIALIZE line; Algorithm 2
    adds nu_0 = 0).  M is m x n, l has m entries, r has n entries."""
    M: np.ndarray
    l: np.ndarray
    r: np.ndarray
    nu: float = 0.0
    t: int = 0

    @staticmethod
    def zeros(m: int, n: int) -> "State":
        return State(np.zeros((m, n)), np.zeros(m), np.zeros(n), 0.0, 0)

    def copy(self) -> "State":
        return State(self.M.copy(), self.l.copy(), self.r.copy(), self.nu, self.t)


# ---------------------------------------------------------------------------
# Statistics and preconditioners
# ---------------------------------------------------------------------------

def row_col_sq_norms(G: np.ndarray):
    """Squared Euclidean norm of every row and every column of G
    (Algorithm 1, the l_t and r_t lines; eq. dp_preconditioner)."""
    G = np.asarray(G, dtype=np.float64)
    return np.sum(G * G, axis=1), np.sum(G * G, axis=0)


def ema(prev: np.ndarray, new: np.ndarray, mu: float) -> np.ndarray:
    """mu * prev + (1 - mu) * new (Algorithm 1, momentum and statistics lines)."""
    return mu * prev + (1.0 - mu) * new


def diag_preconditioner(v: np.ndarray, eps: float) -> np.ndarray:
    """Diagonal of Diag((v + eps)^(-1/8)) (Algorithm 1, L_t / R_t line;
    eq. dp_preconditioner)."""
    return np.power(np.asarray(v, dtype=np.float64) + eps, PRECOND_EXPONENT)


def two_sided(Ld: np.ndarray, X: np.ndarray, Rd: np.ndarray) -> np.ndarray:
    """Diag(Ld) X Diag(Rd): entry (i, j) is Ld_i X_ij Rd_j
    (eq. two_sided_diagonal_preconditioner and the entrywise form below it)."""
    return Ld[:, None] * X * Rd[None, :]


# ---------------------------------------------------------------------------
# Orthogonalisation
# ---------------------------------------------------------------------------

def orth_exact(X: np.ndarray, rank_tol: float = 1e-12) -> np.ndarray:
    """Orth(X) = U V^T from the reduced SVD X = U S V^T (Section 3.1,
    eq. muon-update).  Singular values below rank_tol * s_max map to 0, the
    same convention Newton-Schulz follows for a rank-deficient input."""
    X = np.asarray(X, dtype=np.float64)
    U, S, Vt = np.linalg.svd(X, full_matrices=False)
    if S.size == 0 or S[0] == 0.0:
        return np.zeros_like(X)
    keep = (S > rank_tol * S[0]).astype(np.float64)
    return (U * keep[None, :]) @ Vt


def newton_schulz(X: np.ndarray, steps: int = DEFAULT_NS_STEPS,
                  coeffs=DEFAULT_NS_COEFFS, ns_eps: float = DEFAULT_NS_EPS) -> np.ndarray:
    """Approximate Orth(X) by the quintic Newton-Schulz iteration (Section 3.1
    names the method; the iteration and its constants are reading 1 in the
    module docstring).  Works on the wide orientation: a tall X is transposed
    first and the result transposed back."""
    a, b, c = (float(v) for v in coeffs)
    X = np.asarray(X, dtype=np.float64)
    transposed = X.shape[0] > X.shape[1]
    if transposed:
        X = X.T
    X = X / (np.linalg.norm(X) + ns_eps)
    for _ in range(steps):
        A = X @ X.T
        B = b * A + c * (A @ A)
        X = a * X + B @ X
    return X.T if transposed else X


def ns_scalar_map(x, steps: int = DEFAULT_NS_STEPS, coeffs=DEFAULT_NS_COEFFS):
    """The scalar polynomial p(x) = a x + b x^3 + c x^5 applied `steps` times.
    Newton-Schulz acts on each singular value of the normalised input through
    this map (used by the tests to pin newton_schulz)."""
    a, b, c = (float(v) for v in coeffs)
    x = np.asarray(x, dtype=np.float64)
    for _ in range(steps):
        x = a * x + b * x ** 3 + c * x ** 5
    return x


# ---------------------------------------------------------------------------
# bf16 rounding (the oracle's own; no framework conversion)
# ---------------------------------------------------------------------------

def round_to_bf16(x: np.ndarray) -> np.ndarray:
    """Round fp64 values to the nearest bfloat16 value, ties to even.
    bfloat16 keeps 8 significant bits and fp32's exponent range; below the
    smallest normal (2^-126) its spacing is the subnormal quantum 2^-133."""
    x = np.asarray(x, dtype=np.float64)
    out = np.zeros_like(x)
    nz = x != 0.0
    _, e = np.frexp(x[nz])               # x = f * 2^e, 0.5 <= |f| < 1
    q = np.ldexp(1.0, np.maximum(e - 8, -133))
    out[nz] = np.rint(x[nz] / q) * q     # np.rint rounds half to even
    return out


# ---------------------------------------------------------------------------
# The update
# ---------------------------------------------------------------------------

def malt_step_ref(W: np.ndarray, G: np.ndarray, state: State, hp: Hyper,
                  variant: str = "malt", orth: str = "ns",
                  weight_dtype: str = "f32", force_identity: bool = False):
    """One step of Algorithm 1 (variant="malt") or Algorithm 2 ("malter") on
    one matrix.  Returns (W_new, info) and updates `state` in place.

    W and G are upcast to fp64 as given.  `weight_dtype="bf16"` rounds the new
    W to bf16 (reading 6).  `orth` selects Newton-Schulz ("ns") or the exact
    polar factor ("exact").  `force_identity` replaces L and R by identity
    (plain Muon with EMA momentum and the graft), a test switch."""
    W = np.asarray(W, dtype=np.float64)
    G = np.asarray(G, dtype=np.float64)
    state.t += 1                                             # reading 4
    t = state.t
    # Momentum (Algorithm 1 / 2, M_t line).
    state.M = ema(state.M, G, hp.mu1)
    # Row / column squared-norm statistics (l_t, r_t lines).
    s_row, s_col = row_col_sq_norms(G)
    state.l = ema(state.l, s_row, hp.mu2)
    state.r = ema(state.r, s_col, hp.mu2)
    # Diagonal preconditioners (L_t, R_t line).
    if force_identity:
        Ld, Rd = np.ones(G.shape[0]), np.ones(G.shape[1])
    else:
        Ld = diag_preconditioner(state.l, hp.eps)
        Rd = diag_preconditioner(state.r, hp.eps)
    # Preconditioned momentum, orthogonalisation, back-map.
    Mt = two_sided(Ld, state.M, Rd)
    if orth == "exact":
        O = orth_exact(Mt)
    else:
        O = newton_schulz(Mt, hp.ns_steps, hp.ns_coeffs, hp.ns_eps)
    D = two_sided(Ld, O, Rd)
    norm_O = float(np.linalg.norm(O))
    norm_D = float(np.linalg.norm(D))
    norm_Mt = float(np.linalg.norm(Mt))
    scale = hp.lr * norm_O / (norm_D + hp.eps)               # graft (W_t line)
    alpha = 1.0
    lgr_sq = float("nan")
    if variant == "malter":
        # Algorithm 2: nu_t line, then alpha_t of Section 3.5 (reading 2).
        lgr_sq = float(np.sum(two_sided(Ld, G, Rd) ** 2))
        state.nu = hp.mu2 * state.nu + (1.0 - hp.mu2) * lgr_sq
        alpha = (math.sqrt(1.0 - hp.mu2 ** t) / (1.0 - hp.mu1 ** t + hp.eps)
                 * norm_Mt / (math.sqrt(state.nu) + hp.eps))
        scale *= alpha
    elif variant != "malt":
        raise ValueError(f"unknown variant {variant!r}")
    W_decayed = (1.0 - hp.lr * hp.weight_decay) * W if hp.weight_decay else W
    delta = scale * D
    W_new = W_decayed - delta
    if weight_dtype == "bf16":
        W_new = round_to_bf16(W_new)
    info = dict(L=Ld, R=Rd, Mt=Mt, O=O, D=D, norm_O=norm_O, norm_D=norm_D,
                norm_Mt=norm_Mt, lgr_sq=lgr_sq, alpha=alpha, scale=scale,
                delta=delta, t=t, nu=state.nu)
    return W_new, info


def run_steps(W0, grads, hp: Hyper, variant: str = "malt", weight_dtype: str = "f32",
              orth: str = "ns"):
    """Apply malt_step_ref over a sequence of gradients from zero state
    (Algorithm 1/2 for-loop).  Returns (W_final, state, infos)."""
    W = np.asarray(W0, dtype=np.float64)
    m, n = W.shape
    st = State.zeros(m, n)
    infos = []
    for G in grads:
        W, info = malt_step_ref(W, G, st, hp, variant=variant, orth=orth,
                                weight_dtype=weight_dtype)
        infos.append(info)
    return W, st, infos


def state_floats(m: int, n: int, variant: str = "malt") -> int:
    """Optimizer-state size in floats for one m x n matrix as this oracle holds
    it (M, l, r, plus nu for MALTER): mn + m + n (+1), the complexity table of
    Section 5.5."""
    st = State.zeros(m, n)
    extra = 1 if variant == "malter" else 0
    return st.M.size + st.l.size + st.r.size + extra
