"""Seeded synthetic workloads for the MALT / MALTER update.

This module only draws inputs; it holds none of the update's arithmetic.  Both
the CUDA path (tests, benchmark) and the fp64 oracle receive exactly the
arrays produced here.

Shapes are the 2-D parameter sets of the GPT-2 models the paper trains
(Section 5.1: GPT-2 Small / Medium / Large with NanoGPT), taken literally as
rows x cols, plus a single small matrix and a square/rectangular stress set.
Gradients stand in for the paper's OpenWebText gradients (Section 5.1),
which are not available here: G_ij = z_ij * a_i * b_j with z ~ N(0, 1) drawn
fresh every step and row/column scales a_i, b_j = exp(sigma * N(0, 1)) drawn
once per matrix, the row/column anisotropy that Section 5.4 reports for the
trained model.  Initial weights follow the GPT-2 init N(0, 0.02^2).

Every draw comes from numpy's PCG64 seeded with the tuple
(workload id, matrix index, step + 1, stream tag), so any matrix of any step
can be regenerated on its own.
"""
from __future__ import annotations

import dataclasses
from concurrent.futures import ThreadPoolExecutor

import numpy as np

_TAG_SCALES, _TAG_GRAD, _TAG_WEIGHT = 1, 2, 3


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    wid: int                     # seed component
    shapes: tuple                # ((rows, cols), ...) in matrix order
    weight_dtype: str            # "f32" | "bf16"
    sigma: float                 # log-normal row/col scale spread
    lr: float
    variant: str                 # "malt" | "malter"
    steps: int
    ns_steps: int = 5

    @property
    def elements(self) -> int:
        return int(sum(m * n for m, n in self.shapes))

    def ns_flops_min(self) -> float:
        """Newton-Schulz flops of one step when the symmetry of A = X X^T and
        of the polynomial in A is used: per matrix and iteration p^2 q (Gram,
        one triangle) + p^3 (A A, one triangle) + 2 p^2 q (B X)."""
        tot = 0.0
        for m, n in self.shapes:
            p, q = min(m, n), max(m, n)
            tot += 3.0 * p * p * q + p ** 3
        return tot * self.ns_steps

    def ns_flops_issued(self, tile: int = 256) -> float:
        """Tensor-core flops the Newton-Schulz products issue in one step with
        tile x tile output tiles over the padded NS frame: every tile on or
        above the diagonal of the symmetric Gram and polynomial products (a
        diagonal tile is computed whole), every tile of B X."""
        tot = 0.0
        for m, n in self.shapes:
            p, q = min(m, n), max(m, n)
            tp, tq = -(-p // tile), -(-q // tile)
            sym = tp * (tp + 1) // 2
            tot += 2.0 * tile * tile * (sym * tq * tile + sym * tp * tile + tp * tq * tp * tile)
        return tot * self.ns_steps

    def ns_flops_dense(self) -> float:
        """Dense Newton-Schulz flops of one step: per matrix and iteration
        4 p^2 q + 2 p^3 with p = min(m, n), q = max(m, n)."""
        tot = 0.0
        for m, n in self.shapes:
            p, q = min(m, n), max(m, n)
            tot += 4.0 * p * p * q + 2.0 * p ** 3
        return tot * self.ns_steps


def _gpt2(layers, d):
    # attn.c_attn d x 3d, attn.c_proj d x d, mlp.c_fc d x 4d, mlp.c_proj 4d x d
    per_layer = ((d, 3 * d), (d, d), (d, 4 * d), (4 * d, d))
    return tuple(s for _ in range(layers) for s in per_layer)


WORKLOADS = {
    "single_256x512": Workload("single_256x512", 1, ((256, 512),), "f32", 1.0, 0.02, "malt", 3),
    "gpt2_small": Workload("gpt2_small", 2, _gpt2(12, 768), "bf16", 1.5, 0.0013, "malt", 10),
    "gpt2_medium": Workload("gpt2_medium", 3, _gpt2(24, 1024), "bf16", 1.5, 0.009, "malter", 10),
    "gpt2_large": Workload("gpt2_large", 4, _gpt2(36, 1280), "bf16", 1.5, 0.0007, "malt", 10),
}


def first_layers(wl: Workload, layers: int, per_layer: int = 4) -> Workload:
    """The first `layers` layers of a GPT-2 workload: same shapes, same seeds,
    so matrix i draws the same inputs as in the full set."""
    return dataclasses.replace(wl, name=f"{wl.name}_first{layers}l",
                               shapes=wl.shapes[: layers * per_layer])


def stress_workload(rows: int, cols: int, sigma: float, ns_steps: int) -> Workload:
    """One large matrix in bf16 with fp32 state, 3 MALT steps (stress sweep)."""
    wid = 5_000 + int(sigma * 10) * 10 + ns_steps
    return Workload(f"stress_{rows}x{cols}_s{sigma:g}_k{ns_steps}", wid, ((rows, cols),),
                    "bf16", sigma, 0.02, "malt", 3, ns_steps)


def random_shapes(seed: int, count: int, max_dim: int = 776, multiple: int = 8) -> tuple:
    """`count` seeded (rows, cols) pairs, each a multiple of `multiple` in
    [multiple, max_dim]: wide, tall and square matrices with ragged tiles in
    both directions, and repeated frames (a shared NS shape class) where two
    draws coincide up to orientation."""
    rng = np.random.Generator(np.random.PCG64([7_000 + (multiple != 8), seed]))
    hi = max_dim // multiple
    shapes = [(multiple * int(rng.integers(1, hi + 1)), multiple * int(rng.integers(1, hi + 1)))
              for _ in range(count)]
    if count >= 2:
        shapes[-1] = shapes[0][::-1]          # one tall/wide pair in the same class
    return tuple(shapes)


def _rng(wid: int, idx: int, step: int, tag: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64([wid, idx, step + 1, tag]))


def row_col_scales(wl: Workload, idx: int):
    """(a, b): per-row and per-column log-normal scales of matrix idx, fp32."""
    m, n = wl.shapes[idx]
    rng = _rng(wl.wid, idx, -1, _TAG_SCALES)
    a = np.exp(wl.sigma * rng.standard_normal(m)).astype(np.float32)
    b = np.exp(wl.sigma * rng.standard_normal(n)).astype(np.float32)
    return a, b


def gradient(wl: Workload, idx: int, step: int, scales=None) -> np.ndarray:
    """fp32 gradient of matrix idx at step (0-based): z * a_i * b_j."""
    m, n = wl.shapes[idx]
    a, b = scales if scales is not None else row_col_scales(wl, idx)
    z = _rng(wl.wid, idx, step, _TAG_GRAD).standard_normal((m, n), dtype=np.float32)
    z *= a[:, None]
    z *= b[None, :]
    return z


def bf16_representable(x: np.ndarray) -> np.ndarray:
    """Input preparation only: the bf16 value nearest each fp32 entry
    (ties to even), returned as fp32 so the same bits can go anywhere."""
    u = np.array(x, dtype=np.float32, copy=True).view(np.uint32)   # finite inputs only
    lsb = (u >> 16) & np.uint32(1)
    u += np.uint32(0x7FFF)
    u += lsb
    u &= np.uint32(0xFFFF0000)
    return u.view(np.float32)


def initial_weight(wl: Workload, idx: int) -> np.ndarray:
    """W_0 of matrix idx ~ N(0, 0.02^2); bf16-representable for bf16 weights."""
    m, n = wl.shapes[idx]
    w = _rng(wl.wid, idx, 0, _TAG_WEIGHT).standard_normal((m, n), dtype=np.float32)
    w *= np.float32(0.02)
    return bf16_representable(w) if wl.weight_dtype == "bf16" else w


def gradients_for_step(wl: Workload, step: int, indices=None, workers: int = 8):
    """Gradients of all (or the listed) matrices at one step, drawn in parallel."""
    idxs = list(range(len(wl.shapes))) if indices is None else list(indices)
    with ThreadPoolExecutor(max_workers=workers) as ex:
        return list(ex.map(lambda i: gradient(wl, i, step), idxs))


def initial_weights(wl: Workload, indices=None, workers: int = 8):
    idxs = list(range(len(wl.shapes))) if indices is None else list(indices)
    with ThreadPoolExecutor(max_workers=workers) as ex:
        return list(ex.map(lambda i: initial_weight(wl, i), idxs))


# ---------------------------------------------------------------------------
# The rest of a GPT-2 model: the tensors AdamW updates in the paper's
# parameter grouping (Section 5.1: vectors, scalars, embeddings, output head).
# NanoGPT's layout: token embedding with its padded vocabulary of 50304 rows,
# tied with the output head (one tensor); position embedding over the block
# size 1024; per layer the two LayerNorms' gains and biases and the four
# Linear biases; the final LayerNorm.  Weight decay (appendix table: 0.1)
# goes to the 2-D tensors and not to the vectors, NanoGPT's convention.
# Learning rates: the AdamW column of the Section 5.1 table.
# ---------------------------------------------------------------------------
GPT2_VOCAB = 50304
GPT2_BLOCK = 1024
_TAG_ADAM_SCALES, _TAG_ADAM_GRAD, _TAG_ADAM_INIT = 5, 6, 7


@dataclasses.dataclass(frozen=True)
class AdamWSet:
    name: str
    wid: int                     # seed component
    tensors: tuple               # ((name, shape, weight_decay), ...)
    lr: float
    steps: int
    sigma: float = 1.5

    @property
    def elements(self) -> int:
        return int(sum(int(np.prod(shape)) for _, shape, _ in self.tensors))


def _gpt2_adamw(layers, d):
    t = [("wte", (GPT2_VOCAB, d), 0.1), ("wpe", (GPT2_BLOCK, d), 0.1)]
    for i in range(layers):
        t += [(f"h{i}.ln_1.weight", (d,), 0.0), (f"h{i}.ln_1.bias", (d,), 0.0),
              (f"h{i}.attn.c_attn.bias", (3 * d,), 0.0), (f"h{i}.attn.c_proj.bias", (d,), 0.0),
              (f"h{i}.ln_2.weight", (d,), 0.0), (f"h{i}.ln_2.bias", (d,), 0.0),
              (f"h{i}.mlp.c_fc.bias", (4 * d,), 0.0), (f"h{i}.mlp.c_proj.bias", (d,), 0.0)]
    t += [("ln_f.weight", (d,), 0.0), ("ln_f.bias", (d,), 0.0)]
    return tuple(t)


ADAMW_SETS = {
    "gpt2_small": AdamWSet("gpt2_small_adamw", 12, _gpt2_adamw(12, 768), 0.0013, 10),
    "gpt2_medium": AdamWSet("gpt2_medium_adamw", 13, _gpt2_adamw(24, 1024), 0.0009, 10),
    "gpt2_large": AdamWSet("gpt2_large_adamw", 14, _gpt2_adamw(36, 1280), 0.0009, 10),
}


def adamw_initial(aset: AdamWSet, idx: int) -> np.ndarray:
    """Initial value of tensor idx (fp32): embeddings ~ N(0, 0.02^2), LayerNorm
    gains 1, biases 0 (the GPT-2 / NanoGPT initialisation)."""
    name, shape, _ = aset.tensors[idx]
    if len(shape) == 2:
        w = _rng(aset.wid, idx, 0, _TAG_ADAM_INIT).standard_normal(shape, dtype=np.float32)
        w *= np.float32(0.02)
        return w
    if name.endswith("ln_1.weight") or name.endswith("ln_2.weight") or name == "ln_f.weight":
        return np.ones(shape, dtype=np.float32)
    return np.zeros(shape, dtype=np.float32)


def adamw_gradient(aset: AdamWSet, idx: int, step: int) -> np.ndarray:
    """fp32 gradient of tensor idx at step (0-based): z times log-normal
    scales drawn once per tensor (per row and column for the embeddings, per
    entry for a vector)."""
    _, shape, _ = aset.tensors[idx]
    srng = _rng(aset.wid, idx, -1, _TAG_ADAM_SCALES)
    z = _rng(aset.wid, idx, step, _TAG_ADAM_GRAD).standard_normal(shape, dtype=np.float32)
    if len(shape) == 2:
        z *= np.exp(aset.sigma * srng.standard_normal(shape[0])).astype(np.float32)[:, None]
        z *= np.exp(aset.sigma * srng.standard_normal(shape[1])).astype(np.float32)[None, :]
    else:
        z *= np.exp(aset.sigma * srng.standard_normal(shape)).astype(np.float32)
    return z


def toy_quadratic_problem(kappa: float, n: int = 50, r: int = 5, seed: int = 0):
    """(A, B, C) of the matrix quadratic regression min_X 1/2 ||A X B^T - C||_F^2
    (Appendix B): C = U* S* V*^T of rank r with orthonormal U*, V* (n x r) and a
    random core S* of unit Frobenius norm; A = U* R1, B = V* R2 with r x r
    factors R1, R2 of condition number kappa^(1/4) each, so the Hessian
    (B^T B) kron (A^T A) has condition number cond(R1)^2 cond(R2)^2 = kappa."""
    rng = _rng(9_000, int(round(np.log10(kappa) * 100)), seed, 4)
    U, _ = np.linalg.qr(rng.standard_normal((n, r)))
    V, _ = np.linalg.qr(rng.standard_normal((n, r)))
    S = rng.standard_normal((r, r))
    S /= np.linalg.norm(S)

    def with_condition(c):
        Q1, _ = np.linalg.qr(rng.standard_normal((r, r)))
        Q2, _ = np.linalg.qr(rng.standard_normal((r, r)))
        return Q1 @ np.diag(np.geomspace(1.0, c, r)) @ Q2.T

    c = kappa ** 0.25
    R1, R2 = with_condition(c), with_condition(c)
    return U @ R1, V @ R2, U @ S @ V.T
