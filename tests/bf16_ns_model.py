"""A CPU model of the Newton-Schulz arithmetic the GPU path is required to use
(test infrastructure).

The GPU path computes Newton-Schulz with bf16 operands and fp32 accumulation.  On
most inputs that arithmetic lands well inside the 2e-2 direction bar; on a
few (a thin matrix with three singular values, the very ill-conditioned steps
of the toy quadratic) the arithmetic itself reaches or passes it, whatever
the kernel does.  This model computes the same products in the same
precisions, so a test can tell "the kernel is wrong" from "bf16 operands
cannot resolve this input": where the model's own error is at the bar, the
GPU must be no worse than the model.

The model rounds what the kernels store to bf16 and accumulates each product
in fp32 (numpy float32 matmuls; their summation order differs from the
tensor cores', which only moves results by fp32 ulps):
  X0 = bf16(Mt)                             on the wide orientation
  A  = bf16(k^2 * X X^T)  (first iteration),  bf16(X X^T) after
  B' = bf16(b A + c (A A) + a I)            (aI folded into B', as stored)
  X  = bf16(k * B' X)     (first iteration),  bf16(B' X) after
with k = 1 / (||Mt||_F + ns_eps) in fp32.  It shares no code with the CUDA
path; its bf16 rounding is the oracle's (pinned against torch).
"""
from __future__ import annotations

import numpy as np

import oracle.malt_ref as ref


def _mm(a, b):
    return (np.asarray(a, np.float32) @ np.asarray(b, np.float32)).astype(np.float64)


def newton_schulz_bf16(Mt, steps=ref.DEFAULT_NS_STEPS, coeffs=ref.DEFAULT_NS_COEFFS,
                       ns_eps=ref.DEFAULT_NS_EPS, rounding=ref.round_to_bf16):
    """O = NS_k(Mt) in the arithmetic described in the module docstring.
    `rounding` is the bf16 rounding (identity turns the model into fp32
    Newton-Schulz)."""
    a, b, c = (float(np.float32(v)) for v in coeffs)
    X = np.asarray(Mt, dtype=np.float64)
    transposed = X.shape[0] > X.shape[1]
    if transposed:
        X = X.T
    k = float(np.float32(1.0) / (np.float32(np.linalg.norm(X)) + np.float32(ns_eps)))
    X = rounding(X)
    eye = np.eye(X.shape[0])
    for it in range(steps):
        s = k if it == 0 else 1.0
        A = rounding(_mm(X, X.T) * (s * s))
        B = rounding(b * A + c * _mm(A, A) + a * eye)
        X = rounding(_mm(B, X) * s)
    return X.T if transposed else X


def step_errors(info, hp, steps=None, coeffs=None):
    """Errors of the model against the oracle for one oracle step's info
    (the keys of malt_step_ref): O, ||O||, ||D|| and the update delta, each
    relative as the parity tests measure them."""
    O = newton_schulz_bf16(info["Mt"], steps or hp.ns_steps, coeffs or hp.ns_coeffs, hp.ns_eps)
    D = info["L"][:, None] * O * info["R"][None, :]
    nO, nD = float(np.linalg.norm(O)), float(np.linalg.norm(D))
    delta = (info["scale"] / max(info["norm_O"], 1e-300) * (info["norm_D"] + hp.eps)) \
        * nO / (nD + hp.eps) * D
    rel = lambda x, y: float(np.linalg.norm(x - y) / max(np.linalg.norm(y), 1e-300))
    return dict(O=rel(O, info["O"]),
                norm_o=abs(nO - info["norm_O"]) / max(info["norm_O"], 1e-300),
                norm_d=abs(nD - info["norm_D"]) / max(info["norm_D"], 1e-300),
                dW=rel(delta, info["delta"]))
