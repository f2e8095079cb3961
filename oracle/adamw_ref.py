"""Reference (oracle) implementation of the AdamW update of a whole-optimizer step.

TEST INFRASTRUCTURE ONLY.  This module is a plain, slow, fp64 NumPy restatement
used to check the CUDA library; only the test suite, ``__graft_entry__.smoke()``
and the CPU-baseline leg of ``bench.py`` may import it.  It imports nothing
from the library.

What it computes.  The paper trains its GPT-2 models with MALT / MALTER on the
2-D weight matrices only and hands "the vectors, scalars, embedding layers and
output head layers" to AdamW (Section 5.1, Baselines and Parameter Grouping),
with (beta1, beta2) = (0.9, 0.95) and weight decay 0.1 (appendix
hyperparameter table).  AdamW is the cited decoupled-weight-decay variant of
Adam (Loshchilov and Hutter); per parameter tensor, at step t (1-based, from
zero moments):

    m <- beta1 m + (1 - beta1) g
    v <- beta2 v + (1 - beta2) g^2
    m_hat = m / (1 - beta1^t),   v_hat = v / (1 - beta2^t)
    w <- (1 - lr wd) w - lr m_hat / (sqrt(v_hat) + eps)

Readings of points the paper leaves open (the same in the CUDA path):

1. eps: the table leaves AdamW's damping blank; the usual default 1e-8 is used,
   added to sqrt(v_hat) as in the published algorithm.
2. The decay multiplies the weights the step starts from (decoupled, before
   the Adam step), as in the published algorithm.
3. Weights are kept in fp32 ("master weights"); an optional bf16 copy is the
   round-to-nearest-even of the updated fp32 master.
"""
from __future__ import annotations

import dataclasses

import numpy as np

# Appendix hyperparameter table, AdamW column: momentum (beta1, beta2) and
# weight decay; reading 1 for eps.
DEFAULT_BETAS = (0.9, 0.95)
DEFAULT_WEIGHT_DECAY = 0.1
DEFAULT_EPS = 1e-8


@dataclasses.dataclass
class AdamWHyper:
    lr: float = 1e-3
    beta1: float = DEFAULT_BETAS[0]
    beta2: float = DEFAULT_BETAS[1]
    eps: float = DEFAULT_EPS


@dataclasses.dataclass
class AdamWState:
    """First and second moments of one parameter tensor and the step count
    (zero at the start, as in the published algorithm)."""
    m: np.ndarray
    v: np.ndarray
    t: int = 0

    @staticmethod
    def zeros(shape) -> "AdamWState":
        return AdamWState(np.zeros(shape), np.zeros(shape), 0)


def adamw_step_ref(w: np.ndarray, g: np.ndarray, state: AdamWState, hp: AdamWHyper,
                   weight_decay: float = 0.0):
    """One AdamW step of one parameter tensor in fp64 (the update in the
    module docstring).  Returns (w_new, info) and updates `state` in place."""
    w = np.asarray(w, dtype=np.float64)
    g = np.asarray(g, dtype=np.float64)
    state.t += 1
    t = state.t
    state.m = hp.beta1 * state.m + (1.0 - hp.beta1) * g
    state.v = hp.beta2 * state.v + (1.0 - hp.beta2) * g * g
    m_hat = state.m / (1.0 - hp.beta1 ** t)
    v_hat = state.v / (1.0 - hp.beta2 ** t)
    update = hp.lr * m_hat / (np.sqrt(v_hat) + hp.eps)
    w_new = (1.0 - hp.lr * weight_decay) * w - update
    return w_new, dict(m_hat=m_hat, v_hat=v_hat, update=update, t=t)
