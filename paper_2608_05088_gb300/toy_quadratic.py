"""The matrix quadratic regression of Appendix B on the CUDA engine.

min_X f(X) = 1/2 ||A X B^T - C||_F^2 with A, B in R^{n x r}, X in R^{r x r}
(n = 50, r = 5), gradient A^T (A X B^T - C) B, X_0 = 0, and the paper's
warmup-stable-decay schedule (for 5000 steps: linear warmup to lr_max over
500 steps, constant for 3500, linear decay to 0 over the last 1000).  The optimizer
steps run through the library's C ABI (malt_step or muon_step); the gradient
of the toy loss is the "model" and is formed with torch on the device.

X is passed at its own r x r shape; the library runs matrices whose sizes
are not multiples of 8 on zero-padded copies, with the results of the
unpadded matrix.
"""
from __future__ import annotations

import numpy as np

from . import inputs

def wsd_lr(t: int, total: int = 5000, lr_max: float = 1e-3) -> float:
    """Learning rate of 0-based step t under the warmup-stable-decay schedule:
    linear warmup over the first 10 % of the steps, constant, linear decay to
    0 over the last 20 % (500 / 3500 / 1000 of the paper's 5000)."""
    warmup, decay = max(1, total // 10), max(1, total // 5)
    if t < warmup:
        return lr_max * (t + 1) / warmup
    if t < total - decay:
        return lr_max
    return lr_max * (total - t) / decay


def objective(A, B, C, X) -> float:
    """f(X) = 1/2 ||A X B^T - C||_F^2 (fp64, host)."""
    Rr = A @ X @ B.T - C
    return 0.5 * float(np.sum(Rr * Rr))


def optimum(A, B, C):
    """Closed-form least-squares solution X* = A^+ C (B^+)^T and f(X*)."""
    Xs = np.linalg.pinv(A) @ C @ np.linalg.pinv(B).T
    return Xs, objective(A, B, C, Xs)


def run_gpu(kappa: float, optimizer: str = "malt", steps: int = 5000, lr_max: float = 1e-3,
            record_every: int = 100, seed: int = 0, ns_steps: int = 5):
    """Optimality-gap trace of MALT ("malt") or Muon ("muon") on the toy
    problem, steps on the GPU engine.  Returns (ts, gaps, X_final)."""
    import torch
    from . import malt
    A, B, C = inputs.toy_quadratic_problem(kappa, seed=seed)
    r = A.shape[1]
    dev = torch.device("cuda")
    At = torch.from_numpy(A).float().to(dev)
    Bt = torch.from_numpy(B).float().to(dev)
    Ct = torch.from_numpy(C).float().to(dev)
    X = torch.zeros((r, r), dtype=torch.float32, device=dev)
    G = torch.zeros_like(X)
    M = torch.empty_like(X)
    l = torch.empty(r, dtype=torch.float32, device=dev)
    rr = torch.empty(r, dtype=torch.float32, device=dev)
    opt = malt.MaltOptimizer([(X, G, M, l, rr)])
    _, fstar = optimum(A, B, C)
    ts, gaps = [], []
    for t in range(steps):
        if t % record_every == 0:
            ts.append(t)
            gaps.append(objective(A, B, C, X.double().cpu().numpy()) - fstar)
        G.copy_(torch.mm(torch.mm(At.T, torch.mm(torch.mm(At, X), Bt.T) - Ct), Bt))
        hp = malt.hparams(lr=wsd_lr(t, steps, lr_max=lr_max), ns_steps=ns_steps)
        opt.step(hp, muon=(optimizer == "muon"))
    ts.append(steps)
    Xf = X.double().cpu().numpy()
    gaps.append(objective(A, B, C, Xf) - fstar)
    status = opt.check()
    opt.close()
    if status != malt.MALT_OK:
        raise RuntimeError(f"toy run failed: {malt.status_string(status)}")
    return np.array(ts), np.array(gaps), Xf
