"""Pins that tie the fp64 AdamW oracle to what the published algorithm and the
mathematics fix.  Each check takes the oracle module as an argument, so the
same checks run against the real oracle (test_adamw_oracle.py) and against
copies with planted mistakes.  No check re-types the oracle's formula: each
uses a closed form, exact arithmetic, or a library routine (torch.optim.AdamW
run in float64 on the CPU)."""
from __future__ import annotations

import numpy as np


def _rel(a, b):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def check_first_step_is_lr_sign(ref):
    """From zero moments the bias corrections make m_hat = g and v_hat = g^2
    exactly, so the first step (no decay) is lr * g / (|g| + eps): lr times
    the sign of g up to eps, whatever the betas."""
    rng = np.random.default_rng(31)
    g = rng.standard_normal(1000) * np.exp(3 * rng.standard_normal(1000))
    g[:3] = (0.0, 1e-9, -1e-9)
    w0 = rng.standard_normal(1000)
    for betas in ((0.9, 0.95), (0.5, 0.25), (0.0, 0.0)):
        hp = ref.AdamWHyper(lr=0.01, beta1=betas[0], beta2=betas[1], eps=1e-8)
        st = ref.AdamWState.zeros(g.shape)
        w1, _ = ref.adamw_step_ref(w0, g, st, hp)
        want = w0 - 0.01 * g / (np.abs(g) + 1e-8)
        assert np.allclose(w1, want, rtol=0, atol=1e-15), betas
        assert np.allclose(np.abs(w1[3:] - w0[3:])[np.abs(g[3:]) > 1e-4], 0.01, rtol=1e-4)


def check_constant_gradient(ref):
    """A constant gradient keeps m_hat = g and v_hat = g^2 at every step (the
    bias corrections undo the geometric sums exactly), so each step moves w by
    lr * g / (|g| + eps)."""
    rng = np.random.default_rng(32)
    g = rng.standard_normal(64) + 0.5
    hp = ref.AdamWHyper(lr=3e-3)
    st = ref.AdamWState.zeros(g.shape)
    w = np.zeros(64)
    for t in range(1, 8):
        w, info = ref.adamw_step_ref(w, g, st, hp)
        assert _rel(info["m_hat"], g) < 1e-13 and _rel(info["v_hat"], g * g) < 1e-13
        assert _rel(w, -t * 3e-3 * g / (np.abs(g) + 1e-8)) < 1e-12
    assert st.t == 7


def check_unrolled_moments(ref):
    """Three steps with beta1 = 1/2, beta2 = 1/4 on integer gradients equal the
    unrolled geometric sums exactly (fp64 is exact here)."""
    rng = np.random.default_rng(33)
    gs = [rng.integers(-4, 5, size=20).astype(np.float64) for _ in range(3)]
    hp = ref.AdamWHyper(lr=0.0, beta1=0.5, beta2=0.25)
    st = ref.AdamWState.zeros(20)
    w = np.zeros(20)
    for g in gs:
        w, _ = ref.adamw_step_ref(w, g, st, hp)
    assert np.array_equal(st.m, 0.5 * (0.25 * gs[0] + 0.5 * gs[1] + gs[2]))
    assert np.array_equal(st.v, 0.75 * (0.0625 * gs[0] ** 2 + 0.25 * gs[1] ** 2 + gs[2] ** 2))


def check_zero_gradient_is_pure_decay(ref):
    """g = 0: both moments stay 0, the Adam step is 0 / (0 + eps) = 0, and t
    steps shrink w geometrically, w_t = (1 - lr wd)^t w_0."""
    w0 = np.random.default_rng(34).standard_normal(50)
    hp = ref.AdamWHyper(lr=0.02)
    st = ref.AdamWState.zeros(50)
    w = w0
    for _ in range(6):
        w, _ = ref.adamw_step_ref(w, np.zeros(50), st, hp, weight_decay=0.1)
    assert not np.any(st.m) and not np.any(st.v)
    assert _rel(w, (1 - 0.02 * 0.1) ** 6 * w0) < 1e-15


def check_decay_is_decoupled(ref):
    """The decay neither enters the moments nor the Adam step: with and
    without it the moments agree exactly, and the decayed step removes the
    same Adam step from the shrunk starting weights."""
    rng = np.random.default_rng(35)
    w0 = rng.standard_normal(40)
    g = rng.standard_normal(40)
    hp = ref.AdamWHyper(lr=0.05)
    a, b = ref.AdamWState.zeros(40), ref.AdamWState.zeros(40)
    wa, ia = ref.adamw_step_ref(w0, g, a, hp, weight_decay=0.3)
    wb, ib = ref.adamw_step_ref(w0, g, b, hp, weight_decay=0.0)
    assert np.array_equal(a.m, b.m) and np.array_equal(a.v, b.v)
    assert _rel(wa, (1 - 0.05 * 0.3) * w0 - (w0 - wb)) < 1e-15


def check_against_torch_adamw(ref):
    """Seven steps on random gradients against torch.optim.AdamW (the library
    routine) in float64 on the CPU, with decay, for two learning rates."""
    import torch
    rng = np.random.default_rng(36)
    w0 = rng.standard_normal((12, 7))
    grads = [rng.standard_normal((12, 7)) * np.exp(rng.standard_normal((12, 7))) for _ in range(7)]
    for lr, wd in ((1e-3, 0.1), (0.05, 0.0)):
        p = torch.nn.Parameter(torch.from_numpy(w0.copy()))
        opt = torch.optim.AdamW([p], lr=lr, betas=(0.9, 0.95), eps=1e-8, weight_decay=wd,
                                foreach=False)
        hp = ref.AdamWHyper(lr=lr, beta1=0.9, beta2=0.95, eps=1e-8)
        st = ref.AdamWState.zeros(w0.shape)
        w = w0
        for g in grads:
            p.grad = torch.from_numpy(g.copy())
            opt.step()
            w, _ = ref.adamw_step_ref(w, g, st, hp, weight_decay=wd)
            assert _rel(w, p.detach().numpy()) < 1e-13


def check_defaults_match_paper(ref):
    """The AdamW column of the appendix table: (beta1, beta2) = (0.9, 0.95),
    weight decay 0.1."""
    assert ref.DEFAULT_BETAS == (0.9, 0.95)
    assert ref.DEFAULT_WEIGHT_DECAY == 0.1
    hp = ref.AdamWHyper()
    assert (hp.beta1, hp.beta2) == (0.9, 0.95)


ALL_CHECKS = [
    check_first_step_is_lr_sign,
    check_constant_gradient,
    check_unrolled_moments,
    check_zero_gradient_is_pure_decay,
    check_decay_is_decoupled,
    check_against_torch_adamw,
    check_defaults_match_paper,
]
