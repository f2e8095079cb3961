"""The Appendix B matrix quadratic regression: its construction (CPU) and the
MALT / Muon runs on the GPU engine against the oracle (GPU)."""
import numpy as np
import pytest

from paper_2608_05088_gb300 import inputs
from paper_2608_05088_gb300 import toy_quadratic as tq
from tests import bf16_ns_model


@pytest.mark.parametrize("kappa", [10.0, 100.0, 1e3, 1e4])
def test_problem_has_prescribed_hessian_condition(kappa):
    """The Hessian of vec(X) is (B^T B) kron (A^T A); its condition number must
    be kappa, and C is realisable (f* = 0) as Appendix B constructs it."""
    A, B, C = inputs.toy_quadratic_problem(kappa)
    ev = np.linalg.eigvalsh(np.kron(B.T @ B, A.T @ A))
    assert abs(ev.max() / ev.min() / kappa - 1) < 1e-9
    Xs, fstar = tq.optimum(A, B, C)
    assert fstar < 1e-24
    # the gradient vanishes at X*
    assert np.linalg.norm(A.T @ (A @ Xs @ B.T - C) @ B) < 1e-12


def test_wsd_schedule_shape():
    lr = [tq.wsd_lr(t, 5000) for t in range(5000)]
    assert lr[0] == pytest.approx(2e-6) and lr[499] == pytest.approx(1e-3)
    assert lr[500] == lr[3999] == pytest.approx(1e-3)
    assert lr[4999] == pytest.approx(1e-6) and all(a >= b for a, b in zip(lr[3999:], lr[4000:]))


def _oracle_trace(kappa, optimizer, steps, lr_max, record_every):
    import oracle.malt_ref as ref
    A, B, C = inputs.toy_quadratic_problem(kappa)
    r = A.shape[1]
    X = np.zeros((r, r))
    st = ref.State.zeros(r, r)
    _, fstar = tq.optimum(A, B, C)
    ts, gaps = [], []
    for t in range(steps):
        if t % record_every == 0:
            ts.append(t)
            gaps.append(tq.objective(A, B, C, X) - fstar)
        G = A.T @ (A @ X @ B.T - C) @ B
        hp = ref.Hyper(lr=tq.wsd_lr(t, steps, lr_max))
        X, _ = ref.malt_step_ref(X, G, st, hp, force_identity=(optimizer == "muon"))
    ts.append(steps)
    gaps.append(tq.objective(A, B, C, X) - fstar)
    return np.array(ts), np.array(gaps)


@pytest.mark.gpu
@pytest.mark.parametrize("optimizer", ["malt", "muon"])
@pytest.mark.parametrize("kappa", [10.0, 1e4])
def test_gpu_steps_match_oracle_teacher_forced(kappa, optimizer):
    """600 WSD steps (lr_max 1e-2): both sides get the gradient of the
    oracle's iterate, so their optimizer states see the same inputs; every
    100th GPU update (X at its own 5 x 5 shape, which the library pads to 8 x 8
    inside) is compared with the oracle's update of that step.

    With bf16 Newton-Schulz operands the direction error grows with the
    condition number of Mt: rounding the entries perturbs the weak singular
    directions by about 2^-9 sigma_max / sigma_min relative to themselves, and
    those directions still weigh in O.  Every checked update must be within
    the 2e-2 bar, except where a CPU model of that same bf16 arithmetic
    (tests/bf16_ns_model.py) errs by 1.8e-2 or more on the step (the badly
    conditioned steps of kappa = 1e4, cond(Mt) up to ~1e4); there the GPU's
    update must be no worse than the model's, within 25 % + 2e-3."""
    import torch
    import oracle.malt_ref as ref
    import paper_2608_05088_gb300.malt as malt
    steps, lr_max = 600, 1e-2
    A, B, C = inputs.toy_quadratic_problem(kappa)
    r = A.shape[1]
    dev = torch.device("cuda")
    X = torch.zeros((r, r), dtype=torch.float32, device=dev)
    G = torch.zeros_like(X)
    M = torch.empty_like(X)
    l = torch.empty(r, dtype=torch.float32, device=dev)
    rr = torch.empty(r, dtype=torch.float32, device=dev)
    opt = malt.MaltOptimizer([(X, G, M, l, rr)])
    Xr = np.zeros((r, r))
    st = ref.State.zeros(r, r)
    checked = []
    for t in range(steps):
        Gp = (A.T @ (A @ Xr @ B.T - C) @ B).astype(np.float32)
        G.copy_(torch.from_numpy(Gp))
        lr = tq.wsd_lr(t, steps, lr_max)
        check = t % 100 == 99
        if check:
            X_before = X.double().cpu().numpy()
        opt.step(malt.hparams(lr=lr), muon=(optimizer == "muon"))
        Xr, info = ref.malt_step_ref(Xr, Gp.astype(np.float64), st, ref.Hyper(lr=lr),
                                     force_identity=(optimizer == "muon"))
        if check:
            Xg = X.double().cpu().numpy()
            step_gpu = X_before - Xg
            err = np.linalg.norm(step_gpu - info["delta"]) / np.linalg.norm(info["delta"])
            sv = np.linalg.svd(info["Mt"], compute_uv=False)
            cond = sv[0] / sv[-1]
            checked.append((t, cond, err))
            if err >= 2e-2:
                # bf16 operands cannot resolve this step's weak directions:
                # the GPU must be no worse than a model of that arithmetic
                model = bf16_ns_model.step_errors(info, ref.Hyper(lr=lr))["dW"]
                assert model >= 0.9 * 2e-2 and err <= 1.25 * model + 2e-3, (t, cond, err, model)
    assert opt.check() == malt.MALT_OK
    opt.close()
    assert any(e < 2e-2 for _, _, e in checked), checked    # the paper's bar was exercised


@pytest.mark.gpu
@pytest.mark.parametrize("optimizer", ["malt", "muon"])
@pytest.mark.parametrize("kappa", [10.0, 1e4])
def test_gpu_free_run_converges(kappa, optimizer):
    """The paper's setting (5000 WSD steps, lr_max 1e-3, X_0 = 0) run entirely
    on the GPU engine reaches an optimality gap below 1e-3 of the start."""
    ts, gaps, _ = tq.run_gpu(kappa, optimizer, 5000, 1e-3, 500)
    assert gaps[-1] < 1e-3 * gaps[0], list(zip(ts, gaps))
