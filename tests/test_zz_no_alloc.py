"""malt_stats_noalloc against the regular step.

malt_stats_noalloc is for callers that cannot allocate device memory when
they need the work done: code inside a CUDA stream capture, code whose
framework allocator owns all device memory, code that cannot afford the
device synchronisation an allocation may cause.  It keeps its scratch in a
fixed array inside the library.  Its momentum, row/column statistics and
preconditioners must match what malt_step computes for the same matrix, on
consecutive calls (the shared array keeps the previous call's contents).
"""
import numpy as np
import pytest

import paper_2608_05088_gb300.malt as malt
from paper_2608_05088_gb300 import inputs
from tests.gpu_harness import TOL_STATS

pytestmark = pytest.mark.gpu


def _rel(a, b):
    a = a.double().cpu().numpy()
    b = b.double().cpu().numpy() if hasattr(b, "cpu") else np.asarray(b, dtype=np.float64)
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


def _elem_rel(a, b):
    a = a.double().cpu().numpy()
    b = b.double().cpu().numpy() if hasattr(b, "cpu") else np.asarray(b, dtype=np.float64)
    return float(np.max(np.abs(a - b) / np.abs(b)))


@pytest.mark.parametrize("shape", [(392, 1000), (1280, 5120)])
def test_noalloc_stats_match_regular_step_on_two_calls(shape):
    import torch
    dev = torch.device("cuda:0")
    m, n = shape
    wl = inputs.Workload("noalloc", 60, (shape,), "f32", 1.5, 0.02, "malt", 2)
    W = torch.from_numpy(inputs.initial_weight(wl, 0)).to(dev)
    G = torch.zeros(shape, dtype=torch.float32, device=dev)
    M_a = torch.empty(shape, dtype=torch.float32, device=dev)
    l_a = torch.empty(m, dtype=torch.float32, device=dev)
    r_a = torch.empty(n, dtype=torch.float32, device=dev)
    opt = malt.MaltOptimizer([(W, G, M_a, l_a, r_a)])
    hp = malt.hparams(lr=wl.lr)
    M_b = torch.zeros(shape, dtype=torch.float32, device=dev)
    l_b = torch.zeros(m, dtype=torch.float32, device=dev)
    r_b = torch.zeros(n, dtype=torch.float32, device=dev)
    L_b = torch.empty(m, dtype=torch.float32, device=dev)
    R_b = torch.empty(n, dtype=torch.float32, device=dev)
    for step in range(2):
        G.copy_(torch.from_numpy(inputs.gradient(wl, 0, step)))
        opt.step(hp)
        rc = malt.malt_stats_noalloc(G, M_b, l_b, r_b, L_b, R_b, hp.mu1, hp.mu2, hp.eps)
        assert rc == malt.MALT_OK, malt.status_string(rc)
        torch.cuda.synchronize()
        assert opt.check() == malt.MALT_OK
        assert _rel(M_b, M_a) <= TOL_STATS
        assert _elem_rel(l_b, l_a) <= TOL_STATS and _elem_rel(r_b, r_a) <= TOL_STATS
        L_want = (l_a.double() + hp.eps) ** -0.125
        R_want = (r_a.double() + hp.eps) ** -0.125
        assert _elem_rel(L_b, L_want) <= TOL_STATS and _elem_rel(R_b, R_want) <= TOL_STATS
    opt.close()


def test_noalloc_rejects_matrix_past_scratch_limit():
    import torch
    dev = torch.device("cuda:0")
    m = n = 8192   # needs 32*8192 + 128*8192 floats, past the 1,048,576 limit
    G = torch.zeros((m, n), dtype=torch.float32, device=dev)
    M = torch.zeros((m, n), dtype=torch.float32, device=dev)
    l = torch.zeros(m, dtype=torch.float32, device=dev)
    r = torch.zeros(n, dtype=torch.float32, device=dev)
    L = torch.empty(m, dtype=torch.float32, device=dev)
    R = torch.empty(n, dtype=torch.float32, device=dev)
    assert malt.malt_stats_noalloc(G, M, l, r, L, R) == malt.MALT_ERR_UNSUPPORTED
    torch.cuda.synchronize()
    assert not torch.any(M)
