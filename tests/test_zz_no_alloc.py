"""malt_stats_noalloc against the regular step and the fp64 oracle.

malt_stats_noalloc is for callers that cannot allocate device memory when
they need the work done: code under a framework allocator that owns all
device memory, code that cannot afford the device synchronisation an
allocation may cause, services that reserve all memory at start-up.  It keeps
its scratch in a fixed array inside the library and runs the step's own
statistics and finalize blocks.  So on consecutive calls (the shared array
keeps the previous call's contents) its momentum, row/column statistics and
preconditioners must equal malt_step's for the same matrix bitwise, and the
oracle's (Algorithm 1, M_t, l_t, r_t and L_t / R_t lines) within the 1e-5
statistics bar, and a call must not change the device's free memory.

This file is collected last, so a run that stops at the first failure has
run every other test before it.
"""
import numpy as np
import pytest

import oracle.malt_ref as ref
import paper_2608_05088_gb300.malt as malt
from paper_2608_05088_gb300 import inputs
from tests.gpu_harness import TOL_STATS

pytestmark = pytest.mark.gpu


def _host(t):
    return t.double().cpu().numpy()


def _rel(a, b):
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


def _elem_rel(a, b):
    return float(np.max(np.abs(a - b) / np.abs(b)))


@pytest.mark.parametrize("shape,g_dtype", [((392, 1000), "f32"), ((1280, 5120), "f32"),
                                           ((520, 1544), "bf16")])
def test_noalloc_stats_match_step_and_oracle_on_two_calls(shape, g_dtype):
    import torch
    dev = torch.device("cuda:0")
    m, n = shape
    tdt = torch.float32 if g_dtype == "f32" else torch.bfloat16
    wl = inputs.Workload("noalloc", 60, (shape,), "f32", 1.5, 0.02, "malt", 2)
    W = torch.from_numpy(inputs.initial_weight(wl, 0)).to(dev)
    G = torch.zeros(shape, dtype=tdt, device=dev)
    M_a = torch.empty(shape, dtype=torch.float32, device=dev)
    l_a = torch.empty(m, dtype=torch.float32, device=dev)
    r_a = torch.empty(n, dtype=torch.float32, device=dev)
    opt = malt.MaltOptimizer([(W, G, M_a, l_a, r_a)])
    hp = malt.hparams(lr=wl.lr)
    f32 = lambda v: float(np.float32(v))
    mu1, mu2, eps = f32(hp.mu1), f32(hp.mu2), f32(hp.eps)
    M_b = torch.zeros(shape, dtype=torch.float32, device=dev)
    l_b = torch.zeros(m, dtype=torch.float32, device=dev)
    r_b = torch.zeros(n, dtype=torch.float32, device=dev)
    L_b = torch.empty(m, dtype=torch.float32, device=dev)
    R_b = torch.empty(n, dtype=torch.float32, device=dev)
    M_ref, l_ref, r_ref = np.zeros(shape), np.zeros(m), np.zeros(n)
    for step in range(2):
        g = inputs.gradient(wl, 0, step)
        if g_dtype == "bf16":
            g = inputs.bf16_representable(g)
        G.copy_(torch.from_numpy(g))
        opt.step(hp)
        torch.cuda.synchronize()
        free_before = torch.cuda.mem_get_info()[0]
        allocated_before = torch.cuda.memory_allocated()
        rc = malt.malt_stats_noalloc(G, M_b, l_b, r_b, L_b, R_b, hp.mu1, hp.mu2, hp.eps)
        assert rc == malt.MALT_OK, malt.status_string(rc)
        torch.cuda.synchronize()
        if step > 0:      # the first call on a device may load the library's module
            assert torch.cuda.mem_get_info()[0] == free_before
        # torch's own count may only fall (Python freeing a tensor meanwhile)
        assert torch.cuda.memory_allocated() <= allocated_before
        assert opt.check() == malt.MALT_OK
        L_a, R_a = opt.precond(0)
        torch.cuda.synchronize()
        # the same blocks as the step: bitwise equal
        for x, y in ((M_b, M_a), (l_b, l_a), (r_b, r_a), (L_b, L_a), (R_b, R_a)):
            assert torch.equal(x, y)
        # the oracle's statistics and preconditioners (fp64)
        s_row, s_col = ref.row_col_sq_norms(g.astype(np.float64))
        M_ref = ref.ema(M_ref, g.astype(np.float64), mu1)
        l_ref = ref.ema(l_ref, s_row, mu2)
        r_ref = ref.ema(r_ref, s_col, mu2)
        assert _rel(_host(M_b), M_ref) <= TOL_STATS
        assert _elem_rel(_host(l_b), l_ref) <= TOL_STATS
        assert _elem_rel(_host(r_b), r_ref) <= TOL_STATS
        assert _elem_rel(_host(L_b), ref.diag_preconditioner(l_ref, eps)) <= TOL_STATS
        assert _elem_rel(_host(R_b), ref.diag_preconditioner(r_ref, eps)) <= TOL_STATS
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
