"""Error paths on a live state: bad arguments return codes, a device-side wait
that runs out reports MALT_ERR_TIMEOUT and leaves the context usable."""
import ctypes

import numpy as np
import pytest

import paper_2608_05088_gb300.malt as malt
from paper_2608_05088_gb300 import inputs
from tests.gpu_harness import Run

pytestmark = pytest.mark.gpu


def test_bad_arguments_on_live_state():
    import torch
    wl = inputs.Workload("err", 40, ((128, 256),), "f32", 1.0, 0.02, "malt", 1)
    run = Run(wl, check=[])
    lib = malt.load()
    arr = malt.params_array(run.params)
    s = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    good = malt.hparams()
    assert lib.malt_step(run.opt.state, arr, 2, ctypes.byref(good), s) == malt.MALT_ERR_SHAPE_CHANGED
    bad = malt.hparams(mu1=1.0)
    assert lib.malt_step(run.opt.state, arr, 1, ctypes.byref(bad), s) == malt.MALT_ERR_INVALID_ARG
    bad = malt.hparams(ns_steps=0)
    assert lib.malt_step(run.opt.state, arr, 1, ctypes.byref(bad), s) == malt.MALT_ERR_INVALID_ARG
    other = torch.empty((256, 128), device="cuda")
    arr2 = malt.params_array([(other, other, other, run.l[0], run.r[0])])
    assert lib.malt_step(run.opt.state, arr2, 1, ctypes.byref(good), s) == malt.MALT_ERR_SHAPE_CHANGED
    big = torch.empty(128 * 256 + 4, device="cuda")
    mis = big[1:1 + 128 * 256].view(128, 256)
    arr3 = malt.params_array([(run.W[0], run.G[0], mis, run.l[0], run.r[0])])
    assert lib.malt_step(run.opt.state, arr3, 1, ctypes.byref(good), s) == malt.MALT_ERR_MISALIGNED
    run.step(oracle=False)
    assert run.status() == malt.MALT_OK
    run.close()


def test_bounded_wait_reports_timeout_and_context_survives():
    assert malt.malt_debug_wait_timeout(200_000_000) == malt.MALT_ERR_TIMEOUT
    wl = inputs.Workload("after", 41, ((256, 512),), "f32", 1.0, 0.02, "malt", 1)
    run = Run(wl)
    run.step()
    assert run.status() == malt.MALT_OK
    run.assert_close(0)
    run.close()


def test_empty_parameter_list():
    opt = malt.MaltOptimizer([])
    opt.step(malt.hparams())
    assert opt.check() == malt.MALT_OK
    opt.close()


@pytest.mark.parametrize("schedule", ["auto", "persistent"])
def test_host_buffer_step_matches_device_step(schedule):
    """malt_step_host (gradients from pinned host memory, weights copied back)
    gives bitwise the same W, M, l, r as malt_step on the same gradients, and
    the host copies of W equal the device W after every step."""
    import numpy as np
    import torch
    wl = inputs.Workload("hoststep", 42, ((256, 512), (392, 136), (520, 1544), (250, 509)), "bf16",
                         1.5, 0.02, "malter", 3)
    a = Run(wl, check=[])
    b = Run(wl, check=[])
    if schedule == "persistent":
        b.opt.set_ns_schedule(malt.MALT_NS_PERSISTENT)
    g_host = [torch.empty(s, dtype=torch.float32).pin_memory() for s in wl.shapes]
    w_host = [torch.empty(s, dtype=torch.bfloat16).pin_memory() for s in wl.shapes]
    # alternate two device gradient sets, as a pipelining caller does
    G2 = [torch.empty_like(g) for g in b.G]
    sets = [b.params, list(zip(b.W, G2, b.M, b.l, b.r))]
    for step in range(wl.steps):
        for i in range(len(wl.shapes)):
            g_host[i].copy_(torch.from_numpy(inputs.gradient(wl, i, step)))
        a.step(oracle=False)
        b.opt.step_host(b.hp, g_host, w_host, malter=True, params=sets[step % 2])
        assert a.status() == malt.MALT_OK and b.opt.check() == malt.MALT_OK
        for i in range(len(wl.shapes)):
            assert torch.equal(a.W[i], b.W[i])
            assert torch.equal(w_host[i], b.W[i].cpu())
            for x, y in ((a.M[i], b.M[i]), (a.l[i], b.l[i]), (a.r[i], b.r[i])):
                assert torch.equal(x, y)
    a.close()
    b.close()


def test_host_buffer_steps_run_ahead_over_three_gradient_sets():
    """Six malt_step_host calls queued without a synchronisation in between,
    rotating three device gradient sets (each copy-in must wait for the steps
    that last read its set, also once the set has left the two remembered
    slots) and one pinned gradient buffer per step: the final W, M, l, r
    equal six device steps on the same gradients, bitwise."""
    import numpy as np
    import torch
    wl = inputs.Workload("hostrun", 44, ((256, 512), (392, 136), (520, 1544)), "f32", 1.5, 0.02,
                         "malter", 6)
    a = Run(wl, check=[])
    b = Run(wl, check=[])
    g_host = [[torch.from_numpy(inputs.gradient(wl, i, step)).pin_memory()
               for i in range(len(wl.shapes))] for step in range(wl.steps)]
    w_host = [[torch.empty(s, dtype=torch.float32).pin_memory() for s in wl.shapes]
              for _ in range(wl.steps)]
    sets = [b.params] + [list(zip(b.W, [torch.empty_like(g) for g in b.G], b.M, b.l, b.r))
                         for _ in range(2)]
    for step in range(wl.steps):
        a.step(oracle=False)
        b.opt.step_host(b.hp, g_host[step], w_host[step], malter=True, params=sets[step % 3])
    assert a.status() == malt.MALT_OK and b.opt.check() == malt.MALT_OK
    for i in range(len(wl.shapes)):
        assert torch.equal(a.W[i], b.W[i])
        assert torch.equal(w_host[-1][i], b.W[i].cpu())
        for x, y in ((a.M[i], b.M[i]), (a.l[i], b.l[i]), (a.r[i], b.r[i])):
            assert torch.equal(x, y)
    a.close()
    b.close()


def test_step_replays_from_a_cuda_graph():
    """A step enqueues no host synchronisation and no allocation, so it can
    be captured into a CUDA graph; replays advance the device-side step
    counter and give bitwise the same state as eager steps."""
    import torch
    wl = inputs.Workload("graph", 43, ((256, 512), (392, 136)), "f32", 1.5, 0.02, "malter", 3)
    a = Run(wl, check=[])
    b = Run(wl, check=[])
    grads = [inputs.gradient(wl, i, 0) for i in range(2)]
    for run in (a, b):
        for i in range(2):
            run.G[i].copy_(torch.from_numpy(grads[i]))
    torch.cuda.synchronize()
    for _ in range(3):
        a.opt.step(a.hp, malter=True)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(s):
        with torch.cuda.graph(graph, stream=s):
            b.opt.step(b.hp, malter=True, stream=s)
    torch.cuda.synchronize()
    # Capturing records the work without running it; replay three steps.
    for _ in range(3):
        graph.replay()
    torch.cuda.synchronize()
    assert a.opt.check() == malt.MALT_OK and b.opt.check() == malt.MALT_OK
    for i in range(2):
        for x, y in ((a.W[i], b.W[i]), (a.M[i], b.M[i]), (a.l[i], b.l[i]), (a.r[i], b.r[i])):
            assert torch.equal(x, y)
    nu_a, t_a = a.opt.scalars()
    nu_b, t_b = b.opt.scalars()
    assert t_a == t_b == 3 and np.array_equal(nu_a, nu_b)
    a.close()
    b.close()
