"""Error paths on a live state: bad arguments return codes, a device-side wait
that runs out reports MALT_ERR_TIMEOUT and leaves the context usable."""
import ctypes

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
