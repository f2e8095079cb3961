"""ctypes binding of include/malt.h, names unchanged, argument marshalling only.

Every step of the optimizer runs in libmalt.so's CUDA kernels; this module
turns torch tensors into device pointers and sizes, passes the current CUDA
stream, and raises on non-zero status codes.  Loading fails loudly when the
library has not been built (there is no fallback of any kind).
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from . import build as _build

MALT_OK = 0
MALT_ERR_INVALID_ARG = -1
MALT_ERR_UNSUPPORTED = -2
MALT_ERR_MISALIGNED = -3
MALT_ERR_SHAPE_CHANGED = -4
MALT_ERR_CUDA = -5
MALT_ERR_TIMEOUT = -6
MALT_ERR_OUT_OF_MEMORY = -7
MALT_F32 = 0
MALT_BF16 = 1
SCALARS_PER_MAT = 8

# Exported entry points declared in include/malt.h.
EXPORTS = ("malt_init_state", "malt_step", "malter_step", "malt_get_scalars",
           "malt_set_scalars", "malt_check", "malt_debug_direction", "malt_debug_scalars",
           "malt_debug_wait_timeout", "malt_profile_enable", "malt_profile_read",
           "malt_workspace_bytes", "malt_status_string", "malt_destroy_state",
           "malt_stats_noalloc", "malt_step_host", "muon_step", "malt_set_ns_schedule",
           "malt_ns_schedule", "malt_debug_timeout_site", "malt_debug_precond",
           "malt_set_weight_copies", "malt_adamw_init_state", "malt_adamw_step",
           "malt_adamw_get_step", "malt_adamw_set_step", "malt_adamw_destroy_state",
           "malt_debug_check_guards")
NOALLOC_SCRATCH_FLOATS = 1048576
KIND_NAMES = ("bind", "stats", "finalize", "prescale", "norms", "ns_gram", "ns_poly", "ns_bx",
              "scalars", "apply", "ns_persistent", "pad")
NS_KINDS = ("ns_gram", "ns_poly", "ns_bx", "ns_persistent")
# Newton-Schulz schedules (malt_set_ns_schedule)
MALT_NS_PHASED = 0
MALT_NS_PERSISTENT = 1
MALT_NS_AUTO = 2
# product kinds of malt_ns_schedule
STAGE_KIND_NAMES = ("gram", "poly", "bx")


class malt_param_t(ctypes.Structure):
    _fields_ = [("w", ctypes.c_void_p), ("w_dtype", ctypes.c_int32),
                ("g", ctypes.c_void_p), ("g_dtype", ctypes.c_int32),
                ("m", ctypes.c_void_p), ("l", ctypes.c_void_p), ("r", ctypes.c_void_p),
                ("rows", ctypes.c_int64), ("cols", ctypes.c_int64)]


class malt_hparams_t(ctypes.Structure):
    _fields_ = [("lr", ctypes.c_float), ("mu1", ctypes.c_float), ("mu2", ctypes.c_float),
                ("eps", ctypes.c_float), ("weight_decay", ctypes.c_float),
                ("ns_steps", ctypes.c_int32), ("ns_a", ctypes.c_float),
                ("ns_b", ctypes.c_float), ("ns_c", ctypes.c_float), ("ns_eps", ctypes.c_float)]


class malt_adamw_param_t(ctypes.Structure):
    _fields_ = [("w", ctypes.c_void_p), ("w_copy", ctypes.c_void_p), ("g", ctypes.c_void_p),
                ("g_dtype", ctypes.c_int32), ("m", ctypes.c_void_p), ("v", ctypes.c_void_p),
                ("numel", ctypes.c_int64), ("weight_decay", ctypes.c_float)]


class malt_adamw_hparams_t(ctypes.Structure):
    _fields_ = [("lr", ctypes.c_float), ("beta1", ctypes.c_float), ("beta2", ctypes.c_float),
                ("eps", ctypes.c_float)]


class MaltError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        super().__init__(f"{where}: {status_string(code)} ({code})")


_LIB = None


def library_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = False) -> ctypes.CDLL:
    """Load libmalt.so (built by build.build()).  Raises if it is missing."""
    global _LIB
    if _LIB is not None:
        return _LIB
    path = library_path()
    if not os.path.exists(path):
        if not build_if_missing:
            raise RuntimeError(f"libmalt.so not built ({path}); run paper_2608_05088_gb300.build.build()")
        _build.build()
    lib = ctypes.CDLL(path)
    vp, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    P = ctypes.POINTER
    lib.malt_init_state.argtypes = [P(vp), P(malt_param_t), i32, vp]
    lib.malt_step.argtypes = [vp, P(malt_param_t), i32, P(malt_hparams_t), vp]
    lib.malter_step.argtypes = [vp, P(malt_param_t), i32, P(malt_hparams_t), vp]
    lib.malt_get_scalars.argtypes = [vp, P(ctypes.c_float), i32, P(i64)]
    lib.malt_set_scalars.argtypes = [vp, P(ctypes.c_float), i32, i64]
    lib.malt_check.argtypes = [vp]
    lib.malt_debug_direction.argtypes = [vp, i32, vp, vp]
    lib.malt_debug_precond.argtypes = [vp, i32, vp, vp, vp]
    lib.malt_debug_precond.restype = ctypes.c_int
    lib.malt_debug_scalars.argtypes = [vp, P(ctypes.c_float), i32]
    lib.malt_debug_wait_timeout.argtypes = [i64, vp]
    lib.malt_profile_enable.argtypes = [vp, i32]
    lib.malt_profile_read.argtypes = [vp, P(ctypes.c_double), P(i64), i32]
    lib.malt_workspace_bytes.argtypes = [vp]
    lib.malt_workspace_bytes.restype = ctypes.c_size_t
    lib.malt_status_string.argtypes = [ctypes.c_int]
    lib.malt_status_string.restype = ctypes.c_char_p
    lib.malt_destroy_state.argtypes = [vp]
    lib.malt_destroy_state.restype = None
    lib.muon_step.argtypes = [vp, P(malt_param_t), i32, P(malt_hparams_t), vp]
    lib.muon_step.restype = ctypes.c_int
    lib.malt_step_host.argtypes = [vp, P(malt_param_t), i32, P(malt_hparams_t), i32,
                                   P(vp), P(vp), vp]
    lib.malt_step_host.restype = ctypes.c_int
    f32 = ctypes.c_float
    lib.malt_stats_noalloc.argtypes = [vp, i32, vp, vp, vp, vp, vp, i64, i64, f32, f32, f32, vp]
    lib.malt_stats_noalloc.restype = ctypes.c_int
    lib.malt_debug_timeout_site.argtypes = [vp, P(i32)]
    lib.malt_debug_timeout_site.restype = ctypes.c_int
    lib.malt_set_ns_schedule.argtypes = [vp, i32]
    lib.malt_set_ns_schedule.restype = ctypes.c_int
    lib.malt_ns_schedule.argtypes = [P(malt_param_t), i32, i32, P(i32), i64, P(i64)]
    lib.malt_debug_check_guards.argtypes = [vp, P(i64)]
    lib.malt_debug_check_guards.restype = ctypes.c_int
    lib.malt_set_weight_copies.argtypes = [vp, P(vp), i32]
    lib.malt_set_weight_copies.restype = ctypes.c_int
    lib.malt_adamw_init_state.argtypes = [P(vp), P(malt_adamw_param_t), i32, vp]
    lib.malt_adamw_init_state.restype = ctypes.c_int
    lib.malt_adamw_step.argtypes = [vp, P(malt_adamw_param_t), i32, P(malt_adamw_hparams_t), vp]
    lib.malt_adamw_step.restype = ctypes.c_int
    lib.malt_adamw_get_step.argtypes = [vp, P(i64)]
    lib.malt_adamw_get_step.restype = ctypes.c_int
    lib.malt_adamw_set_step.argtypes = [vp, i64]
    lib.malt_adamw_set_step.restype = ctypes.c_int
    lib.malt_adamw_destroy_state.argtypes = [vp]
    lib.malt_adamw_destroy_state.restype = None
    lib.malt_ns_schedule.restype = ctypes.c_int
    for name in ("malt_init_state", "malt_step", "malter_step", "malt_get_scalars",
                 "malt_set_scalars", "malt_check", "malt_debug_direction",
                 "malt_debug_scalars", "malt_debug_wait_timeout", "malt_profile_enable",
                 "malt_profile_read"):
        getattr(lib, name).restype = ctypes.c_int
    _LIB = lib
    return lib


def status_string(code: int) -> str:
    return load().malt_status_string(int(code)).decode()


def _check(code: int, where: str):
    if code != MALT_OK:
        raise MaltError(code, where)


def hparams(lr=0.02, mu1=0.95, mu2=0.99, eps=1e-8, weight_decay=0.0, ns_steps=5,
            ns_coeffs=(3.4445, -4.7750, 2.0315), ns_eps=1e-7) -> malt_hparams_t:
    a, b, c = ns_coeffs
    return malt_hparams_t(lr, mu1, mu2, eps, weight_decay, ns_steps, a, b, c, ns_eps)


def _dtype_code(t) -> int:
    import torch
    if t.dtype == torch.float32:
        return MALT_F32
    if t.dtype == torch.bfloat16:
        return MALT_BF16
    raise TypeError(f"unsupported dtype {t.dtype}")


def params_array(params):
    """params: sequence of (W, G, M, l, r) CUDA tensors -> ctypes array."""
    arr = (malt_param_t * max(len(params), 1))()
    for i, (W, G, M, l, r) in enumerate(params):
        for t in (W, G, M, l, r):
            if not t.is_contiguous():
                raise ValueError("all tensors must be contiguous")
        rows, cols = W.shape
        arr[i] = malt_param_t(W.data_ptr(), _dtype_code(W), G.data_ptr(), _dtype_code(G),
                              M.data_ptr(), l.data_ptr(), r.data_ptr(), rows, cols)
    return arr


def _stream_handle(stream=None):
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


# --- C-ABI names ------------------------------------------------------------

def malt_init_state(params, stream=None) -> ctypes.c_void_p:
    lib = load()
    st = ctypes.c_void_p()
    arr = params_array(params)
    _check(lib.malt_init_state(ctypes.byref(st), arr, len(params), _stream_handle(stream)),
           "malt_init_state")
    return st


def malt_step(st, params, hp: malt_hparams_t, stream=None):
    arr = params_array(params)
    _check(load().malt_step(st, arr, len(params), ctypes.byref(hp), _stream_handle(stream)),
           "malt_step")


def malter_step(st, params, hp: malt_hparams_t, stream=None):
    arr = params_array(params)
    _check(load().malter_step(st, arr, len(params), ctypes.byref(hp), _stream_handle(stream)),
           "malter_step")


def muon_step(st, params, hp: malt_hparams_t, stream=None):
    arr = params_array(params)
    _check(load().muon_step(st, arr, len(params), ctypes.byref(hp), _stream_handle(stream)),
           "muon_step")


def malt_step_host(st, params, hp: malt_hparams_t, g_host, w_host, malter=False, stream=None):
    """Step with gradients from host tensors g_host[i] (pinned) into the device
    buffers of params, and updated weights copied back into host tensors
    w_host[i]; valid after malt_check."""
    arr = params_array(params)
    n = len(params)
    gp = (ctypes.c_void_p * max(n, 1))(*[t.data_ptr() for t in g_host])
    wp = (ctypes.c_void_p * max(n, 1))(*[t.data_ptr() for t in w_host])
    _check(load().malt_step_host(st, arr, n, ctypes.byref(hp), 1 if malter else 0, gp, wp,
                                 _stream_handle(stream)), "malt_step_host")


def malt_check(st) -> int:
    return load().malt_check(st)


def malt_get_scalars(st, n: int):
    nu = (ctypes.c_float * max(n, 1))()
    t = ctypes.c_int64()
    _check(load().malt_get_scalars(st, nu, n, ctypes.byref(t)), "malt_get_scalars")
    return np.array(nu[:n], dtype=np.float32), int(t.value)


def malt_set_scalars(st, nu, t: int):
    n = len(nu)
    arr = (ctypes.c_float * max(n, 1))(*[float(x) for x in nu])
    _check(load().malt_set_scalars(st, arr, n, int(t)), "malt_set_scalars")


def malt_debug_direction(st, idx: int, out, stream=None):
    _check(load().malt_debug_direction(st, idx, ctypes.c_void_p(out.data_ptr()),
                                       _stream_handle(stream)), "malt_debug_direction")


def malt_debug_precond(st, idx: int, L_out, R_out, stream=None):
    _check(load().malt_debug_precond(st, idx, ctypes.c_void_p(L_out.data_ptr()),
                                     ctypes.c_void_p(R_out.data_ptr()), _stream_handle(stream)),
           "malt_debug_precond")


def malt_debug_check_guards(st) -> int:
    """Corrupted bytes in the workspace's guard regions (0 when no kernel
    wrote past its buffers)."""
    bad = ctypes.c_int64()
    _check(load().malt_debug_check_guards(st, ctypes.byref(bad)), "malt_debug_check_guards")
    return int(bad.value)


def malt_debug_scalars(st, n: int) -> np.ndarray:
    buf = (ctypes.c_float * max(n * SCALARS_PER_MAT, 1))()
    _check(load().malt_debug_scalars(st, buf, n), "malt_debug_scalars")
    return np.array(buf[: n * SCALARS_PER_MAT], dtype=np.float32).reshape(n, SCALARS_PER_MAT)


def malt_debug_wait_timeout(budget_ns: int, stream=None) -> int:
    return load().malt_debug_wait_timeout(int(budget_ns), _stream_handle(stream))


def malt_profile_enable(st, enable: bool = True):
    _check(load().malt_profile_enable(st, 1 if enable else 0), "malt_profile_enable")


def malt_profile_read(st):
    """{kind: (milliseconds, launches)} accumulated since the last read."""
    n = len(KIND_NAMES)
    ms = (ctypes.c_double * n)()
    cnt = (ctypes.c_int64 * n)()
    _check(load().malt_profile_read(st, ms, cnt, n), "malt_profile_read")
    return {KIND_NAMES[k]: (float(ms[k]), int(cnt[k])) for k in range(n)}


def _noalloc_check(G, M, l, r, L_out, R_out):
    """The tensors malt_stats_noalloc hands to its kernels as raw pointers:
    contiguous, on the current CUDA device, with the shapes and dtypes the
    kernels index (M rows x cols fp32, G the same shape in fp32 or bf16, l and
    L_out rows fp32, r and R_out cols fp32).  Raises ValueError otherwise."""
    import torch
    if M.dim() != 2:
        raise ValueError("M must be a 2-D rows x cols tensor")
    rows, cols = M.shape
    want = {"G": (G, (rows, cols), (torch.float32, torch.bfloat16)),
            "M": (M, (rows, cols), (torch.float32,)),
            "l": (l, (rows,), (torch.float32,)), "L_out": (L_out, (rows,), (torch.float32,)),
            "r": (r, (cols,), (torch.float32,)), "R_out": (R_out, (cols,), (torch.float32,))}
    for name, (t, shape, dtypes) in want.items():
        if tuple(t.shape) != shape:
            raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {shape}")
        if t.dtype not in dtypes:
            raise ValueError(f"{name} has dtype {t.dtype}, expected one of {dtypes}")
        if not t.is_contiguous():
            raise ValueError(f"{name} must be contiguous")
    for name, (t, _, _) in want.items():
        if not t.is_cuda:
            raise ValueError(f"{name} must be a CUDA tensor, not on {t.device}")
    dev = torch.cuda.current_device()
    for name, (t, _, _) in want.items():
        if t.device.index != dev:
            raise ValueError(f"{name} must be on the current CUDA device (cuda:{dev}), not {t.device}")
    return rows, cols


def malt_stats_noalloc(G, M, l, r, L_out, R_out, mu1=0.95, mu2=0.99, eps=1e-8, stream=None) -> int:
    """Statistics stage of one matrix with no device allocation (see
    include/malt.h).  Checks the tensors (ValueError on a mismatch), then
    returns the library's status code without raising, so callers can see
    MALT_ERR_UNSUPPORTED for matrices past the scratch limit."""
    rows, cols = _noalloc_check(G, M, l, r, L_out, R_out)
    return load().malt_stats_noalloc(
        ctypes.c_void_p(G.data_ptr()), _dtype_code(G), ctypes.c_void_p(M.data_ptr()),
        ctypes.c_void_p(l.data_ptr()), ctypes.c_void_p(r.data_ptr()),
        ctypes.c_void_p(L_out.data_ptr()), ctypes.c_void_p(R_out.data_ptr()),
        rows, cols, mu1, mu2, eps, _stream_handle(stream))


def malt_set_weight_copies(st, copies, n: int):
    """copies: one bf16 CUDA tensor (the shape of its fp32 W) or None for each
    of the state's n parameters, or None to clear all."""
    if copies is None:
        _check(load().malt_set_weight_copies(st, None, n), "malt_set_weight_copies")
        return
    for c in copies:
        if c is not None and (not c.is_contiguous() or _dtype_code(c) != MALT_BF16):
            raise ValueError("weight copies must be contiguous bf16 tensors")
    arr = (ctypes.c_void_p * max(len(copies), 1))(
        *[None if c is None else c.data_ptr() for c in copies])
    _check(load().malt_set_weight_copies(st, arr, len(copies)), "malt_set_weight_copies")


def adamw_hparams(lr=1e-3, betas=(0.9, 0.95), eps=1e-8) -> malt_adamw_hparams_t:
    return malt_adamw_hparams_t(lr, betas[0], betas[1], eps)


def adamw_params_array(params):
    """params: sequence of (w, w_copy or None, g, m, v, weight_decay) CUDA
    tensors (w, m, v fp32; w_copy bf16) -> ctypes array."""
    arr = (malt_adamw_param_t * max(len(params), 1))()
    for i, (w, wc, g, m, v, wd) in enumerate(params):
        for t in (w, g, m, v) + (() if wc is None else (wc,)):
            if not t.is_contiguous():
                raise ValueError("all tensors must be contiguous")
        n = w.numel()
        if any(t.numel() != n for t in (g, m, v)) or (wc is not None and wc.numel() != n):
            raise ValueError("w, w_copy, g, m and v must have the same number of elements")
        import torch
        if w.dtype != torch.float32 or m.dtype != torch.float32 or v.dtype != torch.float32:
            raise ValueError("w, m and v must be float32")
        if wc is not None and wc.dtype != torch.bfloat16:
            raise ValueError("w_copy must be bfloat16")
        arr[i] = malt_adamw_param_t(w.data_ptr(), None if wc is None else wc.data_ptr(),
                                    g.data_ptr(), _dtype_code(g), m.data_ptr(), v.data_ptr(),
                                    n, float(wd))
    return arr


def malt_adamw_init_state(params, stream=None) -> ctypes.c_void_p:
    st = ctypes.c_void_p()
    _check(load().malt_adamw_init_state(ctypes.byref(st), adamw_params_array(params), len(params),
                                        _stream_handle(stream)), "malt_adamw_init_state")
    return st


def malt_adamw_step(st, params, hp: malt_adamw_hparams_t, stream=None):
    _check(load().malt_adamw_step(st, adamw_params_array(params), len(params), ctypes.byref(hp),
                                  _stream_handle(stream)), "malt_adamw_step")


def malt_adamw_get_step(st) -> int:
    t = ctypes.c_int64()
    _check(load().malt_adamw_get_step(st, ctypes.byref(t)), "malt_adamw_get_step")
    return int(t.value)


def malt_adamw_set_step(st, t: int):
    _check(load().malt_adamw_set_step(st, int(t)), "malt_adamw_set_step")


def malt_adamw_destroy_state(st):
    load().malt_adamw_destroy_state(st)


def malt_workspace_bytes(st) -> int:
    return int(load().malt_workspace_bytes(st))


def malt_destroy_state(st):
    load().malt_destroy_state(st)


def malt_debug_timeout_site(st):
    """(site, item, seq, block, thread) of the last reported device timeout."""
    out = (ctypes.c_int32 * 5)()
    _check(load().malt_debug_timeout_site(st, out), "malt_debug_timeout_site")
    return tuple(int(v) for v in out)


def malt_set_ns_schedule(st, schedule: int):
    _check(load().malt_set_ns_schedule(st, int(schedule)), "malt_set_ns_schedule")


def malt_ns_schedule(shapes, ns_steps: int):
    """The work table of the persistent schedule for these (rows, cols)
    shapes, computed on the host by the library (no GPU): an int32 array of
    shape (items, 8) with columns launch group, stage, product kind
    (STAGE_KIND_NAMES), matrix, tile, counter index, counter target, tiles of
    (stage, matrix)."""
    import numpy as np
    arr = (malt_param_t * max(len(shapes), 1))()
    for i, (rows, cols) in enumerate(shapes):
        arr[i] = malt_param_t(None, MALT_F32, None, MALT_F32, None, None, None, rows, cols)
    lib = load()
    count = ctypes.c_int64(0)
    _check(lib.malt_ns_schedule(arr, len(shapes), ns_steps, None, 0, ctypes.byref(count)),
           "malt_ns_schedule")
    out = np.zeros((count.value, 8), dtype=np.int32)
    _check(lib.malt_ns_schedule(arr, len(shapes), ns_steps,
                                out.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)),
                                count.value, ctypes.byref(count)), "malt_ns_schedule")
    return out


# --- convenience wrapper ------------------------------------------------------

class MaltOptimizer:
    """Owns a malt_state for a fixed list of (W, G, M, l, r) device tensors.
    M, l, r are zeroed at construction (Algorithm 1 INITIALIZE line)."""

    def __init__(self, params, stream=None):
        self.params = list(params)
        self.n = len(self.params)
        self.state = malt_init_state(self.params, stream)

    def step(self, hp: malt_hparams_t, malter: bool = False, stream=None, params=None,
             muon: bool = False):
        ps = self.params if params is None else params
        if muon:
            muon_step(self.state, ps, hp, stream)
        else:
            (malter_step if malter else malt_step)(self.state, ps, hp, stream)

    def step_host(self, hp: malt_hparams_t, g_host, w_host, malter: bool = False, stream=None,
                  params=None):
        ps = self.params if params is None else params
        malt_step_host(self.state, ps, hp, g_host, w_host, malter, stream)

    def check(self) -> int:
        return malt_check(self.state)

    def scalars(self):
        return malt_get_scalars(self.state, self.n)

    def set_scalars(self, nu, t):
        malt_set_scalars(self.state, nu, t)

    def debug_scalars(self):
        return malt_debug_scalars(self.state, self.n)

    def direction(self, idx: int, stream=None):
        import torch
        W = self.params[idx][0]
        out = torch.empty(W.shape, dtype=torch.bfloat16, device=W.device)
        malt_debug_direction(self.state, idx, out, stream)
        return out

    def precond(self, idx: int, stream=None):
        """(L, R) of parameter idx as the last step computed them."""
        import torch
        W = self.params[idx][0]
        L = torch.empty(W.shape[0], dtype=torch.float32, device=W.device)
        R = torch.empty(W.shape[1], dtype=torch.float32, device=W.device)
        malt_debug_precond(self.state, idx, L, R, stream)
        return L, R

    def guard_bytes_corrupted(self) -> int:
        return malt_debug_check_guards(self.state)

    def timeout_site(self):
        return malt_debug_timeout_site(self.state)

    def set_ns_schedule(self, schedule: int):
        malt_set_ns_schedule(self.state, schedule)

    def set_weight_copies(self, copies):
        malt_set_weight_copies(self.state, copies, self.n)

    def profile(self, enable: bool = True):
        malt_profile_enable(self.state, enable)

    def profile_read(self):
        return malt_profile_read(self.state)

    def workspace_bytes(self) -> int:
        return malt_workspace_bytes(self.state)

    def close(self):
        if self.state is not None:
            malt_destroy_state(self.state)
            self.state = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class AdamW:
    """Owns a malt_adamw_state for a fixed list of (w, w_copy or None, g, m, v,
    weight_decay) device tensors; m and v are zeroed at construction."""

    def __init__(self, params, stream=None):
        self.params = list(params)
        self.state = malt_adamw_init_state(self.params, stream)

    def step(self, hp: malt_adamw_hparams_t, stream=None, params=None):
        malt_adamw_step(self.state, self.params if params is None else params, hp, stream)

    def get_step(self) -> int:
        return malt_adamw_get_step(self.state)

    def set_step(self, t: int):
        malt_adamw_set_step(self.state, t)

    def close(self):
        if self.state is not None:
            malt_adamw_destroy_state(self.state)
            self.state = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class WholeOptimizer:
    """A whole-optimizer step of a model (Section 5.1 parameter grouping):
    MALT or MALTER on the 2-D weight matrices, AdamW on every other tensor,
    both enqueued on the same stream.  matrices: (W, G, M, l, r) as for
    MaltOptimizer (fp32 W for master weights); copies: optional bf16 copy per
    matrix (None entries for none); others: (w, w_copy, g, m, v, weight_decay)
    as for AdamW."""

    def __init__(self, matrices, others, copies=None, stream=None):
        self.malt = MaltOptimizer(matrices, stream)
        if copies is not None:
            self.malt.set_weight_copies(copies)
        self.adamw = AdamW(others, stream)

    def step(self, hp: malt_hparams_t, adamw_hp: malt_adamw_hparams_t, malter: bool = False,
             stream=None):
        self.malt.step(hp, malter=malter, stream=stream)
        self.adamw.step(adamw_hp, stream=stream)

    def check(self) -> int:
        return self.malt.check()

    def close(self):
        self.malt.close()
        self.adamw.close()
