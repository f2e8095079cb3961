"""The C ABI library: builds, loads without a GPU, exports every entry point
include/malt.h declares, and validates arguments on the host (CPU only)."""
import ctypes
import os
import re
import subprocess

import pytest

import paper_2608_05088_gb300.malt as malt
from paper_2608_05088_gb300 import build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def header_functions():
    names = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            src = open(os.path.join(ROOT, "include", fn)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            decl = r"^\s*(?:const\s+)?(?:int|void|size_t|char)\s*\**\s*(\w+)\s*\("
            for m in re.finditer(decl, src, flags=re.M):
                names.add(m.group(1))
    return names


@pytest.fixture(scope="module")
def lib():
    build.build()
    return malt.load()


def test_header_declares_the_binding_names():
    assert header_functions() == set(malt.EXPORTS)


def test_library_exports_every_declared_symbol(lib):
    out = subprocess.run(["nm", "-D", "--defined-only", build.LIB], capture_output=True,
                         text=True, check=True).stdout
    exported = {line.split()[-1] for line in out.splitlines() if " T " in line}
    missing = header_functions() - exported
    assert not missing, missing
    for name in header_functions():
        assert hasattr(lib, name)


def test_status_strings(lib):
    for code in (0, -1, -2, -3, -4, -5, -6, -7):
        assert malt.status_string(code) != "unknown status"
    assert malt.status_string(12345) == "unknown status"


def _param(rows=64, cols=64, w=16, g=16, m=16, l=16, r=16, wd=malt.MALT_F32):
    return malt.malt_param_t(w, wd, g, malt.MALT_F32, m, l, r, rows, cols)


def test_host_validation_without_gpu(lib):
    st = ctypes.c_void_p()
    assert lib.malt_init_state(None, None, 0, None) == malt.MALT_ERR_INVALID_ARG
    assert lib.malt_init_state(ctypes.byref(st), None, -1, None) == malt.MALT_ERR_INVALID_ARG
    cases = [
        (_param(rows=0), malt.MALT_ERR_UNSUPPORTED),
        (_param(cols=-3), malt.MALT_ERR_UNSUPPORTED),
        (_param(rows=65536, cols=65536), malt.MALT_ERR_UNSUPPORTED),
        # 46341 x 46337 < 2^31, but rounded up to multiples of 8 it is not
        (_param(rows=46337, cols=46341), malt.MALT_ERR_UNSUPPORTED),
        (_param(w=0), malt.MALT_ERR_INVALID_ARG),
        (_param(m=24), malt.MALT_ERR_MISALIGNED),
        (_param(wd=7), malt.MALT_ERR_UNSUPPORTED),
    ]
    for p, want in cases:
        arr = (malt.malt_param_t * 1)(p)
        assert lib.malt_init_state(ctypes.byref(st), arr, 1, None) == want
        assert not st.value
    hp = malt.hparams()
    assert lib.malt_step(None, None, 0, ctypes.byref(hp), None) == malt.MALT_ERR_INVALID_ARG
    assert lib.malt_debug_wait_timeout(0, None) == malt.MALT_ERR_INVALID_ARG
    assert lib.malt_workspace_bytes(None) == 0
    lib.malt_destroy_state(None)


def test_noalloc_host_validation_without_gpu(lib):
    """malt_stats_noalloc rejects bad arguments, and matrices whose partial
    sums would not fit its fixed scratch, before it touches the GPU."""
    F32, BF16 = malt.MALT_F32, malt.MALT_BF16

    def call(g=16, dt=F32, m=16, l=16, r=16, L=16, R=16, rows=64, cols=64,
             mu1=0.95, mu2=0.99, eps=1e-8):
        return lib.malt_stats_noalloc(g, dt, m, l, r, L, R, rows, cols, mu1, mu2, eps, None)

    assert call(g=None) == malt.MALT_ERR_INVALID_ARG
    assert call(R=None) == malt.MALT_ERR_INVALID_ARG
    assert call(mu1=1.0) == malt.MALT_ERR_INVALID_ARG
    assert call(mu2=-0.5) == malt.MALT_ERR_INVALID_ARG
    assert call(eps=float("nan")) == malt.MALT_ERR_INVALID_ARG
    assert call(dt=5) == malt.MALT_ERR_UNSUPPORTED
    assert call(rows=0) == malt.MALT_ERR_UNSUPPORTED
    assert call(cols=12) == malt.MALT_ERR_UNSUPPORTED
    assert call(rows=65536, cols=32768) == malt.MALT_ERR_UNSUPPORTED
    assert call(l=24) == malt.MALT_ERR_MISALIGNED
    assert call(dt=BF16, g=40) == malt.MALT_ERR_MISALIGNED
    # ceil(n/256)*m (rounded up to 64) + ceil(m/64)*n floats of scratch
    limit = 1048576

    def need(rows, cols):
        return -(-(-(-cols // 256) * rows) // 64) * 64 + (-(-rows // 64)) * cols

    assert need(8192, 8192) > limit
    assert call(rows=8192, cols=8192) == malt.MALT_ERR_UNSUPPORTED
    assert need(4096, 12800) <= limit < need(4096, 13312)
    assert call(rows=4096, cols=13312) == malt.MALT_ERR_UNSUPPORTED


C_CLIENT = r"""
#include <stdio.h>
#include <string.h>
#include "malt.h"
int main(void) {
    malt_state_t* st = 0;
    malt_param_t p;
    memset(&p, 0, sizeof p);
    if (malt_init_state(0, 0, 0, 0) != MALT_ERR_INVALID_ARG) return 1;
    if (malt_init_state(&st, 0, -1, 0) != MALT_ERR_INVALID_ARG || st) return 2;
    if (malt_init_state(&st, &p, 1, 0) != MALT_ERR_INVALID_ARG || st) return 3;
    if (strcmp(malt_status_string(MALT_OK), malt_status_string(MALT_ERR_CUDA)) == 0) return 4;
    if (malt_workspace_bytes(0) != 0) return 5;
    malt_destroy_state(0);
    printf("%s\n", malt_status_string(MALT_ERR_MISALIGNED));
    return 0;
}
"""


def test_header_is_plain_c_and_links_from_c(lib, tmp_path):
    """include/malt.h is a C header (C99, no C++ constructs) and a C program
    links against libmalt.so and calls it; only calls that fail argument
    checks before touching a GPU are made."""
    import shutil
    if shutil.which("gcc") is None:
        pytest.skip("gcc not available")
    inc = os.path.join(ROOT, "include")
    subprocess.run(["gcc", "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror",
                    "-fsyntax-only", "-x", "c", os.path.join(inc, "malt.h")], check=True)
    src = tmp_path / "client.c"
    src.write_text(C_CLIENT)
    exe = tmp_path / "client"
    libdir = os.path.dirname(build.LIB)
    subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", f"-I{inc}", str(src), f"-L{libdir}",
                    "-lmalt", f"-Wl,-rpath,{libdir}", "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True)
    assert out.returncode == 0, out
    assert out.stdout.strip() == "device pointer not 16-byte aligned"


def test_noalloc_binding_checks_tensors_without_gpu():
    """The binding refuses tensors whose shape, dtype, layout or device would
    make the kernels index past them, before any pointer reaches the library."""
    import torch
    m, n = 16, 24

    def t(*shape, dtype=torch.float32):
        return torch.zeros(shape, dtype=dtype)

    good = dict(G=t(m, n), M=t(m, n), l=t(m), r=t(n), L_out=t(m), R_out=t(n))
    bad_cases = [
        dict(G=t(m, n - 8)),                      # G shorter than M
        dict(l=t(m - 8)),                         # row statistics too short
        dict(R_out=t(n + 8)),                     # wrong length
        dict(M=t(m, n, dtype=torch.bfloat16)),    # bf16 momentum
        dict(G=t(m, n, dtype=torch.float16)),     # unsupported gradient type
        dict(M=t(n, m).t()),                      # right shape, not contiguous
        dict(M=t(m * n)),                         # not 2-D
    ]
    for case in bad_cases:
        args = dict(good, **case)
        with pytest.raises(ValueError):
            malt.malt_stats_noalloc(args["G"], args["M"], args["l"], args["r"],
                                    args["L_out"], args["R_out"])
    # well-formed host tensors are refused too: the library takes device pointers
    with pytest.raises(ValueError, match="CUDA"):
        malt.malt_stats_noalloc(*good.values())
