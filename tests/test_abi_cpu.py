"""The C ABI library loads, exports every entry point include/lrar.h declares,
and rejects bad arguments before touching the GPU (no compute calls here)."""
import ctypes
import os
import re

import pytest

from paper_2607_09694_gb300 import build as lrar_build
from paper_2607_09694_gb300 import lrar

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
FAKE = 1 << 20  # a 16-byte aligned address that is never dereferenced
EPS = 1e-6


@pytest.fixture(scope="module")
def lib():
    lrar_build.build()
    return lrar.load()


def _declared(header="lrar.h"):
    text = open(os.path.join(ROOT, "include", header)).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(lrar_[a-z0-9_]+)\s*\(", text)))


def _all_declared():
    headers = sorted(f for f in os.listdir(os.path.join(ROOT, "include")) if f.endswith(".h"))
    return sorted(set(n for h in headers for n in _declared(h)))


def test_every_declared_symbol_is_exported(lib):
    assert set(_declared("lrar.h")) == set(lrar.EXPORTS)
    assert set(_declared("lrar_testing.h")) == set(lrar.TEST_HOOKS)
    for n in _all_declared():
        assert hasattr(lib, n), n


def test_only_declared_symbols_are_exported(lib):
    import subprocess

    out = subprocess.run(["nm", "-D", "--defined-only", lrar.LIB_PATH], capture_output=True, text=True).stdout
    syms = {line.split()[-1] for line in out.splitlines() if " T " in line}
    assert syms == set(_all_declared())


def test_version_and_strings(lib):
    assert lib.lrar_version() == 2
    for code in (0, -1, -2, -3, -4, -5):
        assert lib.lrar_strerror(code)
    assert b"unknown" in lib.lrar_strerror(-99)


def fwd(lib, variant=1, ind=1, outd=1, values=FAKE, keys=None, query=FAKE, n=4, T=8, d=64, r=4, eps=EPS, h=FAKE,
        lse=None):
    return lib.lrar_forward(variant, ind, outd, values, keys, query, n, T, d, r, eps, h, lse, None)


def bwd(lib, variant=1, ind=1, gd=1, values=FAKE, keys=None, query=FAKE, n=4, T=8, d=64, r=4, eps=EPS, dh=FAKE,
        h=None, hd=1, lse=None, dv=FAKE, dk=None, dq=FAKE, acc=0, ws=FAKE, wsb=None, st=None):
    if wsb is None:
        wsb = lib.lrar_backward_workspace_size(variant, n, T, d, r)
    return lib.lrar_backward(variant, ind, gd, values, keys, query, n, T, d, r, eps, dh, h, hd, lse, dv, dk, dq, acc,
                             ws, wsb, st, None)


@pytest.mark.parametrize("kw,code", [
    (dict(variant=3), lrar.ERR_INVALID_ARG),
    (dict(ind=2), lrar.ERR_INVALID_ARG),
    (dict(outd=7), lrar.ERR_INVALID_ARG),
    (dict(n=0), lrar.ERR_INVALID_ARG),
    (dict(n=129), lrar.ERR_UNSUPPORTED),
    (dict(T=-1), lrar.ERR_INVALID_ARG),
    (dict(r=0), lrar.ERR_INVALID_ARG),
    (dict(r=65, d=64), lrar.ERR_INVALID_ARG),
    (dict(variant=0, r=4), lrar.ERR_INVALID_ARG),
    (dict(eps=0.0), lrar.ERR_INVALID_ARG),
    (dict(eps=-1.0), lrar.ERR_INVALID_ARG),
    (dict(eps=float("inf")), lrar.ERR_INVALID_ARG),
    (dict(eps=float("nan")), lrar.ERR_INVALID_ARG),
    (dict(values=None), lrar.ERR_INVALID_ARG),
    (dict(h=None), lrar.ERR_INVALID_ARG),
    (dict(query=None), lrar.ERR_INVALID_ARG),
    (dict(variant=2, keys=None), lrar.ERR_INVALID_ARG),
    (dict(values=FAKE + 8), lrar.ERR_ALIGNMENT),
    (dict(h=FAKE + 4), lrar.ERR_ALIGNMENT),
    (dict(query=FAKE + 2), lrar.ERR_ALIGNMENT),
    (dict(d=60), lrar.ERR_ALIGNMENT),
    (dict(d=4096, r=16), lrar.ERR_UNSUPPORTED),
    (dict(ind=0, d=2048, r=16), lrar.ERR_UNSUPPORTED),
])
def test_forward_rejects(lib, kw, code):
    assert fwd(lib, **kw) == code
    assert lib.lrar_last_error()


def test_forward_empty_is_noop(lib):
    assert fwd(lib, T=0, values=None, h=None) == lrar.OK


@pytest.mark.parametrize("kw,code", [
    (dict(gd=5), lrar.ERR_INVALID_ARG),
    (dict(acc=2), lrar.ERR_INVALID_ARG),
    (dict(dq=None), lrar.ERR_INVALID_ARG),
    (dict(dv=None), lrar.ERR_INVALID_ARG),
    (dict(dh=None), lrar.ERR_INVALID_ARG),
    (dict(variant=2, keys=FAKE, dk=None), lrar.ERR_INVALID_ARG),
    (dict(variant=0, d=64, r=64, h=FAKE, lse=None), lrar.ERR_INVALID_ARG),
    (dict(variant=0, d=64, r=64, h=None, lse=FAKE), lrar.ERR_INVALID_ARG),
    (dict(variant=0, d=64, r=64, h=FAKE, lse=FAKE, hd=3), lrar.ERR_INVALID_ARG),
    (dict(ws=None), lrar.ERR_WORKSPACE),
    (dict(wsb=16), lrar.ERR_WORKSPACE),
    (dict(ws=FAKE + 8), lrar.ERR_ALIGNMENT),
    (dict(dv=FAKE + 2), lrar.ERR_ALIGNMENT),
    (dict(st=FAKE + 2), lrar.ERR_ALIGNMENT),
    (dict(n=200), lrar.ERR_UNSUPPORTED),
])
def test_backward_rejects(lib, kw, code):
    assert bwd(lib, **kw) == code


def test_workspace_size_is_device_independent(lib):
    assert lib.lrar_backward_workspace_size(1, 49, 16384, 1024, 16) == 1024 * 16 * 4
    assert lib.lrar_backward_workspace_size(0, 49, 16384, 1024, 1024) == 1024 * 1024 * 4
    assert lib.lrar_backward_workspace_size(2, 1, 1, 64, 0) == 0


def test_diagnostics_rejects(lib):
    f = lib.lrar_diagnostics
    ws = lib.lrar_diagnostics_workspace_size(4)
    assert ws == 1024 * 4 * 4
    assert f(1, 1, FAKE, None, FAKE, 0, 8, 64, 4, EPS, FAKE, FAKE, FAKE, ws, None) == lrar.ERR_INVALID_ARG
    assert f(1, 1, None, None, FAKE, 4, 8, 64, 4, EPS, FAKE, None, None, 0, None) == lrar.ERR_INVALID_ARG
    assert f(2, 1, FAKE, None, FAKE, 4, 8, 64, 4, EPS, FAKE, None, None, 0, None) == lrar.ERR_INVALID_ARG
    assert f(1, 1, FAKE, None, FAKE, 4, 8, 64, 4, EPS, FAKE, FAKE, None, 0, None) == lrar.ERR_WORKSPACE
    assert f(1, 1, FAKE, None, FAKE, 4, 8, 64, 4, EPS, FAKE, FAKE, FAKE, 16, None) == lrar.ERR_WORKSPACE
    assert f(1, 1, FAKE + 8, None, FAKE, 4, 8, 64, 4, EPS, FAKE, None, None, 0, None) == lrar.ERR_ALIGNMENT
    assert f(1, 1, FAKE, None, FAKE, 4, 8, 64, 4, EPS, None, None, None, 0, None) == lrar.OK  # nothing asked


def test_block_accumulate_rejects(lib):
    f = lib.lrar_block_accumulate
    assert f(3, FAKE, 1, FAKE, 10, 1.0, 1.0, None) == lrar.ERR_INVALID_ARG
    assert f(1, FAKE, 1, FAKE, -1, 1.0, 1.0, None) == lrar.ERR_INVALID_ARG
    assert f(1, None, 1, FAKE, 10, 1.0, 1.0, None) == lrar.ERR_INVALID_ARG
    assert f(0, FAKE + 2, 1, FAKE, 10, 1.0, 1.0, None) == lrar.ERR_ALIGNMENT
    assert f(1, FAKE, 1, FAKE, 10, float("nan"), 1.0, None) == lrar.ERR_INVALID_ARG
    assert f(1, None, 1, None, 0, 1.0, 1.0, None) == lrar.OK


def test_last_error_is_per_thread(lib):
    import threading

    assert fwd(lib, n=0) == lrar.ERR_INVALID_ARG
    seen = {}

    def other():
        seen["msg"] = lib.lrar_last_error()

    t = threading.Thread(target=other)
    t.start()
    t.join()
    assert seen["msg"] == b""
    assert b"n_src" in lib.lrar_last_error()


def test_binding_raises_typed_error(lib):
    import torch

    v = torch.zeros(2, 4, 64)
    with pytest.raises(lrar.LrarError) as ei:
        lrar.forward("sliced", v, None, torch.zeros(4), torch.zeros(4, 64), n_src=0)
    assert ei.value.code == lrar.ERR_INVALID_ARG


def test_missing_library_fails_loudly(tmp_path):
    with pytest.raises(RuntimeError, match="missing"):
        lrar.load(str(tmp_path / "nope.so"))


def test_project_rejects(lib):
    f = lib.lrar_project
    assert f(0, FAKE, FAKE, 8, 64, 64, 16, FAKE, FAKE, None, None) == lrar.ERR_UNSUPPORTED   # float32 operands
    assert f(5, FAKE, FAKE, 8, 64, 64, 16, FAKE, FAKE, None, None) == lrar.ERR_INVALID_ARG   # unknown dtype
    assert f(1, FAKE, FAKE, 8, 64, 0, 0, None, None, None, None) == lrar.ERR_INVALID_ARG    # d + r == 0
    assert f(1, FAKE, FAKE, 8, 0, 64, 16, FAKE, FAKE, None, None) == lrar.ERR_INVALID_ARG   # m == 0
    assert f(1, FAKE, FAKE, 8, 60, 64, 16, FAKE, FAKE, None, None) == lrar.ERR_ALIGNMENT    # m % 8
    assert f(1, FAKE, FAKE, 8, 64, 64, 12, FAKE, FAKE, None, None) == lrar.ERR_ALIGNMENT    # r % 8
    assert f(1, None, FAKE, 8, 64, 64, 16, FAKE, FAKE, None, None) == lrar.ERR_INVALID_ARG
    assert f(1, FAKE, FAKE, 8, 64, 64, 16, None, FAKE, None, None) == lrar.ERR_INVALID_ARG  # o needed when d > 0
    assert f(1, FAKE + 8, FAKE, 8, 64, 64, 16, FAKE, FAKE, None, None) == lrar.ERR_ALIGNMENT
    assert f(1, FAKE, FAKE, 0, 64, 64, 16, FAKE, FAKE, None, None) == lrar.OK                # T == 0: no-op


def test_pointer_tables_rejected_before_launch(lib):
    import ctypes as C

    T, d, r, n = 8, 64, 4, 3
    good = (C.c_void_p * n)(FAKE, FAKE + 4096, FAKE + 8192)
    null_entry = (C.c_void_p * n)(FAKE, None, FAKE)
    odd_entry = (C.c_void_p * n)(FAKE, FAKE + 8, FAKE)
    f = lib.lrar_forward_ptrs
    assert f(1, 1, 1, None, None, FAKE, n, T, d, r, EPS, FAKE, None, None) == lrar.ERR_INVALID_ARG
    assert f(1, 1, 1, null_entry, None, FAKE, n, T, d, r, EPS, FAKE, None, None) == lrar.ERR_INVALID_ARG
    assert f(1, 1, 1, odd_entry, None, FAKE, n, T, d, r, EPS, FAKE, None, None) == lrar.ERR_ALIGNMENT
    assert f(2, 1, 1, good, None, FAKE, n, T, d, r, EPS, FAKE, None, None) == lrar.ERR_INVALID_ARG  # P-LR keys
    assert f(1, 1, 1, good, None, FAKE, 0, T, d, r, EPS, FAKE, None, None) == lrar.ERR_INVALID_ARG  # n_src
    assert f(1, 1, 1, None, None, FAKE, n, 0, d, r, EPS, None, None, None) == lrar.OK  # T == 0
    b = lib.lrar_backward_ptrs
    ws = lib.lrar_backward_workspace_size(1, n, T, d, r)
    assert b(1, 1, 1, good, None, FAKE, n, T, d, r, EPS, FAKE, None, 1, None, None, None, FAKE, 0, FAKE, ws,
             None, None) == lrar.ERR_INVALID_ARG  # dvalues table
    assert b(1, 1, 1, good, None, FAKE, n, T, d, r, EPS, FAKE, None, 1, None, odd_entry, None, FAKE, 0, FAKE, ws,
             None, None) == lrar.ERR_ALIGNMENT
    assert b(1, 1, 1, good, None, FAKE, n, T, d, r, EPS, FAKE, None, 1, None, good, None, FAKE, 0, FAKE, 16,
             None, None) == lrar.ERR_WORKSPACE


def test_binding_rejects_host_and_strided_tensors(lib):
    """The binding hands the library device addresses only: a host tensor or a
    non-contiguous view is refused before any call (no GPU needed to check)."""
    import torch

    v = torch.zeros(2, 4, 64)
    with pytest.raises(lrar.LrarError) as ei:
        lrar.forward("sliced", v, None, torch.zeros(4), torch.zeros(4, 64), n_src=2)
    assert ei.value.code == lrar.ERR_INVALID_ARG
    assert "CUDA" in str(ei.value)


def _no_cuda_device():
    try:
        import torch

        return not torch.cuda.is_available()
    except Exception:  # pragma: no cover
        return True


@pytest.mark.skipif(not _no_cuda_device(), reason="needs a machine without a usable CUDA device")
def test_cuda_failures_surface_as_lrar_err_cuda(lib):
    """A CUDA runtime failure (here: no usable device or driver) is reported as
    LRAR_ERR_CUDA with the CUDA error's name in the thread's message.  Only run
    where no device exists: the arguments are placeholder addresses."""
    assert fwd(lib) == lrar.ERR_CUDA
    assert b"cuda" in lib.lrar_last_error().lower()
    assert bwd(lib) == lrar.ERR_CUDA
    assert lib.lrar_project(1, FAKE, FAKE, 8, 64, 64, 16, FAKE, FAKE, None, None) == lrar.ERR_CUDA


def test_plain_c_client_compiles_links_and_runs(lib, tmp_path):
    """tests/c_client.c includes include/lrar.h as C11 (-pedantic -Werror),
    links against liblrar.so and gets INVALID_ARG back with a message."""
    import shutil
    import subprocess

    if shutil.which("gcc") is None:
        pytest.skip("no C compiler")
    exe = str(tmp_path / "c_client")
    libdir = os.path.dirname(lrar.LIB_PATH)
    subprocess.run(["gcc", "-std=c11", "-Wall", "-Wextra", "-pedantic", "-Werror", "-I", os.path.join(ROOT, "include"),
                    os.path.join(ROOT, "tests", "c_client.c"), "-L", libdir, "-llrar", f"-Wl,-rpath,{libdir}",
                    "-o", exe], check=True)
    out = subprocess.run([exe], capture_output=True, text=True)
    assert out.returncode == 0, out.stdout + out.stderr
    assert "invalid argument" in out.stdout


@pytest.mark.parametrize("kw", [
    dict(gd=5), dict(acc=2), dict(dq=None), dict(dv=None), dict(dh=None), dict(n=0), dict(eps=0.0), dict(st=FAKE + 1),
    dict(variant=2, keys=FAKE, dk=None), dict(variant=0, d=64, r=64, h=FAKE, lse=None), dict(dv=FAKE + 2),
    dict(n=200),
])
def test_noalloc_rejects_like_the_workspace_backward(lib, kw):
    """lrar_backward_noalloc runs lrar_backward's argument checks before it
    looks up its scratch on the device: a bad call returns the same code and
    message as lrar_backward, with or without a device present."""
    code = bwd(lib, **kw)
    msg = lib.lrar_last_error()
    assert code < 0
    a = dict(variant=1, ind=1, gd=1, values=FAKE, keys=None, query=FAKE, n=4, T=8, d=64, r=4, eps=EPS, dh=FAKE,
             h=None, hd=1, lse=None, dv=FAKE, dk=None, dq=FAKE, acc=0, st=None)
    a.update(kw)
    got = lib.lrar_backward_noalloc(a["variant"], a["ind"], a["gd"], a["values"], a["keys"], a["query"], a["n"],
                                    a["T"], a["d"], a["r"], a["eps"], a["dh"], a["h"], a["hd"], a["lse"], a["dv"],
                                    a["dk"], a["dq"], a["acc"], a["st"], None)
    assert got == code
    assert lib.lrar_last_error() == msg


def test_block_phase1_rejects(lib):
    f = lib.lrar_block_phase1
    args = [1, 1, 1, FAKE, None, FAKE, 4, 8, 16, 64, 8, EPS, FAKE, FAKE]
    assert f(*args, FAKE + 2, None) == lrar.ERR_ALIGNMENT           # status
    assert f(0, *args[1:], None, None) == lrar.ERR_UNSUPPORTED     # full keys
    bad = list(args)
    bad[7] = 0
    assert f(*bad, None, None) == lrar.ERR_INVALID_ARG             # n_sites
    bad = list(args)
    bad[3] = None
    assert f(*bad, None, None) == lrar.ERR_INVALID_ARG             # values
    bad = list(args)
    bad[8] = 0
    bad[3] = None
    assert f(*bad, None, None) == lrar.OK                          # T == 0


def test_test_hooks_reject(lib):
    t = lib.lrar_test_project_tile
    assert t(0, 1, FAKE, FAKE, 8, 64, 64, 16, FAKE, FAKE, None, None) == lrar.ERR_INVALID_ARG
    assert t(200, 1, FAKE, FAKE, 8, 64, 64, 16, FAKE, FAKE, None, None) == lrar.ERR_INVALID_ARG
    assert t(160, 1, FAKE, FAKE, 0, 64, 64, 16, FAKE, FAKE, None, None) == lrar.OK  # T == 0
    assert t(2176, 1, FAKE, FAKE, 0, 64, 64, 16, FAKE, FAKE, None, None) == lrar.OK  # CTA-pair form, T == 0
    assert t(2200, 1, FAKE, FAKE, 8, 64, 64, 16, FAKE, FAKE, None, None) == lrar.ERR_INVALID_ARG
    s = lib.lrar_test_block_phase1_stalled
    args = [1, 1, 1, FAKE, None, FAKE, 4, 8, 16, 64, 8, EPS, FAKE, FAKE]
    assert s(*args, None, 1000, None) == lrar.ERR_INVALID_ARG      # status required
    assert s(*args, FAKE, 0, None) == lrar.ERR_INVALID_ARG         # wait bound
    assert s(*args[:9], 64, 7, EPS, FAKE, FAKE, FAKE, 1000, None) == lrar.ERR_UNSUPPORTED  # r = 7: no staging


def test_block_phase2_rejects(lib):
    """Both phase-2 entries check their arguments before any device work."""
    p2 = lib.lrar_block_phase2
    args = [1, 1, 1, 1, FAKE, FAKE, FAKE, None, FAKE, 16, 64, 8, EPS, FAKE, FAKE]
    assert p2(0, *args[1:], None) == lrar.ERR_UNSUPPORTED                         # full keys
    bad = list(args)
    bad[6] = None
    assert p2(*bad, None) == lrar.ERR_INVALID_ARG                                 # partial
    bad = list(args)
    bad[6] = FAKE + 4
    assert p2(*bad, None) == lrar.ERR_ALIGNMENT                                   # partial alignment
    bad = list(args)
    bad[9] = 0
    bad[6] = None
    assert p2(*bad, None) == lrar.OK                                              # T == 0
    pa = lib.lrar_block_phase2_assemble
    args = [1, 1, 1, 1, FAKE, FAKE, FAKE, FAKE, None, None, FAKE, 16, 64, 8, EPS, FAKE, FAKE]
    assert pa(0, *args[1:], None) == lrar.ERR_UNSUPPORTED                         # full keys
    bad = list(args)
    bad[6] = None
    assert pa(*bad, None) == lrar.ERR_INVALID_ARG                                 # prev_partial
    assert b"prev_partial" in lib.lrar_last_error()
    bad = list(args)
    bad[6] = FAKE + 4
    assert pa(*bad, None) == lrar.ERR_ALIGNMENT                                   # prev_partial alignment
    bad = list(args)
    bad[7] = None
    assert pa(*bad, None) == lrar.ERR_INVALID_ARG                                 # member
    proj = [2] + args[1:]
    proj[9] = FAKE
    assert pa(*proj, None) == lrar.ERR_INVALID_ARG                                # projected: prev key
    bad = list(args)
    bad[11] = 0
    bad[6] = bad[7] = None
    assert pa(*bad, None) == lrar.OK                                              # T == 0
