"""Python binding of liblrar.so (include/lrar.h): argument marshalling only.

Every function takes CUDA tensors (or raw integer device pointers), turns them
into the C ABI's pointers, sizes and type codes, and calls the library on the
current torch stream.  All arithmetic happens in the library's CUDA kernels;
there is no fallback, and a missing or unbuilt library raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

FULL, SLICED, PROJECTED = 0, 1, 2
F32, BF16 = 0, 1
VARIANTS = {"full": FULL, "sliced": SLICED, "projected": PROJECTED}
MAX_SOURCES = 128
DEFAULT_EPS = 1e-6

OK = 0
ERR_INVALID_ARG, ERR_ALIGNMENT, ERR_UNSUPPORTED, ERR_CUDA, ERR_WORKSPACE = -1, -2, -3, -4, -5
STATUS_WAIT_TIMEOUT, STATUS_LSE_MISMATCH = 1, 2  # bits of the optional device status words

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "liblrar.so")
EXPORTS = ("lrar_forward", "lrar_backward", "lrar_backward_workspace_size", "lrar_block_accumulate",
           "lrar_strerror", "lrar_last_error", "lrar_version", "lrar_backward_noalloc", "lrar_diagnostics",
           "lrar_diagnostics_workspace_size", "lrar_block_phase1", "lrar_block_phase2", "lrar_project",
           "lrar_forward_ptrs", "lrar_backward_ptrs", "lrar_block_phase1_ptrs", "lrar_block_phase2_assemble")
TEST_HOOKS = ("lrar_test_project_tile", "lrar_test_block_phase1_stalled")  # include/lrar_testing.h
MAX_BLOCK_SITES = 64

_lock = threading.Lock()
_lib = None


class LrarError(RuntimeError):
    def __init__(self, code: int, message: str):
        super().__init__(f"{message} (status {code})")
        self.code = code


def load(path: str | None = None):
    """Load liblrar.so; raises if it has not been built."""
    global _lib
    with _lock:
        if _lib is not None and path is None:
            return _lib
        p = path or LIB_PATH
        if not os.path.exists(p):
            raise RuntimeError(f"{p} is missing: build it with `python -c 'import __graft_entry__ as g; g.build()'`")
        lib = ctypes.CDLL(p)
        vp, i, i64, f32, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t
        lib.lrar_forward.argtypes = [i, i, i, vp, vp, vp, i, i64, i, i, f32, vp, vp, vp]
        lib.lrar_forward.restype = i
        lib.lrar_backward.argtypes = [i, i, i, vp, vp, vp, i, i64, i, i, f32, vp, vp, i, vp, vp, vp, vp, i, vp, sz, vp,
                                      vp]
        lib.lrar_backward.restype = i
        lib.lrar_backward_noalloc.argtypes = [i, i, i, vp, vp, vp, i, i64, i, i, f32, vp, vp, i, vp, vp, vp, vp, i, vp,
                                              vp]
        lib.lrar_backward_noalloc.restype = i
        lib.lrar_block_phase1.argtypes = [i, i, i, vp, vp, vp, i, i, i64, i, i, f32, vp, vp, vp, vp]
        lib.lrar_block_phase1.restype = i
        lib.lrar_block_phase1_ptrs.argtypes = [i, i, i, vp, vp, vp, i, i, i64, i, i, f32, vp, vp, vp, vp]
        lib.lrar_block_phase1_ptrs.restype = i
        lib.lrar_test_block_phase1_stalled.argtypes = [i, i, i, vp, vp, vp, i, i, i64, i, i, f32, vp, vp, vp,
                                                       ctypes.c_longlong, vp]
        lib.lrar_test_block_phase1_stalled.restype = i
        lib.lrar_test_project_tile.argtypes = [i, i, vp, vp, i64, i, i, i, vp, vp, vp, vp]
        lib.lrar_test_project_tile.restype = i
        lib.lrar_block_phase2.argtypes = [i, i, i, i, vp, vp, vp, vp, vp, i64, i, i, f32, vp, vp, vp]
        lib.lrar_block_phase2.restype = i
        lib.lrar_block_phase2_assemble.argtypes = [i, i, i, i, vp, vp, vp, vp, vp, vp, vp, i64, i, i, f32, vp, vp,
                                                   vp]
        lib.lrar_block_phase2_assemble.restype = i
        lib.lrar_diagnostics.argtypes = [i, i, vp, vp, vp, i, i64, i, i, f32, vp, vp, vp, sz, vp]
        lib.lrar_diagnostics.restype = i
        lib.lrar_diagnostics_workspace_size.argtypes = [i]
        lib.lrar_diagnostics_workspace_size.restype = sz
        lib.lrar_backward_workspace_size.argtypes = [i, i, i64, i, i]
        lib.lrar_backward_workspace_size.restype = sz
        lib.lrar_forward_ptrs.argtypes = [i, i, i, vp, vp, vp, i, i64, i, i, f32, vp, vp, vp]
        lib.lrar_forward_ptrs.restype = i
        lib.lrar_backward_ptrs.argtypes = [i, i, i, vp, vp, vp, i, i64, i, i, f32, vp, vp, i, vp, vp, vp, vp, i, vp,
                                           sz, vp, vp]
        lib.lrar_backward_ptrs.restype = i
        lib.lrar_project.argtypes = [i, vp, vp, i64, i, i, i, vp, vp, vp, vp]
        lib.lrar_project.restype = i
        lib.lrar_block_accumulate.argtypes = [i, vp, i, vp, i64, f32, f32, vp]
        lib.lrar_block_accumulate.restype = i
        lib.lrar_strerror.argtypes = [i]
        lib.lrar_strerror.restype = ctypes.c_char_p
        lib.lrar_last_error.argtypes = []
        lib.lrar_last_error.restype = ctypes.c_char_p
        lib.lrar_version.argtypes = []
        lib.lrar_version.restype = i
        if path is None:
            _lib = lib
        return lib


def _check(rc: int) -> None:
    if rc != OK:
        lib = load()
        raise LrarError(rc, lib.lrar_last_error().decode() or lib.lrar_strerror(rc).decode())


def dtype_code(t: torch.Tensor | None, default: int = F32) -> int:
    if t is None:
        return default
    if t.dtype == torch.bfloat16:
        return BF16
    if t.dtype == torch.float32:
        return F32
    raise TypeError(f"unsupported dtype {t.dtype}")


def _ptr(t) -> int | None:
    """Device address of a tensor argument (None -> NULL).  Every tensor the
    library reads or writes must be a contiguous CUDA tensor: a host tensor's
    address would be dereferenced on the GPU."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if not t.is_cuda:
        raise LrarError(ERR_INVALID_ARG, "tensor arguments must be CUDA tensors")
    if not t.is_contiguous():
        raise LrarError(ERR_INVALID_ARG, "tensor arguments must be contiguous")
    return t.data_ptr()


def _stream(stream) -> int | None:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream if torch.cuda.is_available() else None
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _variant(v) -> int:
    return VARIANTS[v] if isinstance(v, str) else int(v)


def forward(variant, values: torch.Tensor, keys: torch.Tensor | None, query: torch.Tensor | None,
            h: torch.Tensor, lse: torch.Tensor | None = None, n_src: int | None = None, r: int | None = None,
            eps: float = DEFAULT_EPS, stream=None) -> None:
    """lrar_forward: h (and lse) of the first n_src sources of the stack `values` [*, T, d]."""
    variant = _variant(variant)
    _, T, d = values.shape
    n = values.shape[0] if n_src is None else n_src
    if r is None:
        r = d if variant == FULL else (keys.shape[-1] if variant == PROJECTED else query.numel())
    _check(load().lrar_forward(variant, dtype_code(values), dtype_code(h), _ptr(values), _ptr(keys), _ptr(query),
                               n, T, d, r, eps, _ptr(h), _ptr(lse), _stream(stream)))


def workspace_size(variant, n_src: int, T: int, d: int, r: int) -> int:
    return int(load().lrar_backward_workspace_size(_variant(variant), n_src, T, d, r))


def backward(variant, values: torch.Tensor, keys: torch.Tensor | None, query: torch.Tensor | None,
             dh: torch.Tensor, dvalues: torch.Tensor, dq: torch.Tensor, workspace: torch.Tensor,
             dkeys: torch.Tensor | None = None, h: torch.Tensor | None = None, lse: torch.Tensor | None = None,
             n_src: int | None = None, r: int | None = None, accumulate: bool = False,
             eps: float = DEFAULT_EPS, status: torch.Tensor | None = None, stream=None) -> None:
    """lrar_backward for the first n_src sources of `values`; gradients go to the
    first n_src slices of `dvalues` (and `dkeys`).  status: optional int32
    device scalar that collects STATUS_LSE_MISMATCH."""
    variant = _variant(variant)
    _, T, d = values.shape
    n = values.shape[0] if n_src is None else n_src
    if r is None:
        r = d if variant == FULL else (keys.shape[-1] if variant == PROJECTED else query.numel())
    ws_bytes = workspace.numel() * workspace.element_size()
    _check(load().lrar_backward(variant, dtype_code(values), dtype_code(dvalues), _ptr(values), _ptr(keys),
                                _ptr(query), n, T, d, r, eps, _ptr(dh), _ptr(h), dtype_code(h), _ptr(lse),
                                _ptr(dvalues), _ptr(dkeys), _ptr(dq), int(bool(accumulate)), _ptr(workspace),
                                ws_bytes, _ptr(status), _stream(stream)))


def _table(ts):
    """Host array of device pointers for a list of source tensors (None -> NULL)."""
    if ts is None:
        return None
    return (ctypes.c_void_p * len(ts))(*[_ptr(t) for t in ts])


def forward_ptrs(variant, values, keys, query: torch.Tensor | None, h: torch.Tensor, lse: torch.Tensor | None = None,
                 r: int | None = None, eps: float = DEFAULT_EPS, stream=None) -> None:
    """lrar_forward_ptrs: like forward, with the sources given as a list of
    separate [T, d] tensors (and P-LR keys as a list of [T, r] tensors)."""
    variant = _variant(variant)
    n = len(values)
    T, d = values[0].shape
    if r is None:
        r = d if variant == FULL else (keys[0].shape[-1] if variant == PROJECTED else query.numel())
    _check(load().lrar_forward_ptrs(variant, dtype_code(values[0]), dtype_code(h), _table(values), _table(keys),
                                    _ptr(query), n, T, d, r, eps, _ptr(h), _ptr(lse), _stream(stream)))


def backward_ptrs(variant, values, keys, query: torch.Tensor | None, dh: torch.Tensor, dvalues, dq: torch.Tensor,
                  workspace: torch.Tensor, dkeys=None, h: torch.Tensor | None = None, lse: torch.Tensor | None = None,
                  r: int | None = None, accumulate: bool = False, eps: float = DEFAULT_EPS,
                  status: torch.Tensor | None = None, stream=None) -> None:
    """lrar_backward_ptrs: like backward, with sources and their gradients as
    lists of separate tensors (gradient i goes to dvalues[i], dkeys[i])."""
    variant = _variant(variant)
    n = len(values)
    T, d = values[0].shape
    if r is None:
        r = d if variant == FULL else (keys[0].shape[-1] if variant == PROJECTED else query.numel())
    ws_bytes = workspace.numel() * workspace.element_size()
    _check(load().lrar_backward_ptrs(variant, dtype_code(values[0]), dtype_code(dvalues[0]), _table(values),
                                     _table(keys), _ptr(query), n, T, d, r, eps, _ptr(dh), _ptr(h), dtype_code(h),
                                     _ptr(lse), _table(dvalues), _table(dkeys), _ptr(dq), int(bool(accumulate)),
                                     _ptr(workspace), ws_bytes, _ptr(status), _stream(stream)))


def backward_noalloc(variant, values: torch.Tensor, keys: torch.Tensor | None, query: torch.Tensor | None,
                     dh: torch.Tensor, dvalues: torch.Tensor, dq: torch.Tensor, dkeys: torch.Tensor | None = None,
                     h: torch.Tensor | None = None, lse: torch.Tensor | None = None, n_src: int | None = None,
                     r: int | None = None, accumulate: bool = False, eps: float = DEFAULT_EPS,
                     status: torch.Tensor | None = None, stream=None) -> None:
    """lrar_backward_noalloc: lrar_backward without a workspace, for callers
    that cannot allocate device memory (scratch is the library's fixed 4 MiB
    array per device; calls that may overlap on the GPU race on it)."""
    variant = _variant(variant)
    _, T, d = values.shape
    n = values.shape[0] if n_src is None else n_src
    if r is None:
        r = d if variant == FULL else (keys.shape[-1] if variant == PROJECTED else query.numel())
    _check(load().lrar_backward_noalloc(variant, dtype_code(values), dtype_code(dvalues), _ptr(values), _ptr(keys),
                                        _ptr(query), n, T, d, r, eps, _ptr(dh), _ptr(h), dtype_code(h), _ptr(lse),
                                        _ptr(dvalues), _ptr(dkeys), _ptr(dq), int(bool(accumulate)),
                                        _ptr(status), _stream(stream)))


def block_phase1(variant, values: torch.Tensor, keys: torch.Tensor | None, queries: torch.Tensor,
                 h_pre: torch.Tensor, lse_pre: torch.Tensor, n_completed: int | None = None,
                 eps: float = DEFAULT_EPS, status: torch.Tensor | None = None, stream=None) -> None:
    """lrar_block_phase1: mixes of the first n_completed sources of `values` for
    every query row of `queries` [n_sites, r] -> h_pre [n_sites, T, d], lse_pre [n_sites, T].
    status: optional int32 device scalar that collects STATUS_WAIT_TIMEOUT."""
    variant = _variant(variant)
    _, T, d = values.shape
    n = values.shape[0] if n_completed is None else n_completed
    c, r = queries.shape
    _check(load().lrar_block_phase1(variant, dtype_code(values), dtype_code(h_pre), _ptr(values), _ptr(keys),
                                    _ptr(queries), n, c, T, d, r, eps, _ptr(h_pre), _ptr(lse_pre), _ptr(status),
                                    _stream(stream)))


def block_phase1_ptrs(variant, values, keys, queries: torch.Tensor, h_pre: torch.Tensor, lse_pre: torch.Tensor,
                      eps: float = DEFAULT_EPS, status: torch.Tensor | None = None, stream=None) -> None:
    """lrar_block_phase1_ptrs: block_phase1 with the completed sources as a list
    of separate [T, d] tensors (and P-LR keys as a list of [T, r] tensors)."""
    variant = _variant(variant)
    n = len(values)
    T, d = values[0].shape
    c, r = queries.shape
    _check(load().lrar_block_phase1_ptrs(variant, dtype_code(values[0]), dtype_code(h_pre), _table(values),
                                         _table(keys), _ptr(queries), n, c, T, d, r, eps, _ptr(h_pre),
                                         _ptr(lse_pre), _ptr(status), _stream(stream)))


def block_phase2(variant, h_pre: torch.Tensor, lse_pre: torch.Tensor, partial: torch.Tensor,
                 partial_key: torch.Tensor | None, query: torch.Tensor, h: torch.Tensor,
                 lse: torch.Tensor | None = None, eps: float = DEFAULT_EPS, stream=None) -> None:
    """lrar_block_phase2: one site's mix = phase-1 result (+) its partial-block summary."""
    variant = _variant(variant)
    T, d = partial.shape
    r = query.numel()
    _check(load().lrar_block_phase2(variant, dtype_code(partial), dtype_code(h_pre), dtype_code(h), _ptr(h_pre),
                                    _ptr(lse_pre), _ptr(partial), _ptr(partial_key), _ptr(query), T, d, r, eps,
                                    _ptr(h), _ptr(lse), _stream(stream)))


def block_phase2_assemble(variant, h_pre: torch.Tensor, lse_pre: torch.Tensor, prev_partial: torch.Tensor,
                          member: torch.Tensor, prev_partial_key: torch.Tensor | None, member_key: torch.Tensor | None,
                          query: torch.Tensor, h: torch.Tensor, lse: torch.Tensor | None = None,
                          eps: float = DEFAULT_EPS, stream=None) -> None:
    """lrar_block_phase2_assemble: member := prev_partial + member (the partial
    summary, Eq. 6; keys likewise for P-LR), then the site's mix as block_phase2."""
    variant = _variant(variant)
    T, d = member.shape
    r = query.numel()
    _check(load().lrar_block_phase2_assemble(variant, dtype_code(member), dtype_code(h_pre), dtype_code(h),
                                             _ptr(h_pre), _ptr(lse_pre), _ptr(prev_partial), _ptr(member),
                                             _ptr(prev_partial_key), _ptr(member_key), _ptr(query), T, d, r, eps,
                                             _ptr(h), _ptr(lse), _stream(stream)))


def diagnostics(variant, values: torch.Tensor, keys: torch.Tensor | None, query: torch.Tensor | None,
                neff: torch.Tensor | None = None, mean_alpha: torch.Tensor | None = None,
                workspace: torch.Tensor | None = None, n_src: int | None = None, r: int | None = None,
                eps: float = DEFAULT_EPS, stream=None) -> None:
    """lrar_diagnostics: per-token N_eff [T] and the token-mean of alpha [n_src] (Eq. 16, §4.5-4.6)."""
    variant = _variant(variant)
    _, T, d = values.shape
    n = values.shape[0] if n_src is None else n_src
    if r is None:
        r = d if variant == FULL else (keys.shape[-1] if variant == PROJECTED else query.numel())
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(load().lrar_diagnostics(variant, dtype_code(values), _ptr(values), _ptr(keys), _ptr(query), n, T, d, r,
                                   eps, _ptr(neff), _ptr(mean_alpha), _ptr(workspace), ws_bytes, _stream(stream)))


def diagnostics_workspace_size(n_src: int) -> int:
    return int(load().lrar_diagnostics_workspace_size(n_src))


def block_accumulate(dst: torch.Tensor, src: torch.Tensor, alpha: float = 1.0, beta: float = 1.0,
                     stream=None) -> None:
    """lrar_block_accumulate: dst = beta * dst + alpha * src (beta == 0 does not read dst)."""
    if dst.numel() != src.numel():
        raise ValueError("dst and src sizes differ")
    _check(load().lrar_block_accumulate(dtype_code(dst), _ptr(dst), dtype_code(src), _ptr(src), dst.numel(),
                                        float(alpha), float(beta), _stream(stream)))


def project(a: torch.Tensor, w: torch.Tensor, o: torch.Tensor | None, keys: torch.Tensor | None,
            status: torch.Tensor | None = None, stream=None) -> None:
    """lrar_project: [o ; keys] = [W_O ; W_K] a per token (§3.3, Eq. 11-12).
    a [T, m], w [d + r, m], o [T, d] (None when d = 0), keys [T, r] (None when r = 0),
    all bfloat16; status: optional int32 device scalar set to 1 if the kernel gave up."""
    T, m = a.shape
    d = 0 if o is None else o.shape[-1]
    r = 0 if keys is None else keys.shape[-1]
    if w.shape[0] != d + r or w.shape[-1] != m:
        raise ValueError(f"w must be [{d + r}, {m}], got {tuple(w.shape)}")
    _check(load().lrar_project(dtype_code(a), _ptr(a), _ptr(w), T, m, d, r, _ptr(o), _ptr(keys), _ptr(status),
                               _stream(stream)))


def version() -> int:
    return int(load().lrar_version())


# ------------------------------------------------------------ test hooks ----
# include/lrar_testing.h: variants of the calls above that let the tests reach
# paths ordinary inputs do not choose.  Not part of the library's interface.
def test_project_tile(tile: int, a: torch.Tensor, w: torch.Tensor, o: torch.Tensor | None,
                      keys: torch.Tensor | None, status: torch.Tensor | None = None, stream=None) -> None:
    """lrar_test_project_tile: project() with the tile width forced."""
    T, m = a.shape
    d = 0 if o is None else o.shape[-1]
    r = 0 if keys is None else keys.shape[-1]
    if w.shape[0] != d + r or w.shape[-1] != m:
        raise ValueError(f"w must be [{d + r}, {m}], got {tuple(w.shape)}")
    _check(load().lrar_test_project_tile(int(tile), dtype_code(a), _ptr(a), _ptr(w), T, m, d, r, _ptr(o),
                                         _ptr(keys), _ptr(status), _stream(stream)))


def test_block_phase1_stalled(variant, values: torch.Tensor, keys: torch.Tensor | None, queries: torch.Tensor,
                              h_pre: torch.Tensor, lse_pre: torch.Tensor, status: torch.Tensor, wait_cycles: int,
                              n_completed: int | None = None, eps: float = DEFAULT_EPS, stream=None) -> None:
    """lrar_test_block_phase1_stalled: block_phase1() whose key waits all run out."""
    variant = _variant(variant)
    _, T, d = values.shape
    n = values.shape[0] if n_completed is None else n_completed
    c, r = queries.shape
    _check(load().lrar_test_block_phase1_stalled(variant, dtype_code(values), dtype_code(h_pre), _ptr(values),
                                                 _ptr(keys), _ptr(queries), n, c, T, d, r, eps, _ptr(h_pre),
                                                 _ptr(lse_pre), _ptr(status), int(wait_cycles), _stream(stream)))
