"""fp64 CPU oracle for the Low-Rank Attention Residuals depth mix.

TEST INFRASTRUCTURE ONLY: the plain, slow, obviously-correct statement of what
the GPU library computes, written in C (``lrar_oracle.c``) from the paper's
equations (Eq. 8-10 for the mix, Eq. 14 for sliced keys, Eq. 2 for AttnRes
keys, Eq. 5-6 for Block AttnRes summaries, Eq. 16 for N_eff).  Only the test
suite, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline leg may
import it.  The product package never does, and the two share no code.

Inputs may be numpy arrays (float64 / float32, or uint16 holding raw bfloat16
words) or CPU torch tensors (float64 / float32 / bfloat16).  Outputs are numpy
float64 arrays.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

FULL, SLICED, PROJECTED = 0, 1, 2
_F64, _F32, _BF16 = 0, 1, 2

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "lrar_oracle.c")
_SO = os.path.join(_HERE, "liblrar_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (OpenMP, no fast-math) and return the .so path."""
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < os.path.getmtime(_SRC):
        tmp = _SO + f".tmp{os.getpid()}"
        subprocess.check_call(
            ["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", _SRC, "-o", tmp, "-lm"]
        )
        os.replace(tmp, _SO)
    return _SO


def _load():
    global _lib
    with _lock:
        if _lib is None:
            # LRAR_ORACLE_LIB points the tests' mutation check at a deliberately broken build.
            lib = ctypes.CDLL(os.environ.get("LRAR_ORACLE_LIB") or build())
            vp, i64p, dp = ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p
            i, i64, dbl = ctypes.c_int, ctypes.c_int64, ctypes.c_double
            lib.oracle_forward.argtypes = [i, i, vp, vp, dp, i, i64, i, i, dbl, i64p, i64, dp, dp, dp]
            lib.oracle_backward.argtypes = [i, i, vp, vp, dp, i, i64, i, i, dbl, vp, i64p, i64, dp, dp, dp, dp, dp]
            lib.oracle_diagnostics.argtypes = [i, i, vp, vp, dp, i, i64, i, i, dbl, i64p, i64, dp, dp]
            lib.oracle_block_sources.argtypes = [i, vp, i, i64, i, i, dp]
            lib.oracle_block_fanout.argtypes = [dp, i, i64, i, i, dp]
            lib.oracle_block_num_sources.argtypes = [i, i]
            lib.oracle_full_num_sources.argtypes = [i]
            lib.oracle_set_threads.argtypes = [i]
            lib.oracle_projection.argtypes = [i, vp, vp, i64, i, i, i64p, i64, dp]
            lib.oracle_set_threads.restype = None
            for f in (lib.oracle_forward, lib.oracle_backward, lib.oracle_diagnostics,
                      lib.oracle_block_sources, lib.oracle_block_fanout,
                      lib.oracle_block_num_sources, lib.oracle_full_num_sources, lib.oracle_get_threads,
                      lib.oracle_projection):
                f.restype = ctypes.c_int
            _lib = lib
    return _lib


def set_threads(n: int) -> None:
    _load().oracle_set_threads(int(n))


def get_threads() -> int:
    return int(_load().oracle_get_threads())


def _as_array(a):
    """Return (contiguous numpy array, element-type code) without changing any value."""
    if a is None:
        return None, _F64
    try:
        import torch

        if isinstance(a, torch.Tensor):
            a = a.detach().cpu().contiguous()
            if a.dtype == torch.bfloat16:
                return a.view(torch.int16).numpy().view(np.uint16), _BF16
            if a.dtype == torch.float32:
                return a.numpy(), _F32
            if a.dtype == torch.float64:
                return a.numpy(), _F64
            raise TypeError(f"unsupported tensor dtype {a.dtype}")
    except ImportError:  # pragma: no cover
        pass
    a = np.ascontiguousarray(a)
    if a.dtype == np.float64:
        return a, _F64
    if a.dtype == np.float32:
        return a, _F32
    if a.dtype == np.uint16:
        return a, _BF16
    raise TypeError(f"unsupported array dtype {a.dtype}")


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _tok(tokens, T):
    if tokens is None:
        return None, T
    t = np.ascontiguousarray(np.asarray(tokens, dtype=np.int64))
    return t, t.size


def _query(q):
    qa, _ = _as_array(q)
    return np.ascontiguousarray(qa.astype(np.float64))


def forward(variant, values, keys, q, eps, r=None, tokens=None, want_alpha=False):
    """Eq. (8)-(10): returns dict(h [n_tok,d], lse [n_tok], alpha [n_tok,n] or None)."""
    va, dt = _as_array(values)
    ka, kdt = _as_array(keys)
    if ka is not None and kdt != dt:
        raise TypeError("values and keys must share an element type")
    n, T, d = va.shape
    if r is None:
        r = ka.shape[-1] if variant == PROJECTED else d
    qa = _query(q)
    tk, n_tok = _tok(tokens, T)
    h = np.zeros((n_tok, d))
    lse = np.zeros(n_tok)
    alpha = np.zeros((n_tok, n)) if want_alpha else None
    rc = _load().oracle_forward(variant, dt, _ptr(va), _ptr(ka), _ptr(qa), n, T, d, r, float(eps),
                                _ptr(tk), n_tok, _ptr(h), _ptr(lse), _ptr(alpha))
    if rc != 0:
        raise ValueError("oracle_forward rejected its arguments")
    return {"h": h, "lse": lse, "alpha": alpha}


def backward(variant, values, keys, q, eps, dh, r=None, tokens=None, want_dvalues=True, want_ds=False):
    """Gradients of sum <dh, h>: dict(dvalues [n,n_tok,d], dkeys [n,n_tok,r], dq [r], ds [n_tok,n],
    dq_abs [r]).  dq_abs[j] = sum over tokens and sources of |ds_i kbar_ij|, the
    magnitude of the terms that dq[j] sums (what bounds the rounding of that sum)."""
    va, dt = _as_array(values)
    ka, kdt = _as_array(keys)
    da, ddt = _as_array(dh)
    if (ka is not None and kdt != dt) or ddt != dt:
        raise TypeError("values, keys and dh must share an element type")
    n, T, d = va.shape
    if r is None:
        r = ka.shape[-1] if variant == PROJECTED else d
    qa = _query(q)
    tk, n_tok = _tok(tokens, T)
    dv = np.zeros((n, n_tok, d)) if want_dvalues else None
    dk = np.zeros((n, n_tok, r)) if variant == PROJECTED else None
    dq = np.zeros(r)
    dq_abs = np.zeros(r)
    ds = np.zeros((n_tok, n)) if want_ds else None
    rc = _load().oracle_backward(variant, dt, _ptr(va), _ptr(ka), _ptr(qa), n, T, d, r, float(eps), _ptr(da),
                                 _ptr(tk), n_tok, _ptr(dv), _ptr(dk), _ptr(dq), _ptr(ds), _ptr(dq_abs))
    if rc != 0:
        raise ValueError("oracle_backward rejected its arguments")
    return {"dvalues": dv, "dkeys": dk, "dq": dq, "ds": ds, "dq_abs": dq_abs}


def diagnostics(variant, values, keys, q, eps, r=None, tokens=None):
    """Eq. (16) N_eff per token and the token-mean of alpha (heatmap row)."""
    va, dt = _as_array(values)
    ka, _ = _as_array(keys)
    n, T, d = va.shape
    if r is None:
        r = ka.shape[-1] if variant == PROJECTED else d
    qa = _query(q)
    tk, n_tok = _tok(tokens, T)
    neff = np.zeros(n_tok)
    mean_alpha = np.zeros(n)
    rc = _load().oracle_diagnostics(variant, dt, _ptr(va), _ptr(ka), _ptr(qa), n, T, d, r, float(eps),
                                    _ptr(tk), n_tok, _ptr(neff), _ptr(mean_alpha))
    if rc != 0:
        raise ValueError("oracle_diagnostics rejected its arguments")
    return {"neff": neff, "mean_alpha": mean_alpha}


def full_num_sources(t: int) -> int:
    return int(_load().oracle_full_num_sources(int(t)))


def block_num_sources(t: int, c: int) -> int:
    return int(_load().oracle_block_num_sources(int(t), int(c)))


def block_sources(outputs, c: int):
    """Eq. (5)-(6): stack [o_0, b_1, ..., b_P] from outputs [t, T, w] (o_0..o_{t-1})."""
    oa, dt = _as_array(outputs)
    t, T, w = oa.shape
    nt = block_num_sources(t, c)
    out = np.zeros((nt, T, w))
    rc = _load().oracle_block_sources(dt, _ptr(oa), t, T, w, int(c), _ptr(out))
    if rc != nt:
        raise ValueError("oracle_block_sources rejected its arguments")
    return out


def block_fanout(dsources, t: int, c: int):
    """Gradient of the Block assembly: dsources [n_t, T, w] -> doutputs [t, T, w]."""
    ds = np.ascontiguousarray(np.asarray(dsources, dtype=np.float64))
    _, T, w = ds.shape
    out = np.zeros((t, T, w))
    rc = _load().oracle_block_fanout(_ptr(ds), int(t), T, w, int(c), _ptr(out))
    if rc != 0:
        raise ValueError("oracle_block_fanout rejected its arguments")
    return out


def projection(a, w, d: int, tokens=None):
    """Eq. (11)-(12): [o; k] = [W_O; W_K] a per token; a [T, m], w [d + r, m].
    Returns dict(o [n_tok, d], keys [n_tok, r]) in float64."""
    aa, dt = _as_array(a)
    wa, wdt = _as_array(w)
    if wdt != dt:
        raise TypeError("a and w must have the same element type")
    T, m = aa.shape
    nrows = wa.shape[0]
    if wa.shape[1] != m or not 0 <= d <= nrows:
        raise ValueError("w must be [d + r, m]")
    tk, n_tok = _tok(tokens, T)
    y = np.zeros((n_tok, nrows))
    rc = _load().oracle_projection(dt, _ptr(aa), _ptr(wa), T, m, nrows, _ptr(tk), n_tok, _ptr(y))
    if rc != 0:
        raise ValueError("oracle_projection rejected its arguments")
    return {"o": y[:, :d], "keys": y[:, d:]}
