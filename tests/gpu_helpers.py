"""Shared helpers of the GPU parity tests: run the C-ABI path on a site's
inputs, run the oracle on the same inputs, and compare."""
from __future__ import annotations

import json
import os

import numpy as np
import torch

import oracle
from paper_2607_09694_gb300 import lrar

EPS = lrar.DEFAULT_EPS
ORACLE_VARIANT = {"full": oracle.FULL, "sliced": oracle.SLICED, "projected": oracle.PROJECTED}
TORCH_DTYPE = {"f32": torch.float32, "bf16": torch.bfloat16}


def rms(a) -> float:
    a = np.asarray(a, dtype=np.float64)
    return float(np.sqrt(np.mean(a * a))) if a.size else 0.0


def max_err(got, ref) -> float:
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    return float(np.max(np.abs(got - ref))) if ref.size else 0.0


def record(name, err, ref, tol):
    """Append one comparison (test, tensor, max abs error, largest exact value,
    bound) to the JSON-lines file named by LRAR_PARITY_LOG, when that is set:
    the measured errors behind the tolerances."""
    path = os.environ.get("LRAR_PARITY_LOG")
    if not path:
        return
    ref = np.asarray(ref, dtype=np.float64)
    line = dict(test=os.environ.get("PYTEST_CURRENT_TEST", "").split(" ")[0], tensor=name, err=float(err),
                max_ref=float(np.max(np.abs(ref))) if ref.size else 0.0, size=int(ref.size), tol=float(tol))
    with open(path, "a") as f:
        f.write(json.dumps(line) + "\n")


def assert_abs(name, got, ref, tol=1e-4):
    e = max_err(got, ref)
    record(name, e, ref, tol)
    assert e <= tol, f"{name}: max abs err {e:.3e} > {tol:.1e}"


U32 = 2.0 ** -24  # unit roundoff of float32 (round to nearest)


def dq_chain(n: int, T: int) -> int:
    """Longest chain of float32 additions a term of dq passes through in the
    backward kernels: each warp holds m = ceil(T / (8 P)) tokens of the P CTAs
    (P = min(ceil(T / 8), CTAs resident) >= min(ceil(T / 8), 152) for one warp
    per token), sums a token's n source terms ((n + 1) m roundings with its
    running sum), combines lanes in at most 5 butterfly steps, the CTA adds
    its 8 warps, and the reduction adds the P CTA partials in CTA order."""
    w = -(-T // 8)
    m = -(-T // (8 * min(w, 152)))
    return (n + 1) * m + 5 + 8 + min(w, 1024)


def assert_dq(name, got, ref, dq_abs, n, T, init=None):
    """Query gradient with float32 storage.  dq is a sum over all T tokens and
    n sources: at |dq| of several hundred one float32 spacing already exceeds
    half of a flat 1e-4, so the bound adds the rounding bound of that sum,
    L u sum |terms| (L = dq_chain(n, T) additions, u = 2^-24, the magnitudes of
    the terms from the oracle); an accumulated initial value adds one rounding."""
    ref = np.asarray(ref, dtype=np.float64)
    mag = np.asarray(dq_abs, dtype=np.float64)
    chain = dq_chain(n, T)
    if init is not None:
        mag = mag + np.abs(np.asarray(init, dtype=np.float64))
        chain += 1
    tol = 1e-4 + chain * U32 * mag
    err = np.abs(np.asarray(got, dtype=np.float64) - ref)
    record(name, float(err.max()) if err.size else 0.0, ref, float(tol.max()) if tol.size else 1e-4)
    bad = err > tol
    assert not bad.any(), (f"{name}: {int(bad.sum())} coordinates beyond 1e-4 + {chain} u sum|terms|, worst "
                           f"err {float(err.max()):.3e} (bound there {float(tol[np.argmax(err)]):.3e})")


def assert_rms(name, got, ref, frac=1e-2):
    e, r = max_err(got, ref), rms(ref)
    assert e <= frac * r, f"{name}: max abs err {e:.3e} > {frac:g} x RMS {r:.3e}"


def bf16_ulp(x):
    """Spacing of bfloat16 numbers at |x| (8 significant bits)."""
    x = np.abs(np.asarray(x, dtype=np.float64))
    _, e = np.frexp(np.where(x > 0, x, 1.0))
    return np.where(x > 0, np.ldexp(1.0, e - 8), np.ldexp(1.0, -133))


def assert_bf16_rounded(name, got, ref, ulps=1.0):
    """A bfloat16 output equals the exact value up to `ulps` bfloat16 spacings
    (plus 1e-5 x RMS for results that cancel to near zero)."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    tol = ulps * bf16_ulp(ref) + 1e-5 * rms(ref)
    bad = np.abs(got - ref) > tol
    assert not bad.any(), (f"{name}: {int(bad.sum())} elements beyond {ulps} ulp, worst "
                           f"{float(np.max(np.abs(got - ref) - tol)):.3e}")


def sample_tokens(T: int, k: int = 48, seed: int = 0) -> np.ndarray:
    """Edges, warp/CTA boundaries of the persistent grid, and random tokens."""
    pts = {0, 1, 7, 8, 9, 255, 256, T - 1, T - 2, T // 2}
    for g in (152, 304, 456, 608):
        pts.update({g * 8 - 1, g * 8, g * 8 + 1})
    rng = np.random.default_rng(seed)
    pts.update(int(t) for t in rng.choice(T, size=min(k, T), replace=False))
    return np.array(sorted(t for t in pts if 0 <= t < T), dtype=np.int64)


def run_gpu(si, out_dtype="f32", grad_dtype="f32", accumulate=False, init=None, n_src=None, eps=EPS,
            stream=None, tokens=None, bwd_lse=True):
    """Forward + backward of one site through the C ABI.  `init` (dict of CPU
    tensors dvalues/dkeys/dq) seeds the gradient buffers when accumulating;
    otherwise they start as NaN so that any element left unwritten shows.
    With `tokens`, only those token rows of h / lse / dvalues / dkeys come back.
    bwd_lse=False calls the backward without the forward's lse (the sliced
    backward then routes first and finishes the key slices in a second pass)."""
    dev = torch.device("cuda")
    n = si.n if n_src is None else n_src
    v = si.values.to(dev)
    k = si.keys.to(dev) if si.keys is not None else None
    q = si.query.to(dev)
    dh = si.dh.to(dev)
    T, d = si.T, si.d
    h = torch.empty(T, d, dtype=TORCH_DTYPE[out_dtype], device=dev)
    lse = torch.empty(T, dtype=torch.float32, device=dev)
    gdt = TORCH_DTYPE[grad_dtype]
    rq = d if si.variant == "full" else si.r
    if accumulate:
        dv = init["dvalues"].to(dev, gdt).clone()
        dk = init["dkeys"].to(dev, gdt).clone() if k is not None else None
        dq = init["dq"].to(dev, torch.float32).clone()
    else:
        dv = torch.full((si.values.shape[0], T, d), float("nan"), dtype=gdt, device=dev)
        dk = torch.full((si.keys.shape[0], T, si.r), float("nan"), dtype=gdt, device=dev) if k is not None else None
        dq = torch.full((rq,), float("nan"), dtype=torch.float32, device=dev)
    ws = torch.empty(max(1, lrar.workspace_size(si.variant, n, T, d, si.r) // 4), dtype=torch.float32, device=dev)
    lrar.forward(si.variant, v, k, q, h, lse, n_src=n, r=si.r, eps=eps, stream=stream)
    lrar.backward(si.variant, v, k, q, dh, dv, dq, ws, dkeys=dk, h=h, lse=lse if bwd_lse else None, n_src=n, r=si.r,
                  accumulate=accumulate, eps=eps, stream=stream)
    torch.cuda.synchronize()
    if tokens is not None:
        idx = torch.as_tensor(tokens, dtype=torch.long, device=dev)
        h, lse, dv = h.index_select(0, idx), lse.index_select(0, idx), dv.index_select(1, idx)
        dk = dk.index_select(1, idx) if dk is not None else None
    out = dict(h=h.double().cpu().numpy(), lse=lse.double().cpu().numpy(), dvalues=dv.double().cpu().numpy(),
               dq=dq.double().cpu().numpy())
    if dk is not None:
        out["dkeys"] = dk.double().cpu().numpy()
    return out


def run_oracle(si, tokens=None, n_src=None, eps=EPS, want_dvalues=True):
    n = si.n if n_src is None else n_src
    ov = ORACLE_VARIANT[si.variant]
    vals = si.values[:n]
    keys = si.keys[:n] if si.keys is not None else None
    f = oracle.forward(ov, vals, keys, si.query, eps, r=si.r, tokens=tokens)
    b = oracle.backward(ov, vals, keys, si.query, eps, si.dh, r=si.r, tokens=tokens, want_dvalues=want_dvalues)
    return dict(h=f["h"], lse=f["lse"], dvalues=b["dvalues"], dkeys=b["dkeys"], dq=b["dq"], dq_abs=b["dq_abs"])
