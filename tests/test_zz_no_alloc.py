"""lrar_backward_noalloc, checked against lrar_backward.

lrar_backward_noalloc is the backward pass for callers that cannot allocate
device memory when they call it -- plugin callbacks that must not allocate
while they run, services held to a fixed device-memory budget, C hosts that
have no device allocator of their own -- and so cannot hand lrar_backward a
workspace.  It uses a fixed scratch array compiled into the library instead.

The file name puts it last in collection, so that a run stopping at the first
failure has already run every other test; it also passes on its own in a
fresh process (the first call on the device does the scratch set-up).
"""
import numpy as np
import pytest
import torch

from paper_2607_09694_gb300 import lrar, synth

pytestmark = pytest.mark.gpu

CASES = [
    dict(config="slr", variant="sliced", n=49, T=1000),
    dict(config="plr", variant="projected", n=17, T=333, r=32),
    dict(config="slr", variant="full", n=9, T=257, d=512),
]


def _site(c):
    kw = {k: v for k, v in c.items() if k not in ("config",)}
    return synth.site(c["config"], **kw)


def _backward(si, noalloc):
    """Forward with the existing entry point, then one backward through either
    lrar_backward (with a workspace) or lrar_backward_noalloc; fp32 gradients."""
    dev = torch.device("cuda")
    v, q, dh = si.values.to(dev), si.query.to(dev), si.dh.to(dev)
    k = si.keys.to(dev) if si.keys is not None else None
    h = torch.empty(si.T, si.d, dtype=torch.float32, device=dev)
    lse = torch.empty(si.T, dtype=torch.float32, device=dev)
    lrar.forward(si.variant, v, k, q, h, lse, r=si.r)
    dv = torch.full(v.shape, float("nan"), dtype=torch.float32, device=dev)
    dk = torch.full(k.shape, float("nan"), dtype=torch.float32, device=dev) if k is not None else None
    dq = torch.full((si.d if si.variant == "full" else si.r,), float("nan"), device=dev)
    if noalloc:
        lrar.backward_noalloc(si.variant, v, k, q, dh, dv, dq, dkeys=dk, h=h, lse=lse, r=si.r)
    else:
        ws = torch.empty(lrar.workspace_size(si.variant, si.n, si.T, si.d, si.r) // 4, device=dev)
        lrar.backward(si.variant, v, k, q, dh, dv, dq, ws, dkeys=dk, h=h, lse=lse, r=si.r)
    torch.cuda.synchronize()
    out = {"dvalues": dv.double().cpu().numpy(), "dq": dq.double().cpu().numpy()}
    if dk is not None:
        out["dkeys"] = dk.double().cpu().numpy()
    return out


def test_consecutive_calls_match_the_workspace_backward():
    """Back-to-back calls with different shapes share the scratch; each result
    equals lrar_backward's on the same inputs bit for bit: both run the same
    kernels on the same grid, and dq's partial sums are reduced in a fixed
    order, so a stale or overlapping partial-sum row would show as a
    difference.  (Accuracy against the oracle is covered by the parity tests.)"""
    sites = [_site(c) for c in CASES]
    refs = [_backward(si, noalloc=False) for si in sites]
    for si, ref in zip(sites + sites[:1], refs + refs[:1]):  # four calls in a row, first case again last
        got = _backward(si, noalloc=True)
        for name in ref:
            assert np.array_equal(got[name], ref[name]), f"{si.variant}:{name}"


def test_rejects_problems_beyond_the_scratch():
    """Full keys with d = 2048 need an 8 MiB workspace, above the 4 MiB scratch."""
    dev = torch.device("cuda")
    d = 2048
    v = torch.zeros(2, 1, d, dtype=torch.bfloat16, device=dev)
    q = torch.zeros(d, device=dev)
    h = torch.zeros(1, d, device=dev)
    lse = torch.zeros(1, device=dev)
    dv = torch.zeros(2, 1, d, device=dev)
    dq = torch.zeros(d, device=dev)
    with pytest.raises(lrar.LrarError) as ei:
        lrar.backward_noalloc("full", v, None, q, v[0], dv, dq, h=h, lse=lse, r=d)
    assert ei.value.code == lrar.ERR_UNSUPPORTED
    assert "4 MiB" in str(ei.value)
