"""The whole-decoder driver (paper_2607_09694_gb300.sweep): every read site over
separate source tensors, forward in order and backward in reverse with each
source's gradient summed over the sites that read it (Eq. 4), eager and as a
replayed CUDA graph, against the stacked calls and the oracle."""
import numpy as np
import pytest
import torch

import gpu_helpers as H
import oracle
from paper_2607_09694_gb300 import lrar, synth
from paper_2607_09694_gb300.sweep import DepthSweep

pytestmark = pytest.mark.gpu


def _model(variant, n_sites, T, d, r, dtype, seed):
    dev = torch.device("cuda")
    vals = synth.values(n_sites, T, d, seed, dtype, (0.5, 2.0))
    keys = synth.keys(n_sites, T, r, seed, dtype) if variant == "projected" else None
    queries = synth.queries(n_sites, d if variant == "full" else r, seed, std=0.5)
    dh = synth.upstream(T, d, seed, dtype, sites=n_sites)
    return vals, keys, queries, dh, dev


def _sweep(variant, vals, keys, queries, dh, dev, r):
    n, T, d = vals.shape
    tdt = vals.dtype
    srcs = [vals[i].to(dev).clone() for i in range(n)]
    ks = [keys[i].to(dev).clone() for i in range(n)] if keys is not None else None
    h = torch.empty(n, T, d, device=dev)
    lse = torch.empty(n, T, device=dev)
    dsrc = [torch.full((T, d), float("nan"), dtype=tdt, device=dev) for _ in range(n)]
    dks = [torch.full((T, r), float("nan"), dtype=tdt, device=dev) for _ in range(n)] if ks is not None else None
    dq = torch.empty(n, queries.shape[-1], device=dev)
    sw = DepthSweep(variant, srcs, queries.to(dev), [dh[t].to(dev) for t in range(n)], h, lse, dsrc, dq, keys=ks,
                    dkeys=dks, r=r)
    return sw


@pytest.mark.parametrize("variant", ["sliced", "projected", "full"])
def test_sweep_against_the_oracle(variant):
    """fp32 storage: each site's h and lse, every source's summed gradient and
    every site's dq against the oracle's per-site mix and backward."""
    n, T, d, r = 6, 96, 128, 8
    vals, keys, queries, dh, dev = _model(variant, n, T, d, r, "f32", 51)
    rr = d if variant == "full" else r
    sw = _sweep(variant, vals, keys, queries, dh, dev, rr)
    sw.step()
    torch.cuda.synchronize()
    ov = H.ORACLE_VARIANT[variant]
    dsum = np.zeros((n, T, d))
    dksum = np.zeros((n, T, r)) if keys is not None else None
    for t in range(1, n + 1):
        q = queries[t - 1] if t > 1 else torch.zeros(queries.shape[-1])
        kk = keys[:t] if keys is not None else None
        ref = oracle.forward(ov, vals[:t], kk, q, H.EPS, r=rr)
        H.assert_abs(f"h[{t}]", sw.h[t - 1].double().cpu().numpy(), ref["h"])
        H.assert_abs(f"lse[{t}]", sw.lse[t - 1].double().cpu().numpy(), ref["lse"], 1e-4)
        g = oracle.backward(ov, vals[:t], kk, q, H.EPS, dh[t - 1], r=rr)
        dsum[:t] += g["dvalues"]
        if dksum is not None:
            dksum[:t] += g["dkeys"]
        if t > 1:
            H.assert_dq(f"dq[{t}]", sw.dq[t - 1].double().cpu().numpy(), g["dq"], g["dq_abs"], t, T)
    got = np.stack([x.double().cpu().numpy() for x in sw.dsources])
    H.assert_abs("summed source gradients", got, dsum)
    if dksum is not None:
        H.assert_abs("summed key gradients", np.stack([x.double().cpu().numpy() for x in sw.dkeys]), dksum)


def test_sweep_equals_the_stacked_calls_and_its_graph():
    """bf16, the S-LR workload's shape at a small T: the driver's eager step
    equals the stacked entry points bit for bit, and so do two graph replays."""
    n, T, d, r = 12, 384, 1024, 16
    vals, _, queries, dh, dev = _model("sliced", n, T, d, r, "bf16", 52)
    sw = _sweep("sliced", vals, None, queries, dh, dev, r)
    sw.step()
    # the stacked calls of the benchmark's step
    v = vals.to(dev)
    h = torch.empty(n, T, d, device=dev)
    lse = torch.empty(n, T, device=dev)
    dv = torch.zeros(n, T, d, dtype=torch.bfloat16, device=dev)
    dq = torch.empty(n, r, device=dev)
    ws = torch.empty(lrar.workspace_size("sliced", n, T, d, r) // 4, device=dev)
    qd, dhd = queries.to(dev), dh.to(dev)
    for t in range(1, n + 1):
        lrar.forward("sliced", v, None, qd[t - 1] if t > 1 else None, h[t - 1], lse[t - 1], n_src=t, r=r)
    dq.zero_()
    for t in range(n, 0, -1):
        lrar.backward("sliced", v, None, qd[t - 1] if t > 1 else None, dhd[t - 1], dv, dq[t - 1], ws, lse=lse[t - 1],
                      n_src=t, r=r, accumulate=t != n)
    torch.cuda.synchronize()
    assert torch.equal(sw.h, h) and torch.equal(sw.lse, lse) and torch.equal(sw.dq, dq)
    assert torch.equal(torch.stack(sw.dsources), dv)
    eager = (sw.h.clone(), sw.lse.clone(), torch.stack(sw.dsources).clone(), sw.dq.clone())
    sw.capture()
    for _ in range(2):
        for x in sw.dsources:
            x.fill_(float("nan"))  # the backward's first site overwrites every gradient
        sw.h.zero_()
        sw.dq.fill_(float("nan"))  # zeroed inside the step
        sw.replay()
        torch.cuda.synchronize()
        assert torch.equal(sw.h, eager[0]) and torch.equal(sw.lse, eager[1])
        assert torch.equal(torch.stack(sw.dsources), eager[2]) and torch.equal(sw.dq, eager[3])
