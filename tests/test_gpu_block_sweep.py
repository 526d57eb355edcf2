"""The Block AttnRes training step (paper_2607_09694_gb300.sweep.BlockSweep):
assembly after every sub-layer (Eq. 5-6), the mix at every read site, the
backward at every site in reverse, and the fan-out of each summary's gradient
to its members -- against the oracle's own assembly (oracle.block_sources),
its mix and backward at each site, and its fan-out (oracle.block_fanout),
summed over the sites."""
import numpy as np
import pytest
import torch

import gpu_helpers as H
import oracle
from paper_2607_09694_gb300 import sites, synth
from paper_2607_09694_gb300.sweep import BlockSweep

pytestmark = pytest.mark.gpu


def _inputs(variant, M, T, d, r, dtype, seed):
    outs = synth.outputs(M + 1, T, d, seed=seed, dtype=dtype)
    keys = synth.randn((M + 1, T, r), seed, "keys").to(outs.dtype) if variant == "projected" else None
    queries = synth.queries(M + 1, d if variant == "full" else r, seed, std=0.5)
    dh = synth.upstream(T, d, seed, dtype, sites=M + 1)
    return outs, keys, queries, dh


def _run(variant, outs, keys, queries, dh, c, r, gdt=None, h_dtype=torch.float32, two_phase=None):
    dev = torch.device("cuda")
    M1, T, d = outs.shape
    gdt = gdt or outs.dtype
    o = [outs[i].to(dev).clone() for i in range(M1)]
    k = [keys[i].to(dev).clone() for i in range(M1)] if keys is not None else None
    h = torch.empty(M1, T, d, dtype=h_dtype, device=dev)
    lse = torch.empty(M1, T, device=dev)
    do = [torch.full((T, d), float("nan"), dtype=gdt, device=dev) for _ in range(M1)]
    dk = [torch.full((T, r), float("nan"), dtype=gdt, device=dev) for _ in range(M1)] if k is not None else None
    sw = BlockSweep(variant, o, queries.to(dev), [dh[t].to(dev) for t in range(M1)], h, lse, do, c, keys=k,
                    dkeys=dk, r=r, two_phase=two_phase)
    sw.step()
    torch.cuda.synchronize()
    return sw


def _oracle(variant, outs, keys, queries, dh, c, r):
    """Per site t: the oracle's Block sources of o_0..o_{t-1}, its mix, its
    backward, and the fan-out of the source gradients to the outputs."""
    M1, T, d = outs.shape
    ov = H.ORACLE_VARIANT[variant]
    res = dict(h=[], lse=[], dq=[], dq_abs=[], n=[], douts=np.zeros((M1, T, d)),
               dkeys=np.zeros((M1, T, r)) if keys is not None else None)
    for t in range(1, M1 + 1):
        src = oracle.block_sources(outs[:t], c)
        ksrc = oracle.block_sources(keys[:t], c) if keys is not None else None
        n = src.shape[0]
        q = queries[t - 1] if n > 1 else torch.zeros(queries.shape[-1])
        f = oracle.forward(ov, src, ksrc, q, H.EPS, r=r)
        b = oracle.backward(ov, src, ksrc, q, H.EPS, dh[t - 1].double(), r=r)
        res["h"].append(f["h"])
        res["lse"].append(f["lse"])
        res["dq"].append(b["dq"])
        res["dq_abs"].append(b["dq_abs"])
        res["n"].append(n)
        res["douts"][:t] += oracle.block_fanout(b["dvalues"], t, c)
        if keys is not None:
            res["dkeys"][:t] += oracle.block_fanout(b["dkeys"], t, c)
    return res


@pytest.mark.parametrize("variant,two_phase", [("sliced", False), ("sliced", True), ("projected", False),
                                               ("projected", True), ("full", False)])
@pytest.mark.parametrize("M,c", [(12, 4), (13, 4)])
def test_block_step_fp32(variant, two_phase, M, c):
    """float32 storage: every site's h and lse, every output's gradient summed
    over the sites that read it, every site's dq; M = 12 fills three blocks of
    four, M = 13 leaves the last block open at the final site.  The forward
    runs site by site, or (low-rank keys) two-phase: phase 1 per block into the
    sites' h and lse, phase 2 in place."""
    T, d, r = 96, 128, 8
    rr = d if variant == "full" else r
    outs, keys, queries, dh = _inputs(variant, M, T, d, r, "f32", seed=61)
    sw = _run(variant, outs, keys, queries, dh, c, rr, two_phase=two_phase)
    ref = _oracle(variant, outs, keys, queries, dh, c, rr)
    for t in range(1, M + 2):
        H.assert_abs(f"h[{t}]", sw.h[t - 1].double().cpu().numpy(), ref["h"][t - 1])
        H.assert_abs(f"lse[{t}]", sw.lse[t - 1].double().cpu().numpy(), ref["lse"][t - 1], 1e-4)
        if ref["n"][t - 1] > 1:
            H.assert_dq(f"dq[{t}]", sw.dq[t - 1].double().cpu().numpy(), ref["dq"][t - 1], ref["dq_abs"][t - 1],
                        ref["n"][t - 1], T)
    H.assert_abs("doutputs", np.stack([x.double().cpu().numpy() for x in sw.doutputs]), ref["douts"])
    if keys is not None:
        H.assert_abs("dkeys", np.stack([x.double().cpu().numpy() for x in sw.dkeys]), ref["dkeys"])
    # every output tensor of the open block's members now holds its running sum (Eq. 6)
    runs = oracle.block_sources(outs, c)
    for i in range(1, M + 1):
        if (i % c == 0) or i == M:
            H.assert_abs(f"summary of o_{i}", sw.outputs[i].double().cpu().numpy(), runs[sites.block_slot(i, c)],
                         1e-4)


def _rounded_running_sums(outs, c):
    """bfloat16 running block sums built on the host the way the assembly
    defines them: each member added to the running sum in float32 and the sum
    stored with one round to nearest even."""
    run = outs.clone()
    for i in range(2, outs.shape[0]):
        if not sites.block_opens_slot(i, c):
            run[i] = (run[i - 1].float() + outs[i].float()).to(outs.dtype)
    return run


def test_block_step_bf16_decoder_shape():
    """The large decoder's shape at a small T (d = 2048, r = 64, c = 8, M = 64
    sub-layers, 65 sites, two-phase forward), bfloat16 outputs and summaries,
    float32 h and gradients: the GPU's running sums equal the host's bf16 running sums bit
    for bit, and the mix and its gradients match the oracle evaluated on those
    sums within 1e-2 x RMS (the bf16-input bound)."""
    M, c, T, d, r = 64, 8, 64, 2048, 64
    outs, _, queries, dh = _inputs("sliced", M, T, d, r, "bf16", seed=62)
    sw = _run("sliced", outs, None, queries, dh, c, r, gdt=torch.float32, two_phase=True)
    run = _rounded_running_sums(outs, c)
    for i in range(1, M + 1):
        assert torch.equal(sw.outputs[i].cpu(), run[i]), i
    ov = oracle.SLICED
    douts = np.zeros((M + 1, T, d))
    for t in range(1, M + 2):
        idx = sw.site_sources(t)
        src = run[idx]
        q = queries[t - 1] if len(idx) > 1 else torch.zeros(r)
        f = oracle.forward(ov, src, None, q, H.EPS, r=r)
        H.assert_rms(f"h[{t}]", sw.h[t - 1].double().cpu().numpy(), f["h"])
        H.assert_abs(f"lse[{t}]", sw.lse[t - 1].double().cpu().numpy(), f["lse"], 1e-4)
        b = oracle.backward(ov, src, None, q, H.EPS, dh[t - 1], r=r)
        if len(idx) > 1:
            H.assert_rms(f"dq[{t}]", sw.dq[t - 1].double().cpu().numpy(), b["dq"])
        douts[:t] += oracle.block_fanout(b["dvalues"], t, c)
    got = np.stack([x.double().cpu().numpy() for x in sw.doutputs])
    for i in range(M + 1):
        H.assert_rms(f"doutputs[{i}]", got[i], douts[i])


@pytest.mark.parametrize("variant", ["sliced", "projected"])
def test_member_gradients_handed_over(variant):
    """The fan-out as a hand-over: the views passed to member_grad as each
    output's gradient completes, copied there on the stream, equal bit for bit
    the doutputs (and dkeys) that the copying fan-out writes; doutputs stay
    untouched."""
    M, c, T, d, r = 13, 4, 96, 128, 8
    outs, keys, queries, dh = _inputs(variant, M, T, d, r, "f32", seed=64)
    ref = _run(variant, outs, keys, queries, dh, c, r)
    dev = torch.device("cuda")
    o = [outs[i].to(dev).clone() for i in range(M + 1)]
    k = [keys[i].to(dev).clone() for i in range(M + 1)] if keys is not None else None
    h = torch.empty(M + 1, T, d, device=dev)
    lse = torch.empty(M + 1, T, device=dev)
    do = [torch.full((T, d), float("nan"), device=dev) for _ in range(M + 1)]
    dk = [torch.full((T, r), float("nan"), device=dev) for _ in range(M + 1)] if k is not None else None
    sw = BlockSweep(variant, o, queries.to(dev), [dh[t].to(dev) for t in range(M + 1)], h, lse, do, c, keys=k,
                    dkeys=dk, r=r)
    got, got_k, order = {}, {}, []

    def take(i, g, gk):
        order.append(i)
        got[i] = g.clone()
        if gk is not None:
            got_k[i] = gk.clone()

    sw.step(member_grad=take)
    torch.cuda.synchronize()
    assert order == list(range(M, -1, -1))
    for i in range(M + 1):
        assert torch.equal(got[i], ref.doutputs[i]), i
        assert torch.isnan(do[i]).all(), i
        if keys is not None:
            assert torch.equal(got_k[i], ref.dkeys[i]), i


def test_forward_runs_once_per_set_of_outputs():
    outs, _, queries, dh = _inputs("sliced", 4, 16, 64, 4, "f32", seed=63)
    sw = _run("sliced", outs, None, queries, dh, 2, 4)
    with pytest.raises(RuntimeError):
        sw.forward()
