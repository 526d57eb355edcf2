"""Block AttnRes (§3.1, Eq. 5-6) on the GPU: source assembly with
lrar_block_accumulate, the mix over the assembled stack, and the gradient
fan-out, each against the oracle's own assembly and mix."""
import numpy as np
import pytest
import torch

import gpu_helpers as H
import oracle
from paper_2607_09694_gb300 import lrar, sites, synth

pytestmark = pytest.mark.gpu


def _assemble(outs_dev, t, c, dst_dtype):
    """Stack [o_0, b_1, ..., b_P] for site t from outputs o_0..o_{t-1}."""
    n = sites.block_num_sources(t, c)
    _, T, w = outs_dev.shape
    stack = torch.empty(n, T, w, dtype=dst_dtype, device=outs_dev.device)
    for i in range(t):
        slot = sites.block_slot(i, c)
        lrar.block_accumulate(stack[slot], outs_dev[i], 1.0, 0.0 if sites.block_opens_slot(i, c) else 1.0)
    return stack


@pytest.mark.parametrize("t,c", [(1, 8), (9, 8), (20, 8), (65, 8), (13, 4)])
def test_assembly_fp32_summaries(t, c):
    outs = synth.outputs(t, 64, 256, seed=5, dtype="bf16")
    stack = _assemble(outs.cuda(), t, c, torch.float32)
    torch.cuda.synchronize()
    ref = oracle.block_sources(outs, c)
    assert stack.shape[0] == ref.shape[0] == sites.block_num_sources(t, c)
    H.assert_abs("stack", stack.double().cpu().numpy(), ref, 1e-5)


def test_assembly_bf16_incremental_rounding_bound():
    """bf16 summaries grow one rounded add at a time; each add is within half
    a bf16 spacing of its exact result, so the total error is bounded by the
    sum of those half-spacings."""
    t, c = 17, 8
    outs = synth.outputs(t, 96, 512, seed=6, dtype="bf16")
    stack = _assemble(outs.cuda(), t, c, torch.bfloat16).double().cpu().numpy()
    ref = oracle.block_sources(outs, c)
    o = outs.double().numpy()
    bound = np.zeros_like(ref)
    for b in range(1, ref.shape[0]):
        members = [i for i in range(1, t) if sites.block_slot(i, c) == b]
        run = np.zeros_like(o[0])
        for k, i in enumerate(members):
            run = run + o[i]
            if k > 0:
                bound[b] += 0.5 * H.bf16_ulp(run) * (1 + 2 ** -7)
    assert np.all(np.abs(stack - ref) <= bound + 1e-12)


@pytest.mark.parametrize("variant", ["sliced", "projected"])
def test_block_mix_fp32(variant):
    """Site t = 21 with c = 8: sources [o_0, b_1, b_2, b_P(4 outputs)]; GPU
    assembly + mix + fan-out against the oracle's assembly + mix + fan-out."""
    t, c, T, d, r = 21, 8, 300, 512, 16
    outs = synth.outputs(t, T, d, seed=7, dtype="f32")
    q = synth.queries(1, r, seed=7)[0].contiguous()
    dh = synth.upstream(T, d, seed=7, dtype="f32")
    okeys = synth.randn((t, T, r), 7, "keys") if variant == "projected" else None
    dev = torch.device("cuda")
    stack = _assemble(outs.to(dev), t, c, torch.float32)
    kstack = _assemble(okeys.to(dev), t, c, torch.float32) if okeys is not None else None
    n = stack.shape[0]
    h = torch.empty(T, d, device=dev)
    lrar.forward(variant, stack, kstack, q.to(dev), h, r=r)
    dstack = torch.empty_like(stack)
    dkst = torch.empty_like(kstack) if kstack is not None else None
    dq = torch.empty(r, device=dev)
    ws = torch.empty(lrar.workspace_size(variant, n, T, d, r) // 4, device=dev)
    lrar.backward(variant, stack, kstack, q.to(dev), dh.to(dev), dstack, dq, ws, dkeys=dkst, r=r)
    # fan the summary gradients back to the members: d(o_i) = d(slot of o_i)
    douts = torch.empty(t, T, d, device=dev)
    for i in range(t):
        lrar.block_accumulate(douts[i], dstack[sites.block_slot(i, c)], 1.0, 0.0)
    torch.cuda.synchronize()

    src = oracle.block_sources(outs, c)
    ksrc = oracle.block_sources(okeys, c) if okeys is not None else None
    ov = H.ORACLE_VARIANT[variant]
    f = oracle.forward(ov, src, ksrc, q, H.EPS, r=r)
    b = oracle.backward(ov, src, ksrc, q, H.EPS, dh.double(), r=r)
    H.assert_abs("h", h.double().cpu().numpy(), f["h"])
    H.assert_dq("dq", dq.double().cpu().numpy(), b["dq"], b["dq_abs"], n, T)
    H.assert_abs("dsources", dstack.double().cpu().numpy(), b["dvalues"])
    fan = oracle.block_fanout(b["dvalues"], t, c)
    H.assert_abs("doutputs", douts.double().cpu().numpy(), fan)
    if variant == "projected":
        H.assert_abs("dkeys", dkst.double().cpu().numpy(), b["dkeys"])


@pytest.mark.parametrize("dst,src", [("f32", "bf16"), ("bf16", "f32"), ("bf16", "bf16"), ("f32", "f32")])
def test_accumulate_dtypes_and_ragged_count(dst, src):
    g = torch.Generator().manual_seed(3)
    count = 8 * 1000 + 5
    a = torch.randn(count, generator=g).to(H.TORCH_DTYPE[dst])
    b = torch.randn(count, generator=g).to(H.TORCH_DTYPE[src])
    d_dev = a.cuda()
    lrar.block_accumulate(d_dev, b.cuda(), 0.5, -2.0)
    torch.cuda.synchronize()
    exact = -2.0 * a.double() + 0.5 * b.double()
    got = d_dev.double().cpu().numpy()
    if dst == "f32":
        H.assert_abs("acc", got, exact.numpy(), 1e-5)
    else:
        H.assert_bf16_rounded("acc", got, exact.numpy())


def test_accumulate_misaligned_view_uses_scalar_path():
    base = torch.zeros(1001, device="cuda")
    src = torch.ones(1000, device="cuda")
    lrar.block_accumulate(base[1:], src, 3.0, 1.0)
    torch.cuda.synchronize()
    assert base[0].item() == 0.0 and torch.all(base[1:] == 3.0)
