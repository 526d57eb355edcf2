"""Sources as separate tensors (lrar_forward_ptrs / lrar_backward_ptrs): the
same mix as the stacked entry points, bit for bit, with sources and gradients
in unrelated allocations; checked against the oracle, and under CUDA-graph
capture and replay."""
import numpy as np
import pytest
import torch

import gpu_helpers as H
import oracle
from paper_2607_09694_gb300 import lrar, synth

pytestmark = pytest.mark.gpu


def _scatter(stack, pad_elems):
    """Copies of the slices of `stack` in separate places: each inside its own
    buffer at a 16-byte aligned offset, so no two are contiguous."""
    outs = []
    for i in range(stack.shape[0]):
        buf = torch.zeros(stack[i].numel() + pad_elems * (i + 1), dtype=stack.dtype, device=stack.device)
        off = pad_elems * (i % 3)
        t = buf[off:off + stack[i].numel()].view(stack[i].shape)
        t.copy_(stack[i])
        outs.append(t)
    return outs


def _case(variant, dtype="bf16", n=9, T=333, d=256, r=16, seed=41):
    si = synth.site("slr", variant=variant, n=n, T=T, d=d, r=r if variant != "full" else None, dtype=dtype, seed=seed)
    dev = torch.device("cuda")
    return si, si.values.to(dev), (si.keys.to(dev) if si.keys is not None else None), si.query.to(dev), si.dh.to(dev)


def _run_both(variant, accumulate, dtype="bf16", **kw):
    si, v, k, q, dh = _case(variant, dtype, **kw)
    dev = v.device
    n, T, d = v.shape
    r = si.r
    pad = 8 if v.dtype == torch.bfloat16 else 4  # 16 bytes
    vs = _scatter(v, pad)
    ks = _scatter(k, pad) if k is not None else None
    g = torch.Generator(device="cpu").manual_seed(5)
    init_dv = torch.randn(v.shape, generator=g).to(v.dtype).to(dev) if accumulate else torch.zeros_like(v)
    init_dk = (torch.randn(k.shape, generator=g).to(k.dtype).to(dev) if accumulate else torch.zeros_like(k)) \
        if k is not None else None
    rq = d if variant == "full" else r
    res = {}
    for mode in ("stacked", "ptrs"):
        h = torch.empty(T, d, device=dev)
        lse = torch.empty(T, device=dev)
        dq = torch.full((rq,), 0.25, device=dev)
        ws = torch.empty(lrar.workspace_size(variant, n, T, d, r) // 4, device=dev)
        if mode == "stacked":
            dv, dk = init_dv.clone(), (init_dk.clone() if k is not None else None)
            lrar.forward(variant, v, k, q, h, lse, r=r)
            lrar.backward(variant, v, k, q, dh, dv, dq, ws, dkeys=dk, h=h, lse=lse, r=r, accumulate=accumulate)
            res[mode] = (h, lse, dv, dk, dq)
        else:
            dvs = _scatter(init_dv, pad)
            dks = _scatter(init_dk, pad) if k is not None else None
            lrar.forward_ptrs(variant, vs, ks, q, h, lse, r=r)
            lrar.backward_ptrs(variant, vs, ks, q, dh, dvs, dq, ws, dkeys=dks, h=h, lse=lse, r=r,
                               accumulate=accumulate)
            res[mode] = (h, lse, torch.stack(dvs), torch.stack(dks) if dks is not None else None, dq)
    torch.cuda.synchronize()
    return si, res


@pytest.mark.parametrize("variant", ["sliced", "projected", "full"])
@pytest.mark.parametrize("accumulate", [False, True])
def test_pointer_tables_match_the_stack_bitwise(variant, accumulate):
    _, res = _run_both(variant, accumulate)
    for a, b, name in zip(res["stacked"], res["ptrs"], ("h", "lse", "dvalues", "dkeys", "dq")):
        if a is None:
            assert b is None
            continue
        assert torch.equal(a, b), name


def test_pointer_tables_fp32_wide_rows():
    """fp32 storage (register backward) and d = 2048 bf16 (split forward rows)."""
    for kw in (dict(dtype="f32", d=128, r=8), dict(d=2048, r=64, T=130)):
        _, res = _run_both("sliced", True, **kw)
        for a, b in zip(res["stacked"], res["ptrs"]):
            if a is not None:
                assert torch.equal(a, b)


def test_pointer_tables_against_the_oracle():
    si, res = _run_both("projected", False, n=6, T=200, d=128, r=8, seed=43)
    h, lse, dv, dk, dq = res["ptrs"]
    ref = H.run_oracle(si)
    H.assert_rms("h", h.double().cpu().numpy(), ref["h"])
    H.assert_abs("lse", lse.double().cpu().numpy(), ref["lse"], 1e-4)
    H.assert_bf16_rounded("dvalues", dv.double().cpu().numpy(), ref["dvalues"], 1.0)
    H.assert_bf16_rounded("dkeys", dk.double().cpu().numpy(), ref["dkeys"], 1.0)
    H.assert_rms("dq", dq.double().cpu().numpy(), ref["dq"])


def test_graph_capture_replays_the_same_mix():
    """The calls allocate nothing and synchronise nothing, so a forward and an
    accumulating backward over separate sources capture into a CUDA graph whose
    replays equal eager execution bit for bit (one and two steps)."""
    si, v, k, q, dh = _case("sliced", n=7, T=512, d=256, r=16, seed=44)
    dev = v.device
    n, T, d = v.shape
    vs = [v[i].clone() for i in range(n)]
    dvs = [torch.zeros(T, d, dtype=v.dtype, device=dev) for _ in range(n)]
    h = torch.empty(T, d, dtype=v.dtype, device=dev)
    lse = torch.empty(T, device=dev)
    dq = torch.zeros(si.r, device=dev)
    ws = torch.empty(lrar.workspace_size("sliced", n, T, d, si.r) // 4, device=dev)
    s = torch.cuda.Stream()

    def step():
        lrar.forward_ptrs("sliced", vs, None, q, h, lse, r=si.r, stream=s.cuda_stream)
        lrar.backward_ptrs("sliced", vs, None, q, dh, dvs, dq, ws, r=si.r, accumulate=True, stream=s.cuda_stream)

    def reset():
        for x in dvs:
            x.zero_()
        dq.zero_()
        torch.cuda.synchronize()

    def snapshot():
        torch.cuda.synchronize()
        return [x.clone() for x in dvs] + [h.clone(), lse.clone(), dq.clone()]

    s.wait_stream(torch.cuda.current_stream())
    eager = []
    with torch.cuda.stream(s):
        for _ in range(2):
            step()
            eager.append(snapshot())
    reset()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=s):
        step()
    reset()  # capture does not execute; start the replays from zero
    for k_ in range(2):
        graph.replay()
        got = snapshot()
        for a, b in zip(eager[k_], got):
            assert torch.equal(a, b), k_
