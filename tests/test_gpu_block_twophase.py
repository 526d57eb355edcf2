"""Block AttnRes two-phase batched sites (§3.5): phase 1 over a block's
completed sources for all of its sites, phase 2 folding in each site's
partial-block summary, against the oracle's plain mix over that site's Block
source set (Eq. 5-6 sums, Eq. 8-10 mix).  Both sides build their own sources:
the GPU with lrar_block_accumulate, the oracle with its own assembly."""
import numpy as np
import pytest
import torch

import gpu_helpers as H
import oracle
from paper_2607_09694_gb300 import lrar, sites, synth

pytestmark = pytest.mark.gpu


def _assemble(outs, t, c, dtype):
    n = sites.block_num_sources(t, c)
    _, T, w = outs.shape
    stack = torch.empty(n, T, w, dtype=dtype, device=outs.device)
    for i in range(t):
        lrar.block_accumulate(stack[sites.block_slot(i, c)], outs[i], 1.0,
                              0.0 if sites.block_opens_slot(i, c) else 1.0)
    return stack


def _to_stack(t32, dtype):
    """fp32 sums -> stack type, one rounding (lrar_block_accumulate with beta = 0)."""
    if dtype == torch.float32:
        return t32
    out = torch.empty(t32.shape, dtype=dtype, device=t32.device)
    lrar.block_accumulate(out, t32, 1.0, 0.0)
    return out


def _oracle_src(x, dtype):
    """The oracle's exact sums, stored like the GPU's stack (one RNE rounding)."""
    t = torch.from_numpy(x)
    return t.to(torch.bfloat16) if dtype == torch.bfloat16 else t


def _run(variant, c, b, T, d, r, store, stack, pre, seed=11):
    """Sites t = b*c + 1 + j, j = 0..c-1, of the block after b completed blocks.
    Yields (j, (h, lse) from the GPU, oracle mix over the site's sources, oracle
    mix over the completed sources only)."""
    t_max = b * c + c  # outputs o_0 .. o_{b*c + c - 1}
    outs = synth.outputs(t_max, T, d, seed=seed, dtype=store)
    okeys = synth.randn((t_max, T, r), seed, "keys").to(outs.dtype) if variant == "projected" else None
    queries = synth.queries(c, r, seed, std=0.5)
    dev = torch.device("cuda")
    sdt = H.TORCH_DTYPE[stack]
    full_stack = _to_stack(_assemble(outs.to(dev), t_max, c, torch.float32), sdt)  # [1 + b + 1, T, d]
    kstack = _to_stack(_assemble(okeys.to(dev), t_max, c, torch.float32), sdt) if okeys is not None else None
    n_c = 1 + b
    h_pre = torch.empty(c, T, d, dtype=H.TORCH_DTYPE[pre], device=dev)
    lse_pre = torch.empty(c, T, device=dev)
    lrar.block_phase1(variant, full_stack, kstack, queries.to(dev), h_pre, lse_pre, n_completed=n_c)
    got = []
    for j in range(c):
        if j == 0:  # empty partial block: the site's mix is the phase-1 result
            got.append((h_pre[0].double().cpu().numpy(), lse_pre[0].double().cpu().numpy()))
            continue
        part = torch.zeros(T, d, device=dev)  # partial summary of the open block's first j outputs
        pkey = torch.zeros(T, r, device=dev) if kstack is not None else None
        for i in range(b * c + 1, b * c + 1 + j):
            lrar.block_accumulate(part, outs[i].to(dev), 1.0, 1.0)
            if pkey is not None:
                lrar.block_accumulate(pkey, okeys[i].to(dev), 1.0, 1.0)
        part = _to_stack(part, sdt)
        pkey = _to_stack(pkey, sdt) if pkey is not None else None
        h = torch.empty(T, d, device=dev)
        lse = torch.empty(T, device=dev)
        lrar.block_phase2(variant, h_pre[j], lse_pre[j], part, pkey, queries[j].to(dev), h, lse)
        got.append((h.double().cpu().numpy(), lse.double().cpu().numpy()))
    torch.cuda.synchronize()
    ov = H.ORACLE_VARIANT[variant]
    for j in range(c):
        t = b * c + 1 + j
        src = _oracle_src(oracle.block_sources(outs[:t], c), sdt)
        ksrc = _oracle_src(oracle.block_sources(okeys[:t], c), sdt) if okeys is not None else None
        assert src.shape[0] == n_c + (1 if j > 0 else 0)
        ref = oracle.forward(ov, src, ksrc, queries[j], H.EPS, r=r)
        pre_ref = oracle.forward(ov, src[:n_c], None if ksrc is None else ksrc[:n_c], queries[j], H.EPS, r=r)
        yield j, got[j], ref, pre_ref


@pytest.mark.parametrize("variant", ["sliced", "projected"])
def test_fp32_sites_of_a_block(variant):
    for j, (h, lse), ref, _ in _run(variant, c=8, b=3, T=300, d=512, r=16, store="f32", stack="f32", pre="f32"):
        H.assert_abs(f"h[site {j}]", h, ref["h"])
        H.assert_abs(f"lse[site {j}]", lse, ref["lse"], 1e-4)


def test_more_sites_than_one_launch_holds():
    """n_sites = 12 > 8 queries per launch: the host splits the queries."""
    for j, (h, lse), ref, _ in _run("sliced", c=12, b=2, T=130, d=256, r=8, store="f32", stack="f32", pre="f32",
                                    seed=12):
        H.assert_abs(f"h[site {j}]", h, ref["h"])
        H.assert_abs(f"lse[site {j}]", lse, ref["lse"], 1e-4)


@pytest.mark.parametrize("b", [0, 1, 7])
def test_bf16_members_d2048(b):
    """The large decoder's shape (d = 2048, r = 64, c = 8): bf16 sub-layer outputs
    and summaries (each summary rounded once), fp32 phase-1 results."""
    for j, (h, lse), ref, _ in _run("sliced", c=8, b=b, T=257, d=2048, r=64, store="bf16", stack="bf16", pre="f32",
                                    seed=13 + b):
        H.assert_rms(f"h[site {j}]", h, ref["h"])
        H.assert_abs(f"lse[site {j}]", lse, ref["lse"], 1e-4)


@pytest.mark.parametrize("variant,r,c,b,T,d", [("sliced", 32, 8, 1, 333, 256), ("sliced", 48, 5, 2, 333, 256),
                                                 ("projected", 32, 8, 2, 333, 256), ("projected", 16, 3, 4, 333, 256),
                                                 ("sliced", 64, 8, 15, 333, 256), ("sliced", 32, 8, 3, 20011, 256),
                                                 ("projected", 48, 2, 30, 3001, 384)])
def test_bf16_key_depths(variant, r, c, b, T, d):
    """bf16 sources with keys of depth 16, 32, 48 and 64 (the phase-1 scores on the
    tensor cores, one to four k-steps), up to 31 completed sources, fewer than 8
    sites, and token counts that leave several tokens per warp and a ragged last
    chunk (T = 20011; T = 3001 with 31 sources).  Both sides mix the same bf16
    sources, so h is held to the fp32 bar."""
    for j, (h, lse), ref, _ in _run(variant, c=c, b=b, T=T, d=d, r=r, store="bf16", stack="bf16", pre="f32",
                                    seed=19 + r + b):
        H.assert_abs(f"h[site {j}]", h, ref["h"])
        H.assert_abs(f"lse[site {j}]", lse, ref["lse"], 1e-4)


def test_weights_wider_than_an_h_pre_row():
    """21 completed sources with a bf16 h_pre of d = 256: a token's 21 x 8 fp32
    weights do not fit one h_pre row, so phase 1 runs as the single fused kernel."""
    for j, (h, lse), ref, pre_ref in _run("sliced", c=4, b=20, T=333, d=256, r=16, store="bf16", stack="bf16",
                                          pre="bf16", seed=23):
        bound = 0.5 * H.bf16_ulp(pre_ref["h"]) + 1e-5 * H.rms(ref["h"])
        assert np.all(np.abs(h - ref["h"]) <= bound), j
        H.assert_abs(f"lse[site {j}]", lse, ref["lse"], 1e-4)


def test_bf16_phase1_outputs_within_one_rounding():
    """With a bf16 h_pre, phase 2 sees the completed-source mix rounded once; its
    weight is at most 1, so h moves by at most half a bf16 spacing of that mix
    (plus fp32 arithmetic)."""
    for j, (h, lse), ref, pre_ref in _run("sliced", c=4, b=2, T=200, d=1024, r=16, store="bf16", stack="bf16",
                                          pre="bf16", seed=17):
        bound = 0.5 * H.bf16_ulp(pre_ref["h"]) + 1e-5 * H.rms(ref["h"])
        assert np.all(np.abs(h - ref["h"]) <= bound), j
        H.assert_abs(f"lse[site {j}]", lse, ref["lse"], 1e-4)


def test_phase2_needs_the_partial_key_for_projected_keys():
    dev = torch.device("cuda")
    T, d, r = 8, 64, 4
    z = torch.zeros(T, d, device=dev)
    with pytest.raises(lrar.LrarError) as ei:
        lrar.block_phase2("projected", z, torch.zeros(T, device=dev), z, None, torch.zeros(r, device=dev),
                          torch.empty(T, d, device=dev))
    assert ei.value.code == lrar.ERR_INVALID_ARG


@pytest.mark.parametrize("d,n_c", [(2048, 9), (512, 3)])
def test_phase1_give_up_is_reported(d, n_c):
    """The test hook diverts every key-staging wait of phase 1 to a barrier that
    nothing completes, with a bound of 2^20 SM cycles (about half a
    millisecond): each wait runs out, the launch reports
    LRAR_STATUS_WAIT_TIMEOUT, drains the bulk copies it issued and returns.
    No fault, no hang: the next launch on the same context is correct."""
    T, r, c = 600, 64, 8
    dev = torch.device("cuda")
    vals = synth.outputs(n_c, T, d, seed=31, dtype="bf16").to(dev)
    qs = synth.queries(c, r, 31, std=0.5).to(dev)
    h_pre = torch.empty(c, T, d, dtype=torch.bfloat16, device=dev)
    lse_pre = torch.empty(c, T, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    lrar.test_block_phase1_stalled("sliced", vals, None, qs, h_pre, lse_pre, status, 1 << 20)
    torch.cuda.synchronize()
    assert status.item() == lrar.STATUS_WAIT_TIMEOUT
    # the context is intact: an ordinary launch right after is exact and reports nothing
    status.zero_()
    lrar.block_phase1("sliced", vals, None, qs, h_pre, lse_pre, status=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    toks = H.sample_tokens(T, k=16, seed=3)
    for j in (0, c - 1):
        ref = oracle.forward(oracle.SLICED, vals.cpu(), None, qs[j].cpu(), H.EPS, r=r, tokens=toks)
        H.assert_abs(f"lse_pre[{j}]", lse_pre[j].cpu().numpy()[toks], ref["lse"], 1e-4)
        H.assert_bf16_rounded(f"h_pre[{j}]", h_pre[j].double().cpu().numpy()[toks], ref["h"])


def test_phase1_status_stays_clear():
    """An ordinary phase-1 launch that stages its keys never writes status."""
    T, d, r, c = 300, 1024, 16, 4
    dev = torch.device("cuda")
    vals = synth.outputs(4, T, d, seed=32, dtype="bf16").to(dev)
    qs = synth.queries(c, r, 32, std=0.5).to(dev)
    status = torch.full((1,), 0x100, dtype=torch.int32, device=dev)  # bits the library must leave alone
    lrar.block_phase1("sliced", vals, None, qs, torch.empty(c, T, d, device=dev), torch.empty(c, T, device=dev),
                      status=status)
    torch.cuda.synchronize()
    assert status.item() == 0x100


@pytest.mark.parametrize("variant,dtype,pre,d,r", [("sliced", "bf16", "bf16", 1024, 16), ("sliced", "f32", "f32", 200, 8),
                                                   ("projected", "bf16", "f32", 512, 32)])
def test_phase2_assemble_equals_accumulate_then_phase2(variant, dtype, pre, d, r):
    """lrar_block_phase2_assemble forms the partial summary (running sum plus
    the newest member) inside phase 2: the summary it writes over the member,
    and h and lse, equal bit for bit lrar_block_accumulate followed by
    lrar_block_phase2 on the same inputs (in place: h is h_pre)."""
    dev = torch.device("cuda")
    T = 333
    sdt, pdt = H.TORCH_DTYPE[dtype], H.TORCH_DTYPE[pre]
    prev = synth.randn((T, d), 31, "values").to(sdt).to(dev)
    member = synth.randn((T, d), 32, "values").to(sdt).to(dev)
    h_pre = synth.randn((T, d), 33, "values").to(pdt).to(dev)
    lse_pre = (synth.randn((T,), 34, "scale") + 2.0).to(dev)
    query = synth.queries(1, r, 35, std=0.5)[0].to(dev)
    pkey = synth.randn((T, r), 36, "keys").to(sdt).to(dev) if variant == "projected" else None
    mkey = synth.randn((T, r), 37, "keys").to(sdt).to(dev) if variant == "projected" else None

    m_a, h_a, l_a = member.clone(), h_pre.clone(), lse_pre.clone()
    k_a = mkey.clone() if mkey is not None else None
    lrar.block_accumulate(m_a, prev, 1.0, 1.0)
    if k_a is not None:
        lrar.block_accumulate(k_a, pkey, 1.0, 1.0)
    lrar.block_phase2(variant, h_a, l_a, m_a, k_a, query, h_a, l_a)

    m_b, h_b, l_b = member.clone(), h_pre.clone(), lse_pre.clone()
    k_b = mkey.clone() if mkey is not None else None
    lrar.block_phase2_assemble(variant, h_b, l_b, prev, m_b, pkey, k_b, query, h_b, l_b)
    torch.cuda.synchronize()
    assert torch.equal(m_a, m_b)
    assert torch.equal(h_a, h_b)
    assert torch.equal(l_a, l_b)
    if k_a is not None:
        assert torch.equal(k_a, k_b)
