"""Host logic of the Block AttnRes driver (sweep.BlockSweep) on the CPU: the
library's entry points are replaced by plain torch stand-ins (assembly as
dst = beta dst + alpha src, phase 2's assembling form as member += prev), so
the order of calls and the tensors each one receives can be checked without a
GPU -- the assembled running sums (Eq. 5-6) against the oracle's own assembly,
each site's sources, and the backward's accumulation flags, gradient slots and
member hand-over order."""
import contextlib
import types

import numpy as np
import pytest
import torch

import oracle
from paper_2607_09694_gb300 import lrar, sites
from paper_2607_09694_gb300.sweep import BlockSweep

STREAM = types.SimpleNamespace(cuda_stream=0)


class FakeLib:
    def __init__(self, sweep_ref):
        self.calls = []
        self.sw = sweep_ref

    def block_accumulate(self, dst, src, alpha, beta, stream=None):
        dst.mul_(beta).add_(src, alpha=alpha)
        self.calls.append(("acc", id(dst), id(src)))

    def block_phase1_ptrs(self, variant, values, keys, queries, h_pre, lse_pre, eps=None, status=None, stream=None):
        self.calls.append(("ph1", [v.clone() for v in values], queries.shape[0]))

    def block_phase2(self, variant, h_pre, lse_pre, partial, pkey, query, h, lse, eps=None, stream=None):
        self.calls.append(("ph2", partial.clone()))

    def block_phase2_assemble(self, variant, h_pre, lse_pre, prev, member, pkey, mkey, query, h, lse, eps=None,
                              stream=None):
        member.add_(prev)
        if mkey is not None:
            mkey.add_(pkey)
        self.calls.append(("ph2a", member.clone()))

    def forward_ptrs(self, variant, values, keys, query, h, lse, r=None, eps=None, stream=None):
        self.calls.append(("fwd", [v.clone() for v in values]))

    def backward_ptrs(self, variant, values, keys, query, dh, dvalues, dq, ws, dkeys=None, h=None, lse=None, r=None,
                      accumulate=False, eps=None, stream=None):
        self.calls.append(("bwd", [id(g) for g in dvalues], bool(accumulate), len(values)))


@pytest.fixture
def fake(monkeypatch):
    lib = FakeLib(None)
    for name in ("block_accumulate", "block_phase1_ptrs", "block_phase2", "block_phase2_assemble", "forward_ptrs",
                 "backward_ptrs"):
        monkeypatch.setattr(lrar, name, getattr(lib, name))
    monkeypatch.setattr(torch.cuda, "stream", lambda s: contextlib.nullcontext())
    return lib


def _sweep(M, c, two_phase, T=3, d=16, r=4, seed=5):
    g = torch.Generator().manual_seed(seed)
    outs = torch.randn(M + 1, T, d, generator=g, dtype=torch.float64)
    o = [outs[i].clone() for i in range(M + 1)]
    q = torch.randn(M + 1, r, generator=g)
    dh = [torch.zeros(T, d) for _ in range(M + 1)]
    h = torch.zeros(M + 1, T, d)
    lse = torch.zeros(M + 1, T)
    do = [torch.zeros(T, d) for _ in range(M + 1)]
    sw = BlockSweep("sliced", o, q, dh, h, lse, do, c, r=r, two_phase=two_phase)
    return sw, outs


@pytest.mark.parametrize("M,c", [(12, 4), (13, 4), (7, 1), (9, 3), (5, 8)])
@pytest.mark.parametrize("two_phase", [False, True])
def test_forward_assembles_the_block_sums_and_feeds_each_site(fake, M, c, two_phase):
    sw, outs = _sweep(M, c, two_phase)
    sw.forward(STREAM)
    # every output tensor ends as its block's running sum (Eq. 5-6)
    run = outs.clone()
    for i in range(1, M + 1):
        if not sites.block_opens_slot(i, c):
            run[i] = run[i - 1] + outs[i]
    for i in range(M + 1):
        assert torch.equal(sw.outputs[i], run[i]), i
    # each site mixes exactly the oracle's Block source set of o_0 .. o_{t-1}
    seen = {}
    if not two_phase:
        fw = [cl for cl in fake.calls if cl[0] == "fwd"]
        assert len(fw) == M + 1
        for t, cl in enumerate(fw, start=1):
            seen[t] = cl[1]
    else:
        t = 1
        for cl in fake.calls:
            if cl[0] == "ph1":
                srcs, ns = cl[1], cl[2]
                seen[t] = srcs  # the block's first site: the completed sources only
                base, t = srcs, t + 1
            elif cl[0] in ("ph2", "ph2a"):
                seen[t] = base + [cl[1]]  # completed sources + the partial summary as phase 2 saw it
                t += 1
        assert t == M + 2
    for t in range(1, M + 2):
        ref = oracle.block_sources(outs[:t].float(), c)
        got = torch.stack([x.float() for x in seen[t]])
        assert got.shape == ref.shape, t
        assert np.allclose(got.numpy(), np.asarray(ref), atol=1e-5), t


@pytest.mark.parametrize("M,c", [(12, 4), (13, 4), (9, 3)])
def test_two_phase_assembles_inside_phase2_where_a_running_sum_exists(fake, M, c):
    sw, _ = _sweep(M, c, True)
    sw.forward(STREAM)
    kinds = [cl[0] for cl in fake.calls if cl[0] in ("ph2", "ph2a")]
    assert kinds.count("ph2a") == sites.block_phase2_assembled_sites(M, c)
    # separate accumulations remain only where a block completes before its phase 1
    n_acc = sum(1 for cl in fake.calls if cl[0] == "acc")
    n_members = sum(1 for i in range(1, M + 1) if not sites.block_opens_slot(i, c))
    assert n_acc + kinds.count("ph2a") == n_members


@pytest.mark.parametrize("M,c", [(12, 4), (13, 4)])
def test_backward_flags_slots_and_member_hand_over(fake, M, c):
    sw, _ = _sweep(M, c, True)
    sw.forward(STREAM)
    fake.calls.clear()
    order = []
    sw.backward(STREAM, member_grad=lambda i, g, gk: order.append((i, id(g))))
    bw = [cl for cl in fake.calls if cl[0] == "bwd"]
    assert len(bw) == M + 1
    for k, (_, grads, acc, n) in enumerate(bw):
        t = M + 1 - k
        idx = sw.site_sources(t)
        assert n == len(idx) == sites.block_num_sources(t, c)
        assert grads == [id(sw.grads[sites.block_slot(i, c)]) for i in idx]
        assert acc == (t != M + 1)  # the first backward writes every slot it reads
    assert [i for i, _ in order] == list(range(M, -1, -1))
    assert all(gid == id(sw.grads[sites.block_slot(i, c)]) for i, gid in order)
    assert not any(cl[0] == "acc" for cl in fake.calls)  # no fan-out copies when handed over


@pytest.mark.parametrize("variant", ["sliced", "projected"])
def test_depth_sweep_order_sources_and_flags(fake, variant):
    """sweep.DepthSweep (Full AttnRes over separate source tensors, Eq. 4): site t
    mixes sources o_0..o_{t-1} with query row t-1 (none at site 1); the backward
    runs t = n..1, the first call writing every gradient and the rest adding,
    each over the same prefix of sources (and keys); dq starts from zero."""
    from paper_2607_09694_gb300.sweep import DepthSweep

    n, T, d, r = 6, 3, 16, 4
    src = [torch.full((T, d), float(i)) for i in range(n)]
    keys = [torch.zeros(T, r) for _ in range(n)] if variant == "projected" else None
    dkeys = [torch.zeros(T, r) for _ in range(n)] if variant == "projected" else None
    q = torch.randn(n, r)
    dq = torch.ones(n, r)
    ds = [torch.zeros(T, d) for _ in range(n)]
    sw = DepthSweep(variant, src, q, [torch.zeros(T, d)] * n, torch.zeros(n, T, d), torch.zeros(n, T), ds, dq,
                    keys=keys, dkeys=dkeys, r=r)
    sw.step(STREAM)
    fw = [cl for cl in fake.calls if cl[0] == "fwd"]
    assert [len(cl[1]) for cl in fw] == list(range(1, n + 1))
    for t, cl in enumerate(fw, start=1):
        assert [float(v[0, 0]) for v in cl[1]] == [float(i) for i in range(t)]
    bw = [cl for cl in fake.calls if cl[0] == "bwd"]
    assert [cl[3] for cl in bw] == list(range(n, 0, -1))
    assert [cl[2] for cl in bw] == [False] + [True] * (n - 1)
    assert all(cl[1] == [id(g) for g in ds[:cl[3]]] for cl in bw)
    assert torch.count_nonzero(dq) == 0
