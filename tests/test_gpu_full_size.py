"""Parity at the workloads' full sizes, in the configuration the benchmark
times (bf16 values, bf16 h, bf16 gradients accumulated into a live buffer).

Every h / lse / dvalues row of a sample of tokens (edges, warp and CTA
boundaries of the persistent grid, random tokens) is compared with the
oracle; dq, a sum over all T tokens, is compared with the oracle's sum over
all T tokens.
"""
import numpy as np
import pytest
import torch

import gpu_helpers as H
import oracle
from paper_2607_09694_gb300 import lrar, synth

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


@pytest.fixture(scope="module")
def slr_values():
    c = synth.CONFIGS["slr"]
    return synth.values(c["n"], c["T"], c["d"], c["seed"], "bf16", c["scale"])


@pytest.fixture(scope="module")
def plr_values():
    c = synth.CONFIGS["plr"]
    return synth.values(c["n"], c["T"], c["d"], c["seed"], "bf16")


def _site(config, values, r=None, variant=None):
    c = synth.CONFIGS[config]
    variant = variant or c["variant"]
    n, T, d = values.shape
    r = d if variant == "full" else (c["r"] if r is None else r)
    seed = c["seed"]
    keys = synth.keys(n, T, r, seed, "bf16") if variant == "projected" else None
    q = synth.queries(1, r, seed)[0].contiguous()
    dh = synth.upstream(T, d, seed, "bf16")
    return synth.SiteInputs(variant, n, T, d, r, values, keys, q, dh)


def _bench_like(si):
    """Accumulate into a buffer that already holds a per-source constant i/64
    (exact in bf16), as the all-sites sweep does."""
    n = si.n
    dv0 = torch.empty(n, si.T, si.d, dtype=torch.bfloat16)
    for i in range(n):
        dv0[i].fill_(i / 64.0)
    init = dict(dvalues=dv0, dq=torch.zeros(si.d if si.variant == "full" else si.r))
    if si.keys is not None:
        init["dkeys"] = torch.zeros(si.keys.shape, dtype=torch.bfloat16)
    toks = H.sample_tokens(si.T)
    h_out = "f32" if si.variant == "full" else "bf16"  # full keys: exact gbar = <dh, h> needs an fp32 h
    got = H.run_gpu(si, h_out, "bf16", accumulate=True, init=init, tokens=toks)
    ov = H.ORACLE_VARIANT[si.variant]
    f = oracle.forward(ov, si.values, si.keys, si.query, H.EPS, r=si.r, tokens=toks)
    b = oracle.backward(ov, si.values, si.keys, si.query, H.EPS, si.dh, r=si.r, tokens=toks)
    dq_all = oracle.backward(ov, si.values, si.keys, si.query, H.EPS, si.dh, r=si.r, want_dvalues=False)["dq"]
    if h_out == "bf16":
        H.assert_bf16_rounded("h", got["h"], f["h"])
    else:
        H.assert_rms("h", got["h"], f["h"], 1e-5)
    H.assert_abs("lse", got["lse"], f["lse"], 1e-4)
    dv_ref = b["dvalues"] + (np.arange(si.n) / 64.0)[:, None, None]
    H.assert_bf16_rounded("dvalues", got["dvalues"], dv_ref)
    if si.keys is not None:
        H.assert_bf16_rounded("dkeys", got["dkeys"], b["dkeys"])
    H.assert_rms("dq", got["dq"], dq_all)
    return got, f, b


def test_slr_d1024_n49_bench_configuration(slr_values):
    _bench_like(_site("slr", slr_values))


def test_slr_d1024_n49_fp32_outputs(slr_values):
    si = _site("slr", slr_values)
    toks = H.sample_tokens(si.T, seed=1)
    got = H.run_gpu(si, "f32", "f32", tokens=toks)
    ref = H.run_oracle(si, tokens=toks)
    H.assert_rms("h", got["h"], ref["h"])
    H.assert_rms("dvalues", got["dvalues"], ref["dvalues"])


def test_full_attnres_d1024_n49(slr_values):
    _bench_like(_site("full", slr_values, variant="full"))


@pytest.mark.parametrize("r", [4, 8, 16, 32, 64])
def test_plr_d1024_n49_rank_sweep(r, plr_values):
    _bench_like(_site("plr", plr_values, r=r))


def test_all_sites_prefixes(slr_values):
    """A few sites of the 24-layer sweep (n = 2, 25, 48) read prefixes of the stack."""
    si = _site("slr", slr_values)
    toks = H.sample_tokens(si.T, k=16, seed=2)
    for n in (2, 25, 48):
        got = H.run_gpu(si, "f32", "f32", n_src=n, tokens=toks)
        ref = H.run_oracle(si, tokens=toks, n_src=n)
        H.assert_rms(f"h[n={n}]", got["h"], ref["h"])
        H.assert_rms(f"dvalues[n={n}]", got["dvalues"][:n], ref["dvalues"])
        assert np.all(np.isnan(got["dvalues"][n:]))


def test_slr_d2048_n65_t32768():
    c = synth.CONFIGS["slr_large"]
    vals = synth.values(c["n"], c["T"], c["d"], c["seed"], "bf16")
    _bench_like(_site("slr_large", vals))


def test_block_two_phase_d2048_t32768():
    """The Block decoder's last block at full size (T = 32768, d = 2048, r = 64,
    c = 8, 9 completed sources, bf16 h_pre as the benchmark's faster setting):
    phase 1 for the block's eight sites, phase 2 for one of them, on sampled
    tokens against the oracle's mix over the site's whole source set."""
    c = synth.CONFIGS["block"]
    T, d, r, cb = c["T"], c["d"], c["r"], c["block_c"]
    n = 9
    dev = torch.device("cuda")
    stack = synth.values(n + 1, T, d, c["seed"], "bf16")  # 9 completed sources, then a partial summary
    qs = synth.queries(cb, r, c["seed"], std=0.5)
    sd = stack.to(dev)
    h_pre = torch.empty(cb, T, d, dtype=torch.bfloat16, device=dev)
    lse_pre = torch.empty(cb, T, device=dev)
    lrar.block_phase1("sliced", sd, None, qs.to(dev), h_pre, lse_pre, n_completed=n)
    h = torch.empty(T, d, device=dev)
    lse = torch.empty(T, device=dev)
    lrar.block_phase2("sliced", h_pre[3], lse_pre[3], sd[n], None, qs[3].to(dev), h, lse)
    torch.cuda.synchronize()
    toks = H.sample_tokens(T, k=24, seed=3)
    idx = torch.as_tensor(toks, dtype=torch.long, device=dev)
    # phase 1 alone: site 0's mix over the completed sources (h_pre rounded to bf16 once)
    ref1 = oracle.forward(oracle.SLICED, stack[:n], None, qs[0], H.EPS, r=r, tokens=toks)
    H.assert_bf16_rounded("h_pre[0]", h_pre[0].index_select(0, idx).double().cpu().numpy(), ref1["h"])
    H.assert_abs("lse_pre[0]", lse_pre[0].index_select(0, idx).double().cpu().numpy(), ref1["lse"], 1e-4)
    # both phases: site 3's mix over the completed sources and the partial summary
    ref = oracle.forward(oracle.SLICED, stack, None, qs[3], H.EPS, r=r, tokens=toks)
    got = h.index_select(0, idx).double().cpu().numpy()
    pre_ref = oracle.forward(oracle.SLICED, stack[:n], None, qs[3], H.EPS, r=r, tokens=toks)
    bound = 0.5 * H.bf16_ulp(pre_ref["h"]) + 1e-5 * H.rms(ref["h"])  # h_pre rounded once, weight <= 1
    assert np.all(np.abs(got - ref["h"]) <= bound)
    H.assert_abs("lse", lse.index_select(0, idx).double().cpu().numpy(), ref["lse"], 1e-4)
