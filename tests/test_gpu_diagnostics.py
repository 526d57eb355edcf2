"""lrar_diagnostics (§4.5-4.6: N_eff of Eq. 16 per token, token-mean of alpha
per site) against the oracle's diagnostics on the same inputs.

Tolerance: both sides compute alpha from identical stored inputs; the GPU in
fp32 (softmax, logs and exps to a few ulp), so N_eff agrees to 1e-5 relative
and the mean to 1e-6 absolute (alpha <= 1).
"""
import numpy as np
import pytest
import torch

import gpu_helpers as H
import oracle
from paper_2607_09694_gb300 import lrar, synth

pytestmark = pytest.mark.gpu


def _gpu_diag(si, want_neff=True, want_mean=True, query=None):
    dev = torch.device("cuda")
    v = si.values.to(dev)
    k = si.keys.to(dev) if si.keys is not None else None
    q = (si.query if query is None else query).to(dev)
    neff = torch.full((si.T,), float("nan"), device=dev) if want_neff else None
    mean = torch.full((si.n,), float("nan"), device=dev) if want_mean else None
    ws = torch.empty(lrar.diagnostics_workspace_size(si.n) // 4, device=dev) if want_mean else None
    lrar.diagnostics(si.variant, v, k, q, neff, mean, ws, r=si.r)
    torch.cuda.synchronize()
    return (neff.double().cpu().numpy() if want_neff else None, mean.double().cpu().numpy() if want_mean else None)


def _ref(si, query=None):
    return oracle.diagnostics(H.ORACLE_VARIANT[si.variant], si.values, si.keys,
                              si.query if query is None else query, H.EPS, r=si.r)


@pytest.mark.parametrize("variant,cfg,kw", [("sliced", "slr", dict(n=49, T=1500)),
                                             ("projected", "plr", dict(n=33, T=777, r=32)),
                                             ("full", "slr", dict(n=17, T=300, d=512)),
                                             ("sliced", "tiny", dict()),
                                             ("sliced", "slr", dict(n=128, T=100, r=4))])
def test_matches_oracle(variant, cfg, kw):
    si = synth.site(cfg, variant=variant, **kw)
    neff, mean = _gpu_diag(si)
    ref = _ref(si)
    assert np.allclose(neff, ref["neff"], rtol=1e-5, atol=1e-6)
    assert np.allclose(mean, ref["mean_alpha"], rtol=0, atol=1e-6)
    assert np.all(neff >= 1 - 1e-5) and np.all(neff <= si.n * (1 + 1e-5))


def test_zero_query_uses_every_source():
    """The paper's zero-initialised queries (§4.1): uniform alpha, N_eff = n."""
    si = synth.site("slr", n=20, T=256)
    neff, mean = _gpu_diag(si, query=torch.zeros(si.r))
    assert np.allclose(neff, 20.0, rtol=1e-5)
    assert np.allclose(mean, 1.0 / 20, atol=1e-7)


def test_sharp_query_selects_one_source():
    si = synth.site("plr", n=6, T=64, r=8)
    keys = torch.zeros(si.keys.shape)
    keys[:, :, 0] = -1.0
    keys[3, :, 0] = 1.0
    si.keys = keys.to(torch.bfloat16)
    q = torch.tensor([500.0] + [0.0] * 7)
    neff, mean = _gpu_diag(si, query=q)
    assert np.allclose(neff, 1.0, atol=1e-5)
    assert abs(mean[3] - 1.0) < 1e-6


def test_outputs_are_optional():
    si = synth.site("slr", n=9, T=200)
    neff, _ = _gpu_diag(si, want_mean=False)
    _, mean = _gpu_diag(si, want_neff=False)
    ref = _ref(si)
    assert np.allclose(neff, ref["neff"], rtol=1e-5)
    assert np.allclose(mean, ref["mean_alpha"], atol=1e-6)


def test_reproducible():
    si = synth.site("slr", n=49, T=3000)
    a = _gpu_diag(si)
    b = _gpu_diag(si)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])
