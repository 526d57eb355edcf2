"""Pins of the fp64 oracle against what the paper and the mathematics fix.

None of these re-type the oracle's formulas: each checks a property, a closed
form of a special case, or a finite difference, chosen so that a plausible
slip in the oracle (a dropped term, a wrong sign, a wrong index, the wrong key
slice, a misplaced epsilon, a transposed operand) fails at least one of them.
"""
import numpy as np
import pytest

import oracle
from oracle import FULL, PROJECTED, SLICED

EPS = 1e-6


def _rng(seed):
    return np.random.default_rng(seed)


def _case(variant, n, T, d, r, seed=0, q_std=1.0):
    g = _rng(seed)
    values = g.standard_normal((n, T, d))
    keys = g.standard_normal((n, T, r)) if variant == PROJECTED else None
    q = g.standard_normal(r) * q_std
    dh = g.standard_normal((T, d))
    return values, keys, q, dh


@pytest.mark.parametrize("variant,d,r", [(SLICED, 16, 4), (PROJECTED, 16, 4), (FULL, 12, 12)])
def test_weights_are_a_distribution(variant, d, r):
    """Eq. (9): alpha is a softmax, so alpha_i > 0 and sum_i alpha_i = 1."""
    v, k, q, _ = _case(variant, 7, 5, d, r, seed=1)
    out = oracle.forward(variant, v, k, q, EPS, r=r, want_alpha=True)
    a = out["alpha"]
    assert np.all(a > 0)
    assert np.max(np.abs(a.sum(axis=1) - 1.0)) < 1e-14


def test_sliced_key_is_the_tail():
    """Eq. (14): identical last-r coordinates give identical keys, whatever the
    first d - r coordinates hold, so the weights are uniform and h is the mean."""
    n, T, d, r = 5, 4, 12, 3
    v, _, q, _ = _case(SLICED, n, T, d, r, seed=2)
    v[:, :, d - r:] = v[0:1, :, d - r:]
    out = oracle.forward(SLICED, v, None, q, EPS, r=r, want_alpha=True)
    assert np.allclose(out["alpha"], 1.0 / n, atol=1e-15)
    assert np.allclose(out["h"], v.mean(axis=0), atol=1e-14)
    # The same values with distinct tails but identical heads are not uniform.
    v2, _, q2, _ = _case(SLICED, n, T, d, r, seed=2)
    v2[:, :, : d - r] = v2[0:1, :, : d - r]
    a2 = oracle.forward(SLICED, v2, None, q2, EPS, r=r, want_alpha=True)["alpha"]
    assert np.max(np.abs(a2 - 1.0 / n)) > 1e-3


def test_identical_projected_keys_give_the_mean():
    n, T, d, r = 6, 3, 8, 4
    v, k, q, _ = _case(PROJECTED, n, T, d, r, seed=3)
    k[:] = k[0:1]
    out = oracle.forward(PROJECTED, v, k, q, EPS, want_alpha=True)
    assert np.allclose(out["alpha"], 1.0 / n, atol=1e-15)
    assert np.allclose(out["h"], v.mean(axis=0), atol=1e-14)


@pytest.mark.parametrize("variant,d,r", [(SLICED, 16, 4), (PROJECTED, 16, 4), (FULL, 8, 8)])
def test_zero_query_is_uniform(variant, d, r):
    """§4.1 initialises the queries to zero: every score is 0, alpha uniform,
    lse = log n, and the value-path gradient is dh / n."""
    n, T = 5, 3
    v, k, _, dh = _case(variant, n, T, d, r, seed=4)
    q = np.zeros(r)
    out = oracle.forward(variant, v, k, q, EPS, r=r, want_alpha=True)
    assert np.allclose(out["alpha"], 1.0 / n, atol=1e-15)
    assert np.allclose(out["lse"], np.log(n), atol=1e-14)


@pytest.mark.parametrize("variant,d,r", [(SLICED, 16, 4), (PROJECTED, 16, 4), (FULL, 8, 8)])
def test_single_source_is_identity(variant, d, r):
    """n = 1 (site 1): h = o_0, dvalues = dh, no key or query gradient."""
    v, k, q, dh = _case(variant, 1, 4, d, r, seed=5)
    f = oracle.forward(variant, v, k, q, EPS, r=r)
    assert np.array_equal(f["h"], v[0])
    b = oracle.backward(variant, v, k, q, EPS, dh, r=r)
    assert np.allclose(b["dvalues"][0], dh, atol=1e-15)
    assert np.max(np.abs(b["dq"])) < 1e-15 and np.max(b["dq_abs"]) < 1e-15
    if variant == PROJECTED:
        assert np.max(np.abs(b["dkeys"])) < 1e-15


def test_two_sources_closed_form():
    """With k_i = c_i u and u in {-1,+1}^r, mean(k_i^2) = c_i^2, so Eq. (8) gives
    kbar_i = c_i / sqrt(c_i^2 + eps) u exactly; Eq. (9) then reduces to the
    logistic alpha_1 = 1 / (1 + exp(s_0 - s_1)) and lse = logaddexp(s_0, s_1).
    Small c_i make the epsilon placement matter."""
    r, d, T = 8, 10, 1
    g = _rng(6)
    u = np.where(g.standard_normal(r) > 0, 1.0, -1.0)
    q = g.standard_normal(r)
    c = np.array([1e-3, -3e-3])
    keys = np.stack([ci * u for ci in c])[:, None, :]
    v = g.standard_normal((2, T, d))
    qu = float(q @ u)
    s = c / np.sqrt(c * c + EPS) * qu
    a1 = 1.0 / (1.0 + np.exp(s[0] - s[1]))
    out = oracle.forward(PROJECTED, v, keys, q, EPS, want_alpha=True)
    assert abs(out["alpha"][0, 1] - a1) < 1e-14
    assert abs(out["lse"][0] - np.logaddexp(s[0], s[1])) < 1e-14
    assert np.allclose(out["h"][0], (1 - a1) * v[0, 0] + a1 * v[1, 0], atol=1e-14)
    # The score gradient of a two-way softmax is the logistic derivative:
    # ds_1 = a1 (1 - a1) (g_1 - g_0) with g_i = <dh, o_i>.
    dh = g.standard_normal((T, d))
    b = oracle.backward(PROJECTED, v, keys, q, EPS, dh, want_ds=True)
    gi = v[:, 0, :] @ dh[0]
    assert abs(b["ds"][0, 1] - a1 * (1 - a1) * (gi[1] - gi[0])) < 1e-13
    # dq = sum_i ds_i kbar_i with ds_0 = -ds_1 and kbar_i = kappa_i u; the two
    # terms share a sign (kappa_0 > 0 > kappa_1), so the magnitude of the terms
    # summed, dq_abs = sum_i |ds_i kbar_i|, equals |dq| here
    kap = c / np.sqrt(c * c + EPS)
    ds1 = a1 * (1 - a1) * (gi[1] - gi[0])
    assert np.allclose(b["dq"], ds1 * (kap[1] - kap[0]) * u, rtol=1e-12, atol=1e-15)
    assert np.allclose(b["dq_abs"], abs(ds1) * (abs(kap[0]) + abs(kap[1])) * np.ones(r), rtol=1e-12, atol=1e-15)


def test_zero_key_scores_zero():
    """A zero key normalises to zero (eps > 0), so its score is 0."""
    r, d = 4, 4
    g = _rng(7)
    keys = g.standard_normal((2, 1, r))
    keys[0] = 0.0
    v = g.standard_normal((2, 1, d))
    q = g.standard_normal(r)
    kb1 = keys[1, 0] / np.sqrt(np.mean(keys[1, 0] ** 2) + EPS)
    a = oracle.forward(PROJECTED, v, keys, q, EPS, want_alpha=True)["alpha"][0]
    assert abs(a[1] - 1.0 / (1.0 + np.exp(0.0 - q @ kb1))) < 1e-14


def test_sliced_rank_d_equals_attnres():
    """§3.4: with r = d, S-LR-AttnRes is AttnRes (keys o_i), forward and backward."""
    n, T, d = 4, 3, 6
    v, _, q, dh = _case(FULL, n, T, d, d, seed=8)
    fs = oracle.forward(SLICED, v, None, q, EPS, r=d)
    ff = oracle.forward(FULL, v, None, q, EPS, r=d)
    assert np.allclose(fs["h"], ff["h"], atol=1e-15) and np.allclose(fs["lse"], ff["lse"], atol=1e-15)
    bs = oracle.backward(SLICED, v, None, q, EPS, dh, r=d)
    bf = oracle.backward(FULL, v, None, q, EPS, dh, r=d)
    assert np.allclose(bs["dvalues"], bf["dvalues"], atol=1e-14)
    assert np.allclose(bs["dq"], bf["dq"], atol=1e-14)


@pytest.mark.parametrize("variant,d,r", [(SLICED, 10, 3), (PROJECTED, 10, 3)])
def test_source_permutation(variant, d, r):
    """Softmax over a set: permuting sources permutes alpha and the value
    gradients and leaves h, lse and dq unchanged."""
    n, T = 6, 4
    v, k, q, dh = _case(variant, n, T, d, r, seed=9)
    p = _rng(10).permutation(n)
    f0 = oracle.forward(variant, v, k, q, EPS, r=r, want_alpha=True)
    f1 = oracle.forward(variant, v[p], None if k is None else k[p], q, EPS, r=r, want_alpha=True)
    assert np.allclose(f0["h"], f1["h"], atol=1e-14)
    assert np.allclose(f0["alpha"][:, p], f1["alpha"], atol=1e-15)
    b0 = oracle.backward(variant, v, k, q, EPS, dh, r=r)
    b1 = oracle.backward(variant, v[p], None if k is None else k[p], q, EPS, dh, r=r)
    assert np.allclose(b0["dvalues"][p], b1["dvalues"], atol=1e-14)
    assert np.allclose(b0["dq"], b1["dq"], atol=1e-13)


@pytest.mark.parametrize("variant,d,r", [(SLICED, 10, 3), (FULL, 8, 8)])
def test_hidden_coordinate_permutation(variant, d, r):
    """§3.4: which r coordinates form the S-LR key is arbitrary up to a
    permutation of the hidden coordinates.  Permuting the head coordinates
    among themselves and the key coordinates among themselves (with the query
    permuted alike) permutes h, the value gradients and dq the same way, and
    leaves lse unchanged; for full keys any permutation does."""
    n, T = 5, 4
    v, _, q, dh = _case(variant, n, T, d, r, seed=12)
    g = _rng(13)
    head, tail = np.arange(d - r), np.arange(d - r, d)
    perm = np.concatenate([g.permutation(head), d - r + g.permutation(r)]) if variant == SLICED \
        else g.permutation(d)
    qperm = perm[d - r:] - (d - r)  # the key slice's own coordinates, in the permuted order
    f0 = oracle.forward(variant, v, None, q, EPS, r=r)
    f1 = oracle.forward(variant, v[:, :, perm], None, q[qperm], EPS, r=r)
    assert np.allclose(f0["h"][:, perm], f1["h"], atol=1e-14)
    assert np.allclose(f0["lse"], f1["lse"], atol=1e-14)
    b0 = oracle.backward(variant, v, None, q, EPS, dh, r=r)
    b1 = oracle.backward(variant, v[:, :, perm], None, q[qperm], EPS, dh[:, perm], r=r)
    assert np.allclose(b0["dvalues"][:, :, perm], b1["dvalues"], atol=1e-13)
    assert np.allclose(b0["dq"][qperm], b1["dq"], atol=1e-13)


def test_key_scale_invariance():
    """RMSNorm makes the score invariant to positive rescaling of a key, up to eps."""
    n, T, d, r = 5, 3, 8, 4
    v, k, q, _ = _case(PROJECTED, n, T, d, r, seed=11)
    k2 = k.copy()
    k2[2] *= 3.7
    k2[4] *= 0.25
    a = oracle.forward(PROJECTED, v, k, q, 1e-14, want_alpha=True)["alpha"]
    b = oracle.forward(PROJECTED, v, k2, q, 1e-14, want_alpha=True)["alpha"]
    assert np.max(np.abs(a - b)) < 1e-11


@pytest.mark.parametrize("variant,d,r", [(SLICED, 12, 4), (PROJECTED, 12, 4), (FULL, 6, 6)])
def test_score_gradients_sum_to_zero(variant, d, r):
    """Softmax is invariant to adding a constant to every score, so sum_i ds_i = 0."""
    v, k, q, dh = _case(variant, 7, 5, d, r, seed=12)
    out = oracle.backward(variant, v, k, q, EPS, dh, r=r, want_ds=True)
    ds = out["ds"]
    assert np.max(np.abs(ds.sum(axis=1))) < 1e-13
    assert np.max(np.abs(ds)) > 1e-3
    # the magnitude of the terms of dq bounds |dq| (triangle inequality) and,
    # over many tokens of mixed sign, exceeds it
    assert np.all(out["dq_abs"] >= np.abs(out["dq"]) - 1e-15)
    assert np.all(out["dq_abs"] > np.abs(out["dq"]))


def test_key_gradient_is_orthogonal_to_key():
    """RMSNorm is scale-invariant as eps -> 0, so <k_i, dL/dk_i> = 0."""
    v, k, q, dh = _case(PROJECTED, 5, 4, 8, 6, seed=13)
    dk = oracle.backward(PROJECTED, v, k, q, 1e-14, dh)["dkeys"]
    dots = np.einsum("ntr,ntr->nt", k, dk)
    assert np.max(np.abs(dots)) < 1e-10
    assert np.max(np.abs(dk)) > 1e-3


def test_linear_in_values_for_fixed_keys():
    """P-LR: with keys fixed, h is linear in the values (Eq. 10)."""
    v, k, q, _ = _case(PROJECTED, 5, 3, 8, 4, seed=14)
    w = _rng(15).standard_normal(v.shape)
    h1 = oracle.forward(PROJECTED, v, k, q, EPS)["h"]
    h2 = oracle.forward(PROJECTED, w, k, q, EPS)["h"]
    h3 = oracle.forward(PROJECTED, 2.0 * v - 0.5 * w, k, q, EPS)["h"]
    assert np.allclose(h3, 2.0 * h1 - 0.5 * h2, atol=1e-13)


def _loss(variant, v, k, q, dh, r):
    return float(np.sum(oracle.forward(variant, v, k, q, EPS, r=r)["h"] * dh))


@pytest.mark.parametrize("variant,n,T,d,r", [(SLICED, 4, 3, 8, 2), (PROJECTED, 4, 3, 8, 2), (FULL, 3, 2, 6, 6)])
def test_gradients_match_central_differences(variant, n, T, d, r):
    """Every gradient the oracle returns equals a central difference of
    L = sum <dh, h> in fp64 (step 1e-6)."""
    v, k, q, dh = _case(variant, n, T, d, r, seed=16)
    b = oracle.backward(variant, v, k, q, EPS, dh, r=r)
    step = 1e-6

    def fd(arr, idx, fn):
        old = arr[idx]
        arr[idx] = old + step
        lp = fn()
        arr[idx] = old - step
        lm = fn()
        arr[idx] = old
        return (lp - lm) / (2 * step)

    L = lambda: _loss(variant, v, k, q, dh, r)  # noqa: E731
    num_v = np.zeros_like(v)
    for idx in np.ndindex(v.shape):
        num_v[idx] = fd(v, idx, L)
    num_q = np.array([fd(q, (j,), L) for j in range(r)])
    scale = max(1.0, np.max(np.abs(b["dvalues"])))
    assert np.max(np.abs(num_v - b["dvalues"])) / scale < 1e-7
    assert np.max(np.abs(num_q - b["dq"])) / max(1.0, np.max(np.abs(b["dq"]))) < 1e-7
    if variant == PROJECTED:
        num_k = np.zeros_like(k)
        for idx in np.ndindex(k.shape):
            num_k[idx] = fd(k, idx, L)
        assert np.max(np.abs(num_k - b["dkeys"])) / max(1.0, np.max(np.abs(b["dkeys"]))) < 1e-7


def test_sampled_tokens_match_full_evaluation():
    """Per-token evaluation: a token list gives the same rows as the full run,
    and dq over a token list is the sum of per-token dq."""
    v, k, q, dh = _case(SLICED, 5, 9, 12, 4, seed=17)
    full = oracle.forward(SLICED, v, None, q, EPS, r=4)
    toks = [8, 0, 3]
    part = oracle.forward(SLICED, v, None, q, EPS, r=4, tokens=toks)
    assert np.array_equal(part["h"], full["h"][toks])
    per = sum(oracle.backward(SLICED, v, None, q, EPS, dh, r=4, tokens=[t])["dq"] for t in range(9))
    allq = oracle.backward(SLICED, v, None, q, EPS, dh, r=4)["dq"]
    assert np.allclose(per, allq, atol=1e-13)


def test_bf16_inputs_decode_exactly():
    """Raw bfloat16 words decode to the exact same doubles as their fp32 widening."""
    import torch

    g = torch.Generator().manual_seed(0)
    vb = torch.randn(3, 4, 16, generator=g).to(torch.bfloat16)
    q = torch.randn(4, generator=g)
    a = oracle.forward(SLICED, vb, None, q, EPS, r=4)
    b = oracle.forward(SLICED, vb.double(), None, q, EPS, r=4)
    assert np.array_equal(a["h"], b["h"])


def test_effective_sources_range():
    """Eq. (16): N_eff = 1 for a one-hot distribution, n for a uniform one,
    and lies in [1, n] otherwise (§4.5)."""
    n, T, d, r = 6, 5, 8, 4
    v, k, q, _ = _case(PROJECTED, n, T, d, r, seed=18)
    uni = oracle.diagnostics(PROJECTED, v, k, np.zeros(r), EPS)
    assert np.allclose(uni["neff"], n, atol=1e-12)
    assert np.allclose(uni["mean_alpha"], 1.0 / n, atol=1e-15)
    sharp_k = np.zeros_like(k)
    sharp_k[:, :, 0] = -1.0
    sharp_k[2, :, 0] = 1.0
    sharp = oracle.diagnostics(PROJECTED, v, sharp_k, np.array([1e4, 0, 0, 0.0]), EPS)
    assert np.allclose(sharp["neff"], 1.0, atol=1e-12)
    assert np.allclose(sharp["mean_alpha"][2], 1.0, atol=1e-12)
    mid = oracle.diagnostics(PROJECTED, v, k, q, EPS)
    assert np.all(mid["neff"] >= 1.0) and np.all(mid["neff"] <= n)


def test_block_assembly_special_cases():
    """Eq. (5)-(6): with c = 1 every output is its own block (the stack is the
    outputs, as in Full AttnRes); with c >= t - 1 the stack is the embedding
    plus one partial sum of all later outputs."""
    g = _rng(19)
    t, T, w = 7, 3, 5
    outs = g.standard_normal((t, T, w))
    assert np.array_equal(oracle.block_sources(outs, 1), outs)
    s = oracle.block_sources(outs, 10)
    assert s.shape == (2, T, w)
    assert np.array_equal(s[0], outs[0])
    assert np.allclose(s[1], outs[1:].sum(axis=0), atol=1e-14)
    s3 = oracle.block_sources(outs, 3)
    assert s3.shape == (3, T, w)
    assert np.allclose(s3[1], outs[1:4].sum(axis=0), atol=1e-14)
    assert np.allclose(s3[2], outs[4:7].sum(axis=0), atol=1e-14)


@pytest.mark.parametrize("t,c", [(1, 3), (5, 2), (9, 4), (10, 4), (13, 3)])
def test_block_fanout_is_the_adjoint(t, c):
    """The fan-out is the transpose of the assembly: <dS, A(o)> = <A^T(dS), o>."""
    g = _rng(20 + t)
    T, w = 2, 3
    outs = g.standard_normal((t, T, w))
    src = oracle.block_sources(outs, c)
    dsrc = g.standard_normal(src.shape)
    dout = oracle.block_fanout(dsrc, t, c)
    assert abs(np.sum(dsrc * src) - np.sum(dout * outs)) < 1e-12
    assert src.shape[0] == oracle.block_num_sources(t, c)


# ------------------------------------------------ P-LR fused projection ----
def test_projection_matches_a_library_matmul():
    """Eq. (11)-(12): [o; k] = [W_O; W_K] a equals numpy's float64 matmul of the
    same operands (an independent routine), split after the first d rows."""
    g = _rng(31)
    T, m, d, r = 9, 24, 10, 6
    a = g.standard_normal((T, m))
    w = g.standard_normal((d + r, m))
    out = oracle.projection(a, w, d)
    y = a @ w.T
    assert np.allclose(out["o"], y[:, :d], rtol=1e-13, atol=1e-13)
    assert np.allclose(out["keys"], y[:, d:], rtol=1e-13, atol=1e-13)


def test_projection_selects_rows():
    """W_O = I gives o = a exactly; each W_K row a unit vector e_j picks a's
    coordinate j (pins the split and catches a transposed operand)."""
    g = _rng(32)
    T, m, r = 4, 6, 3
    a = g.standard_normal((T, m))
    pick = [5, 0, 2]
    w = np.concatenate([np.eye(m), np.eye(m)[pick]], axis=0)
    out = oracle.projection(a, w, m)
    assert np.array_equal(out["o"], a)
    assert np.array_equal(out["keys"], a[:, pick])


def test_projection_embedding_key_and_tokens():
    """d = 0 is Eq. (13)'s embedding key k_0 = W_0^K o_0; evaluating listed
    tokens equals the rows of the full run; bf16 words decode exactly."""
    import torch

    g = _rng(33)
    T, m, r = 7, 16, 4
    a = torch.from_numpy(g.standard_normal((T, m))).to(torch.bfloat16)
    w = torch.from_numpy(g.standard_normal((r, m))).to(torch.bfloat16)
    full = oracle.projection(a, w, 0)
    assert full["o"].shape == (T, 0)
    assert np.allclose(full["keys"], a.double().numpy() @ w.double().numpy().T, rtol=1e-13, atol=1e-13)
    part = oracle.projection(a, w, 0, tokens=[6, 1])
    assert np.array_equal(part["keys"], full["keys"][[6, 1]])
