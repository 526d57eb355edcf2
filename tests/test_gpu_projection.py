"""P-LR fused output projection (§3.3, Eq. 11-12) on the tensor cores
(lrar_project) against the oracle's float64 projection of the same bfloat16
operands: [o; k] = [W_O; W_K] a per token, o and k written to separate slots."""
import numpy as np
import pytest
import torch

import gpu_helpers as H
import oracle
from paper_2607_09694_gb300 import lrar, synth

pytestmark = pytest.mark.gpu


def _operands(T, m, N, seed):
    a = synth.randn((T, m), seed, "proj_a").to(torch.bfloat16)
    w = (synth.randn((N, m), seed, "proj_w") / m ** 0.5).to(torch.bfloat16)
    return a, w


def _run(T, m, d, r, seed=3, tile=0):
    a, w = _operands(T, m, d + r, seed)
    dev = torch.device("cuda")
    o = torch.full((T, d), float("nan"), dtype=torch.bfloat16, device=dev) if d else None
    k = torch.full((T, r), float("nan"), dtype=torch.bfloat16, device=dev) if r else None
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    if tile:
        lrar.test_project_tile(tile, a.to(dev), w.to(dev), o, k, status=status)
    else:
        lrar.project(a.to(dev), w.to(dev), o, k, status=status)
    torch.cuda.synchronize()
    assert status.item() == 0, "a pipeline wait in the projection kernel gave up"
    return a, w, o, k


def _check(name, got, ref, a, w_rows):
    """One bf16 rounding of the exact value (half a spacing) plus the float32
    accumulation over m products (each product of two bf16 is exact in
    float32; m additions, each within one float32 spacing)."""
    got = got.double().cpu().numpy()
    m = a.shape[1]
    absprod = np.abs(a.double().numpy()) @ np.abs(w_rows.double().numpy()).T
    bound = 0.5 * H.bf16_ulp(ref) + m * 2.0 ** -23 * absprod
    err = np.abs(got - ref)
    bad = np.argwhere(~(err <= bound))
    assert bad.size == 0, f"{name}: {bad.shape[0]} elements out of bound, first {bad[:3].tolist()}"
    # and as a whole, no more than rounding: mean error below half the mean spacing
    assert err.mean() <= 0.5 * H.bf16_ulp(ref).mean(), name


def _compare(T, m, d, r, seed=3, tokens=None, tile=0):
    a, w, o, k = _run(T, m, d, r, seed, tile)
    ref = oracle.projection(a if tokens is None else a[tokens], w, d)
    if d:
        _check("o", o.cpu() if tokens is None else o.cpu()[tokens], ref["o"],
               a if tokens is None else a[tokens], w[:d])
    if r:
        _check("keys", k.cpu() if tokens is None else k.cpu()[tokens], ref["keys"],
               a if tokens is None else a[tokens], w[d:])


def test_whole_tiles():
    """T = 256 (one 256-row tile of the CTA-pair form, two 128-row tiles of the
    single-CTA form), m = d = 1024, r = 32 (N = 1056)."""
    _compare(256, 1024, 1024, 32)


def test_ragged_edges():
    """T, m and N that fill no tile: 300 tokens, m = 1000 (not a multiple of the
    64-column K-block), d = 1024 and r = 16 (the key columns start inside a tile)."""
    _compare(300, 1000, 1024, 16, seed=4)


@pytest.mark.parametrize("width", [160, 176, 192, 224, 240, 256])
def test_every_tile_width(width):
    """Each compiled tile width (forced through the lrar_test_project_tile hook)
    on ragged T, m and N, the value/key split falling inside a tile."""
    _compare(300, 1000, 1024, 16, seed=4, tile=width)


@pytest.mark.parametrize("width", [160, 176, 192, 224, 240, 256])
def test_every_pair_tile_width(width):
    """The CTA-pair (two-SM, tcgen05.mma.cta_group::2) form at each width
    (hook code 2000 + width): 256-row tiles split over the two CTAs of a
    cluster, on ragged T, m and N."""
    _compare(300, 1000, 1024, 16, seed=4, tile=2000 + width)


def test_swiglu_output_projection():
    """The FFN's output projection: m = 2816 (the SwiGLU width of the 0.5B decoder)."""
    _compare(256, 2816, 1024, 32, seed=5)


def test_embedding_key_only():
    """d = 0: Eq. 13's embedding key k_0 = W_0^K o_0."""
    _compare(130, 1024, 0, 32, seed=6)


def test_output_only_and_smallest():
    _compare(128, 512, 512, 0, seed=7)
    _compare(1, 8, 8, 8, seed=8)


def test_full_size_sampled_tokens():
    """The P-LR decoder's projection at full size (T = 16384, m = d = 1024,
    r = 32), checked on tokens spread over every row tile."""
    g = np.random.default_rng(9)
    tokens = np.sort(np.concatenate([g.choice(16384, 40, replace=False), [0, 127, 128, 16383]]))
    _compare(16384, 1024, 1024, 32, seed=9, tokens=tokens)


def test_large_decoder_sampled_tokens():
    """The d = 2048 decoder (m = d = 2048, r = 64, T = 32768): d + r = 2112
    columns in 240-wide tiles of the CTA-pair form, the last one partly outside."""
    g = np.random.default_rng(10)
    tokens = np.sort(np.concatenate([g.choice(32768, 24, replace=False), [0, 32767]]))
    _compare(32768, 2048, 2048, 64, seed=10, tokens=tokens)


def test_keys_land_in_the_key_stack_of_the_mix():
    """Projected keys written straight into slot i of a [n, T, r] key stack are
    the keys the mix reads: the forward over that stack equals the oracle's
    forward over the oracle's projected keys (rounded to bf16 once)."""
    n, T, m, d, r = 3, 200, 256, 256, 16
    dev = torch.device("cuda")
    vals = torch.empty(n, T, d, dtype=torch.bfloat16, device=dev)
    keys = torch.empty(n, T, r, dtype=torch.bfloat16, device=dev)
    acts, ws = [], []
    for i in range(n):
        a, w = _operands(T, m, d + r, 20 + i)
        lrar.project(a.to(dev), w.to(dev), vals[i], keys[i])
        acts.append(a)
        ws.append(w)
    q = synth.queries(1, r, 20, std=1.0)[0]
    h = torch.empty(T, d, device=dev)
    lse = torch.empty(T, device=dev)
    lrar.forward("projected", vals, keys, q.to(dev), h, lse, r=r)
    torch.cuda.synchronize()
    ov = np.stack([oracle.projection(acts[i], ws[i], d)["o"] for i in range(n)])
    ok = np.stack([oracle.projection(acts[i], ws[i], d)["keys"] for i in range(n)])
    to_bf16 = lambda x: torch.from_numpy(x).to(torch.bfloat16)  # noqa: E731
    ref = oracle.forward(oracle.PROJECTED, to_bf16(ov), to_bf16(ok), q, H.EPS, r=r)
    # the GPU's projected bf16 values may differ from the oracle's rounding by
    # one spacing where accumulation order decides; the mix is within the rms bar
    H.assert_rms("h", h.double().cpu().numpy(), ref["h"])
