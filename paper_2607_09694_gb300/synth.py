"""Seeded synthetic inputs shaped like the paper's depth-routing workloads.

This module only draws random numbers: it holds none of the method's
arithmetic, and both the oracle-side tests and the GPU path take their inputs
from it.  The paper's model (§4.1: d = 1024, L = 24, 2L = 48 residual-writing
sub-layers, context 2048) trained on a dataset that is not available here;
these tensors stand in for its sub-layer outputs, routing keys, queries and
upstream gradients.

Recipe (fixed order: values -> per-source scale -> keys -> queries -> dh):
  * values  o_i ~ N(0, 1) [n, T, d], optionally times a per-source scale
    s_i ~ U(lo, hi), computed in fp32 and rounded to the storage type once
    (round-to-nearest-even);
  * P-LR keys ~ N(0, 1) [n, T, r];
  * static per-site queries ~ N(0, q_std^2) [r] (the paper initialises them to
    zero, §4.1; zero queries are a separate test case);
  * upstream gradients dh ~ N(0, 1) [T, d].

Generation is split into fixed chunks of the flattened tensor, each with its
own seed, so the numbers do not depend on the thread count and large tensors
are drawn in parallel.  On a CUDA device the same recipe uses the device's
generator (different numbers, same distribution).
"""
from __future__ import annotations

import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field

import torch

_TAGS = {"values": 1, "scale": 2, "keys": 3, "query": 4, "dh": 5, "outputs": 6, "proj_a": 7, "proj_w": 8}
_CHUNK = 1 << 22
_MASK = (1 << 62) - 1

# The five workloads: (1) tiny fp32 case, (2) S-LR at every site of a 24-layer
# decoder, (3) P-LR with learned keys, (4) full AttnRes keys (r = d) on the
# values of (2), (5) a 32-layer, d = 2048 decoder with Block AttnRes, c = 8.
CONFIGS = {
    "tiny": dict(variant="sliced", T=256, d=64, r=4, n=8, seed=0, dtype="f32", scale=None),
    "slr": dict(variant="sliced", T=16384, d=1024, r=16, n=49, seed=1, dtype="bf16", scale=(0.5, 2.0)),
    "plr": dict(variant="projected", T=16384, d=1024, r=32, n=49, seed=2, dtype="bf16", scale=None),
    "full": dict(variant="full", T=16384, d=1024, r=1024, n=49, seed=1, dtype="bf16", scale=(0.5, 2.0)),
    "slr_large": dict(variant="sliced", T=32768, d=2048, r=64, n=65, seed=3, dtype="bf16", scale=None),
    "block": dict(variant="sliced", T=32768, d=2048, r=64, n=9, seed=3, dtype="bf16", scale=None,
                  block_c=8, n_outputs=65),
}
Q_STD = 0.02


def _seed(seed: int, tag: str, k: int) -> int:
    x = (seed * 0x9E3779B97F4A7C15 + _TAGS[tag] * 0xBF58476D1CE4E5B9 + k * 0x94D049BB133111EB) & _MASK
    x ^= x >> 31
    return (x * 0xD6E8FEB86659FD93) & _MASK


def _fill(out: torch.Tensor, seed: int, tag: str, kind: str) -> torch.Tensor:
    flat = out.view(-1)
    nchunks = (flat.numel() + _CHUNK - 1) // _CHUNK
    dev = flat.device

    def work(k: int) -> None:
        g = torch.Generator(device=dev)
        g.manual_seed(_seed(seed, tag, k))
        part = flat[k * _CHUNK:(k + 1) * _CHUNK]
        if kind == "normal":
            part.normal_(generator=g)
        else:
            part.uniform_(generator=g)

    if dev.type == "cpu" and nchunks > 1:
        with ThreadPoolExecutor(max_workers=min(nchunks, os.cpu_count() or 1)) as ex:
            list(ex.map(work, range(nchunks)))
    else:
        for k in range(nchunks):
            work(k)
    return out


def randn(shape, seed: int, tag: str, device="cpu") -> torch.Tensor:
    """fp32 N(0, 1) of the given shape, chunk-seeded."""
    return _fill(torch.empty(shape, dtype=torch.float32, device=device), seed, tag, "normal")


def rand(shape, seed: int, tag: str, device="cpu") -> torch.Tensor:
    """fp32 U[0, 1) of the given shape, chunk-seeded."""
    return _fill(torch.empty(shape, dtype=torch.float32, device=device), seed, tag, "uniform")


def storage_dtype(name: str) -> torch.dtype:
    return {"f32": torch.float32, "bf16": torch.bfloat16}[name]


def values(n: int, T: int, d: int, seed: int, dtype="bf16", scale=None, device="cpu") -> torch.Tensor:
    """Stacked sources [n, T, d]: N(0,1), times s_i ~ U(lo, hi) per source if scale=(lo, hi)."""
    v = randn((n, T, d), seed, "values", device)
    if scale is not None:
        lo, hi = scale
        s = rand((n,), seed, "scale", device) * (hi - lo) + lo
        v.mul_(s.view(n, 1, 1))
    return v.to(storage_dtype(dtype))


def keys(n: int, T: int, r: int, seed: int, dtype="bf16", device="cpu") -> torch.Tensor:
    """Learned-key stand-ins [n, T, r] ~ N(0, 1)."""
    return randn((n, T, r), seed, "keys", device).to(storage_dtype(dtype))


def queries(n_sites: int, r: int, seed: int, std: float = Q_STD, device="cpu") -> torch.Tensor:
    """Static per-site queries [n_sites, r] ~ N(0, std^2), fp32."""
    return randn((n_sites, r), seed, "query", device).mul_(std)


def upstream(T: int, d: int, seed: int, dtype="bf16", sites: int | None = None, device="cpu") -> torch.Tensor:
    """Upstream gradients dh ~ N(0, 1): [T, d], or [sites, T, d]."""
    shape = (T, d) if sites is None else (sites, T, d)
    return randn(shape, seed, "dh", device).to(storage_dtype(dtype))


def outputs(n_outputs: int, T: int, d: int, seed: int, dtype="bf16", device="cpu") -> torch.Tensor:
    """Sub-layer outputs o_0..o_{M} [n_outputs, T, d] ~ N(0, 1) for Block assembly."""
    return randn((n_outputs, T, d), seed, "outputs", device).to(storage_dtype(dtype))


@dataclass
class SiteInputs:
    """Inputs of one residual read site."""

    variant: str
    n: int
    T: int
    d: int
    r: int
    values: torch.Tensor
    keys: torch.Tensor | None
    query: torch.Tensor
    dh: torch.Tensor
    meta: dict = field(default_factory=dict)


def site(config: str, n: int | None = None, T: int | None = None, r: int | None = None,
         dtype: str | None = None, device="cpu", query_std: float = Q_STD, seed: int | None = None,
         variant: str | None = None, d: int | None = None) -> SiteInputs:
    """One site of a named workload, optionally at a different n, T, r, d,
    storage type or key variant (full keys force r = d)."""
    c = dict(CONFIGS[config])
    if variant is not None:
        c["variant"] = variant
    n = c["n"] if n is None else n
    T = c["T"] if T is None else T
    r = c["r"] if r is None else r
    d = c["d"] if d is None else d
    if c["variant"] == "full":
        r = d
    dt = c["dtype"] if dtype is None else dtype
    sd = c["seed"] if seed is None else seed
    v = values(n, T, d, sd, dt, c.get("scale"), device)
    k = keys(n, T, r, sd, dt, device) if c["variant"] == "projected" else None
    q = queries(1, r, sd, query_std, device)[0].contiguous()
    g = upstream(T, d, sd, dt, None, device)
    return SiteInputs(c["variant"], n, T, d, r, v, k, q, g, meta=dict(config=config, seed=sd, dtype=dt))
