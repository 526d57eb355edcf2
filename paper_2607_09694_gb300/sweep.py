"""Whole-decoder driver of the depth mix: every residual read site of a model,
forward over the sites in order and backward in reverse with the gradients of
each source accumulated across the sites that read it (Eq. 4: site t reads
sources 0..t-1).

Sources are separate tensors (one per sub-layer output, as a model produces
them), passed to the library as pointer tables, so nothing is stacked or
copied.  The whole sweep can be captured once into a CUDA graph and replayed:
every call is asynchronous, allocates nothing and synchronises nothing.

The sub-layers between read sites are not part of this library: the driver
runs the mixes of all sites back to back, as a model's depth-attention traffic
with fixed sub-layer outputs (the benchmark's step).
"""
from __future__ import annotations

import torch

from . import lrar


class DepthSweep:
    """All read sites t = 1..n_sites over sources o_0..o_{n_sites-1}.

    sources   list of n_sites tensors [T, d] (o_0 is the embedding)
    queries   [n_sites, r] fp32, row t-1 the static query of site t (row 0,
              site 1, is unused: one source mixes to itself)
    dh        list of n_sites upstream gradients [T, d], one per site
    h, lse    outputs per site: [n_sites, T, d] and [n_sites, T]
    dsources  list of n_sites gradient tensors [T, d] (written, then accumulated)
    dq        [n_sites, r] fp32 query gradients
    keys / dkeys  lists of [T, r] tensors for projected keys
    """

    def __init__(self, variant, sources, queries, dh, h, lse, dsources, dq, keys=None, dkeys=None,
                 r: int | None = None, eps: float = lrar.DEFAULT_EPS):
        self.variant = lrar._variant(variant)
        self.sources, self.keys = list(sources), (list(keys) if keys is not None else None)
        self.dsources, self.dkeys = list(dsources), (list(dkeys) if dkeys is not None else None)
        self.queries, self.dh, self.h, self.lse, self.dq = queries, list(dh), h, lse, dq
        self.n_sites = len(self.sources)
        T, d = self.sources[0].shape
        self.r = d if self.variant == lrar.FULL else (r if r is not None else queries.shape[-1])
        self.eps = eps
        self.ws = torch.empty(max(1, lrar.workspace_size(self.variant, self.n_sites, T, d, self.r) // 4),
                              dtype=torch.float32, device=self.sources[0].device)
        self.graph = None
        self.graph_stream = None

    def _keys(self, ks, t):
        return ks[:t] if ks is not None else None

    def forward(self, stream: torch.cuda.Stream | None = None) -> None:
        s = stream or torch.cuda.current_stream()
        for t in range(1, self.n_sites + 1):
            q = self.queries[t - 1] if t > 1 else None
            lrar.forward_ptrs(self.variant, self.sources[:t], self._keys(self.keys, t), q, self.h[t - 1],
                              self.lse[t - 1], r=self.r, eps=self.eps, stream=s.cuda_stream)

    def backward(self, stream: torch.cuda.Stream | None = None) -> None:
        """Site n_sites writes the gradients of all its sources; every earlier
        site adds into those of its own (a source's gradient sums over the sites
        that read it).  Each site's dq is that step's: the accumulating calls
        add dq too, so dq starts from zero."""
        s = stream or torch.cuda.current_stream()
        with torch.cuda.stream(s):
            self.dq.zero_()
        for t in range(self.n_sites, 0, -1):
            q = self.queries[t - 1] if t > 1 else None
            lrar.backward_ptrs(self.variant, self.sources[:t], self._keys(self.keys, t), q, self.dh[t - 1],
                               self.dsources[:t], self.dq[t - 1], self.ws, dkeys=self._keys(self.dkeys, t),
                               h=self.h[t - 1], lse=self.lse[t - 1], r=self.r, accumulate=t != self.n_sites,
                               eps=self.eps, stream=s.cuda_stream)

    def step(self, stream: torch.cuda.Stream | None = None) -> None:
        self.forward(stream)
        self.backward(stream)

    def capture(self) -> None:
        """Record one step into a CUDA graph (the step is not executed)."""
        self.graph_stream = torch.cuda.Stream(device=self.sources[0].device)
        self.graph_stream.wait_stream(torch.cuda.current_stream())
        self.graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(self.graph, stream=self.graph_stream):
            self.step(self.graph_stream)

    def replay(self) -> None:
        """One step from the captured graph, ordered after the current stream's work."""
        if self.graph is None:
            raise RuntimeError("capture() first")
        self.graph.replay()
