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

from . import lrar, sites


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


class BlockSweep:
    """Block AttnRes (§3.1, Eq. 5-6) over every residual read site t = 1..M+1 of
    a decoder with M residual-writing sub-layers and c outputs per block: the
    assembly after each sub-layer, the mix at every site, the backward at every
    site in reverse, and the fan-out of each summary's gradient to its members.

    Site t has written o_0..o_{t-1}: with k = (t-1) // c completed blocks and
    j = (t-1) % c outputs in the open block, its sources are the embedding o_0,
    the completed summaries b_1..b_k and, when j > 0, the partial summary of
    the open block (Eq. 6).

    outputs   list of M+1 tensors [T, d]: o_0 (the embedding) and o_1..o_M.
              Assembly works in place: once site i+1 has been reached, the
              tensor of o_i (i >= 1) holds its block's running sum through o_i,
              so the tensor of a block's last member holds the completed summary
              (Eq. 5) and every partial summary a site read stays available for
              its backward.  (In Block AttnRes a sub-layer output is read only
              through its block's sums.)  The forward refuses to run twice on
              the same tensors.
    queries   [M+1, r] fp32, row t-1 the static query of site t (row 0 unused)
    dh        list of M+1 upstream gradients [T, d], one per site
    h, lse    per-site outputs [M+1, T, d] and [M+1, T]
    doutputs  list of M+1 tensors [T, d]: the gradient of each output o_i,
              summed over every site that reads it through a summary
    keys / dkeys  P-LR: [T, r] key tensors per output (summed like the
              outputs: a summary's key is the sum of its members' keys) and
              their gradients
    grads / dkgrads  optional gradient accumulators, one [T, d] (keys: [T, r])
              tensor per slot (1 + ceil(M / c)); allocated like doutputs when
              not given.
    """

    def __init__(self, variant, outputs, queries, dh, h, lse, doutputs, c: int, keys=None, dkeys=None,
                 r: int | None = None, eps: float = lrar.DEFAULT_EPS, grads=None, dkgrads=None,
                 two_phase: bool | None = None):
        self.variant = lrar._variant(variant)
        self.outputs, self.keys = list(outputs), (list(keys) if keys is not None else None)
        self.doutputs, self.dkeys = list(doutputs), (list(dkeys) if dkeys is not None else None)
        # site 1 reads one source and has no query (its softmax is 1, its score 0):
        # row 0 is zeroed so that a phase-1 pass over site 1 scores it the same way
        self.queries = queries.clone()
        self.queries[0].zero_()
        self.dh, self.h, self.lse = list(dh), h, lse
        self.c = int(c)
        self.M = len(self.outputs) - 1
        if self.M < 0 or self.c < 1:
            raise ValueError("need at least the embedding and c >= 1")
        self.n_slots = 1 + -(-self.M // self.c)
        T, d = self.outputs[0].shape
        self.r = d if self.variant == lrar.FULL else (r if r is not None else queries.shape[-1])
        self.eps = eps
        dev = self.outputs[0].device
        gdt = self.doutputs[0].dtype
        self.grads = list(grads) if grads is not None else [torch.empty(T, d, dtype=gdt, device=dev)
                                                            for _ in range(self.n_slots)]
        if self.keys is not None:
            kdt = self.dkeys[0].dtype
            self.dkgrads = list(dkgrads) if dkgrads is not None else [torch.empty(T, self.r, dtype=kdt, device=dev)
                                                                      for _ in range(self.n_slots)]
        else:
            self.dkgrads = None
        self.dq = torch.zeros(self.M + 1, self.queries.shape[-1], dtype=torch.float32, device=dev)
        n_max = max(sites.block_num_sources(t, self.c) for t in range(1, self.M + 2))
        self.ws = torch.empty(max(1, lrar.workspace_size(self.variant, n_max, T, d, self.r) // 4),
                              dtype=torch.float32, device=dev)
        self.assembled = False
        self.graph = None
        # the two-phase forward (§3.5) serves low-rank keys; h and its phase-1
        # result share a type because phase 2 updates each site's h in place
        self.two_phase = (self.variant != lrar.FULL) if two_phase is None else bool(two_phase)
        if self.two_phase and self.variant == lrar.FULL:
            raise ValueError("the two-phase path serves low-rank keys (sliced, projected)")

    # slot layout -------------------------------------------------------------
    def site_sources(self, t: int) -> list[int]:
        """Indices of the output tensors that hold site t's sources (after assembly)."""
        k, j = divmod(t - 1, self.c)
        idx = [0] + [b * self.c for b in range(1, k + 1)]
        if j:
            idx.append(k * self.c + j)
        return idx

    def _slot(self, i: int) -> int:
        return sites.block_slot(i, self.c)

    # forward -----------------------------------------------------------------
    def _assemble(self, i: int, s) -> None:
        """o_i joins its block: its tensor becomes the running sum through o_i."""
        if i >= 1 and not sites.block_opens_slot(i, self.c):
            lrar.block_accumulate(self.outputs[i], self.outputs[i - 1], 1.0, 1.0, stream=s.cuda_stream)
            if self.keys is not None:
                lrar.block_accumulate(self.keys[i], self.keys[i - 1], 1.0, 1.0, stream=s.cuda_stream)

    def forward(self, stream: torch.cuda.Stream | None = None) -> None:
        """Site t's mix after o_{t-1} joined its block, for t = 1..M+1: site by
        site, or (two_phase) per block of c sites one phase-1 pass over the
        completed sources written into those sites' h and lse, then each site's
        partial summary folded in by phase 2, in place."""
        if self.assembled:
            raise RuntimeError("the outputs already hold block sums: forward runs once per set of outputs")
        s = stream or torch.cuda.current_stream()
        if self.two_phase:
            self._forward_two_phase(s)
            self.assembled = True
            return
        for t in range(1, self.M + 2):
            self._assemble(t - 1, s)
            idx = self.site_sources(t)
            q = self.queries[t - 1] if len(idx) > 1 else None
            ks = [self.keys[i] for i in idx] if self.keys is not None else None
            lrar.forward_ptrs(self.variant, [self.outputs[i] for i in idx], ks, q, self.h[t - 1], self.lse[t - 1],
                              r=self.r, eps=self.eps, stream=s.cuda_stream)
        self.assembled = True

    def _forward_two_phase(self, s) -> None:
        c = self.c
        for b in range(self.M // c + 1):  # sites t = b c + 1 .. b c + ns share the completed sources
            t0 = b * c + 1
            ns = min(c, self.M + 1 - b * c)
            self._assemble(t0 - 1, s)  # o_{t0-1} completes block b (or is the embedding)
            idx = [0] + [k * c for k in range(1, b + 1)]
            ks = [self.keys[i] for i in idx] if self.keys is not None else None
            lrar.block_phase1_ptrs(self.variant, [self.outputs[i] for i in idx], ks,
                                   self.queries[t0 - 1:t0 - 1 + ns], self.h[t0 - 1:t0 - 1 + ns],
                                   self.lse[t0 - 1:t0 - 1 + ns], eps=self.eps, stream=s.cuda_stream)
            for j in range(1, ns):
                t = t0 + j
                i = t - 1  # the partial summary runs through o_i
                pk = self.keys[i] if self.keys is not None else None
                if sites.block_opens_slot(i, c):  # o_i alone
                    lrar.block_phase2(self.variant, self.h[t - 1], self.lse[t - 1], self.outputs[i], pk,
                                      self.queries[t - 1], self.h[t - 1], self.lse[t - 1], eps=self.eps,
                                      stream=s.cuda_stream)
                else:  # o_i joins its block's running sum inside phase 2 (no separate assembly pass)
                    ppk = self.keys[i - 1] if self.keys is not None else None
                    lrar.block_phase2_assemble(self.variant, self.h[t - 1], self.lse[t - 1], self.outputs[i - 1],
                                               self.outputs[i], ppk, pk, self.queries[t - 1], self.h[t - 1],
                                               self.lse[t - 1], eps=self.eps, stream=s.cuda_stream)

    # backward ----------------------------------------------------------------
    def backward(self, stream: torch.cuda.Stream | None = None, member_grad=None) -> None:
        """Sites in reverse: site t adds the gradients of its sources into the
        accumulators of their slots (site M+1 writes them); right after site
        i+1, the accumulator of o_i's slot holds the whole gradient of o_i
        (every later site reads o_i through that slot), so it is copied to
        doutputs[i] -- the fan-out of the summary gradients to the members.

        member_grad: optional callable(i, dout, dkey), the fan-out as a
        hand-over instead of copies.  It is called as soon as o_i's gradient is
        complete, with views of the slot accumulators that hold it (dkey: the
        key gradient with P-LR keys, else None), and inside the stream's
        context.  The views keep d o_i until the next site's backward, which is
        enqueued after the call returns, so work that the callable enqueues on
        the stream reads them in time: in a training step, the backward of the
        sub-layer that wrote o_i.  doutputs and dkeys are then left untouched,
        and the step moves no fan-out bytes."""
        s = stream or torch.cuda.current_stream()
        with torch.cuda.stream(s):
            self.dq.zero_()
        for t in range(self.M + 1, 0, -1):
            idx = self.site_sources(t)
            slots = [self._slot(i) for i in idx]
            q = self.queries[t - 1] if len(idx) > 1 else None
            ks = [self.keys[i] for i in idx] if self.keys is not None else None
            dks = [self.dkgrads[b] for b in slots] if self.keys is not None else None
            first = t == self.M + 1  # reads every slot: writes the accumulators
            lrar.backward_ptrs(self.variant, [self.outputs[i] for i in idx], ks, q, self.dh[t - 1],
                               [self.grads[b] for b in slots], self.dq[t - 1], self.ws, dkeys=dks,
                               h=self.h[t - 1], lse=self.lse[t - 1], r=self.r, accumulate=not first, eps=self.eps,
                               stream=s.cuda_stream)
            i = t - 1  # o_{t-1} is read by sites t..M+1 only: its gradient is complete
            b = self._slot(i)
            if member_grad is not None:
                with torch.cuda.stream(s):
                    member_grad(i, self.grads[b], self.dkgrads[b] if self.keys is not None else None)
                continue
            lrar.block_accumulate(self.doutputs[i], self.grads[b], 1.0, 0.0, stream=s.cuda_stream)
            if self.keys is not None:
                lrar.block_accumulate(self.dkeys[i], self.dkgrads[b], 1.0, 0.0, stream=s.cuda_stream)

    def rearm(self) -> None:
        """The caller has written new sub-layer outputs (and keys) into the
        output tensors: the next forward assembles them again."""
        self.assembled = False

    def step(self, stream: torch.cuda.Stream | None = None, member_grad=None) -> None:
        self.forward(stream)
        self.backward(stream, member_grad)
