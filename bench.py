"""Benchmark of the depth-attention mix hot path (Low-Rank Attention Residuals).

Workload (one step): every residual read site t = 1..49 of a 24-layer PreNorm
decoder with S-LR-AttnRes keys (last r = 16 of d = 1024 coordinates), T = 16384
tokens (batch 8 x sequence 2048), bf16 storage, fp32 accumulation.  A step is
the forward sweep (site t mixes the first t sources of the stacked buffer) and
the backward sweep t = 49..1, which writes (site 49) and then accumulates
(sites 48..1) the source gradients, as a training step does.  Inputs are
synthetic (normal values with a per-source scale, N(0, 0.02^2) queries, normal
upstream gradients), drawn on the device with a seeded generator.

Metric: algorithmic HBM bytes of the step / step time (GB/s), the fraction of
the measured HBM copy peak, and tokens/s per site.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

With N > 1 (launched by torch.distributed.run) every rank runs its own replica
of the workload on its own GPU (independent token batches, no exchange: weak
scaling); the reported value is all ranks' bytes over the slowest rank's time.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "depth-residual fwd+bwd GB/s and % of GB300 HBM peak; tokens/sec per site"
T_TOK, D, R, N_SITES, SEED, EPS = 16384, 1024, 16, 49, 1, 1e-6
WORKLOAD = ("S-LR-AttnRes fwd+bwd at every residual site (n_src = 1..49) of a 24-layer decoder: "
            "T=16384 (8 x 2048), d=1024, r=16, bf16 storage, fp32 accumulate")
FALLBACK_HBM_GBS = 6800.0


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def _bf16_peak():
    """Measured dense bf16 tensor throughput (burst), TFLOP/s; else the fallback."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops"]), "measured"
    except Exception:
        return 1900.0, "fallback"


def _kernel_source_hash() -> str:
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2607_09694_gb300", "csrc")
    for name in sorted(os.listdir(csrc)):
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(name.encode() + f.read())
    return h.hexdigest()[:16]


def _recorded_traffic(kernel: str):
    """Bytes per launch from a committed ncu summary, if it was taken on the
    current kernel sources (the summary records their hash)."""
    path = os.path.join(ROOT, "profiles", f"{kernel}_traffic.txt")
    if not os.path.exists(path):
        return None
    fields = {}
    with open(path) as f:
        for line in f:
            if ":" in line and not line.startswith("#"):
                k, v = line.split(":", 1)
                fields[k.strip()] = v.strip()
    if fields.get("source_hash") != _kernel_source_hash():
        return None
    try:
        return float(fields["dram_bytes_per_launch_avg"])
    except (KeyError, ValueError):
        return None


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines: list[str] = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, FileNotFoundError):
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        if self.thread:
            self.thread.join(timeout=2)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for name, flag in zip(names, parts[5:9]):
                if flag.lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# --------------------------------------------------------------------------
# The workload
# --------------------------------------------------------------------------


def site_bytes():
    """Algorithmic bytes of each forward and backward call of one step."""
    from paper_2607_09694_gb300 import sites

    fwd = [sites.forward_bytes(sites.SiteShape("sliced", t, T_TOK, D, R)) for t in range(1, N_SITES + 1)]
    bwd = [sites.backward_bytes(sites.SiteShape("sliced", t, T_TOK, D, R, accumulate=0 if t == N_SITES else 1))
           for t in range(1, N_SITES + 1)]
    return fwd, bwd


class Workload:
    def __init__(self, device, T=T_TOK, n_sites=N_SITES):
        import torch

        from paper_2607_09694_gb300 import lrar, synth

        self.torch, self.lrar = torch, lrar
        self.dev = device
        self.T = T
        ns = n_sites
        self.values = synth.values(ns, T, D, SEED, "bf16", (0.5, 2.0), device=device)
        self.queries = synth.queries(ns, R, SEED, device=device)      # row t-1: query of site t
        self.dh = synth.upstream(T, D, SEED, "bf16", sites=ns, device=device)  # row t-1: dL/dh_t
        self.h = torch.empty(ns, T, D, dtype=torch.bfloat16, device=device)
        self.lse = torch.empty(ns, T, dtype=torch.float32, device=device)
        self.dvalues = torch.zeros(ns, T, D, dtype=torch.bfloat16, device=device)
        self.dq = torch.empty(ns, R, dtype=torch.float32, device=device)
        self.ws = torch.empty(lrar.workspace_size("sliced", ns, T, D, R) // 4, dtype=torch.float32,
                              device=device)

    def step(self, events=None, sweeps=None):
        """Forward sweep t = 1..49, then backward sweep t = 49..1 (49 writes, the rest accumulate).
        events: per-call event pairs (an event between two calls ends the overlap of their
        launches); sweeps: one event pair around each sweep."""
        lrar = self.lrar
        if sweeps is not None:
            sweeps["fwd"][0].record()
        for t in range(1, N_SITES + 1):
            q = self.queries[t - 1] if t > 1 else None
            if events is not None:
                events["fwd"][t - 1][0].record()
            lrar.forward(lrar.SLICED, self.values, None, q, self.h[t - 1], self.lse[t - 1], n_src=t, r=R, eps=EPS)
            if events is not None:
                events["fwd"][t - 1][1].record()
        if sweeps is not None:
            sweeps["fwd"][1].record()
            sweeps["bwd"][0].record()
        for t in range(N_SITES, 0, -1):
            q = self.queries[t - 1] if t > 1 else None
            if events is not None:
                events["bwd"][t - 1][0].record()
            lrar.backward(lrar.SLICED, self.values, None, q, self.dh[t - 1], self.dvalues, self.dq[t - 1], self.ws,
                          lse=self.lse[t - 1], n_src=t, r=R, accumulate=(t != N_SITES), eps=EPS)
            if events is not None:
                events["bwd"][t - 1][1].record()
        if sweeps is not None:
            sweeps["bwd"][1].record()

    @staticmethod
    def launches_per_step() -> int:
        return N_SITES + 2 * N_SITES  # forward kernel; backward kernel + dq reduction


def _events(torch):
    mk = lambda: (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))  # noqa: E731
    return {"fwd": [mk() for _ in range(N_SITES)], "bwd": [mk() for _ in range(N_SITES)]}


def _sweep_events(torch):
    mk = lambda: (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))  # noqa: E731
    return {"fwd": mk(), "bwd": mk()}


# --------------------------------------------------------------------------
# CPU oracle baseline (bounded sample)
# --------------------------------------------------------------------------


def oracle_pass(values_cpu, queries_cpu, dh_cpu, ts: int) -> float:
    """Seconds the fp64 oracle takes for all 49 sites (fwd + bwd) on the first ts tokens."""
    import oracle

    v = values_cpu[:, :ts].contiguous()
    d = dh_cpu[:, :ts].contiguous()
    q0 = queries_cpu[0] * 0
    t0 = time.perf_counter()
    for t in range(1, N_SITES + 1):
        q = queries_cpu[t - 1] if t > 1 else q0
        oracle.forward(oracle.SLICED, v[:t], None, q, EPS, r=R)
        oracle.backward(oracle.SLICED, v[:t], None, q, EPS, d[t - 1], r=R)
    return time.perf_counter() - t0


def sample_bytes(ts: int) -> int:
    from paper_2607_09694_gb300 import sites

    nbytes = 0
    for t in range(1, N_SITES + 1):
        nbytes += sites.forward_bytes(sites.SiteShape("sliced", t, ts, D, R))
        nbytes += sites.backward_bytes(sites.SiteShape("sliced", t, ts, D, R, accumulate=0 if t == N_SITES else 1))
    return nbytes


def calibrate(values_cpu, queries_cpu, dh_cpu, target_s: float) -> int:
    """Token count whose oracle pass takes about target_s seconds (capped by the sample held)."""
    import oracle

    oracle.build()
    probe = min(32, values_cpu.shape[1])
    per_tok = oracle_pass(values_cpu, queries_cpu, dh_cpu, probe) / probe
    ts = int(target_s / max(per_tok, 1e-9))
    return max(probe, min(values_cpu.shape[1], ts))


def oracle_sample(values_cpu, queries_cpu, dh_cpu, target_s: float):
    """(GB/s on the sample's algorithmic bytes, seconds, tokens, threads) of one timed oracle pass."""
    import oracle

    ts = calibrate(values_cpu, queries_cpu, dh_cpu, target_s)
    el = oracle_pass(values_cpu, queries_cpu, dh_cpu, ts)
    return sample_bytes(ts) / el / 1e9, el, ts, oracle.get_threads()


# --------------------------------------------------------------------------


def _dist():
    from paper_2607_09694_gb300 import replicas

    return replicas.init_from_env()


def _max_over_ranks(dist, value: float, device) -> float:
    from paper_2607_09694_gb300 import replicas

    return replicas.max_over_ranks(dist, value, device)


def run_ours(args):
    import torch

    from __graft_entry__ import build

    dist, rank, local, world = _dist()
    build()
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    peak, peak_kind = _peaks()
    fwd_b, bwd_b = site_bytes()
    step_bytes = sum(fwd_b) + sum(bwd_b)

    wl = Workload(dev)
    host = e2e_host_buffers(wl)  # the end-to-end leg's pinned buffers, touched before anything is timed
    for _ in range(args.warmup):
        wl.step()
    torch.cuda.synchronize()

    # device-resident timed region: one event pair around each sweep (events
    # between calls would end the overlap of consecutive launches)
    ev = [_sweep_events(torch) for _ in range(args.steps)]
    clocks = ClockSampler(torch.cuda.current_device())
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record()
    for k in range(args.steps):
        wl.step(sweeps=ev[k])
    t1.record()
    torch.cuda.synchronize()
    clk = clocks.stop()
    if dist:
        dist.barrier()
    elapsed = _max_over_ranks(dist, t0.elapsed_time(t1) / 1e3, dev)
    ms_step = elapsed / args.steps * 1e3
    value = world * step_bytes * args.steps / elapsed / 1e9

    fwd_sweep = sum(e["fwd"][0].elapsed_time(e["fwd"][1]) for e in ev) / args.steps
    bwd_sweep = sum(e["bwd"][0].elapsed_time(e["bwd"][1]) for e in ev) / args.steps
    bwd_gbs = sum(bwd_b) / (bwd_sweep / 1e3) / 1e9
    fwd_gbs = sum(fwd_b) / (fwd_sweep / 1e3) / 1e9
    dominant, dom_gbs, dom_bytes, dom_launches = ("lrar_bwd", bwd_gbs, sum(bwd_b), N_SITES) \
        if bwd_sweep >= fwd_sweep else ("lrar_fwd", fwd_gbs, sum(fwd_b), N_SITES)
    traffic = _recorded_traffic(dominant)

    # the last site inside the sweep, from a few untimed steps with an event pair around every call
    pev = [_events(torch) for _ in range(5)]
    for k in range(5):
        wl.step(pev[k])
    torch.cuda.synchronize()
    fwd_t = [sum(e["fwd"][i][0].elapsed_time(e["fwd"][i][1]) for e in pev) / 5 for i in range(N_SITES)]
    bwd_t = [sum(e["bwd"][i][0].elapsed_time(e["bwd"][i][1]) for e in pev) / 5 for i in range(N_SITES)]
    site49 = {"n_src": 49, "fwd_ms": fwd_t[-1], "bwd_ms": bwd_t[-1],
              "fwd_gbs": fwd_b[-1] / (fwd_t[-1] / 1e3) / 1e9, "bwd_gbs": bwd_b[-1] / (bwd_t[-1] / 1e3) / 1e9,
              "fwd_bwd_gbs": (fwd_b[-1] + bwd_b[-1]) / ((fwd_t[-1] + bwd_t[-1]) / 1e3) / 1e9}
    site49["frac"] = site49["fwd_bwd_gbs"] / peak
    site49["tokens_per_s"] = T_TOK / ((fwd_t[-1] + bwd_t[-1]) / 1e3)

    # the headline site on its own: n = 49, accumulate = 1 (every site but the
    # last accumulates), forward and backward each timed with CUDA events
    hf, hb = time_site(wl, N_SITES, True, 20)
    from paper_2607_09694_gb300 import sites as _sites

    hfb = _sites.forward_bytes(_sites.SiteShape("sliced", N_SITES, T_TOK, D, R))
    hbb = _sites.backward_bytes(_sites.SiteShape("sliced", N_SITES, T_TOK, D, R, accumulate=1))
    headline = {"n_src": N_SITES, "accumulate": 1, "fwd_ms": hf, "bwd_ms": hb, "fwd_gbs": hfb / hf / 1e6,
                "bwd_gbs": hbb / hb / 1e6, "fwd_bwd_gbs": (hfb + hbb) / (hf + hb) / 1e6,
                "frac": (hfb + hbb) / (hf + hb) / 1e6 / peak, "tokens_per_s": T_TOK / ((hf + hb) / 1e3)}

    # the same step as separate source tensors through the whole-decoder
    # driver, captured once into a CUDA graph and replayed (one launch per step)
    graph = run_graph(wl, step_bytes)

    # end to end through the public API with host buffers
    e2e = run_e2e(wl, args, dist, dev, step_bytes, world, host)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        vals = wl.values[:, :4096].cpu()
        qs = wl.queries.cpu()
        dhs = wl.dh[:, :4096].cpu()
        gbs, secs, ts, cores = oracle_sample(vals, qs, dhs, args.cpu_seconds)
        cpu = {"value": gbs, "unit": "GB/s", "cores": cores, "kind": "oracle",
               "sample": f"all 49 sites fwd+bwd on {ts} of {T_TOK} tokens ({secs:.1f} s, fp64 C oracle, "
                         f"OpenMP {cores} threads); GB/s on the sample's algorithmic bytes"}

    line = {
        "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": WORKLOAD, "T": T_TOK, "d": D, "r": R, "sites": N_SITES, "variant": "sliced",
                   "storage": "bf16", "accumulate": "f32", "parallelism": f"replicas{world}",
                   "l2": "inputs larger than L2 (1.64 GB of values per step, L2 129 MB)",
                   "bytes_per_step": step_bytes},
        "hbm_frac": value / world / peak,
        "tokens_per_s_per_site": world * T_TOK * N_SITES / (elapsed / args.steps),
        "site49_in_sweep": site49,
        "headline_site": headline,
        "roofline": {"bound": "hbm", "achieved": dom_gbs, "peak": peak, "unit": "GB/s",
                     "frac": dom_gbs / peak, "traffic": traffic, "kernel": dominant,
                     "algorithmic_bytes_per_launch": dom_bytes / dom_launches,
                     "peak_source": f"{peak_kind} hbm_gbs (copy bandwidth)",
                     "fwd_gbs": fwd_gbs, "bwd_gbs": bwd_gbs,
                     "timing": "CUDA events around the 49-call backward sweep (and forward sweep) of every timed step"},
        "e2e": e2e,
        "graph_step": graph,
        "gpu_launches": Workload.launches_per_step() * args.steps,
        "clocks": clk,
    }
    if cpu is not None:
        line["cpu_baseline"] = cpu
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


def time_site(wl, n: int, accumulate: bool, reps: int):
    """Median ms of one site's forward and backward (first n sources), timed
    separately with CUDA events on the launching stream."""
    import torch

    lrar = wl.lrar
    q = wl.queries[n - 1] if n > 1 else None
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(reps)]
    for e in evs:  # back to back: the host stays ahead of the GPU, so no launch gaps are timed
        e[0].record()
        lrar.forward(lrar.SLICED, wl.values, None, q, wl.h[n - 1], wl.lse[n - 1], n_src=n, r=R, eps=EPS)
        e[1].record()
        lrar.backward(lrar.SLICED, wl.values, None, q, wl.dh[n - 1], wl.dvalues, wl.dq[n - 1], wl.ws,
                      lse=wl.lse[n - 1], n_src=n, r=R, accumulate=accumulate, eps=EPS)
        e[2].record()
    torch.cuda.synchronize()
    f_ms = [e[0].elapsed_time(e[1]) for e in evs]
    b_ms = [e[1].elapsed_time(e[2]) for e in evs]
    return statistics.median(f_ms), statistics.median(b_ms)


def run_profile_site(args):
    """Small single-site case for profilers: --profile-site n sources, --tokens T,
    --site-variant / --site-d / --site-r (bf16 storage; accumulating backward,
    or with --site-write a backward that writes the gradients)."""
    import torch

    from __graft_entry__ import build
    from paper_2607_09694_gb300 import lrar, sites, synth

    build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    n, T, d, variant = args.profile_site, args.tokens, args.site_d, args.site_variant
    r = d if variant == "full" else args.site_r
    vals = synth.values(n, T, d, 1, "bf16", (0.5, 2.0), device=dev)
    keys = synth.keys(n, T, r, 2, "bf16", device=dev) if variant == "projected" else None
    q = synth.queries(1, r, 1, device=dev)[0].contiguous()
    dh = synth.upstream(T, d, 1, "bf16", device=dev)
    h = torch.empty(T, d, dtype=torch.bfloat16, device=dev)
    lse = torch.empty(T, device=dev)
    dv = torch.zeros(n, T, d, dtype=torch.bfloat16, device=dev)
    dk = torch.zeros(n, T, r, dtype=torch.bfloat16, device=dev) if keys is not None else None
    dq = torch.empty(r, device=dev)
    ws = torch.empty(max(1, lrar.workspace_size(variant, n, T, d, r) // 4), device=dev)
    fwd = lambda: lrar.forward(variant, vals, keys, q, h, lse, r=r)
    acc = not args.site_write
    bwd = lambda: lrar.backward(variant, vals, keys, q, dh, dv, dq, ws, dkeys=dk, h=h, lse=lse, r=r, accumulate=acc)
    for _ in range(args.warmup):
        fwd()
        bwd()
    f = _median_ms(torch, fwd, args.steps)
    b = _median_ms(torch, bwd, args.steps)
    shp = sites.SiteShape(variant, n, T, d, r, out_bytes=2, accumulate=int(acc))
    fb, bb = sites.forward_bytes(shp), sites.backward_bytes(shp)
    print(json.dumps({"profile_site": n, "variant": variant, "T": T, "d": d, "r": r, "accumulate": int(acc),
                      "fwd_ms": f, "bwd_ms": b,
                      "fwd_gbs": fb / f / 1e6, "bwd_gbs": bb / b / 1e6}), flush=True)


def run_profile_block(args):
    """Small case of the Block two-phase path for profilers: phase 1 over the
    last block of the d = 2048 decoder (9 completed sources, 8 sites, r = 64,
    bf16 h_pre) and phase 2 for one site, --profile-block T tokens."""
    import torch

    from __graft_entry__ import build
    from paper_2607_09694_gb300 import lrar, synth

    build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    T, d, r, c, n = args.profile_block, 2048, 64, 8, 9
    stack = synth.values(n + 1, T, d, 3, "bf16", device=dev)
    qs = synth.queries(c, r, 3, device=dev)
    h_pre = torch.empty(c, T, d, dtype=torch.bfloat16, device=dev)
    lse_pre = torch.empty(c, T, device=dev)
    h = torch.empty(T, d, dtype=torch.bfloat16, device=dev)
    lse = torch.empty(T, device=dev)
    ph1 = lambda: lrar.block_phase1("sliced", stack, None, qs, h_pre, lse_pre, n_completed=n)  # noqa: E731
    ph2 = lambda: lrar.block_phase2("sliced", h_pre[1], lse_pre[1], stack[n], None, qs[1], h, lse)  # noqa: E731
    for _ in range(args.warmup):
        ph1()
        ph2()
    m1 = _median_ms(torch, ph1, args.steps)
    m2 = _median_ms(torch, ph2, args.steps)
    b1 = T * (n * d * 2 + c * (d * 2 + 4))
    b2 = T * (3 * d * 2 + 8)
    print(json.dumps({"profile_block": T, "phase1_ms": m1, "phase1_gbs": b1 / m1 / 1e6, "phase2_ms": m2,
                      "phase2_gbs": b2 / m2 / 1e6}), flush=True)


def run_profile_proj(args):
    """Small case of the fused projection for profilers: --profile-proj m, with
    --tokens T, --site-d d, --site-r r (bf16 operands)."""
    import torch

    from __graft_entry__ import build
    from paper_2607_09694_gb300 import lrar, synth

    build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    T, m, d, r = args.tokens, args.profile_proj, args.site_d, args.site_r
    a = synth.randn((T, m), 1, "proj_a", device=dev).to(torch.bfloat16)
    w = (synth.randn((d + r, m), 1, "proj_w", device=dev) / m ** 0.5).to(torch.bfloat16)
    o = torch.empty(T, d, dtype=torch.bfloat16, device=dev) if d else None
    k = torch.empty(T, r, dtype=torch.bfloat16, device=dev)
    if args.proj_tile:  # form and width forced through the test hook (2000 + width: CTA pair)
        call = lambda: lrar.test_project_tile(args.proj_tile, a, w, o, k)  # noqa: E731
    else:
        call = lambda: lrar.project(a, w, o, k)  # noqa: E731
    for _ in range(args.warmup):
        call()
    ms = _median_ms(torch, call, args.steps)
    flops = 2.0 * T * m * (d + r)
    print(json.dumps({"profile_proj": m, "T": T, "d": d, "r": r, "tile": args.proj_tile or "chosen", "ms": ms,
                      "tflops": flops / ms / 1e9}), flush=True)


def _median_ms(torch, fn, reps):
    """Median CUDA-event time of fn() over reps back-to-back repetitions (after one warm-up)."""
    fn()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
    for a, b in evs:
        a.record()
        fn()
        b.record()
    torch.cuda.synchronize()
    return statistics.median(a.elapsed_time(b) for a, b in evs)


def run_suite(args):
    """Every workload's headline site (not only the benchmark's): P-LR and its
    rank sweep, full AttnRes keys, the d = 2048 decoder, and the Block AttnRes
    forward sweep site by site against the two-phase path.  One JSON line each."""
    import torch

    from __graft_entry__ import build
    from paper_2607_09694_gb300 import lrar, sites, synth

    build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    peak, _ = _peaks()
    reps = max(5, args.steps // 5)

    def emit(d):
        d["peak_gbs"] = peak
        for k in list(d):
            if k.endswith("_gbs") and k != "peak_gbs":
                d[k.replace("_gbs", "_frac")] = d[k] / peak
        print(json.dumps(d), flush=True)

    def fwd_bwd(name, variant, T, d, r, n, seed, scale=None, h_dtype=torch.bfloat16):
        vals = synth.values(n, T, d, seed, "bf16", scale, device=dev)
        keys = synth.keys(n, T, r, seed, "bf16", device=dev) if variant == "projected" else None
        q = synth.queries(1, r, seed, device=dev)[0].contiguous()
        dh = synth.upstream(T, d, seed, "bf16", device=dev)
        h = torch.empty(T, d, dtype=h_dtype, device=dev)
        lse = torch.empty(T, device=dev)
        dv = torch.zeros(n, T, d, dtype=torch.bfloat16, device=dev)
        dk = torch.zeros(n, T, r, dtype=torch.bfloat16, device=dev) if keys is not None else None
        dq = torch.empty(r, device=dev)
        ws = torch.empty(lrar.workspace_size(variant, n, T, d, r) // 4, device=dev)
        f = _median_ms(torch, lambda: lrar.forward(variant, vals, keys, q, h, lse, r=r), reps)
        b = _median_ms(torch, lambda: lrar.backward(variant, vals, keys, q, dh, dv, dq, ws, dkeys=dk, h=h, lse=lse,
                                                    r=r, accumulate=True), reps)
        hb = 4 if h_dtype == torch.float32 else 2
        shp = sites.SiteShape(variant, n, T, d, r, out_bytes=hb)
        fb, bb = sites.forward_bytes(shp), sites.backward_bytes(shp)
        emit({"suite": name, "variant": variant, "T": T, "d": d, "r": r, "n_src": n, "h_bytes": hb,
              "fwd_ms": f, "bwd_ms": b, "fwd_gbs": fb / f / 1e6, "bwd_gbs": bb / b / 1e6,
              "fwd_bwd_gbs": (fb + bb) / (f + b) / 1e6, "tokens_per_s": T / ((f + b) / 1e3)})
        del vals, keys, dh, h, dv, dk
        torch.cuda.empty_cache()

    fwd_bwd("S-LR d1024 n49 r16 (reference for the rows below)", "sliced", 16384, 1024, 16, 49, 1, (0.5, 2.0))
    for r in (4, 8, 16, 32, 64):
        fwd_bwd(f"P-LR d1024 n49 r{r}", "projected", 16384, 1024, r, 49, 2)
    fwd_bwd("full AttnRes keys d1024 n49 (fp32 h: exact gbar)", "full", 16384, 1024, 1024, 49, 1, (0.5, 2.0),
            torch.float32)
    fwd_bwd("full AttnRes keys d1024 n49 (bf16 h)", "full", 16384, 1024, 1024, 49, 1, (0.5, 2.0))
    fwd_bwd("S-LR d2048 n65 r64 T32768", "sliced", 32768, 2048, 64, 65, 3)
    fwd_bwd("Block S-LR site d2048 n9 r64 T32768", "sliced", 32768, 2048, 64, 9, 3)

    # P-LR fused output projection (Eq. 11-12) on the tensor cores, against
    # cuBLAS (torch.matmul) alone and cuBLAS followed by the split of its output
    # into the value and key slots that the fused epilogue writes directly
    tpeak, tsrc = _bf16_peak()
    for T, m, d, r in ((16384, 1024, 1024, 32), (16384, 2816, 1024, 32), (32768, 2048, 2048, 64),
                       (16384, 1024, 0, 32)):
        a = synth.randn((T, m), 1, "proj_a", device=dev).to(torch.bfloat16)
        w = (synth.randn((d + r, m), 1, "proj_w", device=dev) / m ** 0.5).to(torch.bfloat16)
        o = torch.empty(T, d, dtype=torch.bfloat16, device=dev) if d else None
        k = torch.empty(T, r, dtype=torch.bfloat16, device=dev)
        ours = _median_ms(torch, lambda: lrar.project(a, w, o, k), reps)
        wt = w.t()
        cub = _median_ms(torch, lambda: torch.matmul(a, wt), reps)

        def cub_split():
            y = torch.matmul(a, wt)
            if o is not None:
                o.copy_(y[:, :d])
            k.copy_(y[:, d:])

        cubs = _median_ms(torch, cub_split, reps)
        flops = 2.0 * T * m * (d + r)
        emit({"suite": f"P-LR fused projection T{T} m{m} d{d} r{r}", "ms": ours, "tflops": flops / ours / 1e9,
              "tflops_frac": flops / ours / 1e9 / tpeak, "peak_tflops": tpeak, "peak_source": tsrc,
              "cublas_ms": cub, "cublas_tflops": flops / cub / 1e9, "cublas_then_split_ms": cubs})
        del a, w, o, k
        torch.cuda.empty_cache()

    # routing diagnostics (Eq. 16): reads only the keys (the S-LR tails, one 32-byte
    # sector per row at r = 16), writes N_eff per token and the mean alpha per source
    for variant, r, seed in (("sliced", 16, 1), ("projected", 32, 2)):
        T, d, n = 16384, 1024, 49
        vals = synth.values(n, T, d, seed, "bf16", (0.5, 2.0), device=dev)
        keys = synth.keys(n, T, r, seed, "bf16", device=dev) if variant == "projected" else None
        q = synth.queries(1, r, seed, std=1.0, device=dev)[0].contiguous()
        neff = torch.empty(T, device=dev)
        mean_alpha = torch.empty(n, device=dev)
        ws = torch.empty(lrar.diagnostics_workspace_size(n) // 4, device=dev)
        ms = _median_ms(torch, lambda: lrar.diagnostics(variant, vals, keys, q, neff, mean_alpha, ws, r=r), reps)
        key_bytes = T * (n * r * 2 + 4)
        emit({"suite": f"routing diagnostics {variant} d{d} n{n} r{r}", "T": T, "ms": ms, "key_bytes": key_bytes,
              "key_gbs": key_bytes / ms / 1e6, "tokens_per_s": T / (ms / 1e3)})
        del vals, keys
        torch.cuda.empty_cache()

    # Block AttnRes forward sweep of the 32-layer decoder (64 outputs, c = 8):
    # every site on its own versus the two-phase path.
    T, d, r, c, M = 32768, 2048, 64, 8, 64
    stack = synth.values(1 + M // c, T, d, 3, "bf16", device=dev)
    qs = synth.queries(M + 1, r, 3, device=dev)
    h = torch.empty(T, d, dtype=torch.bfloat16, device=dev)
    lse = torch.empty(T, device=dev)

    def naive():
        for t in range(1, M + 2):
            n = sites.block_num_sources(t, c)
            lrar.forward("sliced", stack, None, qs[t - 1] if n > 1 else None, h, lse, n_src=n, r=r)

    naive_bytes = sum(sites.forward_bytes(sites.SiteShape("sliced", sites.block_num_sources(t, c), T, d, r))
                      for t in range(1, M + 2))
    for pre_dtype, pb in ((torch.float32, 4), (torch.bfloat16, 2)):
        h_pre = torch.empty(c, T, d, dtype=pre_dtype, device=dev)
        lse_pre = torch.empty(c, T, device=dev)

        def two_phase():
            for b in range(M // c + 1):
                ns = c if b < M // c else 1  # the final read site forms a block of one
                t0 = b * c + 1
                lrar.block_phase1("sliced", stack, None, qs[t0 - 1:t0 - 1 + ns], h_pre[:ns], lse_pre[:ns],
                                  n_completed=1 + b)
                for j in range(1, ns):
                    lrar.block_phase2("sliced", h_pre[j], lse_pre[j], stack[1 + b], None, qs[t0 - 1 + j], h, lse)

        tp_bytes = sites.block_two_phase_forward_bytes(T, d, r, c, M, pre_bytes=pb)
        tn = _median_ms(torch, naive, max(3, reps // 2))
        tt = _median_ms(torch, two_phase, max(3, reps // 2))
        emit({"suite": "Block S-LR forward sweep, 65 sites, d2048 r64 c8 T32768", "h_pre_bytes": pb,
              "per_site_ms": tn, "two_phase_ms": tt, "speedup": tn / tt, "per_site_bytes": naive_bytes,
              "two_phase_bytes": tp_bytes, "per_site_gbs": naive_bytes / tn / 1e6,
              "two_phase_gbs": tp_bytes / tt / 1e6})
    del stack, h_pre, lse_pre
    torch.cuda.empty_cache()
    run_block_step(emit, dev, max(3, reps // 2))


def run_block_step(emit, dev, reps: int):
    """The Block AttnRes training step of the 32-layer, d = 2048 decoder
    (M = 64 sub-layer outputs, c = 8, S-LR r = 64, T = 32768, bf16 outputs, h
    and gradients) through sweep.BlockSweep: per step the assembly after each
    sub-layer and the two-phase mix of the 65 sites (forward: phase 1 per block,
    phase 2 at each site after a block's first), then the backward
    at each site in reverse and the fan-out of the summary gradients to the
    members, as copies into per-member tensors or handed over as views of the
    slot accumulators (one line each).  The outputs are written afresh before
    every step (untimed), as the sub-layers would; bytes of the mix and of the
    assembly / fan-out (a9) are reported separately."""
    import torch

    from paper_2607_09694_gb300 import sites, synth
    from paper_2607_09694_gb300.sweep import BlockSweep

    T, d, r, c, M = 32768, 2048, 64, 8, 64
    fresh = synth.values(M + 1, T, d, 3, "bf16", device=dev)
    outs = [torch.empty(T, d, dtype=torch.bfloat16, device=dev) for _ in range(M + 1)]
    qs = synth.queries(M + 1, r, 3, device=dev)
    dh = synth.upstream(T, d, 3, "bf16", sites=M + 1, device=dev)
    h = torch.empty(M + 1, T, d, dtype=torch.bfloat16, device=dev)
    lse = torch.empty(M + 1, T, device=dev)
    douts = [torch.empty(T, d, dtype=torch.bfloat16, device=dev) for _ in range(M + 1)]
    sw = BlockSweep("sliced", outs, qs, [dh[t] for t in range(M + 1)], h, lse, douts, c, r=r, two_phase=True)
    mix_f = sites.block_two_phase_forward_bytes(T, d, r, c, M)  # bf16 h serves as h_pre
    mix_b = 0
    for t in range(1, M + 2):
        shp = sites.SiteShape("sliced", sites.block_num_sources(t, c), T, d, r, accumulate=int(t != M + 1))
        mix_b += sites.backward_bytes(shp)
    asm = sum(sites.block_accumulate_bytes(T, d, 2, True) for i in range(1, M + 1) if not sites.block_opens_slot(i, c))
    # where a member joins its running sum inside phase 2, the partial summary is not read a second time
    asm -= sites.block_phase2_assembled_sites(M, c) * T * d * 2
    # the fan-out as copies into doutputs, or handed over as views (member_grad)
    for mode, hand_over in (("fan-out copies", None), ("member gradients handed over", lambda i, g, gk: None)):
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True),
               torch.cuda.Event(enable_timing=True)) for _ in range(reps + 1)]
        for a, b, e in ev:
            for i in range(M + 1):
                outs[i].copy_(fresh[i])
            sw.rearm()
            a.record()
            sw.forward()
            b.record()
            sw.backward(member_grad=hand_over)
            e.record()
        torch.cuda.synchronize()
        fwd = statistics.median(a.elapsed_time(b) for a, b, _ in ev[1:])
        bwd = statistics.median(b.elapsed_time(e) for _, b, e in ev[1:])
        fan = 0 if hand_over else (M + 1) * sites.block_accumulate_bytes(T, d, 2, False)
        emit({"suite": f"Block S-LR training step, 65 sites, d2048 r64 c8 T32768 (two-phase forward, {mode})",
              "fwd_ms": fwd, "bwd_ms": bwd, "step_ms": fwd + bwd, "mix_fwd_bytes": mix_f, "assembly_bytes": asm,
              "mix_bwd_bytes": mix_b, "fanout_bytes": fan, "fwd_gbs": (mix_f + asm) / fwd / 1e6,
              "bwd_gbs": (mix_b + fan) / bwd / 1e6, "step_gbs": (mix_f + asm + mix_b + fan) / (fwd + bwd) / 1e6,
              "tokens_per_s_per_site": T * (M + 1) / ((fwd + bwd) / 1e3)})
    del fresh, outs, dh, h, douts, sw
    torch.cuda.empty_cache()


def run_block_step_only(args):
    import torch

    from __graft_entry__ import build

    build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    peak, _ = _peaks()

    def emit(d):
        d["peak_gbs"] = peak
        for k in list(d):
            if k.endswith("_gbs") and k != "peak_gbs":
                d[k.replace("_gbs", "_frac")] = d[k] / peak
        print(json.dumps(d), flush=True)

    run_block_step(emit, dev, max(3, args.steps))


def run_graph(wl, step_bytes, reps: int = 10):
    """Median ms of one whole step replayed from a CUDA graph of the
    whole-decoder driver (sources as separate tensors: views of the stack)."""
    import torch

    from paper_2607_09694_gb300.sweep import DepthSweep

    ns = wl.values.shape[0]
    sw = DepthSweep("sliced", [wl.values[i] for i in range(ns)], wl.queries, [wl.dh[i] for i in range(ns)], wl.h,
                    wl.lse, [wl.dvalues[i] for i in range(ns)], wl.dq, r=R, eps=EPS)
    sw.capture()
    ms = _median_ms(torch, sw.replay, reps)
    return {"ms_per_step": ms, "gbs": step_bytes / ms / 1e6, "launches_per_replay": 3 * ns + 1,
            "what": "DepthSweep over per-source tensor views, one CUDA graph replay per step (49 forward, "
                    "49 backward, 49 dq sums, one dq zeroing)"}


def e2e_host_buffers(wl):
    """Pinned host buffers of the end-to-end leg: the step's inputs (values,
    queries, upstream gradients, filled from the workload) and its results.
    Allocated and moved across the link once in both directions before anything
    is timed: freshly pinned pages made the first steps through them up to 1.6x
    slower on GB300."""
    import torch

    host = {"values": torch.empty_like(wl.values, device="cpu").pin_memory(),
            "queries": torch.empty_like(wl.queries, device="cpu").pin_memory(),
            "dh": torch.empty_like(wl.dh, device="cpu").pin_memory(),
            "h": torch.empty_like(wl.h, device="cpu").pin_memory(),
            "lse": torch.empty_like(wl.lse, device="cpu").pin_memory(),
            "dvalues": torch.empty_like(wl.dvalues, device="cpu").pin_memory(),
            "dq": torch.empty_like(wl.dq, device="cpu").pin_memory()}
    for k in ("values", "queries", "dh"):
        host[k].copy_(getattr(wl, k))
        getattr(wl, k).copy_(host[k])
    for k in ("h", "lse", "dvalues", "dq"):
        host[k].copy_(getattr(wl, k))
        getattr(wl, k).copy_(host[k])
    torch.cuda.synchronize()
    return host


def run_e2e(wl, args, dist, dev, step_bytes, world, host=None):
    """The step through the public API with pinned host buffers: H2D of values,
    queries and upstream gradients, both sweeps, D2H of h, lse, dvalues and dq,
    all inside the timed region.  The copies run on their own streams and
    overlap the sweeps: forward site t waits only for sources 0..t-1, backward
    site t only for its dh (copied in the backward's order, 49 first), h_t
    leaves as soon as site t is mixed and d(o_{t-1}) as soon as backward site t
    (its last writer) is done.  The device buffers are doubled, so one step's
    inputs arrive while the previous step is still computing."""
    import torch

    lrar = wl.lrar
    host = host if host is not None else e2e_host_buffers(wl)
    hv, hq, hdh = host["values"], host["queries"], host["dh"]
    oh, olse, odv, odq = host["h"], host["lse"], host["dvalues"], host["dq"]
    h2d = sum(x.numel() * x.element_size() for x in (hv, hq, hdh))
    d2h = sum(x.numel() * x.element_size() for x in (oh, olse, odv, odq))

    names = ("values", "queries", "dh", "h", "lse", "dvalues", "dq")
    bufs = [{k: getattr(wl, k) for k in names}, {k: torch.empty_like(getattr(wl, k)) for k in names}]
    comp = torch.cuda.current_stream()
    s_in = torch.cuda.Stream()
    s_out = torch.cuda.Stream()
    ev = lambda: torch.cuda.Event()  # noqa: E731
    sets = []
    for _ in range(2):
        st = {"v_in": [ev() for _ in range(N_SITES)], "dh_in": [ev() for _ in range(N_SITES)], "q_in": ev(),
              "fwd": [ev() for _ in range(N_SITES)], "bwd": [ev() for _ in range(N_SITES)],
              "in_free": ev(), "out_free": ev()}
        st["in_free"].record(comp)
        st["out_free"].record(s_out)
        sets.append(st)
    k_step = [0]

    def one():
        b = k_step[0] % 2
        k_step[0] += 1
        B, E = bufs[b], sets[b]
        s_in.wait_event(E["in_free"])  # the step two back has finished reading these inputs
        with torch.cuda.stream(s_in):
            B["queries"].copy_(hq, non_blocking=True)
            E["q_in"].record(s_in)
            for i in range(N_SITES):
                B["values"][i].copy_(hv[i], non_blocking=True)
                E["v_in"][i].record(s_in)
            for t in range(N_SITES - 1, -1, -1):  # in the backward sweep's order
                B["dh"][t].copy_(hdh[t], non_blocking=True)
                E["dh_in"][t].record(s_in)
        comp.wait_event(E["out_free"])  # the step two back has shipped these outputs
        comp.wait_event(E["q_in"])
        for t in range(1, N_SITES + 1):
            comp.wait_event(E["v_in"][t - 1])
            q = B["queries"][t - 1] if t > 1 else None
            lrar.forward(lrar.SLICED, B["values"], None, q, B["h"][t - 1], B["lse"][t - 1], n_src=t, r=R, eps=EPS)
            E["fwd"][t - 1].record(comp)
            s_out.wait_event(E["fwd"][t - 1])
            with torch.cuda.stream(s_out):
                oh[t - 1].copy_(B["h"][t - 1], non_blocking=True)
        for t in range(N_SITES, 0, -1):
            comp.wait_event(E["dh_in"][t - 1])
            q = B["queries"][t - 1] if t > 1 else None
            lrar.backward(lrar.SLICED, B["values"], None, q, B["dh"][t - 1], B["dvalues"], B["dq"][t - 1], wl.ws,
                          lse=B["lse"][t - 1], n_src=t, r=R, accumulate=(t != N_SITES), eps=EPS)
            E["bwd"][t - 1].record(comp)
            s_out.wait_event(E["bwd"][t - 1])
            with torch.cuda.stream(s_out):
                odv[t - 1].copy_(B["dvalues"][t - 1], non_blocking=True)  # source t-1 is final after site t
        E["in_free"].record(comp)
        s_out.wait_event(E["in_free"])
        with torch.cuda.stream(s_out):
            olse.copy_(B["lse"], non_blocking=True)
            odq.copy_(B["dq"], non_blocking=True)
        E["out_free"].record(s_out)

    for _ in range(max(2, args.warmup)):
        one()
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    s = torch.cuda.Event(enable_timing=True)
    e = torch.cuda.Event(enable_timing=True)
    s.record(comp)
    for _ in range(args.steps):
        one()
    comp.wait_stream(s_out)
    comp.wait_stream(s_in)
    e.record(comp)
    torch.cuda.synchronize()
    el = _max_over_ranks(dist, s.elapsed_time(e) / 1e3, dev)
    return {"value": world * step_bytes * args.steps / el / 1e9, "unit": "GB/s",
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": el / args.steps * 1e3,
            "overlap": "copies on separate H2D / D2H streams ordered per source with CUDA events; "
                       "double-buffered device inputs and outputs"}


def run_reference(args):
    """The fp64 CPU oracle on the same workload's config (rank 0 only): each
    step is a bounded sample (all 49 sites on a slice of tokens)."""
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if rank != 0:
        return
    import oracle
    from paper_2607_09694_gb300 import synth

    ts_max = 2048
    vals = synth.values(N_SITES, ts_max, D, SEED, "bf16", (0.5, 2.0))
    qs = synth.queries(N_SITES, R, SEED)
    dhs = synth.upstream(ts_max, D, SEED, "bf16", sites=N_SITES)
    ts = calibrate(vals, qs, dhs, args.ref_step_seconds)
    for _ in range(args.warmup):
        oracle_pass(vals, qs, dhs, ts)
    secs = [oracle_pass(vals, qs, dhs, ts) for _ in range(args.steps)]
    total = sum(secs)
    value = sample_bytes(ts) * args.steps / total / 1e9
    cores = oracle.get_threads()
    sample = (f"all 49 sites fwd+bwd on {ts} of {T_TOK} tokens per step (fp64 C oracle, OpenMP {cores} threads); "
              f"GB/s on the sample's algorithmic bytes")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": total / args.steps * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": WORKLOAD, "T": T_TOK, "d": D, "r": R, "sites": N_SITES, "variant": "sliced",
                       "sample_tokens": ts},
            "cpu_baseline": {"value": value, "unit": "GB/s", "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--cpu-seconds", type=float, default=12.0, help="target length of the CPU oracle sample")
    ap.add_argument("--ref-step-seconds", type=float, default=4.0, help="target length of one reference step")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--profile-site", type=int, default=0, help="time one site with this many sources (profiling)")
    ap.add_argument("--tokens", type=int, default=4096, help="tokens of the --profile-site case")
    ap.add_argument("--site-variant", choices=["sliced", "projected", "full"], default="sliced",
                    help="key variant of the --profile-site case")
    ap.add_argument("--site-d", type=int, default=D, help="width d of the --profile-site case")
    ap.add_argument("--site-r", type=int, default=R, help="key rank r of the --profile-site case (not full)")
    ap.add_argument("--site-write", action="store_true", help="--profile-site: the backward writes the gradients")
    ap.add_argument("--suite", action="store_true", help="time every workload's headline site (JSON line each)")
    ap.add_argument("--block-step", action="store_true",
                    help="time only the Block AttnRes training step of the d = 2048 decoder (a --suite line)")
    ap.add_argument("--profile-block", type=int, default=0,
                    help="time the Block two-phase path on this many tokens (profiling)")
    ap.add_argument("--profile-proj", type=int, default=0,
                    help="time the fused projection with this input width m (profiling; --tokens, --site-d, --site-r)")
    ap.add_argument("--proj-tile", type=int, default=0,
                    help="--profile-proj: force the tile width (160..256, or 2000 + width for the CTA-pair form)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.block_step:
        run_block_step_only(args)
        return
    if args.suite:
        run_suite(args)
    elif args.profile_site:
        run_profile_site(args)
    elif args.profile_proj:
        run_profile_proj(args)
    elif args.profile_block:
        run_profile_block(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
