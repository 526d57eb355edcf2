"""Table 1's added-FLOPs column and App. A.6's worked numbers, re-derived from
the closed forms of App. A.

These pin the source-set definitions (Full: n_t = t; Block: embedding +
completed blocks + non-empty partial block) that both the product's host logic
and the oracle use: a different reading of the source sets changes S_src and
breaks the 4-decimal match of all 19 rows.
"""
import os

import pytest

import oracle
from paper_2607_09694_gb300 import sites

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
L, D, M_FFN = 24, 1024, 2816


def _table1():
    rows = []
    with open(os.path.join(GOLDEN, "table1_added_flops.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            method, blocks, rank, val = line.split()
            rows.append((method, blocks, None if rank == "-" else int(rank), val))
    return rows


def _a6():
    out = {}
    with open(os.path.join(GOLDEN, "appendix_a6_numbers.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            name, val, dec = line.split()
            out[name] = (float(val), int(dec))
    return out


@pytest.mark.parametrize("row", _table1(), ids=lambda r: f"{r[0]}-{r[1]}-{r[2]}")
def test_table1_added_flops(row):
    method, blocks, r, printed = row
    mode, N = ("full", None) if blocks == "full" else ("block", int(blocks))
    pct = sites.added_flops_percent(method, L, D, M_FFN, mode, N, r)
    assert f"{pct:.4f}" == printed


def test_source_read_totals():
    """S_src = 1224 (Full, sites 2..49) and 168 / 264 / 456 (Block N = 4/8/16)."""
    assert sites.s_src(48, "full") == 1224
    assert [sites.s_src(48, "block", N) for N in (4, 8, 16)] == [168, 264, 456]


def test_oracle_source_sets_agree():
    """The oracle's independent source-set sizes give the same totals."""
    assert sum(oracle.full_num_sources(t) for t in range(2, 50)) == 1224
    for N, want in ((4, 168), (8, 264), (16, 456)):
        c = 48 // N
        assert sum(oracle.block_num_sources(t, c) for t in range(2, 50)) == want
    for t in range(1, 66):
        for c in (1, 2, 3, 8, 12, 64):
            assert oracle.block_num_sources(t, c) == sites.block_num_sources(t, c)


def test_block_source_counts_of_the_large_decoder():
    """32-layer decoder (M = 64) with c = 8: at most 1 + 8 = 9 sources."""
    counts = sites.source_counts(64, "block", 8, first_site=1)
    assert max(counts) == 9 and counts[0] == 1 and counts[-1] == 9


def test_appendix_a6_numbers():
    a6 = _a6()
    r = 32

    def same(name, value):
        want, dec = a6[name]
        assert round(value, dec) == pytest.approx(want, abs=10 ** -(dec + 3)), name

    same("kernel_reduction_percent", sites.kernel_reduction_percent(D, r))
    same("projected_key_macs_per_token", sites.projected_key_path(L, D, M_FFN, r))
    same("projected_param_increase", sites.projected_params(L, D, M_FFN, r))
    same("sliced_param_increase", sites.sliced_params(L, r))
    same("projected_cache_increase_pct", 100.0 * r / D)
    same("projected_param_overhead_pct", 100.0 * r / D * (1 + M_FFN / D) / (4 + 3 * M_FFN / D))
    key_pct = 100.0 * sites.projected_key_path(L, D, M_FFN, r) / sites.base_core(L, D, M_FFN)
    same("projected_key_path_pct", key_pct)
    full_kernel = 100.0 * sites.lr_kernel(D, r, sites.s_src(48, "full")) / sites.base_core(L, D, M_FFN)
    same("full_projected_r32_total_pct", round(full_kernel, 4) + round(key_pct, 4))
    blk_kernel = 100.0 * sites.lr_kernel(D, r, sites.s_src(48, "block", 8)) / sites.base_core(L, D, M_FFN)
    same("block8_projected_kernel_pct", blk_kernel)
    same("block8_projected_total_pct", round(blk_kernel, 4) + round(key_pct, 4))


def test_byte_model_headline():
    """The algorithmic bytes of the headline site (S-LR, n = 49, T = 16384,
    d = 1024, bf16, accumulate): 1.678 GB forward, 4.966 GB backward."""
    s = sites.SiteShape("sliced", 49, 16384, 1024, 16)
    assert abs(sites.forward_bytes(s) / 1e9 - 1.678) < 1e-3
    assert abs(sites.backward_bytes(s) / 1e9 - 4.966) < 1e-3


@pytest.mark.parametrize("variant,pre", [("sliced", 2), ("sliced", 4), ("projected", 2)])
def test_two_phase_bytes_with_one_site_per_block(variant, pre):
    """With c = 1 every block holds one site and has no phase 2: the two-phase
    forward moves exactly the bytes of the per-site forwards over the same
    source counts (h_pre is then the site's h)."""
    T, d, r, M = 64, 256, 16, 7
    per_site = sum(sites.forward_bytes(sites.SiteShape(variant, sites.block_num_sources(t, 1), T, d, r,
                                                       out_bytes=pre)) for t in range(1, M + 2))
    assert sites.block_two_phase_forward_bytes(T, d, r, 1, M, variant, pre_bytes=pre) == per_site


def test_two_phase_bytes_of_the_large_decoder():
    """The d = 2048 decoder (M = 64, c = 8, r = 64, T = 32768, bf16 h_pre): 8
    blocks of 8 sites and the final read site alone.  Phase 1 reads sum(1 + b)
    source rows per token over the 9 blocks and writes 65 h_pre rows; phase 2 runs
    at 56 sites, each reading an h_pre row and a partial summary and writing h."""
    T, d = 32768, 2048
    row = d * 2
    ph1 = T * (sum(1 + b for b in range(9)) * row + 65 * (row + 4))
    ph2 = 56 * T * (row + 4 + row + row + 4)
    assert sites.block_two_phase_forward_bytes(T, d, 64, 8, 64) == ph1 + ph2
    # against the site-by-site forward of the same sites: 56.1 GB
    naive = sum(sites.forward_bytes(sites.SiteShape("sliced", sites.block_num_sources(t, 8), T, d, 64))
                for t in range(1, 66))
    assert abs(naive / 1e9 - 56.11) < 0.01 and abs((ph1 + ph2) / 1e9 - 37.34) < 0.01


@pytest.mark.parametrize("M,c,expect", [(64, 8, 48), (13, 4, 6), (7, 1, 0), (12, 4, 6), (5, 8, 4)])
def test_sites_assembled_inside_phase2(M, c, expect):
    """Blocks of ns sites fold the assembly of members 2..ns-1 of the open block
    into phase 2: M = 64, c = 8 has eight full blocks of 8 sites (6 each) and a
    final block of one; M = 5, c = 8 one block of 6 sites."""
    assert sites.block_phase2_assembled_sites(M, c) == expect
    brute = 0
    for b in range(M // c + 1):
        t0 = b * c + 1
        for t in range(t0 + 1, min(t0 + c, M + 2)):
            i = t - 1
            brute += int(not sites.block_opens_slot(i, c))
    assert brute == expect
