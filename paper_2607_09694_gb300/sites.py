"""Host-side logic of the depth path: which sources each residual read site
sees, the Block AttnRes slot layout, the bytes a site must move, and the
paper's closed-form cost accounting.

Residual read sites are t = 1..M+1 for a decoder with M = 2L residual-writing
sub-layers (§3.1).  Site t reads sources written before it: the embedding o_0
and the outputs o_1..o_{t-1}.

* Full AttnRes, Eq. (4): S_t = {0, ..., t-1}, so n_t = t.
* Block AttnRes (§3.1, Eq. 5-6) with c outputs per block: the embedding, every
  completed block summary b_B = sum of its c outputs, and the partial-block
  summary when it is non-empty.  In the stacked source buffer the summaries
  occupy slots 1, 2, ...; output o_i (i >= 1) is summed into slot
  1 + (i - 1) // c, so the sources of site t are the first n_t slots.

Site 1 reads one source (its softmax is identically 1); the paper's cost
accounting counts sites t = 2..M+1 only (this reproduces every added-FLOPs
entry of Table 1), and those 2L sites carry the 2L static queries (App. A.5).
"""
from __future__ import annotations

from dataclasses import dataclass

VARIANTS = {"full": 0, "sliced": 1, "projected": 2}
DTYPE_BYTES = {"f32": 4, "bf16": 2}


def full_num_sources(t: int) -> int:
    """|S_t| for Full AttnRes (Eq. 4)."""
    if t < 1:
        raise ValueError("sites are numbered from 1")
    return t


def block_num_sources(t: int, c: int) -> int:
    """|S_t| for Block AttnRes with c outputs per block (Eq. 5-6)."""
    if t < 1 or c < 1:
        raise ValueError("need t >= 1 and c >= 1")
    written = t - 1
    completed, partial = divmod(written, c)
    return 1 + completed + (1 if partial else 0)


def block_slot(i: int, c: int) -> int:
    """Slot of the stacked Block source buffer that output o_i is summed into."""
    if i < 0 or c < 1:
        raise ValueError("need i >= 0 and c >= 1")
    return 0 if i == 0 else 1 + (i - 1) // c


def block_opens_slot(i: int, c: int) -> bool:
    """True when o_i is the first member of its slot (the slot is copied, not added to)."""
    return i == 0 or (i - 1) % c == 0


def source_counts(M: int, mode: str = "full", c: int | None = None, first_site: int = 2) -> list[int]:
    """n_t for sites t = first_site..M+1."""
    if mode == "full":
        return [full_num_sources(t) for t in range(first_site, M + 2)]
    if mode == "block":
        return [block_num_sources(t, c) for t in range(first_site, M + 2)]
    raise ValueError(mode)


def s_src(M: int, mode: str = "full", N: int | None = None) -> int:
    """S_src = sum over read sites of |S_t| (App. A), sites t = 2..M+1; Block with N blocks of c = M/N."""
    if mode == "full":
        return sum(source_counts(M, "full"))
    if M % N:
        raise ValueError("M must be a multiple of N")
    return sum(source_counts(M, "block", M // N))


# ---------------------------------------------------------------------------
# Algorithmic bytes: what one call must move through HBM at minimum.
# ---------------------------------------------------------------------------


@dataclass(frozen=True)
class SiteShape:
    variant: str
    n: int
    T: int
    d: int
    r: int
    in_bytes: int = 2     # values / keys / dh (and h when read back)
    out_bytes: int = 2    # h
    grad_bytes: int = 2   # dvalues / dkeys
    accumulate: int = 1


def forward_bytes(s: SiteShape) -> int:
    """Forward: read n value rows (+ n P-LR keys), write h and lse."""
    rp = s.r if s.variant == "projected" else 0
    return s.T * (s.n * (s.d + rp) * s.in_bytes + s.d * s.out_bytes + 4)


def backward_bytes(s: SiteShape) -> int:
    """Backward: read values (+keys), dh (+h for full keys) and lse; write (or
    read-modify-write when accumulating) the value and key gradients."""
    rp = s.r if s.variant == "projected" else 0
    per_tok = (s.n * (s.d + rp) * s.in_bytes + s.d * s.in_bytes + 4
               + (1 + s.accumulate) * s.n * (s.d + rp) * s.grad_bytes)
    if s.variant == "full":
        per_tok += s.d * s.out_bytes
    return s.T * per_tok


def block_two_phase_forward_bytes(T: int, d: int, r: int, c: int, M: int, variant: str = "sliced",
                                  in_bytes: int = 2, pre_bytes: int = 2, out_bytes: int = 2) -> int:
    """Two-phase Block forward (§3.5) over sites t = 1..M+1 in blocks of c sites:
    per block b, phase 1 reads the 1 + b completed sources (+ their P-LR keys)
    and writes h_pre and lse_pre of each of the block's ns sites; phase 2, at
    every site of the block after the first, reads h_pre, lse_pre and the
    partial summary (+ its key) and writes h and lse."""
    rp = r if variant == "projected" else 0
    total = 0
    for b in range(M // c + 1):
        ns = min(c, M + 1 - b * c)
        total += T * ((1 + b) * (d + rp) * in_bytes + ns * (d * pre_bytes + 4))
        total += (ns - 1) * T * (d * pre_bytes + 4 + (d + rp) * in_bytes + d * out_bytes + 4)
    return total


def block_phase2_assembled_sites(M: int, c: int) -> int:
    """Sites of the two-phase forward whose partial summary is assembled inside
    phase 2 (lrar_block_phase2_assemble): every site of a block after its second,
    where the newest member joins a running sum of at least one member."""
    return sum(max(0, min(c, M + 1 - b * c) - 2) for b in range(M // c + 1))


def block_accumulate_bytes(T: int, width: int, elem_bytes: int, beta_nonzero: bool) -> int:
    """dst = beta*dst + alpha*src: read src (+ dst when beta != 0), write dst."""
    return T * width * elem_bytes * (3 if beta_nonzero else 2)


# ---------------------------------------------------------------------------
# Closed-form cost accounting of App. A (multiply-adds per token).
# ---------------------------------------------------------------------------


def base_core(L: int, d: int, m: int) -> int:
    """C_base = L (4 d^2 + 3 d m), the non-embedding dense SwiGLU core (App. A.6)."""
    return L * (4 * d * d + 3 * d * m)


def attnres_kernel(d: int, S: int) -> int:
    """C_AttnRes = 2 d S_src (App. A.1)."""
    return 2 * d * S


def lr_kernel(d: int, r: int, S: int) -> int:
    """C_LR,kernel = (d + r) S_src (App. A.1); also S-LR's total (App. A.3)."""
    return (d + r) * S


def projected_key_path(L: int, d: int, m: int, r: int) -> int:
    """C_P,key-proj = r [L (d + m) + d] (App. A.2)."""
    return r * (L * (d + m) + d)


def kernel_reduction_percent(d: int, r: int) -> float:
    """100 (d - r) / (2 d), the low-rank kernel saving (App. A.1)."""
    return 100.0 * (d - r) / (2 * d)


def projected_params(L: int, d: int, m: int, r: int) -> int:
    """Delta P_P = r [L (d + m) + d + 2L] (App. A.5)."""
    return r * (L * (d + m) + d + 2 * L)


def sliced_params(L: int, r: int) -> int:
    """Delta P_S = 2 L r (App. A.5)."""
    return 2 * L * r


def added_flops_percent(method: str, L: int, d: int, m: int, mode: str = "full", N: int | None = None,
                        r: int | None = None) -> float:
    """The Added-FLOPs column of Table 1 for one row (percent of C_base)."""
    S = s_src(2 * L, mode, N)
    if method == "attnres":
        c = attnres_kernel(d, S)
    elif method == "sliced":
        c = lr_kernel(d, r, S)
    elif method == "projected":
        c = lr_kernel(d, r, S) + projected_key_path(L, d, m, r)
    else:
        raise ValueError(method)
    return 100.0 * c / base_core(L, d, m)
