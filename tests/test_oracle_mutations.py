"""The oracle's pins catch plausible mistakes.

Each case plants one mistake in a copy of oracle/lrar_oracle.c (on the CPU),
builds it, and runs the pin suites (test_oracle_pins.py, test_accounting.py)
against it in a subprocess: every mutant must make at least one pin fail.
"""
import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "lrar_oracle.c")

# (name, original text, mutated text, occurrence to replace)
MUTANTS = [
    ("eps dropped from RMSNorm", "sqrt(sumsq / (double)r + eps)", "sqrt(sumsq / (double)r + 1e-300)", 0),
    ("sum instead of mean in RMSNorm", "sumsq / (double)r + eps", "sumsq + eps", 0),
    ("sliced key from the head", "value_at(values, dtype, T, d, i, x, d - r + j)",
     "value_at(values, dtype, T, d, i, x, j)", 0),
    ("full key from source 0", "k[j] = value_at(values, dtype, T, d, i, x, j);",
     "k[j] = value_at(values, dtype, T, d, 0, x, j);", 0),
    ("1/sqrt(r) temperature", "s += q[j] * kbi[j];", "s += q[j] * kbi[j] / sqrt((double)r);", 0),
    ("softmax not normalised", "exp(w->s[i] - m) / Z", "exp(w->s[i] - m)", 0),
    ("lse without the max", "return m + log(Z);", "return log(Z);", 0),
    ("mix with a transposed weight index", "acc += w.alpha[i] * value_at(", "acc += w.alpha[n - 1 - i] * value_at(", 0),
    ("gbar dropped", "w.alpha[i] * (w.g[i] - gbar)", "w.alpha[i] * w.g[i]", 0),
    ("gbar without the weights", "gbar += w.alpha[k] * w.g[k];", "gbar += w.g[k] / n;", 0),
    ("value gradient of the wrong source", "= w.alpha[i] * w.dh[j];", "= w.alpha[0] * w.dh[j];", 0),
    ("RMSNorm Jacobian sign", "- (rho * rho * rho / (double)r)", "+ (rho * rho * rho / (double)r)", 0),
    ("RMSNorm Jacobian power", "(rho * rho * rho / (double)r)", "(rho * rho / (double)r)", 0),
    ("dq from the raw key", "dqp[j] += w.ds[i] * kbi[j];", "dqp[j] += w.ds[i] * ki[j];", 0),
    ("sliced key gradient into the head", "int off = (variant == OR_SLICED) ? d - r : 0;", "int off = 0;", 0),
    ("empty partial block counted", "return 1 + completed + (partial > 0 ? 1 : 0);", "return 1 + completed + 1;", 0),
    ("block slot off by one", "int slot = (i == 0) ? 0 : 1 + (i - 1) / c;", "int slot = (i == 0) ? 0 : 1 + i / c;", 0),
    ("fan-out slot off by one", "int slot = (i == 0) ? 0 : 1 + (i - 1) / c;", "int slot = (i == 0) ? 0 : 1 + i / c;", 1),
    ("N_eff without exp", "neff[u] = exp(H);", "neff[u] = H;", 0),
    ("projection with a transposed weight", "elem(w, dtype, (int64_t)j * m + c)", "elem(w, dtype, (int64_t)c * nrows + j)", 0),
    ("projection drops the last input column", "for (int c = 0; c < m; ++c) acc +=", "for (int c = 0; c < m - 1; ++c) acc +=", 0),
    ("projection reads token 0", "elem(a, dtype, x * m + c)", "elem(a, dtype, c)", 0),
]


def _mutate(text, old, new, occurrence):
    start = -1
    for _ in range(occurrence + 1):
        start = text.index(old, start + 1)
    return text[:start] + new + text[start + len(old):]


def _run(case, tmp):
    name, old, new, occ = case
    src = open(SRC).read()
    assert src.count(old) > occ, f"{name}: target text not found in the oracle"
    tag = "".join(ch if ch.isalnum() else "_" for ch in name)
    c_path = os.path.join(tmp, f"{tag}.c")
    so_path = os.path.join(tmp, f"{tag}.so")
    with open(c_path, "w") as f:
        f.write(_mutate(src, old, new, occ))
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", c_path, "-o", so_path, "-lm"])
    env = dict(os.environ, LRAR_ORACLE_LIB=so_path, OMP_NUM_THREADS="1")
    res = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                          os.path.join(ROOT, "tests", "test_oracle_pins.py"),
                          os.path.join(ROOT, "tests", "test_accounting.py")],
                         cwd=ROOT, env=env, capture_output=True, text=True)
    return name, res.returncode


def test_every_mutant_is_caught(tmp_path):
    with ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 1)) as ex:
        results = list(ex.map(lambda c: _run(c, str(tmp_path)), MUTANTS))
    survivors = [name for name, rc in results if rc == 0]
    assert not survivors, f"mutants not caught by any pin: {survivors}"


def test_unmutated_oracle_passes_the_same_way(tmp_path):
    """Control: the same subprocess route on the unmodified oracle passes."""
    name, rc = _run(("control", "sqrt(sumsq", "sqrt(sumsq", 0), str(tmp_path))
    assert rc == 0
