"""The multi-rank host logic of bench.py on CPU: world_size-2 gloo process
groups on 127.0.0.1 (no GPU involved)."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

from paper_2607_09694_gb300 import replicas  # noqa: E402


def _free_port() -> int:
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist, r, local, w = replicas.init_from_env()
    assert dist is not None and (r, local, w) == (rank, rank, world)
    dist.barrier()
    slowest = replicas.max_over_ranks(dist, 1.5 + rank)  # rank 1 is the slowest
    start, stop = replicas.token_range(16384, rank, world)
    with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
        json.dump({"max": slowest, "range": [start, stop]}, f)
    dist.destroy_process_group()


def test_max_over_ranks_and_barrier_with_gloo(tmp_path):
    port = _free_port()
    mp.start_processes(_worker, args=(2, port, str(tmp_path)), nprocs=2, start_method="spawn", join=True)
    res = [json.load(open(tmp_path / f"rank{r}.json")) for r in range(2)]
    assert all(x["max"] == 2.5 for x in res)
    assert res[0]["range"] == [0, 8192] and res[1]["range"] == [8192, 16384]


def test_single_rank_needs_no_group(monkeypatch):
    for k in ("WORLD_SIZE", "RANK", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)
    dist, rank, local, world = replicas.init_from_env()
    assert dist is None and (rank, local, world) == (0, 0, 1)
    assert replicas.max_over_ranks(None, 3.0) == 3.0


@pytest.mark.parametrize("T,world", [(10, 3), (7, 7), (0, 2), (16383, 4)])
def test_token_ranges_tile_the_batch(T, world):
    spans = [replicas.token_range(T, r, world) for r in range(world)]
    assert spans[0][0] == 0 and spans[-1][1] == T
    assert all(a[1] == b[0] for a, b in zip(spans, spans[1:]))
    assert max(b - a for a, b in spans) - min(b - a for a, b in spans) <= 1


def test_reference_arm_under_torchrun_prints_once():
    """`bench.py --impl reference` launched like the driver does for N = 2: rank 0
    alone runs the oracle and prints one JSON line; rank 1 exits 0 silently."""
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "3", "--ref-step-seconds", "0.2"]
    res = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert res.returncode == 0, res.stderr[-2000:]
    lines = [ln for ln in res.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["n_gpus"] == 2 and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle"
