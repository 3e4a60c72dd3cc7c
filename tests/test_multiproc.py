"""The multi-process host path of bench.py on CPU (gloo, world size 2).

bench.py runs one process per GPU; the path does not shard inside a pass, so
the ranks are independent replicas (each decodes its own seeded prompts) and
the only collectives are host-side: a barrier on both sides of the timed
region and the max of the ranks' times.  These tests run those pieces in two
CPU processes with the gloo backend (no GPU), and the reference arm under
torch.distributed.run, where rank 0 alone times the oracle and prints the
line while rank 1 exits without work.
"""

from __future__ import annotations

import json
import os
import socket
import subprocess
import sys

import numpy as np
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank: int, ws: int, port: int, out: str) -> None:
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(ws), LOCAL_RANK=str(rank), MASTER_ADDR="127.0.0.1",
                      MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import bench
    import torch.distributed as dist

    got_ws, got_rank, _ = bench.dist_setup()
    bench.dist_barrier(got_ws)
    slowest = bench.dist_max(1.5 + rank, got_ws)  # rank r "took" 1.5 + r ms
    bench.dist_barrier(got_ws)
    with open(os.path.join(out, f"rank{rank}.json"), "w") as f:
        json.dump({"ws": got_ws, "rank": got_rank, "max": slowest}, f)
    dist.destroy_process_group()


def test_barrier_and_max_over_ranks_gloo(tmp_path):
    ws = 2
    mp.start_processes(_worker, args=(ws, _free_port(), str(tmp_path)), nprocs=ws, start_method="spawn")
    res = [json.load(open(tmp_path / f"rank{r}.json")) for r in range(ws)]
    assert [r["rank"] for r in res] == [0, 1] and all(r["ws"] == ws for r in res)
    assert all(r["max"] == 2.5 for r in res)  # every rank sees the slowest rank's time


def test_replicas_decode_distinct_prompts():
    """Rank r's prompts are seeded with prompt_seed + 7919 r: replicas never
    decode the same sequences, so the job's tokens are the ranks' sum."""
    from paper_2608_11235_gb300 import configs, synth
    cfg = configs.PRESETS["llada8b-shape-256+256"]
    p0 = synth.prompts(cfg["prompt_seed"], 1, cfg["prompt_len"], cfg["mask_id"])
    p1 = synth.prompts(cfg["prompt_seed"] + 7919, 1, cfg["prompt_len"], cfg["mask_id"])
    assert not np.array_equal(p0, p1)
    assert p0.min() >= 0 and p0.max() < cfg["mask_id"]


def test_reference_arm_rank0_only_under_torchrun():
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()), os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--workload", "tiny-2L-d256", "--steps", "1", "--warmup", "0"]
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=300,
                       env=dict(os.environ, OMP_NUM_THREADS="2"))
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["value"] > 0 and d["cpu_baseline"]["kind"] == "oracle"
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["higher_is_better"] is True
