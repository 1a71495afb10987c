"""bench.py's multi-process path on CPU with gloo, world size 2: the decode
step does not shard (each GPU would run an independent replica of the whole
step), so the only cross-rank work is the barrier around the timed region,
the max over ranks of the elapsed time, and rank 0 printing the line."""
import json
import os
import socket
import subprocess
import sys
from pathlib import Path

import pytest
import torch.multiprocessing as mp

ROOT = Path(__file__).resolve().parent.parent


def free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE="2", LOCAL_RANK=str(rank))
    sys.path.insert(0, str(ROOT))
    import bench
    r, world, local = bench.dist_setup(2)
    bench.barrier(world)
    elapsed = bench.reduce_max(10.0 * (rank + 1), world)      # rank 1 is the slower one
    import numpy as np
    _, sets, active = bench.make_step_inputs(rank)
    Path(out_dir, f"rank{rank}.json").write_text(json.dumps({
        "rank": r, "world": world, "local": local, "elapsed": elapsed,
        "sets_sum": int(sets[:2].astype(np.int64).sum()), "active0": int(active[0])}))
    import torch.distributed as dist
    dist.destroy_process_group()


def test_barrier_and_max_over_ranks(tmp_path):
    mp.spawn(_rank_main, args=(free_port(), str(tmp_path)), nprocs=2, join=True)
    r0 = json.loads((tmp_path / "rank0.json").read_text())
    r1 = json.loads((tmp_path / "rank1.json").read_text())
    assert (r0["rank"], r1["rank"], r0["world"]) == (0, 1, 2)
    assert r0["elapsed"] == r1["elapsed"] == 20.0               # every rank reports the max
    # replicas run independent spike sets (weak scaling: per-rank work fixed)
    assert r0["sets_sum"] != r1["sets_sum"]
    assert r0["active0"] > 0 and r1["active0"] > 0


@pytest.mark.timeout(600)
def test_reference_arm_under_torchrun():
    """`bench.py --impl reference` launched like the driver launches N > 1:
    rank 0 alone times the oracle and prints one JSON line; rank 1 exits 0."""
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node=2",
           "--master-addr=127.0.0.1", f"--master-port={free_port()}", str(ROOT / "bench.py"),
           "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "0"]
    env = dict(os.environ, OMP_NUM_THREADS="1")
    res = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600, env=env)
    assert res.returncode == 0, res.stderr[-2000:]
    lines = [l for l in res.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, res.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle" and d["e2e"]["h2d_bytes_per_step"] == 0
