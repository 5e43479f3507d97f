"""Multi-process host logic of bench.py, on CPU with the gloo backend.

Streams are independent, so N ranks decode N disjoint blocks of B streams
with no collective on the data path; the only exchange is the maximum of the
timed-region durations over ranks.  These tests run that logic with
world_size 2 on CPU, and the reference arm under torchrun.
"""
from __future__ import annotations

import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_rank_streams_partition():
    B, ws = 5, 4
    seen = []
    for r in range(ws):
        got = bench.rank_streams(r, B)
        assert len(got) == B
        seen.extend(got)
    assert sorted(seen) == list(range(B * ws))


def test_max_over_ranks_single_rank_is_identity():
    assert bench.max_over_ranks([1.5, 2.0], 1) == [1.5, 2.0]


def _rank_main(rank, ws, port, out_dir):
    import torch.distributed as dist

    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=ws)
    try:
        # rank r "took" (r + 1) ms and (10 - r) ms on two timers
        got = bench.max_over_ranks([rank + 1.0, 10.0 - rank], ws)
        streams = bench.rank_streams(rank, 3)
        with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
            json.dump({"max": got, "streams": streams}, f)
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_gloo_world2(tmp_path):
    import torch.multiprocessing as mp

    ws = 2
    mp.start_processes(_rank_main, args=(ws, _free_port(), str(tmp_path)), nprocs=ws, join=True,
                       start_method="spawn")
    res = [json.load(open(tmp_path / f"rank{r}.json")) for r in range(ws)]
    for r in range(ws):
        assert res[r]["max"] == [2.0, 10.0]  # every rank sees the slowest rank's time
    assert set(res[0]["streams"]).isdisjoint(res[1]["streams"])
    assert sorted(res[0]["streams"] + res[1]["streams"]) == list(range(6))


def test_reference_arm_under_torchrun_prints_once():
    """`bench.py --impl reference` launched the way the driver launches N>1:
    rank 0 times the oracle and prints one JSON line, the other rank exits 0
    without work."""
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()), os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--gpus", "2", "--config", "0", "--steps", "1", "--warmup", "3",
           "--ref-streams", "2"]
    env = dict(os.environ, OMP_NUM_THREADS="1")
    p = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600, env=env)
    assert p.returncode == 0, p.stderr[-2000:]
    lines = [ln for ln in p.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, p.stdout
    rec = json.loads(lines[0])
    assert rec["impl"] == "reference" and rec["n_gpus"] == 2
    assert rec["value"] > 0 and rec["unit"] == "frames/s" and rec["higher_is_better"] is True
    assert rec["cpu_baseline"]["kind"] == "oracle" and rec["cpu_baseline"]["value"] == rec["value"]
    assert rec["e2e"] == {"value": rec["value"], "unit": "frames/s", "h2d_bytes_per_step": 0,
                          "d2h_bytes_per_step": 0}


@pytest.mark.parametrize("streams", [1, 16])
def test_workload_stream_override(streams):
    w = bench.workload(4, streams)
    assert w.B == streams and f"B={streams}" in w.name
    base = bench.workload(4)
    assert (w.V, w.H, w.T, w.lm_total, w.seed) == (base.V, base.H, base.T, base.lm_total, base.seed)
