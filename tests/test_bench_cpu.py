"""The benchmark's host logic without a GPU: the reference arm's JSON line (the fp64
oracle timed on the host cores), its multi-rank launch (rank 0 alone prints, every rank
exits 0) and the max-over-ranks timing reduction, on world_size 2 with gloo."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _json_lines(out: str):
    return [json.loads(l) for l in out.splitlines() if l.startswith("{")]


def test_reference_arm_prints_the_contract_line():
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--config", "tiny",
                        "--steps", "1", "--warmup", "0"], cwd=ROOT, capture_output=True,
                       text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = _json_lines(r.stdout)
    assert len(lines) == 1
    d = lines[0]
    assert d["impl"] == "reference" and d["unit"] == "TFLOP/s" and d["value"] > 0
    assert d["higher_is_better"] is True and d["warmup"] >= 3 and d["steps"] == 1
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"] == {"value": d["value"], "unit": "TFLOP/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}
    assert d["config"]["T"] == 128 and d["metric"].startswith("FlashRelation fwd+bwd")


def test_reference_arm_two_ranks_only_rank0_prints():
    env = dict(os.environ, OMP_NUM_THREADS="1")
    r = subprocess.run([sys.executable, "-m", "torch.distributed.run", "--nnodes=1",
                        "--nproc-per-node", "2", "--master-addr", "127.0.0.1", "--master-port",
                        str(_free_port()), "bench.py", "--impl", "reference", "--config", "tiny",
                        "--gpus", "2", "--steps", "1", "--warmup", "0"],
                       cwd=ROOT, capture_output=True, text=True, timeout=300, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = _json_lines(r.stdout)
    assert len(lines) == 1 and lines[0]["impl"] == "reference"


def _worker(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        dev = torch.device("cpu")
        bench._barrier(dist, dev)
        got = bench._max_over_ranks(dist, 1.5 * (rank + 1), dev)
        with open(os.path.join(out_dir, f"r{rank}"), "w") as f:
            f.write(repr(got))
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_gloo(tmp_path):
    world = 2
    mp.start_processes(_worker, args=(world, _free_port(), str(tmp_path)), nprocs=world,
                       join=True, start_method="spawn")
    for r in range(world):
        assert float(open(tmp_path / f"r{r}").read()) == 3.0


def test_max_over_ranks_single_process_is_identity():
    assert bench._max_over_ranks(None, 2.25, torch.device("cpu")) == 2.25


def test_sdpa_context_runs_on_cpu():
    """The context measurement's code path (PyTorch SDPA fwd+bwd, same flop convention)."""
    from paper_2608_20172_gb300 import workloads
    w = workloads.custom(1, 2, 64, 16, "fp32")
    r = bench.sdpa_context(w, torch.device("cpu"), steps=2, warmup=1)
    assert r["ms_per_step"] > 0 and r["tflops"] > 0
    assert "context only" in r["note"]


def test_oracle_timing_on_one_thread():
    """The single-thread leg of the CPU baseline: the oracle with nthreads = 1 over a
    sample one head wide, reported with cores = 1."""
    from paper_2608_20172_gb300 import workloads
    w = workloads.WORKLOADS["tiny"]
    one = bench.cpu_oracle_run(w, n_heads=1, t_rows=64, nthreads=1)
    assert one["cores"] == 1 and one["heads"] == 1 and one["rows"] == 64
    assert one["tflops"] > 0 and one["reps"] >= 1
    assert bench._sample_text(w, one) == "1 of 2 heads over their first 64 of 128 rows"
